"""Shared helpers of the GPU tests: seeded inputs through both sides, comparison with the oracle.

Inputs are drawn as bf16 bit patterns by mlkv_synth.gen; the GPU receives the bits, the oracle
their exact float64 widening.  Tolerances (per the decode contract for bf16 K/V with fp32
accumulation): max |err| <= 2e-2 and mean |err| <= 2e-3 against the fp64 oracle.
"""
import numpy as np

import oracle
from mlkv_synth import gen

MAX_ABS = 2e-2
MEAN_ABS = 2e-3

# The decode step in the cross-layer fused form (option step_fused 2) on a device of 152 SMs:
# layout, the plan's key tiles of 128 positions per unit (kc) and units, and the query tiles of a
# unit (1: the block's L x G rows fit one tile at head_dim 64; 2: two tiles).
FUSED_STEP_SMS = 152
FUSED_STEP_CASES = [
    # owner, h, g, d, b, L, kc, units, tiles
    ([0] * 6 + [6] * 6, 12, 1, 64, 64, 2048, 16, 128, 1),  # the benchmark's shape: 72 rows a unit
    ([0, 0, 2, 2, 4, 4, 6, 6, 8, 8, 10, 10], 12, 1, 64, 1, 128, 1, 6, 1),   # one tile per block
    ([0] * 12, 12, 1, 64, 4, 3000, 1, 96, 2),              # 144 rows: query tiles A and B
    ([0, 0, 2, 2], 12, 1, 64, 40, 700, 6, 80, 1),           # ragged last tile
    ([0, 0, 2, 2], 4, 4, 64, 8, 333, 2, 128, 1),            # one head per KV head: two rows a unit
    ([0, 0, 0, 3, 3, 3], 12, 4, 64, 16, 1000, 8, 128, 1),   # GQA groups of 3 under MLKV: 9 rows
    ([0, 0, 2, 2], 32, 8, 128, 8, 1500, 12, 128, 2),        # head_dim 128, groups of 4: 8 rows
    ([0] * 20, 16, 2, 128, 2, 600, 1, 20, 2),               # head_dim 128, 160 rows in two tiles
    ([0, 0, 0], 16, 2, 64, 3, 1, 1, 6, 1),                  # a single position
    # few long segments: every segment in chunks, partial records, one merge launch
    ([0] * 6 + [6] * 6, 12, 1, 64, 1, 131072, 14, 148, 1),  # 74 chunks of 14 tiles a segment
    ([0, 0, 2, 2], 12, 4, 64, 2, 9000, 8, 144, 1),          # ragged last tile in the last chunk
    ([0, 0, 2, 2], 32, 8, 128, 1, 30000, 27, 144, 2),       # head_dim 128
    ([0, 1, 2, 3], 12, 1, 64, 3, 5000, 4, 120, 1),          # blocks of one layer (forced)
]


def to_dev(bits):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(
        torch.bfloat16).cuda()


def from_dev(t):
    return t.float().cpu().numpy().astype(np.float64)


def errors(got, expect):
    e = np.abs(got - expect)
    return float(e.max()), float(e.mean())


def run_small_case(owner, h, g, d, b, seq_lens, max_seq, seed, options=None, new_tokens=True,
                   fused=False, expect=None):
    """Full (every output) comparison of all layers of one decode step.

    Owner caches are prefilled with generator values for positions [0, max_seq); when
    new_tokens is set, each owner then appends a different token (another seed) at L-1, through
    mlkv_append on the GPU (or, with fused, mlkv_append_decode_attention) and oracle_append on
    the host.  `expect` maps read-only launch options ("last_cluster_k", ...) to the values the
    decode launches must report.  Returns the worst (max, mean) error.
    """
    import paper_2406_09297_gb300 as mlkv
    import torch

    seq_lens = np.asarray(seq_lens, dtype=np.int32)
    l = len(owner)
    worst = (0.0, 0.0)
    with mlkv.MLKVCache(l, h, d, owner, g, b, max_seq) as cache:
        for k, v in (options or {}).items():
            cache.set_option(k, v)
        ref = oracle.OracleCache(owner, h, g, d, b, max_seq)
        for n in sorted(set(owner)):
            kb = gen.gen_kv(seed, n, 0, b, g, max_seq, d)
            vb = gen.gen_kv(seed, n, 1, b, g, max_seq, d)
            cache.load_prefix(n, to_dev(kb), to_dev(vb), max_seq)
            ref.load_prefix(n, gen.bf16_bits_to_f64(kb), gen.bf16_bits_to_f64(vb), max_seq)
        for n in range(l):
            qb = gen.gen_q(seed, n, b, h, d)
            out = torch.full((b, h, d), float("nan"), dtype=torch.bfloat16, device="cuda")
            kd = vd = None
            if new_tokens:
                kn = gen.gen_bf16(seed + 1, gen.TID_K + n, range(b * g), d).reshape(b, g, d)
                vn = gen.gen_bf16(seed + 1, gen.TID_V + n, range(b * g), d).reshape(b, g, d)
                kd, vd = to_dev(kn), to_dev(vn)
                if not fused:
                    cache.append(n, kd, vd, seq_lens)
                ref.append(n, gen.bf16_bits_to_f64(kn), gen.bf16_bits_to_f64(vn), seq_lens)
            if fused:
                cache.append_decode_attention(n, kd, vd, to_dev(qb), out, seq_lens)
            else:
                cache.decode_attention(n, to_dev(qb), out, seq_lens)
            for key, want in (expect or {}).items():
                assert cache.get_option(key) == want, (key, cache.get_option(key), want)
            ref_out = ref.decode(n, gen.bf16_bits_to_f64(qb), seq_lens)
            got = from_dev(out)
            mx, mean = errors(got, ref_out)
            assert np.isfinite(got).all(), f"layer {n}: non-finite output"
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (
                f"layer {n}: max abs {mx:.3e} mean abs {mean:.3e}")
            worst = (max(worst[0], mx), max(worst[1], mean))
        cache.sync_status()
    return worst
