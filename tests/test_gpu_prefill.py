"""GPU causal prefill (mlkv_prefill, tcgen05 kernel) against the fp64 oracle's prefill.

Every layer of a model is prefilled in order (owner layers store the prompt's K/V, every layer
attends causally over its owner's slot); all rows of every prompt are compared.  Prompt lengths
straddle the 128-position blocks of the kernel; rows past a prompt's length must stay untouched.
A decode step then continues every sequence from the prefilled cache.
"""
import numpy as np
import pytest

import oracle
from mlkv_synth import gen
from tests.mlkv_cases import MAX_ABS, MEAN_ABS, errors, from_dev, to_dev

pytestmark = pytest.mark.gpu

EDGE_PROMPTS = [1, 127, 128, 129, 300]


def _prefill_model(owner, h, g, d, b, prompt_lens, s_max, max_seq, seed, cache, ref, nthreads=4):
    """Prefills every layer of the model on the GPU and in the oracle; returns the worst error."""
    import torch

    l = len(owner)
    prompt_lens = np.asarray(prompt_lens, dtype=np.int32)
    worst = (0.0, 0.0)
    for n in range(l):
        qb = gen.gen_bf16(seed, gen.TID_Q + n, range(b * s_max), h * d).reshape(b, s_max, h, d)
        kd = vd = None
        if owner[n] == n:
            kb = gen.gen_kv(seed, n, 0, b, g, s_max, d)
            vb = gen.gen_kv(seed, n, 1, b, g, s_max, d)
            kd, vd = to_dev(kb), to_dev(vb)
            ref.load_prefix(n, gen.bf16_bits_to_f64(kb), gen.bf16_bits_to_f64(vb), s_max)
        out = torch.full((b, s_max, h, d), float("nan"), dtype=torch.bfloat16, device="cuda")
        cache.prefill(n, to_dev(qb), kd, vd, out, prompt_lens)
        torch.cuda.synchronize()
        expect = ref.prefill(n, gen.bf16_bits_to_f64(qb), prompt_lens, nthreads=nthreads)
        got = from_dev(out)
        for beta in range(b):
            S = int(prompt_lens[beta])
            assert np.isfinite(got[beta, :S]).all(), f"layer {n} seq {beta}: non-finite output"
            assert np.isnan(got[beta, S:]).all(), f"layer {n} seq {beta}: rows past the prompt written"
            mx, mean = errors(got[beta, :S], expect[beta, :S])
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (n, beta, mx, mean)
            worst = (max(worst[0], mx), max(worst[1], mean))
    cache.sync_status()
    return worst


@pytest.mark.parametrize("name,owner,h,g", [
    ("mha", [0, 1, 2], 4, 4),
    ("gqa", [0, 1, 2], 12, 4),
    ("mqa", [0, 1], 12, 1),
    ("mlkv-block", [0, 0, 2, 2], 12, 3),
    ("mlkv-1", [0, 0, 0], 16, 1),
    ("non-uniform", [0, 0, 0, 3, 4, 4], 8, 2),
])
@pytest.mark.parametrize("d", [64, 128])
def test_prefill_maps_and_edges(name, owner, h, g, d):
    import paper_2406_09297_gb300 as mlkv
    b, s_max = len(EDGE_PROMPTS), 300
    with mlkv.MLKVCache(len(owner), h, d, owner, g, b, s_max) as cache:
        ref = oracle.OracleCache(owner, h, g, d, b, s_max)
        _prefill_model(owner, h, g, d, b, EDGE_PROMPTS, s_max, s_max, 51, cache, ref)


@pytest.mark.parametrize("d", [64, 128])
def test_prefill_long_prompts(d):
    # 16 blocks of 128 positions per prompt: the causal triangle's tiles, longest blocks first
    import paper_2406_09297_gb300 as mlkv
    owner, h, g, b, s_max = [0, 0], 12, 1, 2, 2048
    with mlkv.MLKVCache(2, h, d, owner, g, b, s_max) as cache:
        ref = oracle.OracleCache(owner, h, g, d, b, s_max)
        _prefill_model(owner, h, g, d, b, [2048, 1500], s_max, s_max, 52, cache, ref, nthreads=2)


def test_prefill_long_prompt_every_row():
    # A 6000-position prompt: 47 key tiles per query block, units of very different lengths.
    import paper_2406_09297_gb300 as mlkv
    owner, h, g, d = [0], 4, 1, 64
    with mlkv.MLKVCache(1, h, d, owner, g, 1, 6000) as cache:
        ref = oracle.OracleCache(owner, h, g, d, 1, 6000)
        _prefill_model(owner, h, g, d, 1, [6000], 6000, 6000, 54, cache, ref, nthreads=8)


def test_prefill_then_decode_continues():
    # The cache a prefill leaves is the cache decoding continues from (Sec. 4.5: a prompt, then
    # tokens one by one): one decode step at length prompt + 1 in every layer.
    import torch

    import paper_2406_09297_gb300 as mlkv
    owner, h, g, d, b = [0, 0, 2, 2], 12, 3, 64, 3
    prompts = np.array([100, 257, 40], dtype=np.int32)
    s_max, max_seq = 257, 320
    seed = 53
    with mlkv.MLKVCache(len(owner), h, d, owner, g, b, max_seq) as cache:
        ref = oracle.OracleCache(owner, h, g, d, b, max_seq)
        _prefill_model(owner, h, g, d, b, prompts, s_max, max_seq, seed, cache, ref)
        lens = prompts + 1
        owners = sorted(set(owner))
        qb = np.stack([gen.gen_q(seed + 7, n, b, h, d) for n in range(len(owner))])
        kn = np.stack([gen.gen_bf16(seed + 8, gen.TID_K + n, range(b * g), d).reshape(b, g, d)
                       for n in owners])
        vn = np.stack([gen.gen_bf16(seed + 8, gen.TID_V + n, range(b * g), d).reshape(b, g, d)
                       for n in owners])
        out = torch.full((len(owner), b, h, d), float("nan"), dtype=torch.bfloat16, device="cuda")
        cache.decode_step(to_dev(qb), to_dev(kn), to_dev(vn), out, lens)
        torch.cuda.synchronize()
        for n in range(len(owner)):
            if owner[n] == n:
                k = owners.index(n)
                ref.append(n, gen.bf16_bits_to_f64(kn[k]), gen.bf16_bits_to_f64(vn[k]), lens)
            expect = ref.decode(n, gen.bf16_bits_to_f64(qb[n]), lens)
            mx, mean = errors(from_dev(out[n]), expect)
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (n, mx, mean)
        cache.sync_status()


def test_prefill_rejects_bad_arguments():
    import torch

    import paper_2406_09297_gb300 as mlkv
    with mlkv.MLKVCache(2, 4, 64, [0, 0], 2, 2, 256) as cache:
        q = torch.zeros((2, 256, 4, 64), dtype=torch.bfloat16, device="cuda")
        kv = torch.zeros((2, 2, 256, 64), dtype=torch.bfloat16, device="cuda")
        out = torch.zeros_like(q)
        for lens in ([0, 5], [257, 5]):
            with pytest.raises(mlkv.MLKVError) as e:
                cache.prefill(0, q, kv, kv, out, lens)
            assert e.value.code == mlkv.MLKV_ERR_RANGE
        with pytest.raises(mlkv.MLKVError) as e:
            cache.prefill(0, q, None, None, out, [5, 5])   # an owner layer needs its K/V
        assert e.value.code == mlkv.MLKV_ERR_INVALID_ARG
        with pytest.raises(mlkv.MLKVError) as e:
            cache.prefill(1, q, None, None, q, [5, 5])     # out overlapping Q
        assert e.value.code == mlkv.MLKV_ERR_INVALID_ARG
        cache.prefill(1, q, None, None, out, [5, 5])       # a non-owner layer needs no K/V
        cache.sync_status()
