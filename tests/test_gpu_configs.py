"""Full-size workloads in the bench's launch configuration, checked on sampled outputs.

Every workload of the benchmark suite (the Pythia-160M and Llama-2-7B shaped MLKV / GQA maps at
their full batch and context) runs one decode step exactly as bench.py does: owner layers through
mlkv_append_decode_attention, the others through mlkv_decode_attention, default options.  For
sampled (sequence, KV head) pairs -- first, last and seeded random sequences -- the fp64 oracle
recomputes the outputs of that KV head's query group in every layer, from the generator's inputs
rebuilt on the host, and every sampled output must match within the parity tolerance.
"""
import numpy as np
import pytest

import oracle
from mlkv_synth import gen, workloads
from tests.mlkv_cases import MAX_ABS, MEAN_ABS, errors

pytestmark = pytest.mark.gpu


def _sample_pairs(w, n_betas, rng):
    betas = sorted({0, w.b - 1} | set(int(x) for x in rng.integers(0, w.b, size=n_betas)))
    return [(beta, int(rng.integers(0, w.g))) for beta in betas]


def run_full_size(w, n_betas=4, seed=0):
    import torch

    import paper_2406_09297_gb300 as mlkv
    from mlkv_synth import device

    rng = np.random.default_rng(seed)
    with mlkv.MLKVCache(w.l, w.h, w.d, w.owner, w.g, w.b, w.max_seq) as cache:
        seq_lens, Q, Kn, Vn = device.workload_inputs(w, cache)
        outs = []
        for n in range(w.l):
            out = torch.full((w.b, w.h, w.d), float("nan"), dtype=torch.bfloat16, device="cuda")
            if n in Kn:
                cache.append_decode_attention(n, Kn[n], Vn[n], Q[n], out, seq_lens)
            else:
                cache.decode_attention(n, Q[n], out, seq_lens)
            outs.append(out)
        torch.cuda.synchronize()
        cache.sync_status()
        pairs = _sample_pairs(w, n_betas, rng)
        G = w.h // w.g
        worst = 0.0
        for own in w.owners():
            for beta, j in pairs:
                L = int(seq_lens[beta])
                k = gen.bf16_bits_to_f64(gen.gen_kv(w.seed, own, 0, w.b, w.g, L, w.d, w.sigma_k,
                                                    betas=[beta], heads=[j]))
                v = gen.bf16_bits_to_f64(gen.gen_kv(w.seed, own, 1, w.b, w.g, L, w.d, w.sigma_v,
                                                    betas=[beta], heads=[j]))
                for n in range(w.l):
                    if w.owner[n] != own:
                        continue
                    q = gen.bf16_bits_to_f64(gen.gen_q(w.seed, n, w.b, w.h, w.d, w.sigma_q,
                                                       betas=[beta]))[:, j * G:(j + 1) * G]
                    # the query group of KV head j alone: h' = G query heads over one KV head
                    expect = oracle.decode_layer(n, w.owner, G, 1, w.d, [L], q, k, v)
                    got = outs[n][beta, j * G:(j + 1) * G].float().cpu().numpy()[None]
                    mx, mean = errors(got.astype(np.float64), expect)
                    assert np.isfinite(got).all()
                    assert mx <= MAX_ABS and mean <= MEAN_ABS, (w.name, n, beta, j, mx, mean)
                    worst = max(worst, mx)
        return worst


@pytest.mark.parametrize("index", [1, 2, 3, 4])
def test_config_full_size(index):
    run_full_size(workloads.config(index), seed=index)


@pytest.mark.parametrize("name", [w.name for w in workloads.sweep(False)])
def test_sweep_b256_L8192(name):
    run_full_size(workloads.by_name(name), n_betas=3, seed=5)


@pytest.mark.parametrize("name", [w.name for w in workloads.sweep(True)])
def test_sweep_b1_L131072(name):
    run_full_size(workloads.by_name(name), n_betas=0, seed=6)
