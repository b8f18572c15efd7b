"""mlkv_decode_step at the benchmark's full sizes, against the fp64 oracle on sampled outputs.

The benchmark times mlkv_decode_step: one call per step that issues every layer with the step's
own launch shapes (whole segments per CTA, a long single segment on 64 CTAs, clusters or a
stream-K split), lets each layer's grid start before the previous one ends (the later layers of a
block take the owner's new token from the step's input instead of from the cache), prefetches
slots into L2, and replays the whole step from a recorded CUDA graph.  These tests run exactly
that call on every workload of the benchmark suite at full batch and context:

  * the cache holds the generator's K/V at every position; the step's new tokens come from
    another seed, so the newest row (position L-1) of every owner's slot changes in the step and
    a layer that read it from the cache before its owner stored it would be caught;
  * the first call is issued directly, the second records the graph, the third replays it (with
    the default step_graph 2 a step that runs as one multi-layer launch is issued directly every
    time); the outputs of the first and of the third call are both checked;
  * for sampled (sequence, KV head) pairs -- the first and last sequence and seeded random ones
    -- the oracle recomputes that KV head's query group in every layer (Eqs. 2-3 with the maps of
    Eqs. 15 and 18) from the generator's values rebuilt on the host, and every sampled output must
    match within the parity tolerance.
"""
import numpy as np
import pytest

import oracle
from mlkv_synth import gen, workloads
from tests.mlkv_cases import MAX_ABS, MEAN_ABS, errors

pytestmark = pytest.mark.gpu

NEW_SEED_OFFSET = 77   # the step's new tokens: another seed than the cache's contents


def _sample_pairs(w, n_betas, rng):
    betas = sorted({0, w.b - 1} | set(int(x) for x in rng.integers(0, w.b, size=n_betas)))
    return [(beta, int(rng.integers(0, w.g))) for beta in betas]


def _step_inputs(w, cache):
    """Device tensors of one step: Q [l][b][h][d], new K/V [m][b][g][d] (slot order) drawn from
    another seed than the cache, and the lengths."""
    import torch

    from mlkv_synth import device

    seq_lens, Q, _, _ = device.workload_inputs(w, cache)
    owners = w.owners()
    s2 = w.seed + NEW_SEED_OFFSET
    Ks = torch.stack([device.kv_token(s2, n, 0, w.b, w.g, w.d, seq_lens, w.sigma_k)
                      for n in owners])
    Vs = torch.stack([device.kv_token(s2, n, 1, w.b, w.g, w.d, seq_lens, w.sigma_v)
                      for n in owners])
    return seq_lens, torch.stack(Q), Ks, Vs


def _oracle_group(w, n, beta, j, L, kv_rows):
    """The oracle's output of layer n for the query group of KV head j of sequence beta."""
    G = w.h // w.g
    k, v = kv_rows
    q = gen.bf16_bits_to_f64(gen.gen_q(w.seed, n, w.b, w.h, w.d, w.sigma_q,
                                       betas=[beta]))[:, j * G:(j + 1) * G]
    # the query group of KV head j alone: h' = G query heads over one KV head
    return oracle.decode_layer(n, w.owner, G, 1, w.d, [L], q, k, v)


def _kv_rows(w, own, beta, j, L):
    """Host copy of owner `own`'s K and V rows [0, L) of (beta, j) after the step: the cache's
    generator values, the newest row replaced by the step's new token."""
    s2 = w.seed + NEW_SEED_OFFSET
    out = []
    for kv, sigma in ((0, w.sigma_k), (1, w.sigma_v)):
        bits = gen.gen_kv(w.seed, own, kv, w.b, w.g, L, w.d, sigma, betas=[beta], heads=[j])
        bits[:, :, L - 1, :] = gen.gen_kv(s2, own, kv, w.b, w.g, 1, w.d, sigma, betas=[beta],
                                          heads=[j], t0=L - 1)[:, :, 0, :]
        out.append(gen.bf16_bits_to_f64(bits))
    return tuple(out)


def check_step_full_size(w, n_betas=4, seed=0, options=None, host_buffers=False):
    import torch

    import paper_2406_09297_gb300 as mlkv

    rng = np.random.default_rng(seed)
    with mlkv.MLKVCache(w.l, w.h, w.d, w.owner, w.g, w.b, w.max_seq) as cache:
        for key, val in (options or {}).items():
            cache.set_option(key, val)
        seq_lens, Q, K, V = _step_inputs(w, cache)
        shape = (w.l, w.b, w.h, w.d)
        # One output buffer for the three calls (the graph is recorded for these arguments); the
        # first call's result is copied out before the second.
        checked = []
        if host_buffers:
            Qh, Kh, Vh = Q.cpu().pin_memory(), K.cpu().pin_memory(), V.cpu().pin_memory()
            out = torch.empty(shape, dtype=torch.bfloat16).pin_memory()
            for rep in range(3):   # direct, record, replay
                out.fill_(float("nan"))
                cache.decode_step_host(Qh, Kh, Vh, out, seq_lens)
                torch.cuda.synchronize()
                if rep != 1:
                    checked.append(out.float().numpy().copy())
        else:
            out = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
            for rep in range(3):   # direct, record, replay (or three direct launches)
                out.fill_(float("nan"))
                cache.decode_step(Q, K, V, out, seq_lens)
                torch.cuda.synchronize()
                if rep != 1:
                    checked.append(out.float().cpu().numpy())
            # step_graph 2 (default) issues one multi-layer launch directly, else it replays
            direct = (cache.get_option("step_graph") == 2 and
                      cache.get_option("last_step_kernel") == 1)
            assert cache.get_option("step_graph_replays") == (0 if direct else 2)
        fused = cache.get_option("last_step_fused")
        sm_count = cache.get_option("sm_count")
        cache.sync_status()
        worst = 0.0
        for own in w.owners():
            for beta, j in _sample_pairs(w, n_betas, rng):
                L = int(seq_lens[beta])
                rows = _kv_rows(w, own, beta, j, L)
                G = w.h // w.g
                for n in range(w.l):
                    if w.owner[n] != own:
                        continue
                    expect = _oracle_group(w, n, beta, j, L, rows)
                    for got_all in checked:
                        got = got_all[n, beta, j * G:(j + 1) * G][None].astype(np.float64)
                        assert np.isfinite(got).all(), (w.name, n, beta, j)
                        mx, mean = errors(got, expect)
                        assert mx <= MAX_ABS and mean <= MEAN_ABS, (w.name, n, beta, j, mx, mean)
                        worst = max(worst, mx)
        return worst, fused, sm_count


# Which benchmark configurations run the step in the cross-layer fused form by default (blocks of
# >= 3 layers where its cost estimate beats the decode kernel's): MLKV-2 b64, GQA-4 + MLKV-4 b128
# and the Llama-2-7B shapes do; the batch-1 MLKV-6 map of pairs does not.
FUSED_BY_DEFAULT = {1: 0, 2: 1, 3: 1, 4: 1}


@pytest.mark.parametrize("index", [1, 2, 3, 4])
def test_step_config_full_size(index):
    w = workloads.config(index)
    _, fused, _ = check_step_full_size(w, seed=index)
    assert fused == FUSED_BY_DEFAULT[index]


@pytest.mark.parametrize("name", [w.name for w in workloads.sweep(False)])
def test_step_sweep_b256_L8192(name):
    check_step_full_size(workloads.by_name(name), n_betas=3, seed=5)


@pytest.mark.parametrize("name", [w.name for w in workloads.sweep(True)])
def test_step_sweep_b1_L131072(name):
    check_step_full_size(workloads.by_name(name), n_betas=0, seed=6)


def test_step_host_buffers_config2_full_size():
    """mlkv_decode_step_host (the e2e leg of the benchmark: inputs read from pinned host memory,
    outputs written back to it) on the benchmark's default workload."""
    check_step_full_size(workloads.config(2), seed=12, host_buffers=True)


@pytest.mark.parametrize("options", [{"l2_prefetch": 0}, {"l2_persist": 1}, {"step_kernel": 0},
                                     {"step_graph": 1}, {"step_kernel": 0, "early_fetch": 0},
                                     {"step_kernel": 0, "early_fetch": 2},
                                     {"step_kernel": 0, "pdl": 0}, {"step_fused": 0},
                                     {"step_fused": 0, "step_graph": 1}])
def test_step_options_full_size(options):
    """Options that change where bytes come from or how the step is launched, never the result:
    the default workload and the varied-length GQA workload (slots larger than L2) with the L2
    prefetch off, with L2 persistence on, with per-layer launches instead of one multi-layer launch (overlapping; with
    no read, or only the first cache tile, before the previous layer's end; in plain stream
    order), with the multi-layer decode launch instead of the fused form, and with the step
    replayed from a recorded graph."""
    import paper_2406_09297_gb300 as mlkv
    for index in (2, 3):
        try:
            check_step_full_size(workloads.config(index), seed=20 + index, options=options)
        except mlkv.MLKVError as e:
            if e.code == mlkv.MLKV_ERR_UNSUPPORTED and "l2_persist" in options:
                pytest.skip(f"no persisting L2 set-aside on this device: {e}")
            raise
