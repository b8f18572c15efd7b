"""mlkv_decode_step (every layer of a decode step in one call, replayed from a recorded CUDA graph)
against the per-layer calls and the oracle."""
import numpy as np
import pytest

import oracle
from mlkv_synth import gen
from tests.mlkv_cases import (FUSED_STEP_CASES, FUSED_STEP_SMS, MAX_ABS, MEAN_ABS, errors,
                              from_dev, to_dev)

pytestmark = pytest.mark.gpu


def _inputs(owner, h, g, d, b, lens, max_seq, seed, cache, ref):
    m = len(set(owner))
    for n in sorted(set(owner)):
        kb = gen.gen_kv(seed, n, 0, b, g, max_seq, d)
        vb = gen.gen_kv(seed, n, 1, b, g, max_seq, d)
        cache.load_prefix(n, to_dev(kb), to_dev(vb), max_seq)
        if ref is not None:
            ref.load_prefix(n, gen.bf16_bits_to_f64(kb), gen.bf16_bits_to_f64(vb), max_seq)
    qb = np.stack([gen.gen_q(seed, n, b, h, d) for n in range(len(owner))])
    owners = sorted(set(owner))
    kn = np.stack([gen.gen_bf16(seed + 1, gen.TID_K + n, range(b * g), d).reshape(b, g, d)
                   for n in owners])
    vn = np.stack([gen.gen_bf16(seed + 1, gen.TID_V + n, range(b * g), d).reshape(b, g, d)
                   for n in owners])
    return qb, kn, vn


def _fused_applies(owner, h, g):
    """Maps the step can run in the cross-layer fused form (option step_fused 2 forces it there):
    equal contiguous owner blocks whose L * G query rows fit two tiles of 128."""
    l, m = len(owner), len(set(owner))
    L, G = l // m, h // g
    return (L * m == l and all(owner[n] == n - n % L for n in range(l)) and
            128 // G >= 1 and L <= 2 * (128 // G))


@pytest.mark.parametrize("fused", [2, 0])
@pytest.mark.parametrize("owner,h,g,d,b,lens,max_seq", [
    ([0, 0, 2, 2, 2, 5], 12, 2, 64, 5, [1, 300, 1000, 77, 640], 1024),
    ([0, 0, 0, 0], 12, 1, 64, 64, [2048] * 64, 2048),            # whole segments per CTA
    # the benchmark's map (owner change at layer 6) with one length: whole segments per CTA,
    # the later layers taking the owner's new token from the step input, slot 1 prefetched
    ([0] * 6 + [6] * 6, 12, 1, 64, 64, [1024] * 64, 1024),
    ([0, 0, 2], 16, 4, 128, 3, [5000, 20, 4096], 5000),
])
def test_step_matches_oracle_and_layer_calls(owner, h, g, d, b, lens, max_seq, fused):
    import torch

    import paper_2406_09297_gb300 as mlkv
    seed = 31
    lens = np.asarray(lens, dtype=np.int32)
    l = len(owner)
    with mlkv.MLKVCache(l, h, d, owner, g, b, max_seq) as cache, \
            mlkv.MLKVCache(l, h, d, owner, g, b, max_seq) as cache2:
        ref = oracle.OracleCache(owner, h, g, d, b, max_seq)
        qb, kn, vn = _inputs(owner, h, g, d, b, lens, max_seq, seed, cache, ref)
        _inputs(owner, h, g, d, b, lens, max_seq, seed, cache2, None)
        Q, K, V = to_dev(qb), to_dev(kn), to_dev(vn)
        out = torch.full((l, b, h, d), float("nan"), dtype=torch.bfloat16, device="cuda")
        cache.set_option("step_graph", 1)   # always through the recorded graph
        cache.set_option("step_fused", fused)
        for rep in range(4):   # direct, record, then replay twice
            out.fill_(float("nan"))
            cache.decode_step(Q, K, V, out, lens)
        torch.cuda.synchronize()
        assert cache.get_option("step_graph_replays") == 3
        assert cache.get_option("last_step_fused") == int(fused > 0 and _fused_applies(owner, h, g))
        # the same layer calls one by one on a second cache
        owners = sorted(set(owner))
        out2 = torch.full_like(out, float("nan"))
        for n in range(l):
            if owner[n] == n:
                s = owners.index(n)
                cache2.append_decode_attention(n, K[s], V[s], Q[n], out2[n], lens)
            else:
                cache2.decode_attention(n, Q[n], out2[n], lens)
        torch.cuda.synchronize()
        if cache.get_option("last_step_kernel"):
            # The step is one multi-layer launch of whole segments (no merge), while the layer
            # calls split segments over CTAs: same results up to rounding.
            assert cache.get_option("last_cluster_k") == 0
        else:
            # per-layer launches of the step: the layer calls' shapes, bit for bit
            assert torch.equal(out.view(torch.int16), out2.view(torch.int16))
        if bool((lens == lens[0]).all()):
            assert cache.get_option("last_step_kernel") == 1
        for n in range(l):
            if owner[n] == n:
                s = owners.index(n)
                ref.append(n, gen.bf16_bits_to_f64(kn[s]), gen.bf16_bits_to_f64(vn[s]), lens)
            expect = ref.decode(n, gen.bf16_bits_to_f64(qb[n]), lens)
            for o in (out, out2):
                mx, mean = errors(from_dev(o[n]), expect)
                assert mx <= MAX_ABS and mean <= MEAN_ABS, (n, mx, mean)
        cache.sync_status()
        cache2.sync_status()


def test_step_rerecords_on_new_lengths_and_buffers():
    import torch

    import paper_2406_09297_gb300 as mlkv
    owner, h, g, d, b, max_seq = [0, 0, 2, 2], 8, 2, 64, 4, 700
    with mlkv.MLKVCache(4, h, d, owner, g, b, max_seq) as cache:
        qb, kn, vn = _inputs(owner, h, g, d, b, None, max_seq, 41, cache, None)
        Q, K, V = to_dev(qb), to_dev(kn), to_dev(vn)
        outs = []
        for lens in ([300, 1, 700, 64], [301, 2, 700, 65], [301, 2, 700, 65]):
            lens = np.asarray(lens, dtype=np.int32)
            out = torch.empty((4, b, h, d), dtype=torch.bfloat16, device="cuda")
            cache.decode_step(Q, K, V, out, lens)
            outs.append((lens, out))
        torch.cuda.synchronize()
        with mlkv.MLKVCache(4, h, d, owner, g, b, max_seq) as check:
            _inputs(owner, h, g, d, b, None, max_seq, 41, check, None)
            check.set_option("step_graph", 0)
            for lens, out in outs:
                ref = torch.empty_like(out)
                check.decode_step(Q, K, V, ref, lens)
                torch.cuda.synchronize()
                assert torch.equal(out.view(torch.int16), ref.view(torch.int16))


def test_step_inside_a_caller_graph():
    import torch

    import paper_2406_09297_gb300 as mlkv
    owner, h, g, d, b, max_seq = [0, 0], 12, 1, 64, 8, 512
    lens = np.full(b, 512, dtype=np.int32)
    with mlkv.MLKVCache(2, h, d, owner, g, b, max_seq) as cache:
        qb, kn, vn = _inputs(owner, h, g, d, b, lens, max_seq, 51, cache, None)
        Q, K, V = to_dev(qb), to_dev(kn), to_dev(vn)
        out = torch.empty((2, b, h, d), dtype=torch.bfloat16, device="cuda")
        ref = torch.empty_like(out)
        cache.set_option("step_graph", 0)
        cache.decode_step(Q, K, V, ref, lens)
        cache.set_option("step_graph", 1)
        graph = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            cache.decode_step(Q, K, V, out, lens)
        torch.cuda.current_stream().wait_stream(s)
        with torch.cuda.graph(graph):
            cache.decode_step(Q, K, V, out, lens)
        out.zero_()
        graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(out.view(torch.int16), ref.view(torch.int16))


@pytest.mark.parametrize("owner,h,g,d,b,prefix", [
    ([0, 0, 2, 2], 8, 2, 64, 3, [100, 257, 512]),
    ([0, 0, 0, 0, 0, 0], 12, 1, 64, 8, [2000] * 8),   # the decode-loop benchmark's shape, shortened
])
def test_decode_loop_growing_lengths(owner, h, g, d, b, prefix):
    # Autoregressive decode as in the paper's throughput measurement (Sec. 4.5): from a
    # pre-filled cache, every step appends a new token per owner layer (lengths grow by one) and
    # attends over the cache in every layer; every step of every layer is checked.
    import torch

    import paper_2406_09297_gb300 as mlkv
    seed, steps = 41, 5
    l = len(owner)
    owners = sorted(set(owner))
    max_seq = max(prefix) + steps
    with mlkv.MLKVCache(l, h, d, owner, g, b, max_seq) as cache:
        ref = oracle.OracleCache(owner, h, g, d, b, max_seq)
        for n in owners:
            kb = gen.gen_kv(seed, n, 0, b, g, max_seq, d)
            vb = gen.gen_kv(seed, n, 1, b, g, max_seq, d)
            cache.load_prefix(n, to_dev(kb), to_dev(vb), max_seq)
            ref.load_prefix(n, gen.bf16_bits_to_f64(kb), gen.bf16_bits_to_f64(vb), max_seq)
        out = torch.empty((l, b, h, d), dtype=torch.bfloat16, device="cuda")
        for s in range(steps):
            lens = np.asarray(prefix, dtype=np.int32) + s + 1
            qb = np.stack([gen.gen_q(seed + 100 + s, n, b, h, d) for n in range(l)])
            kn = np.stack([gen.gen_bf16(seed + 200 + s, gen.TID_K + n, range(b * g), d)
                           .reshape(b, g, d) for n in owners])
            vn = np.stack([gen.gen_bf16(seed + 200 + s, gen.TID_V + n, range(b * g), d)
                           .reshape(b, g, d) for n in owners])
            out.fill_(float("nan"))
            cache.decode_step(to_dev(qb), to_dev(kn), to_dev(vn), out, lens)
            torch.cuda.synchronize()
            for n in range(l):
                if owner[n] == n:
                    k = owners.index(n)
                    ref.append(n, gen.bf16_bits_to_f64(kn[k]), gen.bf16_bits_to_f64(vn[k]), lens)
                expect = ref.decode(n, gen.bf16_bits_to_f64(qb[n]), lens)
                mx, mean = errors(from_dev(out[n]), expect)
                assert mx <= MAX_ABS and mean <= MEAN_ABS, (s, n, mx, mean)
        cache.sync_status()


def test_step_host_buffers_match_device_step():
    # mlkv_decode_step_host: the same step with Q, K, V and out in host memory; pinned buffers are
    # replayed from a graph from the second call on (recorded then), pageable ones run directly.
    import torch

    import paper_2406_09297_gb300 as mlkv
    from mlkv_synth import device, workloads
    w = workloads.config(1)
    with mlkv.MLKVCache(w.l, w.h, w.d, w.owner, w.g, w.b, w.max_seq) as cache:
        seq_lens, Q, Kn, Vn = device.workload_inputs(w, cache)
        owners = w.owners()
        Qs = torch.stack(Q)
        Ks = torch.stack([Kn[n] for n in owners])
        Vs = torch.stack([Vn[n] for n in owners])
        ref = torch.empty((w.l, w.b, w.h, w.d), dtype=torch.bfloat16, device="cuda")
        cache.decode_step(Qs, Ks, Vs, ref, seq_lens)
        torch.cuda.synchronize()
        want = ref.cpu()
        for pinned in (True, False):
            hq, hk, hv = Qs.cpu(), Ks.cpu(), Vs.cpu()
            out = torch.full((w.l, w.b, w.h, w.d), float("nan"), dtype=torch.bfloat16)
            if pinned:
                hq, hk, hv, out = hq.pin_memory(), hk.pin_memory(), hv.pin_memory(), out.pin_memory()
            for graph in (1, 2):   # always recorded; the default (direct for one launch)
                cache.set_option("step_graph", graph)
                before = cache.get_option("step_graph_replays")
                for _ in range(4):
                    out.fill_(float("nan"))
                    cache.decode_step_host(hq, hk, hv, out, seq_lens)
                    torch.cuda.synchronize()
                    assert torch.equal(out.view(torch.int16), want.view(torch.int16))
                replays = cache.get_option("step_graph_replays") - before
                direct = graph == 2 and cache.get_option("last_step_kernel") == 1
                assert replays == (3 if pinned and not direct else 0), (pinned, graph, replays)
        cache.sync_status()


@pytest.mark.parametrize("step_kernel", [1, 0])
def test_step_single_long_segment(step_kernel):
    # Batch 1, one KV head, 16384 positions.  One multi-layer launch splits every layer's
    # segment into 8 chunks of 8 tiles of 256 positions (24 CTAs), each a partial record, and
    # one combine launch merges them; per-layer launches (step_kernel 0) run the later layers'
    # 128-position tile over 64 CTAs with a merge launch per layer.
    import torch

    import paper_2406_09297_gb300 as mlkv
    owner, h, g, d, b, L = [0, 0, 0], 12, 1, 64, 1, 16384
    lens = np.full(b, L, dtype=np.int32)
    with mlkv.MLKVCache(len(owner), h, d, owner, g, b, L) as cache:
        cache.set_option("step_kernel", step_kernel)
        cache.set_option("step_fused", 0)   # the decode kernel's launch shapes
        ref = oracle.OracleCache(owner, h, g, d, b, L)
        qb, kn, vn = _inputs(owner, h, g, d, b, lens, L, 61, cache, ref)
        out = torch.full((len(owner), b, h, d), float("nan"), dtype=torch.bfloat16, device="cuda")
        cache.decode_step(to_dev(qb), to_dev(kn), to_dev(vn), out, lens)
        torch.cuda.synchronize()
        assert cache.get_option("last_step_kernel") == step_kernel
        assert cache.get_option("last_tile_tokens") == (256 if step_kernel else 128)
        assert cache.get_option("last_deferred_merge") == 1
        assert cache.get_option("last_grid") == (24 if step_kernel else 64)
        ref.append(0, gen.bf16_bits_to_f64(kn[0]), gen.bf16_bits_to_f64(vn[0]), lens)
        for n in range(len(owner)):
            expect = ref.decode(n, gen.bf16_bits_to_f64(qb[n]), lens)
            mx, mean = errors(from_dev(out[n]), expect)
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (n, mx, mean)
        cache.sync_status()


@pytest.mark.parametrize("b,g,L,grid,tile", [
    (128, 2, 512, 128, 128),    # 256 segments of 4 tiles of 128: 128 CTAs of two segments
    (64, 4, 4352, 64, 256),     # 256 segments of 17 tiles of 256: 64 CTAs of four segments
])
def test_step_whole_segments_per_cta(b, g, L, grid, tile):
    # With per-layer launches (option step_kernel 0) the later layers of a step run whole
    # segments per CTA, several per CTA here: each later segment's queries arrive with its first
    # tile.
    import torch

    import paper_2406_09297_gb300 as mlkv
    owner, h, d = [0, 0, 0], 12, 64
    lens = np.full(b, L, dtype=np.int32)
    with mlkv.MLKVCache(len(owner), h, d, owner, g, b, L) as cache:
        cache.set_option("step_kernel", 0)
        ref = oracle.OracleCache(owner, h, g, d, b, L)
        qb, kn, vn = _inputs(owner, h, g, d, b, lens, L, 71, cache, ref)
        out = torch.full((len(owner), b, h, d), float("nan"), dtype=torch.bfloat16, device="cuda")
        cache.decode_step(to_dev(qb), to_dev(kn), to_dev(vn), out, lens)
        torch.cuda.synchronize()
        assert cache.get_option("last_grid") == grid
        assert cache.get_option("last_tile_tokens") == tile
        assert cache.get_option("last_cluster_k") == 0
        ref.append(0, gen.bf16_bits_to_f64(kn[0]), gen.bf16_bits_to_f64(vn[0]), lens)
        for n in range(len(owner)):
            expect = ref.decode(n, gen.bf16_bits_to_f64(qb[n]), lens, nthreads=8)
            mx, mean = errors(from_dev(out[n]), expect)
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (n, mx, mean)
        cache.sync_status()


@pytest.mark.parametrize("owner,h,g,d,b,L,grid", [
    ([0] * 6 + [6] * 6, 12, 1, 64, 64, 2048, 256),     # the benchmark's shape: 768 items, 3 a CTA
    ([0, 1, 2, 3], 12, 1, 64, 40, 700, 160),           # every layer an owner (MQA), ragged last tile
    ([0, 0, 0, 3, 3, 3], 12, 4, 64, 16, 1000, 192),    # GQA groups of 3 under MLKV
    ([0, 0, 2, 2], 32, 8, 128, 8, 1500, 128),          # head_dim 128, groups of 4
    ([0, 0, 2, 2, 4, 4, 6, 6, 8, 8, 10, 10], 12, 1, 64, 1, 128, 12),   # short context: one wave
    ([0, 0, 0], 16, 2, 64, 100, 77, 300),              # one partly visible tile per item
    ([0] * 6, 12, 1, 64, 8, 2001, 48),                 # batch 8: one 256-position-tile item a CTA
    # few long segments: every segment in chunks, partial records, one merge launch
    ([0] * 6 + [6] * 6, 12, 1, 64, 1, 131072, 152),    # 38 chunks of 13-14 256-tiles: 3 waves
    ([0, 0, 2, 2], 12, 4, 64, 2, 9000, 128),           # ragged last tile in the last chunk
    ([0, 0, 2, 2], 32, 8, 128, 1, 30000, 152),         # head_dim 128: 19 chunks, 4 waves of 152
])
def test_multi_layer_step_kernel(owner, h, g, d, b, L, grid):
    # One launch for the whole step: CTA c takes the (layer, segment) items c, c + P, ..., each a
    # whole segment; every layer replaces its newest rows from the step's new tokens and owner
    # layers store them.  Every output of every layer against the oracle; graph replay too.
    import torch

    import paper_2406_09297_gb300 as mlkv
    lens = np.full(b, L, dtype=np.int32)
    l = len(owner)
    owners = sorted(set(owner))
    with mlkv.MLKVCache(l, h, d, owner, g, b, L) as cache:
        ref = oracle.OracleCache(owner, h, g, d, b, L)
        qb, kn, vn = _inputs(owner, h, g, d, b, lens, L, 81, cache, ref)
        Q, K, V = to_dev(qb), to_dev(kn), to_dev(vn)
        out = torch.empty((l, b, h, d), dtype=torch.bfloat16, device="cuda")
        cache.set_option("step_graph", 1)   # always through the recorded graph
        cache.set_option("step_fused", 0)   # the decode kernel's multi-layer launch
        results = []
        for rep in range(3):   # direct, record, replay
            out.fill_(float("nan"))
            cache.decode_step(Q, K, V, out, lens)
            torch.cuda.synchronize()
            results.append(out.clone())
            assert cache.get_option("last_step_kernel") == 1
            assert cache.get_option("last_step_fused") == 0
            assert cache.get_option("last_grid") == grid
        assert cache.get_option("step_graph_replays") == 2
        for r in results[1:]:
            assert torch.equal(r.view(torch.int16), results[0].view(torch.int16))
        for n in range(l):
            if owner[n] == n:
                k = owners.index(n)
                ref.append(n, gen.bf16_bits_to_f64(kn[k]), gen.bf16_bits_to_f64(vn[k]), lens)
            expect = ref.decode(n, gen.bf16_bits_to_f64(qb[n]), lens, nthreads=8)
            mx, mean = errors(from_dev(results[0][n]), expect)
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (n, mx, mean)
        # the owners' new tokens are in the cache afterwards, at position L - 1, K and V
        from tests.test_gpu_cache import _read_cache
        whole = _read_cache(cache, b, g, L, d)          # int16 [m][2][b][g][L][d]
        for k, n in enumerate(owners):
            assert (whole[cache.owner_slot(n)[1], 0, :, :, L - 1] == kn[k].view(np.int16)).all()
            assert (whole[cache.owner_slot(n)[1], 1, :, :, L - 1] == vn[k].view(np.int16)).all()
        cache.sync_status()



@pytest.mark.parametrize("fused", [2, 0])
@pytest.mark.parametrize("owner,h,g,d,lens", [
    # varied lengths: segments sorted longest first and dealt in a snake round-robin
    ([0, 0, 0, 3, 3, 3], 12, 4, 64, [1, 127, 128, 129, 3000, 64, 700, 2048, 5, 1999] * 4),
    ([0, 0, 2, 2], 32, 8, 128, [300, 1, 1500, 900, 64, 65, 1024, 777]),
    ([0, 1, 1, 3], 12, 1, 64, [int(x) for x in np.random.default_rng(7).integers(1, 4097, 96)]),
])
def test_multi_layer_step_varied_lengths(owner, h, g, d, lens, fused):
    import torch

    import paper_2406_09297_gb300 as mlkv
    lens = np.asarray(lens, dtype=np.int32)
    b, max_seq, l = len(lens), int(lens.max()), len(owner)
    owners = sorted(set(owner))
    with mlkv.MLKVCache(l, h, d, owner, g, b, max_seq) as cache:
        ref = oracle.OracleCache(owner, h, g, d, b, max_seq)
        qb, kn, vn = _inputs(owner, h, g, d, b, lens, max_seq, 91, cache, ref)
        Q, K, V = to_dev(qb), to_dev(kn), to_dev(vn)
        out = torch.empty((l, b, h, d), dtype=torch.bfloat16, device="cuda")
        cache.set_option("step_fused", fused)
        results = []
        for rep in range(3):   # direct, record, replay
            out.fill_(float("nan"))
            cache.decode_step(Q, K, V, out, lens)
            torch.cuda.synchronize()
            results.append(out.clone())
            assert cache.get_option("last_step_kernel") == 1
            assert cache.get_option("last_step_fused") == int(fused > 0 and
                                                               _fused_applies(owner, h, g))
        for r in results[1:]:
            assert torch.equal(r.view(torch.int16), results[0].view(torch.int16))
        for n in range(l):
            if owner[n] == n:
                k = owners.index(n)
                ref.append(n, gen.bf16_bits_to_f64(kn[k]), gen.bf16_bits_to_f64(vn[k]), lens)
            expect = ref.decode(n, gen.bf16_bits_to_f64(qb[n]), lens, nthreads=8)
            mx, mean = errors(from_dev(results[0][n]), expect)
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (n, mx, mean)
        cache.sync_status()


@pytest.mark.parametrize("owner,h,g,d,b,L,kc,units,tiles", FUSED_STEP_CASES)
@pytest.mark.parametrize("deep", [1, 0])
def test_fused_step(owner, h, g, d, b, L, kc, units, tiles, deep):
    # The step in the cross-layer fused form (forced: option step_fused 2): one launch storing
    # every owner's new token, then units of (sequence, KV head, owner block, chunk of the
    # context), each loading every K/V tile of its chunk once for the L * G query rows of its
    # block's layers, the context split only as far as the units fit one per SM (152), and a
    # merge launch when a segment has several chunks.  Every output of every layer against the
    # oracle; the new tokens in the cache; the recorded graph's replay bit for bit.
    import torch

    import paper_2406_09297_gb300 as mlkv
    lens = np.full(b, L, dtype=np.int32)
    l = len(owner)
    owners = sorted(set(owner))
    with mlkv.MLKVCache(l, h, d, owner, g, b, L) as cache:
        ref = oracle.OracleCache(owner, h, g, d, b, L)
        qb, kn, vn = _inputs(owner, h, g, d, b, lens, L, 83, cache, ref)
        Q, K, V = to_dev(qb), to_dev(kn), to_dev(vn)
        out = torch.empty((l, b, h, d), dtype=torch.bfloat16, device="cuda")
        cache.set_option("step_graph", 1)   # direct, record, replay
        cache.set_option("step_fused", 2)   # wherever the map allows it
        # head_dim 64 with the block's rows in one tile: one CTA per SM with a 12-tile ring and two
        # S buffers when the units fit one per SM (deep), else two CTAs per SM
        cache.set_option("fused_deep", deep)
        # the host planner's decision for this device (the table holds the one for 152 SMs)
        sms = cache.get_option("sm_count")
        plan = mlkv.mlkv_plan_step(owner, h, d, g, lens, L, sms, step_fused=2, fused_deep=deep)
        if sms == FUSED_STEP_SMS:
            assert (plan["kc"], plan["units"]) == (kc, units)
        kc, units = plan["kc"], plan["units"]
        assert plan["fused"] == 1 and plan["form"] == (0 if tiles == 2 else 2 if deep and
                                                       units <= sms else 1)
        results = []
        for rep in range(3):
            out.fill_(float("nan"))
            cache.decode_step(Q, K, V, out, lens)
            torch.cuda.synchronize()
            results.append(out.clone())
            assert cache.get_option("last_step_fused") == 1
            assert cache.get_option("last_fused_kc") == kc
            assert cache.get_option("last_grid") == units
            assert cache.get_option("last_deferred_merge") == int(kc < (L + 127) // 128)
            assert cache.get_option("last_step_launches") == 2 + int(kc < (L + 127) // 128)
        assert cache.get_option("step_graph_replays") == 2
        for r in results[1:]:
            assert torch.equal(r.view(torch.int16), results[0].view(torch.int16))
        for n in range(l):
            if owner[n] == n:
                k = owners.index(n)
                ref.append(n, gen.bf16_bits_to_f64(kn[k]), gen.bf16_bits_to_f64(vn[k]), lens)
            expect = ref.decode(n, gen.bf16_bits_to_f64(qb[n]), lens, nthreads=8)
            mx, mean = errors(from_dev(results[0][n]), expect)
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (n, mx, mean)
        from tests.test_gpu_cache import _read_cache
        whole = _read_cache(cache, b, g, L, d)          # int16 [m][2][b][g][L][d]
        for k, n in enumerate(owners):
            assert (whole[cache.owner_slot(n)[1], 0, :, :, L - 1] == kn[k].view(np.int16)).all()
            assert (whole[cache.owner_slot(n)[1], 1, :, :, L - 1] == vn[k].view(np.int16)).all()
        cache.sync_status()


@pytest.mark.parametrize("chunked", [False, True])
def test_fused_step_host_buffers(chunked):
    # mlkv_decode_step_host in the fused form: the store launch lets the fused launch go at once,
    # which fetches cache tiles while the step's inputs are still being copied in and waits before
    # the queries and the newest tile; its results equal the device-buffer step's bit for bit.
    import torch

    import paper_2406_09297_gb300 as mlkv
    owner, h, g, d = [0] * 6 + [6] * 6, 12, 1, 64
    b, L = (1, 20000) if chunked else (16, 1000)
    lens = np.full(b, L, dtype=np.int32)
    l = len(owner)
    with mlkv.MLKVCache(l, h, d, owner, g, b, L) as cache, \
            mlkv.MLKVCache(l, h, d, owner, g, b, L) as cache2:
        ref = oracle.OracleCache(owner, h, g, d, b, L)
        qb, kn, vn = _inputs(owner, h, g, d, b, lens, L, 89, cache, ref)
        _inputs(owner, h, g, d, b, lens, L, 89, cache2, None)
        for c in (cache, cache2):
            c.set_option("step_fused", 2)
        Q, K, V = to_dev(qb), to_dev(kn), to_dev(vn)
        want = torch.empty((l, b, h, d), dtype=torch.bfloat16, device="cuda")
        cache2.decode_step(Q, K, V, want, lens)
        torch.cuda.synchronize()
        hq, hk, hv = Q.cpu().pin_memory(), K.cpu().pin_memory(), V.cpu().pin_memory()
        out = torch.full((l, b, h, d), float("nan"), dtype=torch.bfloat16).pin_memory()
        for _ in range(3):
            out.fill_(float("nan"))
            cache.decode_step_host(hq, hk, hv, out, lens)
            torch.cuda.synchronize()
            assert cache.get_option("last_step_fused") == 1
            assert torch.equal(out.view(torch.int16), want.cpu().view(torch.int16))
        owners = sorted(set(owner))
        for n in range(l):
            if owner[n] == n:
                k = owners.index(n)
                ref.append(n, gen.bf16_bits_to_f64(kn[k]), gen.bf16_bits_to_f64(vn[k]), lens)
            expect = ref.decode(n, gen.bf16_bits_to_f64(qb[n]), lens, nthreads=8)
            mx, mean = errors(out[n].float().numpy().astype(np.float64), expect)
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (n, mx, mean)
        cache.sync_status()
        cache2.sync_status()
