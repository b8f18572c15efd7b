"""GPU decode attention against the fp64 oracle on small, fully checked cases.

Sizes span several tiles with ragged tails; the grid option forces segments to be split across
CTAs so that the partial-merge path runs; maps cover MHA, GQA, MQA, MLKV blocks and non-uniform
owner maps; head_dim 64 and 128; every tile variant.
"""
import numpy as np
import pytest

from tests.mlkv_cases import run_small_case

pytestmark = pytest.mark.gpu

TILE_EDGE_LENS = [1, 2, 15, 16, 17, 63, 64, 65, 127, 128, 129, 191, 256, 257, 300]


@pytest.mark.parametrize("d,tile", [(64, 128), (64, 64), (64, 256), (128, 64), (128, 128)])
@pytest.mark.parametrize("fused", [False, True])
def test_tile_edges_single_layer(d, tile, fused):
    b = len(TILE_EDGE_LENS)
    run_small_case([0], 4, 2, d, b, TILE_EDGE_LENS, 300, seed=11, options={"tile_tokens": tile},
                   fused=fused)


# The tcgen05 kernel (option "tc"): 128- and 256-position tiles, both head sizes, ragged lengths,
# split segments (stream-K records, inline and deferred merges) and DSMEM clusters.
@pytest.mark.parametrize("d,tile", [(64, 128), (64, 256), (128, 128)])
@pytest.mark.parametrize("fused", [False, True])
def test_tc_tile_edges(d, tile, fused):
    b = len(TILE_EDGE_LENS)
    run_small_case([0], 4, 2, d, b, TILE_EDGE_LENS, 300, seed=21,
                   options={"tile_tokens": tile, "tc": 1}, fused=fused, expect={"last_tc": 1})


@pytest.mark.parametrize("grid", [3, 7, 64, 600])
def test_tc_split_merges(grid):
    lens = [700, 1, 129, 1000]
    run_small_case([0, 0], 16, 1, 64, len(lens), lens, 1024, seed=22,
                   options={"grid": grid, "tile_tokens": 128, "tc": 1}, fused=True,
                   expect={"last_tc": 1})


@pytest.mark.parametrize("name,owner,h,g,d", [
    ("mha", [0, 1, 2], 4, 4, 64), ("gqa-mlkv", [0, 0, 0, 3, 3, 3], 12, 4, 64),
    ("mqa-g16", [0, 1], 16, 1, 128), ("non-uniform", [0, 0, 0, 3, 4, 4], 8, 2, 128)])
def test_tc_maps(name, owner, h, g, d):
    lens = [5, 130, 77, 260]
    run_small_case(owner, h, g, d, len(lens), lens, 320, seed=23,
                   options={"tc": 1, "tile_tokens": 128}, expect={"last_tc": 1})


def test_tc_cluster_merge():
    run_small_case([0, 0, 2], 12, 1, 64, 64, [2048] * 64, 2048, seed=24, fused=True,
                   options={"tc": 1}, expect={"last_tc": 1, "last_cluster_k": 2})


@pytest.mark.parametrize("lens", [[2048] * 4, [512, 1, 77, 2048], [600] * 3])
def test_default_tile_choice(lens):
    # the default tile length depends on the mean length; both choices are checked
    run_small_case([0, 0, 2], 12, 1, 64, len(lens), lens, 2048, seed=14, fused=True)


@pytest.mark.parametrize("grid", [1, 2, 3, 7, 64, 200, 600])
@pytest.mark.parametrize("fused", [False, True])
def test_split_merge_paths(grid, fused):
    # Many CTAs over few tiles: segments split across up to hundreds of CTAs (the largest grids
    # exceed the shared-memory merge capacity and take the fallback merge).
    lens = [700, 1, 129, 1000]
    run_small_case([0, 0], 16, 1, 64, len(lens), lens, 1024, seed=12,
                   options={"grid": grid, "tile_tokens": 64}, fused=fused)


@pytest.mark.parametrize("name,owner,h,g", [
    ("mha", [0, 1, 2], 4, 4),
    ("gqa", [0, 1, 2], 12, 4),
    ("mqa-g12", [0, 1], 12, 1),
    ("mqa-g16", [0, 1], 16, 1),
    ("mlkv-pairs", [0, 0, 2, 2], 12, 1),
    ("mlkv-1", [0, 0, 0, 0], 12, 1),
    ("gqa-mlkv", [0, 0, 0, 3, 3, 3], 12, 4),
    ("non-uniform", [0, 0, 0, 3, 4, 4], 8, 2),
    ("g8", [0, 0], 16, 2),
])
@pytest.mark.parametrize("d", [64, 128])
def test_maps(name, owner, h, g, d):
    lens = [5, 130, 77, 260]
    run_small_case(owner, h, g, d, len(lens), lens, 320, seed=13)


def test_random_fuzz():
    rng = np.random.default_rng(2024)
    for trial in range(12):
        l = int(rng.integers(1, 7))
        owner = []
        for n in range(l):
            o = int(rng.integers(0, n + 1))
            owner.append(o if (o == n or owner[o] == o) else n)
        h = int(rng.choice([1, 2, 3, 4, 6, 8, 12, 16]))
        divs = [x for x in range(1, h + 1) if h % x == 0]
        g = int(rng.choice(divs))
        d = int(rng.choice([64, 128]))
        b = int(rng.integers(1, 6))
        max_seq = int(rng.choice([1, 7, 64, 129, 333]))
        lens = rng.integers(1, max_seq + 1, size=b)
        opts = {"grid": int(rng.choice([0, 1, 5, 50]))}
        run_small_case(owner, h, g, d, b, lens, max_seq, seed=100 + trial, options=opts,
                       fused=bool(trial % 2))


def test_config1_full():
    from mlkv_synth import workloads
    w = workloads.config(1)
    run_small_case(w.owner, w.h, w.g, w.d, w.b, w.seq_lens(), w.max_seq, seed=w.seed)


def test_non_finite_cache_contents_beyond_length_do_not_leak():
    """Positions >= L of the cache may hold anything (here NaN); outputs stay finite."""
    import torch

    import paper_2406_09297_gb300 as mlkv
    from tests.mlkv_cases import errors, from_dev, to_dev
    import oracle
    from mlkv_synth import gen

    b, g, h, d, max_seq = 2, 1, 4, 64, 200
    lens = np.array([70, 3], dtype=np.int32)
    with mlkv.MLKVCache(1, h, d, [0], g, b, max_seq) as cache:
        kb = gen.gen_kv(5, 0, 0, b, g, max_seq, d)
        vb = gen.gen_kv(5, 0, 1, b, g, max_seq, d)
        kd, vd = to_dev(kb), to_dev(vb)
        kd[:, :, 100:] = float("nan")
        vd[:, :, 100:] = float("nan")
        kd[1, :, 3:] = float("inf")
        vd[1, :, 3:] = float("nan")
        cache.load_prefix(0, kd, vd, max_seq)
        qb = gen.gen_q(5, 0, b, h, d)
        out = torch.empty((b, h, d), dtype=torch.bfloat16, device="cuda")
        cache.decode_attention(0, to_dev(qb), out, lens)
        ref = oracle.OracleCache([0], h, g, d, b, max_seq)
        ref.load_prefix(0, gen.bf16_bits_to_f64(kb), gen.bf16_bits_to_f64(vb), max_seq)
        expect = ref.decode(0, gen.bf16_bits_to_f64(qb), lens)
        got = from_dev(out)
        assert np.isfinite(got).all()
        mx, mean = errors(got, expect)
        assert mx <= 2e-2 and mean <= 2e-3
        cache.sync_status()


@pytest.mark.parametrize("d", [64, 128])
def test_merge_of_hundreds_of_pieces(d):
    # one segment of 313 tiles over 313 CTAs: the decode launch writes partials only and the
    # combine kernel merges them
    run_small_case([0], 16, 1, d, 1, [20000], 20000, seed=15,
                   options={"grid": 600, "tile_tokens": 64}, expect={"last_deferred_merge": 1})
    run_small_case([0], 16, 1, d, 1, [20000], 20000, seed=16,
                   options={"grid": 600, "tile_tokens": 64}, fused=True,
                   expect={"last_deferred_merge": 1})


def test_long_single_segments_default_launch():
    # batch 2 x 2 KV heads of 30000 positions: four segments over the whole GPU
    run_small_case([0, 0], 8, 2, 64, 2, [30000, 29999], 30000, seed=19, fused=True,
                   expect={"last_deferred_merge": 1})


def test_few_pieces_merge_inline():
    run_small_case([0], 8, 2, 64, 4, [700, 1, 129, 1000], 1024, seed=20,
                   options={"grid": 3, "tile_tokens": 64}, expect={"last_deferred_merge": 0})


@pytest.mark.parametrize("b,L,tile,k,want_tile", [(64, 2048, 256, 2, 256), (64, 2048, 0, 4, 128),
                                                   (32, 2048, 0, 4, 128), (64, 256, 64, 4, 64)])
@pytest.mark.parametrize("fused", [False, True])
def test_cluster_merge(b, L, tile, k, want_tile, fused):
    # One length for every sequence, layer calls one by one.  64 segments of 8 tiles of 256: 2-CTA
    # clusters keep the one-wave makespan; by default 64 segments of 16 tiles of 128 (two CTAs per
    # SM): 4-CTA clusters; 32 such segments: 4-CTA clusters; 64 segments of 4 tiles of 64: 4-CTA
    # clusters.  The pieces of a segment are merged through DSMEM.
    opts = {"tile_tokens": tile} if tile else None
    run_small_case([0, 0, 2], 12, 1, 64, b, [L] * b, L, seed=17, fused=fused, options=opts,
                   expect={"last_cluster_k": k, "last_tile_tokens": want_tile})


def test_cluster_mode_off_matches():
    run_small_case([0, 0], 12, 1, 64, 64, [2048] * 64, 2048, seed=18,
                   options={"cluster": 0}, expect={"last_cluster_k": 0})


@pytest.mark.parametrize("k", [2, 4])
def test_cluster_size_forced(k):
    # The "cluster" option may name the cluster size: 2-CTA clusters of 8 tiles of 128 each (half
    # the CTAs of the default shape), or 4-CTA clusters.
    run_small_case([0, 0, 2], 12, 1, 64, 64, [2048] * 64, 2048, seed=21,
                   options={"cluster": k}, expect={"last_cluster_k": k, "last_tile_tokens": 128})


def test_cluster_rule_keeps_a_streaming_grid():
    # One long segment on the two-CTA-per-SM tile: a cluster of its pieces would be a grid of a
    # few CTAs, so the stream-K split over the SMs (and the separate merge) is kept.
    run_small_case([0, 0], 8, 1, 64, 1, [8192], 8192, seed=22, options={"tile_tokens": 128},
                   expect={"last_cluster_k": 0, "last_deferred_merge": 1})
