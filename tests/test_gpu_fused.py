"""GPU cross-layer fused decode (mlkv_decode_block_fused) against the oracle's per-layer decode.

Every layer of an owner block is decoded in one launch that reads each K/V tile once.  It is not
a step of sequential decoding (a model never has all the block's queries at once); its outputs
must equal, layer by layer, the decode attention of Eqs. 2-3 over the owner's slot.
"""
import numpy as np
import pytest

import oracle
from mlkv_synth import gen
from tests.mlkv_cases import MAX_ABS, MEAN_ABS, errors, from_dev, to_dev

pytestmark = pytest.mark.gpu


def _run(owner, h, g, d, lens, max_seq, seed):
    import torch

    import paper_2406_09297_gb300 as mlkv
    l, b = len(owner), len(lens)
    lens = np.asarray(lens, dtype=np.int32)
    worst = (0.0, 0.0)
    with mlkv.MLKVCache(l, h, d, owner, g, b, max_seq) as cache:
        ref = oracle.OracleCache(owner, h, g, d, b, max_seq)
        for o in sorted(set(owner)):
            kb = gen.gen_kv(seed, o, 0, b, g, max_seq, d)
            vb = gen.gen_kv(seed, o, 1, b, g, max_seq, d)
            cache.load_prefix(o, to_dev(kb), to_dev(vb), max_seq)
            ref.load_prefix(o, gen.bf16_bits_to_f64(kb), gen.bf16_bits_to_f64(vb), max_seq)
        qb = [gen.gen_q(seed + 1, n, b, h, d) for n in range(l)]
        for o in sorted(set(owner)):
            block = [n for n in range(l) if owner[n] == o]
            Q = to_dev(np.stack([qb[n] for n in block]))
            out = torch.full((len(block), b, h, d), float("nan"), dtype=torch.bfloat16,
                             device="cuda")
            cache.decode_block_fused(o, Q, out, lens)
            torch.cuda.synchronize()
            got = from_dev(out)
            for k, n in enumerate(block):
                expect = ref.decode(n, gen.bf16_bits_to_f64(qb[n]), lens)
                mx, mean = errors(got[k], expect)
                assert mx <= MAX_ABS and mean <= MEAN_ABS, (o, n, mx, mean)
                worst = (max(worst[0], mx), max(worst[1], mean))
        cache.sync_status()
    return worst


LENS = [1, 127, 128, 129, 700, 1000]


@pytest.mark.parametrize("name,owner,h,g,d", [
    ("mlkv-2 (G 12, 6 layers: one tile of 72 rows)", [0] * 6 + [6] * 6, 12, 1, 64),
    ("mlkv-1 (G 12, 12 layers: tiles of 120 and 24 rows)", [0] * 12, 12, 1, 64),
    ("gqa-4 mlkv-4 (G 3, blocks of 3)", [0, 0, 0, 3, 3, 3], 12, 4, 64),
    ("mha identity (one row a tile)", [0, 1], 4, 4, 64),
    ("llama-shaped (d 128, G 4, blocks of 4)", [0, 0, 0, 0, 4, 4, 4, 4], 32, 8, 128),
    ("non-uniform blocks", [0, 0, 2, 2, 2, 5], 8, 2, 128),
    ("d 128, two tiles (G 16: 8 + 4 layers)", [0] * 12, 16, 1, 128),
])
def test_fused_equals_per_layer_decode(name, owner, h, g, d):
    _run(owner, h, g, d, LENS, 1000, 71)


def test_fused_long_context():
    _run([0] * 6, 12, 1, 64, [4096, 3000], 4096, 72)


def test_fused_rejects_bad_arguments():
    import torch

    import paper_2406_09297_gb300 as mlkv
    with mlkv.MLKVCache(2, 4, 64, [0, 0], 1, 2, 256) as cache:
        q = torch.zeros((2, 2, 4, 64), dtype=torch.bfloat16, device="cuda")
        out = torch.zeros_like(q)
        with pytest.raises(mlkv.MLKVError) as e:
            cache.decode_block_fused(1, q, out, [5, 5])        # layer 1 is not an owner
        assert e.value.code == mlkv.MLKV_ERR_INVALID_ARG
        for lens in ([0, 5], [257, 5]):
            with pytest.raises(mlkv.MLKVError) as e:
                cache.decode_block_fused(0, q, out, lens)
            assert e.value.code == mlkv.MLKV_ERR_RANGE
        with pytest.raises(mlkv.MLKVError) as e:
            cache.decode_block_fused(0, q, q, [5, 5])          # out overlapping Q
        assert e.value.code == mlkv.MLKV_ERR_INVALID_ARG
    # 17 layers of 16 heads per KV head: more than two tiles of whole layers
    with mlkv.MLKVCache(17, 16, 64, [0] * 17, 1, 1, 128) as cache:
        q = torch.zeros((17, 1, 16, 64), dtype=torch.bfloat16, device="cuda")
        out = torch.zeros_like(q)
        with pytest.raises(mlkv.MLKVError) as e:
            cache.decode_block_fused(0, q, out, [5])
        assert e.value.code == mlkv.MLKV_ERR_UNSUPPORTED


def test_fused_unsplit_context():
    # b * g >= 152 (SMs): one unit per (sequence, KV head), no merge of context chunks.
    rng = np.random.default_rng(73)
    lens = list(rng.integers(1, 600, 40))
    _run([0, 0, 0], 8, 4, 64, lens, 600, 73)
