"""GPU KV-weight merge (mlkv_merge_kv_weights, Sec. 4.2) against the oracle, bit for bit.

The oracle averages in float64 (exact sums for these inputs) and rounds to bf16 to nearest, ties
to even; the kernel carries its sums as pairs of floats.  They must agree on every element except
where the exact mean lies within 2^-30 (relative) of a bf16 rounding boundary -- none of the seeded
inputs comes that close, and the constructed ties below are decided exactly.
"""
import numpy as np
import pytest

import oracle
from mlkv_synth import gen
from tests.mlkv_cases import to_dev

pytestmark = pytest.mark.gpu


def _weights(seed, l, h, row, col0=0):
    return np.stack([gen.gen_bf16(seed, gen.TID_W + n, range(h), row, col0=col0) for n in range(l)])


def _bits_of(t):
    import torch
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def _near_boundary(mean, rel=2.0 ** -30):
    """True where mean lies within rel of a midpoint between adjacent bf16 values."""
    a = np.abs(mean)
    e = np.floor(np.log2(np.where(a > 0, a, 1.0)))
    q = 2.0 ** np.maximum(e - 7, -133)          # bf16 quantum at mean
    frac = a / q - np.floor(a / q)
    return np.abs(frac - 0.5) * q <= rel * a


def _check(owner, h, g, W_bits, got_bits):
    mean = oracle.merge_kv(owner, h, g, gen.bf16_bits_to_f64(W_bits))
    want = oracle.bf16_rne(mean)
    bad = got_bits != want
    assert not (bad & ~_near_boundary(mean)).any(), (
        int(bad.sum()), np.argwhere(bad)[:5].tolist())


def _merge(owner, h, g, W_bits):
    import torch
    import paper_2406_09297_gb300 as mlkv
    l, _, row = W_bits.shape
    m = len(set(owner))
    W = to_dev(W_bits)
    out = torch.full((m, g, row), float("nan"), dtype=torch.bfloat16, device="cuda")
    mlkv.mlkv_merge_kv_weights(owner, h, g, W, out)
    torch.cuda.synchronize()
    return _bits_of(out)


@pytest.mark.parametrize("name,owner,h,g", [
    ("mlkv-2 of 12 (Table 2)", [0] * 6 + [6] * 6, 12, 1),
    ("mlkv-12 (Table 2)", [0, 0, 0, 3, 3, 3, 6, 6, 6, 9, 9, 9], 12, 3),
    ("gqa-4 (identity map)", list(range(4)), 12, 4),
    ("mqa (identity map)", list(range(3)), 8, 1),
    ("non-uniform blocks", [0, 0, 0, 3, 4, 4, 4], 8, 2),
    ("mha identity", list(range(3)), 4, 4),
    ("16 members a head", [0, 0], 8, 1),        # small rows: members split over 2 slices
    ("32 members a head", [0, 0, 0, 0], 8, 1),  # over 4 slices
])
@pytest.mark.parametrize("row", [8, 64, 8 * 1001, 64 * 768])
def test_merge_matches_oracle(name, owner, h, g, row):
    W = _weights(61 + row, len(owner), h, row)
    _check(owner, h, g, W, _merge(owner, h, g, W))


def test_identity_map_copies_bits():
    W = _weights(62, 3, 6, 256)
    np.testing.assert_array_equal(_merge([0, 1, 2], 6, 6, W), W)


def _bf16(x):
    return oracle.bf16_rne(np.asarray(x, dtype=np.float64))


def test_constructed_ties():
    # Four heads per group, one layer; each row of 8 columns holds a tie or a near-tie.
    one, up1, up2 = 1.0, 1.0 + 2.0 ** -7, 1.0 + 2.0 ** -6
    cols = [
        ([one, up1, 0.0, 0.0], 0x3F00),                   # mean 0.5 + 2^-9: exact tie, to even 0.5
        ([up1, up2, 0.0, 0.0], 0x3F02),                   # 0.5 + 3 2^-9: tie, up to even
        ([one, up1, 2.0 ** -30, 0.0], 0x3F01),            # a hair above the tie: up
        ([one, up1, -(2.0 ** -30), 0.0], 0x3F00),         # a hair below: down
        ([-one, -up1, 0.0, 0.0], 0xBF00),                 # negative tie, to even
        ([-one, -up1, -(2.0 ** -30), 0.0], 0xBF01),       # negative, past the tie in magnitude
        ([2.0 ** -126, 2.0 ** -126, 2.0 ** -126, 0.0], 0x0060),   # 0.75 2^-126: a subnormal
        ([3.0e37, 2.0e37, -1.0e37, 4.0e37], None),        # large (sums stay below float's max)
    ]
    W = np.zeros((1, 4, 8), dtype=np.uint16)
    for c, (vals, _) in enumerate(cols):
        W[0, :, c] = _bf16(vals)
    got = _merge([0], 4, 1, W)[0, 0]
    for c, (vals, want) in enumerate(cols):
        exact = np.mean(gen.bf16_bits_to_f64(W[0, :, c]))
        if want is None:
            want = int(_bf16([exact])[0])
        assert int(got[c]) == want, (c, hex(int(got[c])), hex(want))


def test_llama7b_shapes_sampled_columns():
    # Llama-2-7B: 32 layers x 32 heads, head rows 128 x 4096 (1 GiB of K weights), MLKV-8 GQA-4
    # (blocks of 4 layers, g = 8).  The whole tensor goes through the kernel; the oracle checks
    # 8 windows of 64 columns of every merged head (a merge is column-wise).
    import torch
    import paper_2406_09297_gb300 as mlkv
    from mlkv_synth import device
    l, h, g, row, seed = 32, 32, 8, 128 * 4096, 63
    owner = [4 * (n // 4) for n in range(l)]
    W = torch.empty((l, h, row), dtype=torch.bfloat16, device="cuda")
    for n in range(l):
        device.fill_(W[n], seed, gen.TID_W + n)
    out = torch.empty((l // 4, g, row), dtype=torch.bfloat16, device="cuda")
    mlkv.mlkv_merge_kv_weights(owner, h, g, W, out)
    torch.cuda.synchronize()
    got = _bits_of(out)
    rng = np.random.default_rng(64)
    for c0 in sorted(rng.choice(row // 64, 8, replace=False) * 64):
        Wc = _weights(seed, l, h, 64, col0=int(c0))
        np.testing.assert_array_equal(_bits_of(W[:, :, c0:c0 + 64]), Wc)   # same inputs
        _check(owner, h, g, Wc, got[:, :, c0:c0 + 64])


def test_rejects_bad_arguments():
    import torch
    import paper_2406_09297_gb300 as mlkv
    W = torch.zeros((2, 4, 64), dtype=torch.bfloat16, device="cuda")
    out = torch.zeros((1, 2, 64), dtype=torch.bfloat16, device="cuda")
    cases = [
        (([0, 0], 4, 3, W, out), mlkv.MLKV_ERR_MAP),          # g does not divide h
        (([0, 2], 4, 2, W, out), mlkv.MLKV_ERR_MAP),          # owner after the layer
        (([1, 1], 4, 2, W, out), mlkv.MLKV_ERR_MAP),          # owner that does not own itself
        (([0, 0], 4, 2, None, out), mlkv.MLKV_ERR_INVALID_ARG),
        (([0, 0], 4, 2, W, W), mlkv.MLKV_ERR_INVALID_ARG),    # output overlaps input
    ]
    for args, code in cases:
        with pytest.raises(mlkv.MLKVError) as e:
            mlkv.mlkv_merge_kv_weights(*args)
        assert e.value.code == code, args
    Wodd = torch.zeros((2, 4, 12), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(mlkv.MLKVError) as e:                   # 12 elements: not a multiple of 8
        mlkv.mlkv_merge_kv_weights([0, 0], 4, 2, Wodd, out)
    assert e.value.code == mlkv.MLKV_ERR_INVALID_ARG


def test_k_and_v_in_one_call():
    """K and V of a model merged by one call, stacked as 2 l layers with V's layers owned by
    owner + l (the benchmark's form): the output is K's merged heads then V's, bit for bit those
    of one call per projection, and both agree with the oracle."""
    owner, h, g, row = [0] * 6 + [6] * 6, 12, 1, 64 * 768
    l = len(owner)
    Wk = _weights(31, l, h, row)
    Wv = _weights(32, l, h, row)
    both = _merge(owner + [o + l for o in owner], h, g, np.concatenate([Wk, Wv]))
    m = len(set(owner))
    assert np.array_equal(both[:m], _merge(owner, h, g, Wk))
    assert np.array_equal(both[m:], _merge(owner, h, g, Wv))
    _check(owner, h, g, Wk, both[:m])
    _check(owner, h, g, Wv, both[m:])
