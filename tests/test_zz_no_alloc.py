"""mlkv_decode_attention_static: the decode entry point for callers that cannot allocate device
memory (a runtime whose allocator owns all device memory, or a serving loop that must not call
cudaMalloc while it runs).  It keeps its merge scratch in an array compiled into the library.

Each case calls it twice in a row through the C ABI and compares every output with the regular
entry point's (mlkv_decode_attention) on the same inputs, within the parity tolerance of the other
GPU tests, and reads the static error record (mlkv_static_status) after each call.  This file is
named to be collected last.
"""
import numpy as np
import pytest

from mlkv_synth import gen
from tests.mlkv_cases import MAX_ABS, MEAN_ABS, errors, from_dev, to_dev

pytestmark = pytest.mark.gpu


def _check_two_calls(owner, h, g, d, b, lens, max_seq, seed):
    import torch

    import paper_2406_09297_gb300 as mlkv
    lens = np.asarray(lens, dtype=np.int32)
    with mlkv.MLKVCache(len(owner), h, d, owner, g, b, max_seq) as cache:
        for n in sorted(set(owner)):
            kb = gen.gen_kv(seed, n, 0, b, g, max_seq, d)
            vb = gen.gen_kv(seed, n, 1, b, g, max_seq, d)
            cache.load_prefix(n, to_dev(kb), to_dev(vb), max_seq)
        for n in range(len(owner)):          # two calls in a row, one per layer
            q = to_dev(gen.gen_q(seed, n, b, h, d))
            ref = torch.full((b, h, d), float("nan"), dtype=torch.bfloat16, device="cuda")
            got = torch.full_like(ref, float("nan"))
            cache.decode_attention(n, q, ref, lens)
            slot = cache.owner_slot(n)[1]
            k_base, v_base, _ = cache.kv_ptr(slot)
            assert v_base == k_base + b * g * max_seq * d * 2    # [2][b][g][max_seq][d] block
            mlkv.mlkv_decode_attention_static(k_base, b, h, g, d, max_seq, q, got, lens)
            torch.cuda.synchronize()
            r, s = from_dev(ref), from_dev(got)
            assert np.isfinite(s).all()
            mx, mean = errors(s, r)
            assert mx <= MAX_ABS and mean <= MEAN_ABS, (n, mx, mean)
            # no bounded wait expired in the static kernels (their error word lives in the
            # static array; reading it allocates nothing either)
            assert mlkv.mlkv_static_status() == mlkv.MLKV_OK
        cache.sync_status()


def test_static_entry_matches_regular_varied_lengths():
    # varied lengths, segments split across CTAs: the partial-merge scratch is exercised
    _check_two_calls([0, 0], 12, 2, 64, 6, [1, 300, 1000, 77, 2048, 513], 2048, seed=21)


def test_static_entry_matches_regular_uniform_d128():
    _check_two_calls([0, 0], 32, 8, 128, 4, [1500] * 4, 1500, seed=22)


def test_static_entry_rejects_requests_beyond_its_scratch():
    import torch

    import paper_2406_09297_gb300 as mlkv
    slot = torch.zeros((2, 1024, 16, 1, 128), dtype=torch.bfloat16, device="cuda")
    q = torch.zeros((1024, 16, 128), dtype=torch.bfloat16, device="cuda")
    out = torch.zeros_like(q)
    lens = np.ones(1024, dtype=np.int32)
    # 1024 sequences x 16 KV heads x (128 + 1) floats: more records than the 8 MiB scratch holds
    with pytest.raises(mlkv.MLKVError) as e:
        mlkv.mlkv_decode_attention_static(slot.data_ptr(), 1024, 16, 16, 128, 1, q, out, lens)
    assert e.value.code == mlkv.MLKV_ERR_UNSUPPORTED
    assert "SCRATCH" in mlkv.mlkv_last_error()


def test_static_entry_rejects_out_overlapping_q():
    import torch

    import paper_2406_09297_gb300 as mlkv
    b, h, g, d, max_seq = 2, 12, 1, 64, 128
    slot = torch.zeros((2, b, g, max_seq, d), dtype=torch.bfloat16, device="cuda")
    buf = torch.zeros((2 * b * h * d,), dtype=torch.bfloat16, device="cuda")
    lens = np.full(b, 16, dtype=np.int32)
    with pytest.raises(mlkv.MLKVError) as e:   # out starts inside Q
        mlkv.mlkv_decode_attention_static(slot.data_ptr(), b, h, g, d, max_seq, buf,
                                          buf[b * h * d // 2:], lens)
    assert e.value.code == mlkv.MLKV_ERR_INVALID_ARG
    assert "overlap" in mlkv.mlkv_last_error()
    assert mlkv.mlkv_static_status() == mlkv.MLKV_OK
