"""Bit-exact checks of the cache layout, append placement, owner-only appends, prefix loads, the
device input generator, and the error paths of the GPU entry points."""
import numpy as np
import pytest

import oracle
from mlkv_synth import gen
from tests.mlkv_cases import to_dev

pytestmark = pytest.mark.gpu


class _DevArray:
    """Exposes raw device memory to torch through the CUDA array interface."""

    def __init__(self, ptr, nelem, typestr="<i2"):
        self.__cuda_array_interface__ = {"shape": (nelem,), "typestr": typestr,
                                         "data": (ptr, False), "version": 2, "strides": None}


def _read_cache(cache, b, g, max_seq, d):
    """Copies the whole device cache to the host: int16 [m][2][b][g][max_seq][d]."""
    import torch
    m = cache.num_slots()
    nbytes = cache.cache_bytes()
    assert nbytes == 2 * b * max_seq * m * g * d * 2
    k0, _, _ = cache.kv_ptr(0)
    torch.cuda.synchronize()
    t = torch.as_tensor(_DevArray(k0, nbytes // 2), device="cuda")
    return t.cpu().numpy().reshape(m, 2, b, g, max_seq, d)


def test_cache_bytes_and_slots_follow_the_paper():
    import paper_2406_09297_gb300 as mlkv
    owner = [0, 0, 2, 2, 2, 5]
    b, h, g, d, s = 3, 8, 2, 64, 40
    with mlkv.MLKVCache(len(owner), h, d, owner, g, b, s) as c:
        m, slot = oracle.slots(owner)
        assert c.num_slots() == m
        assert c.cache_bytes() == oracle.cache_elements(b, s, m, g, d) * 2
        for n in range(len(owner)):
            assert c.owner_slot(n) == (owner[n], int(slot[n]))


def test_append_and_prefix_placement_bit_exact():
    import torch

    import paper_2406_09297_gb300 as mlkv
    owner = [0, 0, 2, 3, 3]
    b, h, g, d, s = 3, 4, 2, 64, 37
    lens = np.array([37, 1, 20], dtype=np.int32)
    with mlkv.MLKVCache(len(owner), h, d, owner, g, b, s) as c:
        m, slot = oracle.slots(owner)
        expect = np.zeros((m, 2, b, g, s, d), dtype=np.int16)
        # prefix of length 30 into owner 3 only
        kb = gen.gen_kv(9, 3, 0, b, g, 30, d)
        vb = gen.gen_kv(9, 3, 1, b, g, 30, d)
        c.load_prefix(3, to_dev(kb), to_dev(vb), 30)
        c.load_prefix(1, to_dev(kb), to_dev(vb), 30)      # non-owner: no-op
        expect[slot[3], 0, :, :, :30] = kb.view(np.int16)
        expect[slot[3], 1, :, :, :30] = vb.view(np.int16)
        torch.cuda.synchronize()
        assert np.array_equal(_read_cache(c, b, g, s, d), expect)
        # appends: owners write at L-1, non-owners write nothing
        for n in range(len(owner)):
            kn = gen.gen_bf16(3, gen.TID_K + n, range(b * g), d).reshape(b, g, d)
            vn = gen.gen_bf16(3, gen.TID_V + n, range(b * g), d).reshape(b, g, d)
            before = _read_cache(c, b, g, s, d)
            c.append(n, to_dev(kn), to_dev(vn), lens)
            torch.cuda.synchronize()
            after = _read_cache(c, b, g, s, d)
            if owner[n] != n:
                assert np.array_equal(before, after), f"non-owner layer {n} wrote the cache"
                continue
            for beta in range(b):
                t = lens[beta] - 1
                expect[slot[n], 0, beta, :, t] = kn[beta].view(np.int16)
                expect[slot[n], 1, beta, :, t] = vn[beta].view(np.int16)
            assert np.array_equal(after, expect), f"layer {n}"
        c.sync_status()


def test_device_generator_matches_host_bits():
    import torch

    from mlkv_synth import device
    t = torch.empty((5, 777), dtype=torch.bfloat16, device="cuda")
    device.fill_(t, 1234, 0x305, sigma=0.5, row0=17, col0=3)
    got = t.view(torch.int16).cpu().numpy().view(np.uint16)
    expect = gen.gen_bf16(1234, 0x305, range(17, 22), 777, sigma=0.5, col0=3)
    assert np.array_equal(got, expect)
    # pitched fill into a slot-like layout
    big = torch.zeros((3, 50, 64), dtype=torch.bfloat16, device="cuda")
    device.fill_ptr(big.data_ptr(), 3, 20 * 64, 50 * 64, 77, 0x201, 1.0)
    host = big.view(torch.int16).cpu().numpy().view(np.uint16)
    expect = gen.gen_bf16(77, 0x201, range(3), 20 * 64).reshape(3, 20, 64)
    assert np.array_equal(host[:, :20], expect)
    assert not host[:, 20:].any()


def test_error_paths_do_not_touch_the_device():
    import torch

    import paper_2406_09297_gb300 as mlkv
    b, h, g, d, s = 2, 4, 2, 64, 16
    with mlkv.MLKVCache(2, h, d, [0, 0], g, b, s) as c:
        q = torch.zeros((b, h, d), dtype=torch.bfloat16, device="cuda")
        out = torch.zeros_like(q)
        kv = torch.zeros((b, g, d), dtype=torch.bfloat16, device="cuda")
        for lens in ([0, 3], [3, 17], [-1, 1]):
            with pytest.raises(mlkv.MLKVError) as e:
                c.decode_attention(0, q, out, lens)
            assert e.value.code == mlkv.MLKV_ERR_RANGE
            with pytest.raises(mlkv.MLKVError) as e:
                c.append(0, kv, kv, lens)
            assert e.value.code == mlkv.MLKV_ERR_RANGE
        with pytest.raises(mlkv.MLKVError) as e:
            c.decode_attention(2, q, out, [1, 1])
        assert e.value.code == mlkv.MLKV_ERR_INVALID_ARG
        with pytest.raises(mlkv.MLKVError) as e:
            c.decode_attention(0, q, q, [1, 1])                   # out aliases Q
        assert e.value.code == mlkv.MLKV_ERR_INVALID_ARG
        with pytest.raises(mlkv.MLKVError) as e:
            c.set_option("tile_tokens", 96)
        assert e.value.code == mlkv.MLKV_ERR_INVALID_ARG
        with pytest.raises(mlkv.MLKVError) as e:
            c.load_prefix(0, kv, kv, s + 1)
        assert e.value.code == mlkv.MLKV_ERR_RANGE
        assert c.sync_status() == 0


def test_out_of_memory_is_reported():
    import paper_2406_09297_gb300 as mlkv
    # 2 * 1024 * 2**30 * 1 * 16 * 128 * 2 bytes: far beyond any device
    with pytest.raises(mlkv.MLKVError) as e:
        mlkv.MLKVCache(1, 16, 128, [0], 16, 1024, 1 << 30)
    assert e.value.code in (mlkv.MLKV_ERR_OOM, mlkv.MLKV_ERR_UNSUPPORTED)
