"""The C ABI library loads, exports every entry point of include/mlkv.h, and rejects invalid
requests on the host before touching the device (no GPU needed)."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
import paper_2406_09297_gb300 as mlkv

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared(header):
    text = open(os.path.join(ROOT, "include", header)).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mlkv_[a-z_0-9]+)\s*\(", text)))


def test_every_declared_symbol_is_exported():
    names = _declared("mlkv.h")
    assert "mlkv_decode_attention" in names and "mlkv_append" in names
    lib = ctypes.CDLL(mlkv.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(mlkv.EXPORTED) == names


def test_block_owner_map_matches_oracle():
    for l in (1, 2, 6, 12, 24, 32):
        for m in range(1, l + 1):
            if l % m:
                with pytest.raises(mlkv.MLKVError) as e:
                    mlkv.mlkv_block_owner_map(l, m)
                assert e.value.code == mlkv.MLKV_ERR_MAP
            else:
                assert np.array_equal(mlkv.mlkv_block_owner_map(l, m),
                                      oracle.block_owner_map(l, m))


@pytest.mark.parametrize("args,code", [
    ((3, 4, 64, [0, 2, 2], 2, 1, 16), mlkv.MLKV_ERR_MAP),      # owner after its layer
    ((3, 4, 64, [0, 0, 1], 2, 1, 16), mlkv.MLKV_ERR_MAP),      # owner not self-owned
    ((3, 6, 64, [0, 0, 0], 4, 1, 16), mlkv.MLKV_ERR_MAP),      # g does not divide h
    ((3, 4, 64, [0, 0, 0], 8, 1, 16), mlkv.MLKV_ERR_MAP),      # g > h
    ((3, 4, 96, [0, 0, 0], 2, 1, 16), mlkv.MLKV_ERR_UNSUPPORTED),   # head_dim
    ((2, 64, 64, [0, 0], 2, 1, 16), mlkv.MLKV_ERR_UNSUPPORTED),     # group of 32 > 16
    ((2, 4, 64, [0, 0], 2, 2000, 16), mlkv.MLKV_ERR_UNSUPPORTED),   # batch above the limit
    ((0, 4, 64, [], 2, 1, 16), mlkv.MLKV_ERR_INVALID_ARG),
    ((2, 4, 64, [0, 0], 2, 0, 16), mlkv.MLKV_ERR_INVALID_ARG),
    ((2, 4, 64, [0, 0], 2, 1, 0), mlkv.MLKV_ERR_INVALID_ARG),
])
def test_create_rejects_invalid_layouts(args, code):
    with pytest.raises(mlkv.MLKVError) as e:
        mlkv.mlkv_cache_create(*args)
    assert e.value.code == code
    assert mlkv.mlkv_last_error()


def test_null_handle_calls_fail_cleanly():
    null = ctypes.c_void_p(0)
    lens = np.ones(1, dtype=np.int32)
    for fn, args in [
        (mlkv.lib.mlkv_decode_attention, (null, 0, None, None,
                                          lens.ctypes.data_as(ctypes.POINTER(ctypes.c_int)),
                                          None)),
        (mlkv.lib.mlkv_append, (null, 0, None, None,
                                lens.ctypes.data_as(ctypes.POINTER(ctypes.c_int)), None)),
        (mlkv.lib.mlkv_num_slots, (null,)),
        (mlkv.lib.mlkv_sync_status, (null,)),
        (mlkv.lib.mlkv_set_option, (null, b"grid", 1)),
    ]:
        assert fn(*args) == mlkv.MLKV_ERR_INVALID_ARG
    assert mlkv.lib.mlkv_cache_destroy(null) == mlkv.MLKV_OK


def test_validation_agrees_with_oracle_on_random_maps():
    """Map validation of the library and of the oracle accept and reject the same layouts.  A
    valid layout goes on to the device: without a GPU that fails with MLKV_ERR_CUDA, with one
    the tiny cache is created and destroyed again."""
    rng = np.random.default_rng(0)
    for _ in range(300):
        l = int(rng.integers(1, 7))
        owner = [int(rng.integers(0, n + 1)) for n in range(l)]
        if rng.random() < 0.7:   # bias toward valid maps: redirect to self-owned owners
            owner = [o if owner[o] == o else n for n, o in enumerate(owner)]
        h = int(rng.choice([1, 2, 3, 4, 6, 8, 12]))
        g = int(rng.integers(1, h + 1))
        handle = ctypes.c_void_p()
        code = mlkv.lib.mlkv_cache_create(ctypes.byref(handle), l, h, 64,
                                          np.asarray(owner, dtype=np.int32).ctypes.data_as(
                                              ctypes.POINTER(ctypes.c_int)), g, 1, 8)
        if code == mlkv.MLKV_OK:
            mlkv.lib.mlkv_cache_destroy(handle)
        if oracle.validate(owner, h, g, 64) == 0:
            assert code in (mlkv.MLKV_OK, mlkv.MLKV_ERR_CUDA), (owner, h, g, code)
        else:
            assert code == mlkv.MLKV_ERR_MAP, (owner, h, g, code)
