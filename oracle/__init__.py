"""MLKV decode-attention oracle: numpy-facing wrapper of oracle/mlkv_oracle.c.

TEST INFRASTRUCTURE ONLY.  Only the test suite, ``__graft_entry__.smoke()`` and bench.py's
CPU-baseline / reference legs may import this package.  It shares no code with the CUDA library in
``paper_2406_09297_gb300`` and never imports it; the library never imports this package.

All arrays are float64.  Inputs the GPU receives as bf16 are widened exactly to float64 before
they reach the oracle (see ``mlkv_synth.gen.bf16_bits_to_f64``).
"""
import ctypes
import os

import numpy as np

from . import build as _build

_lib = None

ORACLE_OK = 0
ORACLE_ERR_ARG = -1
ORACLE_ERR_MAP = -2
ORACLE_ERR_RANGE = -3
ORACLE_ERR_OOM = -4

_ip = ctypes.POINTER(ctypes.c_int)
_dp = ctypes.POINTER(ctypes.c_double)


def load(path):
    """Opens an oracle shared library at ``path`` and declares its signatures."""
    L = ctypes.CDLL(path)
    L.oracle_block_owner_map.argtypes = [ctypes.c_int, ctypes.c_int, _ip]
    L.oracle_kv_head_of.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int]
    L.oracle_validate.argtypes = [ctypes.c_int, _ip, ctypes.c_int, ctypes.c_int, ctypes.c_int]
    L.oracle_slots.argtypes = [ctypes.c_int, _ip, _ip]
    L.oracle_cache_elements.argtypes = [ctypes.c_longlong] * 5
    L.oracle_cache_elements.restype = ctypes.c_longlong
    L.oracle_decode_layer.argtypes = [
        ctypes.c_int, ctypes.c_int, _ip, ctypes.c_int, ctypes.c_int, ctypes.c_int,
        ctypes.c_int, _ip, ctypes.c_int, _dp, ctypes.POINTER(_dp), ctypes.POINTER(_dp), _dp,
        ctypes.c_int]
    L.oracle_prefill_layer.argtypes = [
        ctypes.c_int, ctypes.c_int, _ip, ctypes.c_int, ctypes.c_int, ctypes.c_int,
        ctypes.c_int, _ip, ctypes.c_int, ctypes.c_int, _dp, ctypes.POINTER(_dp),
        ctypes.POINTER(_dp), _dp, ctypes.c_int]
    L.oracle_append.argtypes = [
        ctypes.c_int, ctypes.c_int, _ip, ctypes.c_int, ctypes.c_int, ctypes.c_int, _ip,
        ctypes.c_int, _dp, _dp, ctypes.POINTER(_dp), ctypes.POINTER(_dp)]
    L.oracle_merge_kv.argtypes = [ctypes.c_int, _ip, ctypes.c_int, ctypes.c_int, ctypes.c_longlong,
                                  _dp, _dp]
    L.oracle_bf16_rne.argtypes = [ctypes.c_double]
    L.oracle_bf16_rne.restype = ctypes.c_uint
    L.oracle_bf16_rne_array.argtypes = [_dp, ctypes.c_longlong, ctypes.POINTER(ctypes.c_uint16)]
    return L


def lib():
    """Loads (building first if needed) the oracle shared library."""
    global _lib
    if _lib is None:
        _lib = load(_build.build())
    return _lib


def _ints(a):
    a = np.ascontiguousarray(np.asarray(a, dtype=np.int32))
    return a, a.ctypes.data_as(_ip)


def _f64(a):
    a = np.ascontiguousarray(a, dtype=np.float64)
    return a, a.ctypes.data_as(_dp)


def block_owner_map(l, m):
    """Eq. 18 block map (0-based owners); raises ValueError if m does not divide l."""
    owner = np.zeros(l, dtype=np.int32)
    rc = lib().oracle_block_owner_map(l, m, owner.ctypes.data_as(_ip))
    if rc != ORACLE_OK:
        raise ValueError(f"block map undefined for l={l}, m={m}")
    return owner


def kv_head_of(h, g, i):
    """Eq. 12 group map, 0-based."""
    return lib().oracle_kv_head_of(h, g, i)


def validate(owner, h, g, d=64):
    """Returns 0 or a negative oracle error code for a layer->owner map and head counts."""
    owner, op = _ints(owner)
    return lib().oracle_validate(len(owner), op, h, g, d)


def slots(owner):
    """Returns (m, slot[]) for a layer->owner map (slot = rank of the owner among owners)."""
    owner, op = _ints(owner)
    slot = np.full(len(owner), -1, dtype=np.int32)
    m = lib().oracle_slots(len(owner), op, slot.ctypes.data_as(_ip))
    return m, slot


def cache_elements(b, s, m, g, dk):
    """Sec. 3 / Table 1 cache element count 2*b*s*m*g*d_k."""
    return lib().oracle_cache_elements(b, s, m, g, dk)


class OracleCache:
    """Owner-indexed host KV cache in float64 plus the per-layer decode of Sec. 3.

    ``K[n]`` / ``V[n]`` exist only for layers n that own themselves; shape [b][g][max_seq][d].
    """

    def __init__(self, owner, h, g, d, b, max_seq):
        self.owner = np.ascontiguousarray(np.asarray(owner, dtype=np.int32))
        self.l = len(self.owner)
        self.h, self.g, self.d, self.b, self.max_seq = h, g, d, b, max_seq
        rc = validate(self.owner, h, g, d)
        if rc != ORACLE_OK:
            raise ValueError(f"invalid MLKV map (oracle code {rc})")
        self.K = {}
        self.V = {}
        for n in range(self.l):
            if self.owner[n] == n:
                self.K[n] = np.zeros((b, g, max_seq, d), dtype=np.float64)
                self.V[n] = np.zeros((b, g, max_seq, d), dtype=np.float64)

    def _ptr_arrays(self):
        karr = (_dp * self.l)()
        varr = (_dp * self.l)()
        for n in range(self.l):
            if n in self.K:
                karr[n] = self.K[n].ctypes.data_as(_dp)
                varr[n] = self.V[n].ctypes.data_as(_dp)
        return karr, varr

    def load_prefix(self, layer, K, V, length):
        """Stores positions [0, length) of an owner layer's K/V ([b][g][length][d]); no-op for a
        non-owner layer."""
        if self.owner[layer] != layer:
            return 0
        self.K[layer][:, :, :length, :] = K
        self.V[layer][:, :, :length, :] = V
        return 1

    def append(self, layer, K_new, V_new, seq_lens):
        """Sec. 3 append: owner layers store the new token at position seq_lens-1."""
        sl, sp = _ints(seq_lens)
        K_new, kp = _f64(K_new)
        V_new, vp = _f64(V_new)
        karr, varr = self._ptr_arrays()
        rc = lib().oracle_append(layer, self.l, self.owner.ctypes.data_as(_ip), self.g, self.d,
                                 self.b, sp, self.max_seq, kp, vp, karr, varr)
        if rc < 0:
            raise ValueError(f"oracle_append failed ({rc})")
        return rc

    def decode(self, layer, Q, seq_lens, nthreads=1):
        """Per-layer decode attention; Q [b][h][d] -> out [b][h][d]."""
        sl, sp = _ints(seq_lens)
        Q, qp = _f64(Q)
        out = np.zeros((self.b, self.h, self.d), dtype=np.float64)
        karr, varr = self._ptr_arrays()
        rc = lib().oracle_decode_layer(layer, self.l, self.owner.ctypes.data_as(_ip), self.h,
                                       self.g, self.d, self.b, sp, self.max_seq, qp, karr, varr,
                                       out.ctypes.data_as(_dp), nthreads)
        if rc != ORACLE_OK:
            raise ValueError(f"oracle_decode_layer failed ({rc})")
        return out


    def prefill(self, layer, Q, prompt_lens, nthreads=1):
        """Causal prefill of one layer; Q [b][s_max][h][d] -> out [b][s_max][h][d] (rows past a
        prompt's length stay zero).  The owner's cache must hold the prompt's K/V."""
        pl, pp = _ints(prompt_lens)
        Q, qp = _f64(Q)
        b, s_max, h, d = Q.shape
        assert b == self.b and h == self.h and d == self.d
        out = np.zeros((b, s_max, h, d), dtype=np.float64)
        karr, varr = self._ptr_arrays()
        rc = lib().oracle_prefill_layer(layer, self.l, self.owner.ctypes.data_as(_ip), self.h,
                                        self.g, self.d, self.b, pp, s_max, self.max_seq, qp,
                                        karr, varr, out.ctypes.data_as(_dp), nthreads)
        if rc != ORACLE_OK:
            raise ValueError(f"oracle_prefill_layer failed ({rc})")
        return out


def decode_layer(layer, owner, h, g, d, seq_lens, Q, K_owner, V_owner, nthreads=1):
    """Decode of one layer when only the owner's cache is at hand.

    K_owner / V_owner: [b][g][max_seq][d] caches of layer owner[layer]; Q: [b][h][d].
    """
    owner = np.ascontiguousarray(np.asarray(owner, dtype=np.int32))
    l = len(owner)
    K_owner, kp = _f64(K_owner)
    V_owner, vp = _f64(V_owner)
    b, g_, max_seq, d_ = K_owner.shape
    assert g_ == g and d_ == d
    sl, sp = _ints(seq_lens)
    Q, qp = _f64(Q)
    karr = (_dp * l)()
    varr = (_dp * l)()
    karr[int(owner[layer])] = kp
    varr[int(owner[layer])] = vp
    out = np.zeros((b, h, d), dtype=np.float64)
    rc = lib().oracle_decode_layer(layer, l, owner.ctypes.data_as(_ip), h, g, d, b, sp, max_seq,
                                   qp, karr, varr, out.ctypes.data_as(_dp), nthreads)
    if rc != ORACLE_OK:
        raise ValueError(f"oracle_decode_layer failed ({rc})")
    return out


def merge_kv(owner, h, g, W):
    """Sec. 4.2 KV-weight merge: W [l][h][row] float64 -> [m][g][row] float64 means (owner order)."""
    owner, op = _ints(owner)
    W, wp = _f64(W)
    l, h_, row = W.shape
    assert h_ == h and l == len(owner)
    m, _ = slots(owner)
    if m < 1:
        raise ValueError(f"invalid owner map ({m})")
    out = np.zeros((m, g, row), dtype=np.float64)
    rc = lib().oracle_merge_kv(l, op, h, g, row, wp, out.ctypes.data_as(_dp))
    if rc != ORACLE_OK:
        raise ValueError(f"oracle_merge_kv failed ({rc})")
    return out


def bf16_rne(x):
    """Round-to-nearest-even of float64 values to bfloat16; returns the uint16 bit patterns."""
    x, xp = _f64(x)
    out = np.zeros(x.shape, dtype=np.uint16)
    lib().oracle_bf16_rne_array(xp, x.size, out.ctypes.data_as(ctypes.POINTER(ctypes.c_uint16)))
    return out
