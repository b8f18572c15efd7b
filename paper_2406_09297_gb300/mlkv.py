"""Thin Python binding of libmlkv (include/mlkv.h): argument marshalling only.

Every function has the name of the C entry point it calls and the same argument order; torch
tensors stand in for device pointers and the stream defaults to torch's current stream.  No step
of the decode path runs in Python: every call goes to the CUDA library, and importing this module
fails loudly when the library is missing.
"""
import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmlkv.so")

MLKV_OK = 0
MLKV_ERR_INVALID_ARG = -1
MLKV_ERR_MAP = -2
MLKV_ERR_RANGE = -3
MLKV_ERR_OOM = -4
MLKV_ERR_CUDA = -5
MLKV_ERR_UNSUPPORTED = -6
MLKV_ERR_DEVICE = -7
MLKV_MAX_BATCH = 1024
MLKV_MAX_GROUP = 16

EXPORTED = [
    "mlkv_cache_create", "mlkv_cache_destroy", "mlkv_append", "mlkv_decode_attention",
    "mlkv_append_decode_attention", "mlkv_decode_step",
    "mlkv_load_prefix", "mlkv_cache_bytes", "mlkv_num_slots", "mlkv_owner_slot", "mlkv_kv_ptr",
    "mlkv_set_option", "mlkv_get_option", "mlkv_sync_status", "mlkv_last_error",
    "mlkv_block_owner_map", "mlkv_version", "mlkv_decode_attention_static", "mlkv_prefill",
    "mlkv_merge_kv_weights", "mlkv_decode_block_fused", "mlkv_decode_step_host",
    "mlkv_static_status", "mlkv_read_bandwidth_probe", "mlkv_plan_step",
]


class MLKVError(RuntimeError):
    def __init__(self, code, message):
        super().__init__(f"[{code}] {message}")
        self.code = code


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(
            f"{LIB_PATH} is not built; run `python -c 'import __graft_entry__ as g; g.build()'`")
    L = ctypes.CDLL(LIB_PATH)
    vp, ip, i64 = ctypes.c_void_p, ctypes.POINTER(ctypes.c_int), ctypes.c_int64
    ci = ctypes.c_int
    L.mlkv_cache_create.argtypes = [ctypes.POINTER(vp), ci, ci, ci, ip, ci, ci, ci]
    L.mlkv_cache_destroy.argtypes = [vp]
    L.mlkv_append.argtypes = [vp, ci, vp, vp, ip, vp]
    L.mlkv_decode_attention.argtypes = [vp, ci, vp, vp, ip, vp]
    L.mlkv_append_decode_attention.argtypes = [vp, ci, vp, vp, vp, vp, ip, vp]
    L.mlkv_decode_step.argtypes = [vp, vp, vp, vp, vp, ip, vp]
    L.mlkv_decode_step_host.argtypes = [vp, vp, vp, vp, vp, ip, vp]
    L.mlkv_load_prefix.argtypes = [vp, ci, vp, vp, ci, vp]
    L.mlkv_cache_bytes.argtypes = [vp]
    L.mlkv_cache_bytes.restype = i64
    L.mlkv_num_slots.argtypes = [vp]
    L.mlkv_owner_slot.argtypes = [vp, ci, ip, ip]
    L.mlkv_kv_ptr.argtypes = [vp, ci, ctypes.POINTER(vp), ctypes.POINTER(vp),
                              ctypes.POINTER(i64)]
    L.mlkv_set_option.argtypes = [vp, ctypes.c_char_p, i64]
    L.mlkv_get_option.argtypes = [vp, ctypes.c_char_p, ctypes.POINTER(i64)]
    L.mlkv_sync_status.argtypes = [vp]
    L.mlkv_last_error.argtypes = []
    L.mlkv_last_error.restype = ctypes.c_char_p
    L.mlkv_block_owner_map.argtypes = [ci, ci, ip]
    L.mlkv_version.argtypes = []
    L.mlkv_decode_attention_static.argtypes = [vp, ci, ci, ci, ci, ci, vp, vp, ip, vp]
    L.mlkv_static_status.argtypes = [vp]
    L.mlkv_read_bandwidth_probe.argtypes = [vp, i64, ci, ctypes.POINTER(i64), vp]
    L.mlkv_prefill.argtypes = [vp, ci, vp, vp, vp, vp, ip, ci, vp]
    L.mlkv_merge_kv_weights.argtypes = [ip, ci, ci, ci, i64, vp, vp, vp]
    L.mlkv_decode_block_fused.argtypes = [vp, ci, vp, vp, ip, vp]
    L.mlkv_plan_step.argtypes = [ci, ci, ci, ip, ci, ci, ci, ip, ci, ci, ci, ci,
                                 ctypes.POINTER(i64)]
    return L


lib = _load()


def _check(rc):
    if rc < 0:
        raise MLKVError(rc, lib.mlkv_last_error().decode())
    return rc


def _stream(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr(t):
    return ctypes.c_void_p(0 if t is None else t.data_ptr())


def as_seq_lens(seq_lens):
    """int32 contiguous host array (keep it to avoid a conversion on every call)."""
    a = np.ascontiguousarray(np.asarray(seq_lens, dtype=np.int32))
    return a


def _lens_ptr(seq_lens):
    a = seq_lens if (isinstance(seq_lens, np.ndarray) and seq_lens.dtype == np.int32
                     and seq_lens.flags.c_contiguous) else as_seq_lens(seq_lens)
    return a, a.ctypes.data_as(ctypes.POINTER(ctypes.c_int))


def mlkv_cache_create(n_layers, n_q_heads, head_dim, layer_owner, kv_heads_per_owner, batch,
                      max_seq):
    owner = np.ascontiguousarray(np.asarray(layer_owner, dtype=np.int32))
    if len(owner) != n_layers:
        raise MLKVError(MLKV_ERR_INVALID_ARG, "layer_owner must have n_layers entries")
    h = ctypes.c_void_p()
    _check(lib.mlkv_cache_create(ctypes.byref(h), n_layers, n_q_heads, head_dim,
                                 owner.ctypes.data_as(ctypes.POINTER(ctypes.c_int)),
                                 kv_heads_per_owner, batch, max_seq))
    return h


def mlkv_cache_destroy(handle):
    return _check(lib.mlkv_cache_destroy(handle))


def mlkv_append(handle, layer, K, V, seq_lens, stream=None):
    a, p = _lens_ptr(seq_lens)
    return _check(lib.mlkv_append(handle, layer, _ptr(K), _ptr(V), p, _stream(stream)))


def mlkv_decode_attention(handle, layer, Q, out, seq_lens, stream=None):
    a, p = _lens_ptr(seq_lens)
    return _check(lib.mlkv_decode_attention(handle, layer, _ptr(Q), _ptr(out), p,
                                            _stream(stream)))


def mlkv_append_decode_attention(handle, layer, K, V, Q, out, seq_lens, stream=None):
    a, p = _lens_ptr(seq_lens)
    return _check(lib.mlkv_append_decode_attention(handle, layer, _ptr(K), _ptr(V), _ptr(Q),
                                                   _ptr(out), p, _stream(stream)))


def mlkv_decode_step(handle, Q, K, V, out, seq_lens, stream=None):
    a, p = _lens_ptr(seq_lens)
    return _check(lib.mlkv_decode_step(handle, _ptr(Q), _ptr(K), _ptr(V), _ptr(out), p,
                                       _stream(stream)))


def mlkv_decode_step_host(handle, Q, K, V, out, seq_lens, stream=None):
    """mlkv_decode_step with Q, K, V and out in host memory (page-locked for the graph replay)."""
    a, p = _lens_ptr(seq_lens)
    return _check(lib.mlkv_decode_step_host(handle, _ptr(Q), _ptr(K), _ptr(V), _ptr(out), p,
                                            _stream(stream)))


def mlkv_prefill(handle, layer, Q, K, V, out, prompt_lens, s_max, stream=None):
    a, p = _lens_ptr(prompt_lens)
    return _check(lib.mlkv_prefill(handle, layer, _ptr(Q), _ptr(K), _ptr(V), _ptr(out), p, s_max,
                                   _stream(stream)))


def mlkv_load_prefix(handle, layer, K, V, length, stream=None):
    return _check(lib.mlkv_load_prefix(handle, layer, _ptr(K), _ptr(V), length, _stream(stream)))


def mlkv_cache_bytes(handle):
    return _check(lib.mlkv_cache_bytes(handle))


def mlkv_num_slots(handle):
    return _check(lib.mlkv_num_slots(handle))


def mlkv_owner_slot(handle, layer):
    o, s = ctypes.c_int(), ctypes.c_int()
    _check(lib.mlkv_owner_slot(handle, layer, ctypes.byref(o), ctypes.byref(s)))
    return o.value, s.value


def mlkv_kv_ptr(handle, slot):
    k, v = ctypes.c_void_p(), ctypes.c_void_p()
    st = (ctypes.c_int64 * 4)()
    _check(lib.mlkv_kv_ptr(handle, slot, ctypes.byref(k), ctypes.byref(v), st))
    return k.value, v.value, tuple(st)


def mlkv_set_option(handle, key, value):
    return _check(lib.mlkv_set_option(handle, key.encode(), int(value)))


def mlkv_get_option(handle, key):
    v = ctypes.c_int64()
    _check(lib.mlkv_get_option(handle, key.encode(), ctypes.byref(v)))
    return v.value


def mlkv_sync_status(handle):
    return _check(lib.mlkv_sync_status(handle))


def mlkv_last_error():
    return lib.mlkv_last_error().decode()


def mlkv_block_owner_map(n_layers, n_owners):
    out = np.zeros(n_layers, dtype=np.int32)
    _check(lib.mlkv_block_owner_map(n_layers, n_owners,
                                    out.ctypes.data_as(ctypes.POINTER(ctypes.c_int))))
    return out


def mlkv_version():
    return lib.mlkv_version()


def mlkv_plan_step(layer_owner, n_q_heads, head_dim, kv_heads_per_owner, seq_lens, max_seq,
                   sm_count, step_fused=-1, fused_kc=-1, fused_deep=-1):
    """The form mlkv_decode_step takes (no GPU needed): dict of fused (0/1), form (-1, 0, 1, 2),
    kc (key tiles of 128 positions per unit) and units of the fused launch."""
    owner = np.ascontiguousarray(np.asarray(layer_owner, dtype=np.int32))
    a, p = _lens_ptr(seq_lens)
    plan = (ctypes.c_int64 * 4)()
    _check(lib.mlkv_plan_step(len(owner), n_q_heads, head_dim,
                              owner.ctypes.data_as(ctypes.POINTER(ctypes.c_int)),
                              kv_heads_per_owner, len(a), max_seq, p, sm_count, step_fused,
                              fused_kc, fused_deep, plan))
    return {"fused": int(plan[0]), "form": int(plan[1]), "kc": int(plan[2]),
            "units": int(plan[3])}


def mlkv_decode_attention_static(kv_slot, batch, n_q_heads, kv_heads, head_dim, max_seq, Q, out,
                                 seq_lens, stream=None):
    """kv_slot: device address (int) of a [2][batch][kv_heads][max_seq][head_dim] bf16 block."""
    a, p = _lens_ptr(seq_lens)
    return _check(lib.mlkv_decode_attention_static(
        ctypes.c_void_p(kv_slot), batch, n_q_heads, kv_heads, head_dim, max_seq, _ptr(Q),
        _ptr(out), p, _stream(stream)))


def mlkv_read_bandwidth_probe(buf, reps, stream=None):
    """Queues the read-bandwidth probe over the device tensor buf; returns the bytes it reads."""
    n = ctypes.c_int64(0)
    _check(lib.mlkv_read_bandwidth_probe(_ptr(buf), buf.numel() * buf.element_size(), reps,
                                         ctypes.byref(n), _stream(stream)))
    return n.value


def mlkv_static_status(stream=None):
    """Error record of mlkv_decode_attention_static on the current device (waits for stream)."""
    return _check(lib.mlkv_static_status(_stream(stream)))


def mlkv_decode_block_fused(handle, owner_layer, Q, out, seq_lens, stream=None):
    """Every layer of one owner block in one launch (benchmark only; Q, out [L][b][h][d])."""
    a, p = _lens_ptr(seq_lens)
    return _check(lib.mlkv_decode_block_fused(handle, owner_layer, _ptr(Q), _ptr(out), p,
                                              _stream(stream)))


def mlkv_merge_kv_weights(layer_owner, n_q_heads, n_kv_heads, W, out, stream=None):
    """Sec. 4.2 merge of one projection: W bf16 [l][h][row] -> out bf16 [m][g][row] (device)."""
    owner = np.ascontiguousarray(np.asarray(layer_owner, dtype=np.int32))
    row = W.numel() // (len(owner) * n_q_heads) if W is not None else 0
    return _check(lib.mlkv_merge_kv_weights(
        owner.ctypes.data_as(ctypes.POINTER(ctypes.c_int)), len(owner), n_q_heads, n_kv_heads,
        row, _ptr(W), _ptr(out), _stream(stream)))


class MLKVCache:
    """Owning wrapper around an mlkv_cache_t handle."""

    def __init__(self, n_layers, n_q_heads, head_dim, layer_owner, kv_heads_per_owner, batch,
                 max_seq):
        self.l, self.h, self.d = n_layers, n_q_heads, head_dim
        self.owner = [int(o) for o in layer_owner]
        self.g, self.b, self.max_seq = kv_heads_per_owner, batch, max_seq
        self.handle = mlkv_cache_create(n_layers, n_q_heads, head_dim, layer_owner,
                                        kv_heads_per_owner, batch, max_seq)

    def close(self):
        if self.handle is not None:
            mlkv_cache_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def append(self, layer, K, V, seq_lens, stream=None):
        return mlkv_append(self.handle, layer, K, V, seq_lens, stream)

    def decode_attention(self, layer, Q, out, seq_lens, stream=None):
        return mlkv_decode_attention(self.handle, layer, Q, out, seq_lens, stream)

    def append_decode_attention(self, layer, K, V, Q, out, seq_lens, stream=None):
        return mlkv_append_decode_attention(self.handle, layer, K, V, Q, out, seq_lens, stream)

    def decode_step(self, Q, K, V, out, seq_lens, stream=None):
        return mlkv_decode_step(self.handle, Q, K, V, out, seq_lens, stream)

    def prefill(self, layer, Q, K, V, out, prompt_lens, stream=None):
        """Causal prefill of one layer; Q / out [b][s_max][h][d], K / V [b][g][s_max][d]."""
        return mlkv_prefill(self.handle, layer, Q, K, V, out, prompt_lens, int(Q.shape[1]), stream)

    def decode_step_host(self, Q, K, V, out, seq_lens, stream=None):
        return mlkv_decode_step_host(self.handle, Q, K, V, out, seq_lens, stream)

    def decode_block_fused(self, owner_layer, Q, out, seq_lens, stream=None):
        return mlkv_decode_block_fused(self.handle, owner_layer, Q, out, seq_lens, stream)

    def load_prefix(self, layer, K, V, length, stream=None):
        return mlkv_load_prefix(self.handle, layer, K, V, length, stream)

    def cache_bytes(self):
        return mlkv_cache_bytes(self.handle)

    def num_slots(self):
        return mlkv_num_slots(self.handle)

    def owner_slot(self, layer):
        return mlkv_owner_slot(self.handle, layer)

    def kv_ptr(self, slot):
        return mlkv_kv_ptr(self.handle, slot)

    def set_option(self, key, value):
        return mlkv_set_option(self.handle, key, value)

    def get_option(self, key):
        return mlkv_get_option(self.handle, key)

    def sync_status(self):
        return mlkv_sync_status(self.handle)
