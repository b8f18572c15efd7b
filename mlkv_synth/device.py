"""Device side of the seeded input generator (libmlkv_synth.so), for torch bf16 tensors."""
import ctypes
import os

from . import gen

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmlkv_synth.so")
_lib = None


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is not built")
        L = ctypes.CDLL(LIB_PATH)
        ll = ctypes.c_longlong
        L.synth_fill_bf16.argtypes = [ctypes.c_void_p, ll, ll, ll, ll, ll, ctypes.c_ulonglong,
                                      ctypes.c_ulonglong, ctypes.c_float, ctypes.c_void_p]
        _lib = L
    return _lib


def fill_ptr(ptr, rows, cols, pitch, seed, tensor_id, sigma=1.0, row0=0, col0=0, stream=None):
    """dst[r*pitch + c] = generator(seed, tensor_id, row0 + r, col0 + c) for bf16 dst at ptr."""
    import torch
    s = torch.cuda.current_stream().cuda_stream if stream is None else stream
    rc = lib().synth_fill_bf16(ctypes.c_void_p(ptr), rows, cols, pitch, row0, col0, seed,
                               tensor_id, sigma, ctypes.c_void_p(s))
    if rc != 0:
        raise RuntimeError(f"synth_fill_bf16 failed ({rc})")


def fill_(t, seed, tensor_id, sigma=1.0, row0=0, col0=0):
    """Fills a contiguous bf16 tensor viewed as [rows][cols] (rows = all leading dims)."""
    import torch
    assert t.dtype == torch.bfloat16 and t.is_cuda and t.is_contiguous()
    cols = t.shape[-1]
    rows = t.numel() // cols if cols else 0
    fill_ptr(t.data_ptr(), rows, cols, cols, seed, tensor_id, sigma, row0, col0)
    return t


def q_tensor(seed, layer, b, h, d, sigma=1.0):
    import torch
    t = torch.empty((b, h * d), dtype=torch.bfloat16, device="cuda")
    fill_(t, seed, gen.TID_Q + layer, sigma)
    return t.view(b, h, d)


def kv_token(seed, owner_layer, kv, b, g, d, seq_lens, sigma=1.0):
    """The new token's K (kv=0) or V (kv=1), [b][g][d]: value at position L_beta - 1."""
    import torch
    t = torch.empty((b, g, d), dtype=torch.bfloat16, device="cuda")
    tid = (gen.TID_K if kv == 0 else gen.TID_V) + owner_layer
    lens = [int(x) for x in seq_lens]
    if all(x == lens[0] for x in lens):          # one launch when every sequence has one length
        fill_ptr(t.data_ptr(), b * g, d, d, seed, tid, sigma, row0=0, col0=(lens[0] - 1) * d)
        return t
    for beta in range(b):
        pos = int(seq_lens[beta]) - 1
        fill_ptr(t[beta].data_ptr(), g, d, d, seed, tid, sigma, row0=beta * g, col0=pos * d)
    return t


def fill_slot(k_base, v_base, strides, seed, owner_layer, b, g, d, length, sigma_k=1.0,
              sigma_v=1.0):
    """Writes positions [0, length) of an owner slot in place (cache layout [b][g][max_seq][d],
    strides from mlkv_kv_ptr)."""
    pitch = strides[1]   # elements between consecutive (beta, j) rows
    fill_ptr(k_base, b * g, length * d, pitch, seed, gen.TID_K + owner_layer, sigma_k)
    fill_ptr(v_base, b * g, length * d, pitch, seed, gen.TID_V + owner_layer, sigma_v)


def workload_inputs(w, cache):
    """Device inputs of one decode step of workload `w` on an mlkv cache (the bench's and the
    full-size tests' set-up): every owner slot holds the generator's K/V at positions
    [0, max_seq); Q of every layer; the new token of every owner (the generator's value at L-1,
    so re-appending it is idempotent).  Returns (seq_lens, Q list, K_new dict, V_new dict)."""
    seq_lens = w.seq_lens()
    for n in w.owners():
        slot = cache.owner_slot(n)[1]
        kp, vp, strides = cache.kv_ptr(slot)
        fill_slot(kp, vp, strides, w.seed, n, w.b, w.g, w.d, w.max_seq, w.sigma_k, w.sigma_v)
    Q = [q_tensor(w.seed, n, w.b, w.h, w.d, w.sigma_q) for n in range(w.l)]
    Kn = {n: kv_token(w.seed, n, 0, w.b, w.g, w.d, seq_lens, w.sigma_k) for n in w.owners()}
    Vn = {n: kv_token(w.seed, n, 1, w.b, w.g, w.d, seq_lens, w.sigma_v) for n in w.owners()}
    return seq_lens, Q, Kn, Vn
