"""Seeded, counter-based synthetic inputs (host side, numpy).

This module holds no attention arithmetic: it only draws the bf16 bit patterns that both the
oracle and the CUDA library consume.  ``mlkv_synth/synth_gpu.cu`` implements the same generator
for the device so that caches of many GiB can be filled in place; a GPU test checks that both
produce identical bits.

Generator
---------
SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014,
with the 64-bit finaliser constants of Vigna's public-domain reference version):

    out(s, n) = mix64(s + (n + 1) * GAMMA)            n-th output of the stream seeded with s

Element (seed, tensor_id, row, col):

    s_tensor = out(seed, tensor_id)
    s_row    = out(s_tensor, row)
    x_k      = out(s_row, 3*col + k),   k = 0, 1, 2
    u_0..u_11 = the four 16-bit fields of x_0, x_1, x_2   (least significant first)
    z        = (sum(u) - 6 * 65536) / 65536               Irwin-Hall(12): mean ~0, variance ~1
    value    = bf16_rne(sigma * z)                        sigma a power of two

All steps up to z are exact (integers below 2**20), so the host and the device agree bit for bit.
|z| <= 6, so no value overflows or is NaN.
"""
import sys

import numpy as np

GAMMA = 0x9E3779B97F4A7C15
MIX1 = 0xBF58476D1CE4E5B9
MIX2 = 0x94D049BB133111EB
MASK64 = (1 << 64) - 1

assert sys.byteorder == "little", "the uint16 view of the 64-bit draws assumes little-endian"

# tensor ids (the device generator uses the same numbers, passed in by the caller)
TID_Q = 0x100      # + layer          rows: beta,          cols: i*d + e
TID_K = 0x200      # + owner layer    rows: beta*g + j,    cols: t*d + e
TID_V = 0x300      # + owner layer    rows: beta*g + j,    cols: t*d + e
TID_LEN = 0x400    #                  output n = beta: sequence length draw
TID_W = 0x500      # + layer          rows: head i,        cols: element of the head's rows


def mix64_int(z):
    """SplitMix64 finaliser on a Python int."""
    z &= MASK64
    z = ((z ^ (z >> 30)) * MIX1) & MASK64
    z = ((z ^ (z >> 27)) * MIX2) & MASK64
    return z ^ (z >> 31)


def out_int(s, n):
    """n-th (0-based) output of the SplitMix64 stream seeded with s (Python ints)."""
    return mix64_int((s + (n + 1) * GAMMA) & MASK64)


def _mix64_np(z):
    z = z ^ (z >> np.uint64(30))
    z = z * np.uint64(MIX1)
    z = z ^ (z >> np.uint64(27))
    z = z * np.uint64(MIX2)
    return z ^ (z >> np.uint64(31))


def row_seed(seed, tensor_id, row):
    return out_int(out_int(seed, tensor_id), row)


def f32_to_bf16_bits(v):
    """Round-to-nearest-even float32 -> bf16 bit pattern (finite inputs)."""
    b = np.ascontiguousarray(v, dtype=np.float32).view(np.uint32)
    r = (b + np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f64(bits):
    """Exact widening of bf16 bit patterns to float64."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def bf16_bits_to_f32(bits):
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32)


_host_lib = None


def _host():
    """The C implementation of this generator (synth_host.c), or None if it cannot be built."""
    global _host_lib
    if _host_lib is None:
        import ctypes
        try:
            from . import build as _b
            L = ctypes.CDLL(_b.build_host())
            L.synth_host_fill_bf16.argtypes = [
                ctypes.c_void_p, ctypes.c_longlong, ctypes.c_longlong, ctypes.c_longlong,
                ctypes.c_void_p, ctypes.c_longlong, ctypes.c_ulonglong, ctypes.c_ulonglong,
                ctypes.c_float]
            _host_lib = L
        except Exception:
            _host_lib = False
    return _host_lib or None


def gen_bf16(seed, tensor_id, rows, ncols, sigma=1.0, col0=0, impl="auto"):
    """bf16 bit patterns [len(rows)][ncols] of the generator at the given row ids and columns
    [col0, col0 + ncols).  impl: "numpy", "c" or "auto" (C when available)."""
    rows = [int(r) for r in np.atleast_1d(rows)]
    host = _host() if impl in ("auto", "c") else None
    if impl == "c" and host is None:
        raise RuntimeError("the C generator is not available")
    if host is not None:
        out = np.empty((len(rows), ncols), dtype=np.uint16)
        ids = np.asarray(rows, dtype=np.int64)
        host.synth_host_fill_bf16(out.ctypes.data, len(rows), ncols, ncols, ids.ctypes.data,
                                  col0, seed, tensor_id, sigma)
        return out
    out = np.empty((len(rows), ncols), dtype=np.uint16)
    k = np.arange(3 * col0, 3 * (col0 + ncols), dtype=np.uint64) + np.uint64(1)
    with np.errstate(over="ignore"):
        step = k * np.uint64(GAMMA)                       # (n + 1) * GAMMA mod 2**64
        for ri, r in enumerate(rows):
            s = np.uint64(row_seed(seed, tensor_id, r))
            x = _mix64_np(step + s)                       # x_k for all columns, [3*ncols]
            u = x.view(np.uint16).reshape(ncols, 12)      # 12 uniforms per element
            ssum = u.sum(axis=1, dtype=np.int32) - np.int32(6 * 65536)
            z = ssum.astype(np.float32) * np.float32(1.0 / 65536.0)
            out[ri] = f32_to_bf16_bits(z * np.float32(sigma))
    return out


def gen_seq_lens(seed, b, max_len):
    """Sequence lengths uniform in [1, max_len]: 1 + out(out(seed, TID_LEN), beta) mod max_len."""
    s = out_int(seed, TID_LEN)
    return np.array([1 + out_int(s, beta) % max_len for beta in range(b)], dtype=np.int32)


def gen_q(seed, layer, b, h, d, sigma=1.0, betas=None):
    """Queries of one layer, bf16 bits [len(betas)][h][d]."""
    betas = range(b) if betas is None else betas
    return gen_bf16(seed, TID_Q + layer, list(betas), h * d, sigma).reshape(-1, h, d)


def gen_kv(seed, owner_layer, kv, b, g, length, d, sigma=1.0, betas=None, heads=None, t0=0):
    """K (kv=0) or V (kv=1) cache content of an owner layer, bf16 bits
    [len(betas)][len(heads)][length][d] for positions [t0, t0 + length)."""
    betas = list(range(b)) if betas is None else list(betas)
    heads = list(range(g)) if heads is None else list(heads)
    rows = [beta * g + j for beta in betas for j in heads]
    tid = (TID_K if kv == 0 else TID_V) + owner_layer
    bits = gen_bf16(seed, tid, rows, length * d, sigma, col0=t0 * d)
    return bits.reshape(len(betas), len(heads), length, d)


def gen_kv_token(seed, owner_layer, kv, b, g, d, seq_lens, sigma=1.0):
    """The new token's K or V for every (beta, j): the generator's value at position L_beta - 1,
    bf16 bits [b][g][d]."""
    out = np.empty((b, g, d), dtype=np.uint16)
    for beta in range(b):
        t = int(seq_lens[beta]) - 1
        out[beta] = gen_kv(seed, owner_layer, kv, b, g, 1, d, sigma, betas=[beta], t0=t)[0, :, 0]
    return out
