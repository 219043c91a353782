"""numpy wrapper of the C oracle (layer_math.c) -- TEST INFRASTRUCTURE ONLY.

Arrays in, arrays out. Activations are bit patterns: uint16 for bf16/fp16, uint32 for
fp32. Every function returns fresh arrays and leaves its inputs unchanged. The layer
chain at the bottom is the composition of the single-step oracles, as its definition
states (add+RMSNorm, RoPE+KV append, add+RMSNorm on the rounded residual, SwiGLU).
"""
import ctypes
import os

import numpy as np

from . import build_oracle

BF16, FP16, FP32 = 1, 2, 3

_lib = None
_parallel = False


def set_parallel(parallel):
    """Use the OpenMP build of the C oracle (all host cores; same values) from now on, or
    the serial default again. For timing the oracle only."""
    global _lib, _parallel
    if bool(parallel) != _parallel:
        _parallel = bool(parallel)
        _lib = None


def threads():
    """Threads the C oracle's loops run on (1 for the serial build)."""
    return int(lib().orc_threads())


def lib():
    global _lib
    if _lib is None:
        path = build_oracle.build(parallel=_parallel)
        L = ctypes.CDLL(path)
        L.orc_threads.restype = ctypes.c_int
        L.orc_threads.argtypes = []
        P = ctypes.c_void_p
        i64, c_int, dbl = ctypes.c_int64, ctypes.c_int, ctypes.c_double
        L.orc_widen.restype = dbl
        L.orc_widen.argtypes = [ctypes.c_uint32, c_int]
        L.orc_round.restype = ctypes.c_uint32
        L.orc_round.argtypes = [dbl, c_int]
        L.orc_add_rmsnorm.restype = None
        L.orc_add_rmsnorm.argtypes = [i64, i64, c_int, P, P, P, dbl, P, P, P]
        L.orc_rmsnorm.restype = None
        L.orc_rmsnorm.argtypes = [i64, i64, c_int, P, P, dbl, P, P]
        L.orc_rms_scale.restype = None
        L.orc_rms_scale.argtypes = [i64, P, P, dbl]
        L.orc_rope_apply.restype = None
        L.orc_rope_apply.argtypes = [i64, P, i64, dbl]
        L.orc_rope_kv.restype = c_int
        L.orc_rope_kv.argtypes = [i64, i64, i64, i64, i64, c_int, dbl, c_int, P, P, dbl,
                                  P, P, P, P, P, P, P, P]
        for name, nin in (("orc_silu", 1), ("orc_neg", 1), ("orc_add", 2)):
            f = getattr(L, name)
            f.restype = None
            f.argtypes = [i64, c_int] + [P] * nin + [P, P]
        L.orc_masked_fill.restype = None
        L.orc_masked_fill.argtypes = [i64, c_int, P, P, dbl, P, P]
        L.orc_swiglu.restype = None
        L.orc_swiglu.argtypes = [i64, c_int, P, P, P, P]
        _lib = L
    return _lib


def _bits_dtype(dtype):
    return np.uint32 if dtype == FP32 else np.uint16


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def _p(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def widen(bits, dtype):
    """Exact value of each bit pattern, as float64."""
    b = np.asarray(bits)
    L = lib()
    flat = b.reshape(-1)
    out = np.empty(flat.shape, np.float64)
    for i, v in enumerate(flat):
        out[i] = L.orc_widen(int(v), dtype)
    return out.reshape(b.shape)


def round_bits(values, dtype):
    """Round-to-nearest-even bit patterns of float64 values in `dtype`."""
    v = np.asarray(values, np.float64)
    L = lib()
    flat = v.reshape(-1)
    out = np.empty(flat.shape, _bits_dtype(dtype))
    for i, x in enumerate(flat):
        out[i] = L.orc_round(float(x), dtype)
    return out.reshape(v.shape)


def add_rmsnorm(x, r, gamma, eps, dtype):
    """x, r: [T,H] bits; gamma: [H] float32. Returns (y_ref f64, y bits, r_out bits)."""
    bd = _bits_dtype(dtype)
    x, r = _c(x, bd), _c(r, bd)
    gamma = _c(gamma, np.float32)
    T, H = x.shape
    y_ref = np.empty((T, H), np.float64)
    y = np.empty((T, H), bd)
    r_out = np.empty((T, H), bd)
    lib().orc_add_rmsnorm(T, H, dtype, _p(x), _p(r), _p(gamma), float(eps), _p(y_ref), _p(y),
                          _p(r_out))
    return y_ref, y, r_out


def rmsnorm(x, gamma, eps, dtype):
    """x: [T,H] bits; gamma: [H] float32. Returns (y_ref f64, y bits)."""
    bd = _bits_dtype(dtype)
    x = _c(x, bd)
    gamma = _c(gamma, np.float32)
    T, H = x.shape
    y_ref = np.empty((T, H), np.float64)
    y = np.empty((T, H), bd)
    lib().orc_rmsnorm(T, H, dtype, _p(x), _p(gamma), float(eps), _p(y_ref), _p(y))
    return y_ref, y


def rms_scale(x, gamma, eps):
    """One vector x (float64) RMS-normalised and scaled by gamma (float32), in fp64."""
    x = np.array(x, np.float64)
    gamma = _c(gamma, np.float32)
    lib().orc_rms_scale(x.shape[0], _p(x), _p(gamma), float(eps))
    return x


def rope_apply(x, pos, theta):
    """One head vector x (float64, length D) rotated at `pos`, in fp64."""
    x = np.array(x, np.float64)
    lib().orc_rope_apply(x.shape[0], _p(x), int(pos), float(theta))
    return x


def rope_kv(q, k, v, pos, k_cache, v_cache, theta, dtype, qknorm=False, gamma_q=None,
            gamma_k=None, eps=1e-6):
    """q [T,Hq,D], k/v [T,Hkv,D] bits; pos [T] int32; caches [Hkv,S,D] bits.
    Returns dict(q, q_ref, k_ref, k_cache, v_cache, bad)."""
    bd = _bits_dtype(dtype)
    q = np.array(q, bd)  # copy: rotated in place
    k, v = _c(k, bd), _c(v, bd)
    pos = _c(pos, np.int32)
    kc, vc = np.array(k_cache, bd), np.array(v_cache, bd)
    T, Hq, D = q.shape
    Hkv = k.shape[1]
    S = kc.shape[1]
    q_ref = np.empty(q.shape, np.float64)
    k_ref = np.empty(k.shape, np.float64)
    gq = _c(gamma_q if gamma_q is not None else np.ones(D), np.float32)
    gk = _c(gamma_k if gamma_k is not None else np.ones(D), np.float32)
    bad = lib().orc_rope_kv(T, Hq, Hkv, D, S, dtype, float(theta), 1 if qknorm else 0, _p(gq),
                            _p(gk), float(eps), _p(q), _p(q_ref), _p(k), _p(v), _p(pos), _p(kc),
                            _p(vc), _p(k_ref))
    if bad < 0:
        raise ValueError("head_dim too large for the oracle")
    return dict(q=q, q_ref=q_ref, k_ref=k_ref, k_cache=kc, v_cache=vc, bad=bad)


def _pointwise(name, dtype, *arrays):
    bd = _bits_dtype(dtype)
    arrs = [_c(a, bd) for a in arrays]
    ref = np.empty(arrs[0].shape, np.float64)
    out = np.empty(arrs[0].shape, bd)
    getattr(lib(), name)(arrs[0].size, dtype, *[_p(a) for a in arrs], _p(ref), _p(out))
    return ref, out


def silu(x, dtype):
    """Returns (ref f64, out bits) of x / (1 + exp(-x))."""
    return _pointwise("orc_silu", dtype, x)


def neg(x, dtype):
    return _pointwise("orc_neg", dtype, x)


def add(a, b, dtype):
    """a + b summed in fp32, then rounded to dtype."""
    return _pointwise("orc_add", dtype, a, b)


def masked_fill(x, mask, value, dtype):
    """mask != 0 -> value (rounded once to dtype), else x."""
    bd = _bits_dtype(dtype)
    x = _c(x, bd)
    m = _c(mask, np.uint8)
    ref = np.empty(x.shape, np.float64)
    out = np.empty(x.shape, bd)
    lib().orc_masked_fill(x.size, dtype, _p(x), _p(m), float(value), _p(ref), _p(out))
    return ref, out


def swiglu(g, u, dtype):
    """g, u: bits of equal shape. Returns (ref f64, out bits)."""
    bd = _bits_dtype(dtype)
    g, u = _c(g, bd), _c(u, bd)
    ref = np.empty(g.shape, np.float64)
    out = np.empty(g.shape, bd)
    lib().orc_swiglu(g.size, dtype, _p(g), _p(u), _p(ref), _p(out))
    return ref, out


def layer_chain(inp, theta, eps, dtype, qknorm=False):
    """One decoder layer's non-GEMM chain as the composition of the step oracles.
    inp: dict with h, r0, gamma_attn, q, k, v, pos, k_cache, v_cache, attn_out,
    gamma_mlp, g, u (and gamma_q, gamma_k when qknorm). Returns every output."""
    x1_ref, x1, r1 = add_rmsnorm(inp["h"], inp["r0"], inp["gamma_attn"], eps, dtype)
    rk = rope_kv(inp["q"], inp["k"], inp["v"], inp["pos"], inp["k_cache"], inp["v_cache"],
                 theta, dtype, qknorm=qknorm, gamma_q=inp.get("gamma_q"),
                 gamma_k=inp.get("gamma_k"), eps=eps)
    x2_ref, x2, r2 = add_rmsnorm(inp["attn_out"], r1, inp["gamma_mlp"], eps, dtype)
    o_ref, o = swiglu(inp["g"], inp["u"], dtype)
    return dict(x1_ref=x1_ref, x1=x1, r1=r1, q=rk["q"], q_ref=rk["q_ref"], k_ref=rk["k_ref"],
                k_cache=rk["k_cache"], v_cache=rk["v_cache"], bad=rk["bad"], x2_ref=x2_ref,
                x2=x2, r2=r2, o_ref=o_ref, o=o)
