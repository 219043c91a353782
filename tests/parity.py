"""Comparison helpers for GPU-vs-oracle parity tests.

Tolerances: bf16/fp16 outputs |got - ref| <= 1e-2 + 1.6e-2 |ref| against the oracle's
unrounded fp64 value, and additionally within one unit in the last place of the oracle's
own round-to-nearest-even result. fp32 outputs |got - ref| <= 1e-5 |ref| + 1e-5 rms(row).
Bit-copied data (v into the cache, untouched cache slots) must match exactly.
"""
import numpy as np
import torch

from paper_2609_37241_gb300 import synth

BF16, FP16, FP32 = 1, 2, 3


def widen_bits(bits, dtype):
    return synth.bits_to_torch(bits, dtype).double().numpy()


def ordered(bits, dtype):
    """Map bit patterns to integers whose difference counts representable steps."""
    b = np.asarray(bits).astype(np.int64)
    if dtype == FP32:
        sign, mag = (b >> 31) & 1, b & 0x7FFFFFFF
    else:
        sign, mag = (b >> 15) & 1, b & 0x7FFF
    return np.where(sign == 1, -mag, mag)


def ulp_diff(a_bits, b_bits, dtype):
    return np.abs(ordered(a_bits, dtype) - ordered(b_bits, dtype))


def check_act(got_bits, ref, ref_bits, dtype, name, exact_frac=None):
    got_bits = np.asarray(got_bits)
    got = widen_bits(got_bits, dtype)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    err = np.abs(got - ref)
    if dtype == FP32:
        rms = np.sqrt(np.mean(ref ** 2, axis=-1, keepdims=True))
        tol = 1e-5 * np.abs(ref) + 1e-5 * rms
    else:
        tol = 1e-2 + 1.6e-2 * np.abs(ref)
    bad = err > tol
    assert not bad.any(), f"{name}: {bad.sum()} elements out of tolerance, max err {err.max()}"
    if dtype != FP32:
        # tighter than the contract: one unit in the last place of the reference, plus the
        # fp32 arithmetic error of the kernel relative to the row's scale (outputs that
        # cancel toward zero, e.g. a rotated pair, carry the inputs' absolute error)
        scale = np.max(np.abs(ref), axis=-1, keepdims=True)
        strict = ulp_of(ref, dtype) + 2.0 ** -18 * scale
        worst = np.argmax(err - strict)
        assert (err <= strict).all(), (f"{name}: {(err > strict).sum()} elements beyond 1 ulp + "
                                       f"2^-18 row scale; worst ref {ref.flat[worst]} got {got.flat[worst]}")
        if exact_frac is not None:
            u = ulp_diff(got_bits, ref_bits, dtype)
            frac = float((u == 0).mean())
            assert frac >= exact_frac, f"{name}: only {frac:.5f} bit-exact"


def ulp_of(v, dtype):
    """Spacing of the activation format at |v| (its subnormal spacing below the normal range)."""
    a = np.abs(np.asarray(v, np.float64))
    mant, minexp = (8, -126) if dtype == BF16 else (11, -14)
    e = np.floor(np.log2(np.where(a > 0, a, 1.0)))
    e = np.maximum(e, minexp)
    return np.exp2(e - (mant - 1))


def dev(bits, dtype, device="cuda"):
    return synth.bits_to_torch(bits, dtype).to(device)


def host_bits(t, dtype):
    return synth.torch_to_bits(t, dtype)


def padded(bits, dtype, pad, device="cuda"):
    """A row-strided device view [T, W] (row stride W + pad) holding `bits`."""
    T, W = bits.shape
    buf = torch.zeros((T, W + pad), dtype=synth._TORCH_DT[dtype], device=device)
    view = buf[:, :W]
    view.copy_(dev(bits, dtype, device))
    return view


def check_rope(ref, got, inputs, dtype=BF16):
    """RoPE + KV append against the oracle (`oracle.layer.rope_kv` output `ref`): q and the
    written k-cache rows within tolerance, tokens with a position outside the cache left
    untouched, every other cache slot still the sentinel, the v cache a bit copy, and the
    k / v inputs unchanged. got: host bit arrays q, k_cache, v_cache, k, v."""
    q, k, v, pos = inputs
    valid = (pos >= 0) & (pos < ref["k_cache"].shape[1])
    check_act(got["q"][valid], ref["q_ref"][valid], ref["q"][valid], dtype, "q", exact_frac=0.99)
    assert np.array_equal(got["q"][~valid], q[~valid])  # skipped tokens untouched
    # k cache: rotated rows at the valid positions, sentinel (bit-exact) everywhere else
    kc_ref_rows = ref["k_cache"][:, pos[valid], :]
    kc_got_rows = got["k_cache"][:, pos[valid], :]
    check_act(kc_got_rows.transpose(1, 0, 2), ref["k_ref"][valid], kc_ref_rows.transpose(1, 0, 2),
              dtype, "k_cache", exact_frac=0.99)
    written = np.zeros(ref["k_cache"].shape[1], bool)
    written[pos[valid]] = True
    assert np.all(got["k_cache"][:, ~written, :] == synth.CACHE_SENTINEL)
    assert np.array_equal(got["v_cache"], ref["v_cache"])  # bit copy + sentinel
    assert np.array_equal(got["k"], k) and np.array_equal(got["v"], v)  # inputs unchanged
