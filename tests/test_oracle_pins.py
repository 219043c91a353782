"""Pins of the CPU oracle against facts that do not come from the oracle itself:
hand-computed values, closed forms, invariants, library conversion routines and
hand-written selection cases read off Algorithm 1 / Fig. 4. CPU only."""
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import guards as G
from oracle import layer as L
from paper_2609_37241_gb300 import synth
from tests import cases

BF16, FP16, FP32 = 1, 2, 3
HERE = os.path.dirname(os.path.abspath(__file__))


# ---------------------------------------------------------------------------- rounding
@pytest.mark.parametrize("value,bits", [
    (1.0, 0x3F80), (-2.0, 0xC000), (1.0 + 2 ** -7, 0x3F81),
    (1.0 + 2 ** -8, 0x3F80),          # tie -> even (down)
    (1.0 + 3 * 2 ** -8, 0x3F82),      # tie -> even (up)
    (1.0 + 2 ** -8 + 2 ** -30, 0x3F81),  # just above the tie
    (2.0 ** -133, 0x0001),            # smallest subnormal
    (2.0 ** -134, 0x0000),            # half of it: tie -> even zero
    (3 * 2.0 ** -134, 0x0002),        # 1.5 quanta: tie -> even
    ((2 - 2 ** -7) * 2.0 ** 127, 0x7F7F),  # max finite
    ((2 - 2 ** -8) * 2.0 ** 127, 0x7F80),  # tie above max -> inf
    (-0.0, 0x8000),
])
def test_bf16_round_hand_values(value, bits):
    assert L.round_bits([value], BF16)[0] == bits


@pytest.mark.parametrize("value,bits", [
    (1.0, 0x3C00), (65504.0, 0x7BFF), (65520.0, 0x7C00), (65519.99, 0x7BFF),
    (2.0 ** -24, 0x0001), (2.0 ** -14, 0x0400), (-1.5, 0xBE00), (1.0 + 2 ** -11, 0x3C00),
    (1.0 + 3 * 2 ** -11, 0x3C02),
])
def test_fp16_round_hand_values(value, bits):
    assert L.round_bits([value], FP16)[0] == bits


def test_bf16_round_matches_torch_cast():
    """For fp32-representable inputs the bf16 RNE cast of torch is the same function."""
    g = np.random.default_rng(1)
    mant = g.uniform(-2, 2, 20000)
    expo = g.integers(-140, 128, 20000)
    f = (mant * np.exp2(expo.astype(np.float64))).astype(np.float32)
    f = f[np.isfinite(f)]
    want = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = L.round_bits(f.astype(np.float64), BF16)
    assert np.array_equal(got, want)


def test_fp16_round_matches_numpy_cast():
    g = np.random.default_rng(2)
    mant = g.uniform(-2, 2, 20000)
    expo = g.integers(-30, 17, 20000)
    f = mant * np.exp2(expo.astype(np.float64))
    with np.errstate(over="ignore"):
        want = f.astype(np.float16).view(np.uint16)
    got = L.round_bits(f, FP16)
    assert np.array_equal(got, want)


def test_widen_all_bf16_and_fp16_patterns():
    allbits = np.arange(65536, dtype=np.uint32)
    keep = ~(((allbits & 0x7F80) == 0x7F80) & ((allbits & 0x7F) != 0))  # drop NaNs
    bf = allbits[keep]
    want = torch.from_numpy(bf.astype(np.uint16).view(np.int16)).view(torch.bfloat16).float()
    got = L.widen(bf, BF16)
    assert np.array_equal(got, want.double().numpy())
    keep16 = ~(((allbits & 0x7C00) == 0x7C00) & ((allbits & 0x3FF) != 0))
    h = allbits[keep16]
    assert np.array_equal(L.widen(h, FP16), h.astype(np.uint16).view(np.float16).astype(np.float64))


# ---------------------------------------------------------------------------- add + RMSNorm
def test_add_rmsnorm_hand_example():
    x = synth.to_bits(np.array([[1, 2, 3, 4]], np.float32), BF16)
    r = synth.to_bits(np.array([[0.5, 0, -1, 0]], np.float32), BF16)
    gamma = np.array([1, 2, 0.5, 1], np.float32)
    y_ref, y, r_out = L.add_rmsnorm(x, r, gamma, 0.0, BF16)
    s = [1.5, 2.0, 2.0, 4.0]
    rms = math.sqrt((1.5 ** 2 + 4 + 4 + 16) / 4)  # 2.5617376914898995
    want = [1.5 / rms * 1, 2 / rms * 2, 2 / rms * 0.5, 4 / rms * 1]
    assert np.allclose(y_ref[0], want, rtol=1e-15, atol=0)
    assert list(L.widen(r_out[0], BF16)) == s


def test_add_rmsnorm_constant_row_closed_form():
    H, c, eps = 64, 1.5, 1e-6
    x = synth.to_bits(np.full((1, H), c, np.float32), BF16)
    r = synth.to_bits(np.zeros((1, H), np.float32), BF16)
    gamma = np.linspace(0.5, 1.5, H).astype(np.float32)
    y_ref, _, _ = L.add_rmsnorm(x, r, gamma, eps, BF16)
    want = c / math.sqrt(c * c + eps) * gamma.astype(np.float64)
    assert np.allclose(y_ref[0], want, rtol=1e-14, atol=0)
    # eps inside the square root: with eps = 1 the constant row gives c / sqrt(c^2 + 1)
    y1, _, _ = L.add_rmsnorm(x, r, np.ones(H, np.float32), 1.0, BF16)
    assert np.allclose(y1[0], c / math.sqrt(c * c + 1.0), rtol=1e-14)


def test_add_rmsnorm_scale_invariance_and_symmetry():
    g = np.random.default_rng(3)
    H = 256
    xf = g.normal(size=(3, H)).astype(np.float32)
    rf = g.normal(size=(3, H)).astype(np.float32)
    x, r = synth.to_bits(xf, BF16), synth.to_bits(rf, BF16)
    x2 = synth.to_bits(2 * L.widen(x, BF16).astype(np.float32), BF16)  # exact doubling
    r2 = synth.to_bits(2 * L.widen(r, BF16).astype(np.float32), BF16)
    gam = synth.gamma(g, H)
    ya, _, _ = L.add_rmsnorm(x, r, gam, 0.0, BF16)
    yb, _, _ = L.add_rmsnorm(x2, r2, gam, 0.0, BF16)
    assert np.array_equal(ya, yb)
    yc, _, rc = L.add_rmsnorm(r, x, gam, 1e-6, BF16)
    yd, _, rd = L.add_rmsnorm(x, r, gam, 1e-6, BF16)
    assert np.array_equal(yc, yd) and np.array_equal(rc, rd)
    # with gamma = 1, RMS(y) = sqrt(ms / (ms + eps))
    eps = 0.25
    y1, _, r1 = L.add_rmsnorm(x, r, np.ones(H, np.float32), eps, BF16)
    s = L.widen(x, BF16) + L.widen(r, BF16)
    ms = (s * s).mean(axis=1)
    assert np.allclose(np.sqrt((y1 * y1).mean(axis=1)), np.sqrt(ms / (ms + eps)), rtol=1e-12)


def test_add_rmsnorm_column_permutation_equivariance():
    g = np.random.default_rng(4)
    H = 128
    x, r = synth.act(g, (2, H), BF16), synth.act(g, (2, H), BF16)
    gam = synth.gamma(g, H)
    perm = g.permutation(H)
    ya, yba, ra = L.add_rmsnorm(x, r, gam, 1e-6, BF16)
    yb, ybb, rb = L.add_rmsnorm(x[:, perm], r[:, perm], gam[perm], 1e-6, BF16)
    assert np.allclose(ya[:, perm], yb, rtol=1e-14)
    assert np.array_equal(ra[:, perm], rb)


def test_add_rmsnorm_residual_zero_passes_x_through():
    g = np.random.default_rng(5)
    for dt in (BF16, FP16, FP32):
        x = synth.act(g, (2, 64), dt)
        zero = synth.to_bits(np.zeros((2, 64), np.float32), dt)
        _, _, r_out = L.add_rmsnorm(x, zero, np.ones(64, np.float32), 1e-6, dt)
        assert np.array_equal(r_out, x)


# ---------------------------------------------------------------------------- RMSNorm
def test_rmsnorm_hand_example_and_closed_forms():
    x = synth.to_bits(np.array([[3, 4, 0, 0]], np.float32), BF16)     # mean(x^2) = 25/4
    gamma = np.array([1, 2, 3, 4], np.float32)
    y_ref, y = L.rmsnorm(x, gamma, 0.0, BF16)
    assert np.allclose(y_ref[0], [3 / 2.5, 4 / 2.5 * 2, 0, 0], rtol=1e-15, atol=0)
    c, H, eps = -0.75, 128, 1e-6
    xc = synth.to_bits(np.full((1, H), c, np.float32), BF16)
    yc, _ = L.rmsnorm(xc, np.ones(H, np.float32), eps, BF16)
    assert np.allclose(yc[0], c / math.sqrt(c * c + eps), rtol=1e-14)


def test_rmsnorm_equals_add_rmsnorm_with_zero_residual():
    """Two oracle functions, one definition: rms_norm(x) = add+RMSNorm(x, 0).y, bit for bit."""
    g = np.random.default_rng(14)
    for dt in (BF16, FP16, FP32):
        x = synth.act(g, (5, 128), dt)
        zero = synth.to_bits(np.zeros((5, 128), np.float32), dt)
        gam = synth.gamma(g, 128)
        a_ref, a = L.rmsnorm(x, gam, 1e-6, dt)
        b_ref, b, _ = L.add_rmsnorm(x, zero, gam, 1e-6, dt)
        assert np.array_equal(a, b) and np.allclose(a_ref, b_ref, rtol=1e-15, atol=0)


# ---------------------------------------------------------------------------- RoPE
def test_rope_position_zero_is_identity():
    g = np.random.default_rng(6)
    x = g.normal(size=128)
    assert np.array_equal(L.rope_apply(x, 0, 500000.0), x)


def test_rope_direction_and_frequency_hand_values():
    D, theta = 128, 500000.0
    e0 = np.zeros(D); e0[0] = 1.0
    y = L.rope_apply(e0, 1, theta)          # angle 1 rad at i = 0
    assert y[0] == pytest.approx(math.cos(1.0), abs=1e-15)
    assert y[64] == pytest.approx(math.sin(1.0), abs=1e-15)
    assert np.count_nonzero(np.abs(y) > 1e-300) == 2
    e32 = np.zeros(D); e32[32] = 1.0        # i = 32: inv_freq = theta^(-64/128) = 1/sqrt(theta)
    a = 1000.0 / math.sqrt(theta)
    y = L.rope_apply(e32, 1000, theta)
    assert y[32] == pytest.approx(math.cos(a), abs=1e-14)
    assert y[96] == pytest.approx(math.sin(a), abs=1e-14)
    e96 = np.zeros(D); e96[96] = 1.0        # upper half rotates the other way
    y = L.rope_apply(e96, 1000, theta)
    assert y[32] == pytest.approx(-math.sin(a), abs=1e-14)
    assert y[96] == pytest.approx(math.cos(a), abs=1e-14)


def test_rope_norm_composition_and_complex_form():
    g = np.random.default_rng(7)
    D, theta = 128, 1e6
    for _ in range(20):
        x = g.normal(size=D)
        p1, p2 = (int(v) for v in g.integers(0, 4096, 2))
        y = L.rope_apply(x, p1, theta)
        pair_in = x[:64] ** 2 + x[64:] ** 2
        pair_out = y[:64] ** 2 + y[64:] ** 2
        assert np.allclose(pair_in, pair_out, rtol=1e-12)
        assert np.allclose(L.rope_apply(y, p2, theta), L.rope_apply(x, p1 + p2, theta),
                           rtol=1e-9, atol=1e-9)
        i = np.arange(64)
        z = (x[:64] + 1j * x[64:]) * np.exp(1j * p1 * theta ** (-2.0 * i / D))
        assert np.allclose(y[:64], z.real, atol=1e-10) and np.allclose(y[64:], z.imag, atol=1e-10)


def test_rope_kv_append_sentinel_copy_and_bad_position():
    g = np.random.default_rng(8)
    T, Hq, Hkv, D, S = 5, 4, 2, 16, 32
    q, k, v = (synth.act(g, (T, h, D), BF16) for h in (Hq, Hkv, Hkv))
    pos = synth.positions(g, T, S)
    kc, vc = synth.cache(Hkv, S, D), synth.cache(Hkv, S, D)
    out = L.rope_kv(q, k, v, pos, kc, vc, 10000.0, BF16)
    assert out["bad"] == 0
    written = np.zeros(S, bool); written[pos] = True
    assert np.all(out["k_cache"][:, ~written, :] == synth.CACHE_SENTINEL)
    assert np.all(out["v_cache"][:, ~written, :] == synth.CACHE_SENTINEL)
    for t in range(T):
        assert np.array_equal(out["v_cache"][:, pos[t], :], v[t])
        assert np.array_equal(out["k_cache"][:, pos[t], :], L.round_bits(out["k_ref"][t], BF16))
    # a position outside [0, S): flagged, that token skipped entirely
    bad_pos = pos.copy(); bad_pos[2] = S
    out2 = L.rope_kv(q, k, v, bad_pos, kc, vc, 10000.0, BF16)
    assert out2["bad"] == 1
    assert np.array_equal(out2["q"][2], q[2])
    keep = np.ones(T, bool); keep[2] = False
    assert np.array_equal(out2["q"][keep], out["q"][keep])
    assert np.all(out2["k_cache"][:, S - 1, :] == synth.CACHE_SENTINEL) or pos.max() == S - 1


def test_qknorm_then_rope_keeps_normalised_rms():
    """Norm first, then a norm-preserving rotation: with gamma = 1 every rotated head has
    RMS sqrt(ms / (ms + eps))."""
    g = np.random.default_rng(9)
    T, Hq, Hkv, D, S, eps = 3, 4, 2, 128, 64, 0.5
    q, k, v = (synth.act(g, (T, h, D), BF16) for h in (Hq, Hkv, Hkv))
    pos = synth.positions(g, T, S)
    out = L.rope_kv(q, k, v, pos, synth.cache(Hkv, S, D), synth.cache(Hkv, S, D), 1e6, BF16,
                    qknorm=True, gamma_q=np.ones(D), gamma_k=np.ones(D), eps=eps)
    for src, ref in ((q, out["q_ref"]), (k, out["k_ref"])):
        w = L.widen(src, BF16)
        ms = (w * w).mean(axis=2)
        got = np.sqrt((ref * ref).mean(axis=2))
        assert np.allclose(got, np.sqrt(ms / (ms + eps)), rtol=1e-12)


def test_qknorm_weights_each_head_element_before_the_rotation():
    """Distinct, non-uniform q and k norm weights. At position 0 (the identity rotation) each
    head's output divided by its own weights is proportional to the input head with RMS
    sqrt(ms / (ms + eps)); at any position the rotation keeps the norm of each rotated pair
    (i, i + D/2) equal to that of the weighted, normalised inputs. Swapped q/k weights,
    weights applied after the rotation, or weights indexed from the wrong half fail one of
    these."""
    g = np.random.default_rng(21)
    T, Hq, Hkv, D, S, eps = 4, 3, 2, 64, 64, 1e-3
    q, k, v = (synth.act(g, (T, h, D), BF16) for h in (Hq, Hkv, Hkv))
    pos = np.array([0, 17, 0, 63], np.int32)
    gq = (1.0 + 0.3 * g.standard_normal(D)).astype(np.float32)
    gk = (1.0 - 0.4 * g.standard_normal(D)).astype(np.float32)
    out = L.rope_kv(q, k, v, pos, synth.cache(Hkv, S, D), synth.cache(Hkv, S, D), 1e6, BF16,
                    qknorm=True, gamma_q=gq, gamma_k=gk, eps=eps)
    half = D // 2
    for src, ref, gam in ((q, out["q_ref"], gq), (k, out["k_ref"], gk)):
        w = L.widen(src, BF16)
        gam = gam.astype(np.float64)
        ms = (w * w).mean(axis=2, keepdims=True)
        for t in np.flatnonzero(pos == 0):
            unweighted = ref[t] / gam
            assert np.allclose(np.sqrt((unweighted ** 2).mean(axis=1)), np.sqrt(ms[t, :, 0] / (ms[t, :, 0] + eps)),
                               rtol=1e-12)
            ratio = unweighted / w[t]
            assert np.allclose(ratio, ratio[:, :1], rtol=1e-12)
        weighted = w * gam / np.sqrt(ms + eps)
        pair_in = weighted[..., :half] ** 2 + weighted[..., half:] ** 2
        pair_out = ref[..., :half] ** 2 + ref[..., half:] ** 2
        assert np.allclose(pair_out, pair_in, rtol=1e-12)


# ---------------------------------------------------------------------------- SwiGLU
def test_swiglu_closed_forms():
    vals = np.array([0.0, 1.0, -1.0, 20.0, -30.0, 3.0], np.float32)
    g = synth.to_bits(vals, FP32)
    one = synth.to_bits(np.ones_like(vals), FP32)
    zero = synth.to_bits(np.zeros_like(vals), FP32)
    ref, _ = L.swiglu(g, one, FP32)
    assert ref[0] == 0.0
    assert ref[1] == pytest.approx(0.7310585786300049, rel=1e-15)  # sigmoid(1)
    assert ref[3] == pytest.approx(20.0 * (1 - math.exp(-20.0)), rel=1e-14)
    assert abs(ref[4]) < 1e-11 and ref[4] < 0
    ref0, _ = L.swiglu(g, zero, FP32)
    assert np.all(ref0 == 0.0)
    # silu(g) - silu(-g) = g
    gn = synth.to_bits(-vals, FP32)
    refn, _ = L.swiglu(gn, one, FP32)
    assert np.allclose(ref - refn, vals.astype(np.float64), rtol=1e-14, atol=1e-300)
    # u scales linearly
    three = synth.to_bits(np.full_like(vals, 3.0), FP32)
    ref3, _ = L.swiglu(g, three, FP32)
    assert np.allclose(ref3, 3 * ref, rtol=1e-15)


# ---------------------------------------------------------------------------- pointwise
def test_pointwise_closed_forms_and_library_casts():
    g = np.random.default_rng(15)
    xf = (g.normal(size=4000) * 3).astype(np.float32)
    for dt in (BF16, FP16, FP32):
        x = synth.to_bits(xf, dt)
        xv = L.widen(x[:64], dt)
        # silu against its closed form at special points and the SwiGLU oracle with u = 1
        one = synth.to_bits(np.ones_like(xf), dt)
        s_ref, s = L.silu(x, dt)
        w_ref, w = L.swiglu(x, one, dt)
        assert np.array_equal(s, w) and np.allclose(s_ref, w_ref, rtol=1e-15, atol=0)
        # neg is exact: it flips the sign bit
        n_ref, n = L.neg(x, dt)
        signbit = 0x80000000 if dt == FP32 else 0x8000
        assert np.array_equal(n, x ^ np.array(signbit, x.dtype))
        # add: commutative; x + 0 = x; x + x = 2x exactly
        zero = synth.to_bits(np.zeros_like(xf), dt)
        assert np.array_equal(L.add(x, zero, dt)[1], np.where(L.widen(x, dt) == 0, L.add(x, zero, dt)[1], x))
        y = synth.to_bits(g.normal(size=4000).astype(np.float32), dt)
        assert np.array_equal(L.add(x, y, dt)[1], L.add(y, x, dt)[1])
        two_x, _ = L.add(x, x, dt)
        assert np.array_equal(two_x, 2 * L.widen(x, dt))
    # add against torch's bf16 addition (fp32 sum, one rounding): a library routine
    a = synth.to_bits(xf, BF16)
    b = synth.to_bits((xf[::-1] * 0.37).copy(), BF16)
    want = (synth.bits_to_torch(a, BF16).float() + synth.bits_to_torch(b, BF16).float()).to(torch.bfloat16)
    assert np.array_equal(L.add(a, b, BF16)[1], want.view(torch.int16).numpy().view(np.uint16))


def test_masked_fill_semantics():
    g = np.random.default_rng(16)
    x = synth.act(g, (4, 32), BF16)
    mask = (g.random((4, 32)) < 0.3).astype(np.uint8)
    ref, out = L.masked_fill(x, mask, -1e4, BF16)
    assert np.array_equal(out[mask == 0], x[mask == 0])
    fill = synth.to_bits(np.array([-1e4], np.float32), BF16)[0]  # -10000 rounds to -9984
    assert np.all(out[mask == 1] == fill) and L.widen([fill], BF16)[0] == -9984.0
    _, inf_out = L.masked_fill(x, mask, float("-inf"), BF16)
    assert np.all(inf_out[mask == 1] == 0xFF80)


# ---------------------------------------------------------------------------- layer chain
def test_layer_chain_second_norm_reads_rounded_residual():
    g = np.random.default_rng(10)
    cfg = dict(synth.LLAMA, H=64, Hq=4, Hkv=2, D=16, S=32, I=48)
    inp = synth.layer_inputs(g, 3, cfg)
    out = L.layer_chain(inp, cfg["theta"], 1e-6, BF16)
    _, x1, r1 = L.add_rmsnorm(inp["h"], inp["r0"], inp["gamma_attn"], 1e-6, BF16)
    _, x2, r2 = L.add_rmsnorm(inp["attn_out"], r1, inp["gamma_mlp"], 1e-6, BF16)
    assert np.array_equal(out["r2"], r2) and np.array_equal(out["x2"], x2)
    # r2 = round(attn_out + round(h + r0)) in fp32
    hw, rw, aw = (L.widen(inp[n], BF16).astype(np.float32) for n in ("h", "r0", "attn_out"))
    r1f = L.widen(synth.to_bits(hw + rw, BF16), BF16).astype(np.float32)
    assert np.array_equal(out["r2"], synth.to_bits(aw + r1f, BF16))


# ---------------------------------------------------------------------------- selection
def _golden():
    with open(os.path.join(HERE, "golden", "guard_cases.json")) as f:
        return json.load(f)["cases"]


@pytest.mark.parametrize("case", _golden(), ids=lambda c: c["cite"])
def test_selection_golden_cases(case):
    table = [cases.make_spec(s) for s in case["table"]]
    args = cases.make_args(case["args"])
    assert list(G.select(table, args)) == case["expect"]


def _matching_pair():
    spec = cases.make_spec({"op": 1, "dtype": "bf16", "fixed": [64], "tok": [2, 8]})
    args = cases.make_args({"op": 1, "dtype": "bf16", "T": 4, "H": 64})
    return spec, args


def test_every_guarded_field_can_cause_a_miss():
    """Mutating any single guarded field of a matching pair gives MISS: no guard term is
    silently dropped."""
    spec, args = _matching_pair()
    assert G.select([spec], args) == (G.OK, 0)
    mutations = {
        "op": lambda s, a: s.update(op=4),
        "device": lambda s, a: a["tensors"][2].update(device=1),
        "dtype act": lambda s, a: s.update(dtype=2),
        "dtype gamma": lambda s, a: a["tensors"][2].update(dtype=1),
        "rank": lambda s, a: s.update(rank=3),
        "H": lambda s, a: s.update(fixed=(72,)),
        "gamma size": lambda s, a: a["tensors"][2].update(shape=(63,)),
        "y rows": lambda s, a: a["tensors"][3].update(shape=(3, 64)),
        "T low": lambda s, a: s.update(tok_lo=5),
        "T high": lambda s, a: s.update(tok_hi=3),
        "layout": lambda s, a: s.update(layout=1),
        "inner stride": lambda s, a: a["tensors"][1].update(stride=(128, 2)),
        "gamma stride": lambda s, a: a["tensors"][2].update(stride=(2,)),
        "align ptr": lambda s, a: a["tensors"][4].update(addr=a["tensors"][4]["addr"] + 2),
        "align row": lambda s, a: a["tensors"][0].update(stride=(68, 1)),
    }
    for name, mut in mutations.items():
        s, a = _matching_pair()
        mut(s, a)
        assert G.select([s], a) == (G.MISS, -1), name


def test_first_match_order_properties():
    """Algorithm 1: appending versions never changes a hit; the selected version is the
    lowest index whose guard holds; a table of only failing versions misses."""
    g = np.random.default_rng(11)
    buckets = [(1, 1), (2, 2), (3, 4), (1, 4)]
    for _ in range(300):
        table = []
        for _ in range(g.integers(0, 5)):
            lo, hi = buckets[g.integers(0, 4)]
            table.append(cases.make_spec({"op": 1, "dtype": ["bf16", "fp16"][g.integers(0, 2)],
                                          "fixed": [64], "tok": [lo, hi],
                                          "layout": ["contig", "strided", "any"][g.integers(0, 3)],
                                          "align": [2, 16][g.integers(0, 2)]}))
        args = cases.make_args({"op": 1, "dtype": ["bf16", "fp16"][g.integers(0, 2)],
                                "T": int(g.integers(1, 5)), "H": 64,
                                "layout": ["contig", "strided"][g.integers(0, 2)],
                                "misalign": bool(g.integers(0, 2))})
        st, idx = G.select(table, args)
        holds = [G.guard(s, args) for s in table]
        if st == G.OK:
            assert holds[idx] and not any(holds[:idx])
            extra = cases.make_spec({"op": 1, "dtype": "bf16", "fixed": [64], "tok": [1, 4],
                                     "layout": "any", "align": 2})
            assert G.select(table + [extra], args) == (st, idx)
        else:
            assert st == G.MISS and not any(holds)


def test_overlap_precondition_brute_force():
    base = 0x10000
    x = cases.tensor(base, 1, (4, 8))
    # in place y = x: allowed for ADD_RMSNORM
    gam = cases.tensor(0x90000, 3, (8,))
    r = cases.tensor(0x20000, 1, (4, 8))
    args = dict(op=1, tensors=[x, r, gam, dict(x), cases.tensor(0x30000, 1, (4, 8))], eps=0.0,
                theta=0.0, flags=0)
    assert G.launch_precondition(args)
    # y shifted by one element overlaps x partially: not allowed
    args["tensors"][3] = cases.tensor(base + 2, 1, (4, 8))
    assert not G.launch_precondition(args)
    # y interleaved with x in the gaps of a strided x: disjoint bytes, allowed
    xs = cases.tensor(base, 1, (4, 8), (16, 1))
    ys = cases.tensor(base + 16, 1, (4, 8), (16, 1))
    args["tensors"][0], args["tensors"][3] = xs, ys
    assert G.launch_precondition(args)
    # r_out equal to x (not an in-place pair): not allowed
    args["tensors"][0], args["tensors"][3] = x, cases.tensor(0x40000, 1, (4, 8))
    args["tensors"][4] = dict(x)
    assert not G.launch_precondition(args)


def test_calls_independent_hand_cases():
    """Independence of whole calls: disjoint buffers, shared inputs, a read of another
    call's output, a write-write clash, and a one-byte overlap at a row edge."""
    def norm_call(x, r, y, ro, gam=0x90000):
        return dict(op=1, tensors=[cases.tensor(x, 1, (2, 8)), cases.tensor(r, 1, (2, 8)),
                                   cases.tensor(gam, 3, (8,)), cases.tensor(y, 1, (2, 8)),
                                   cases.tensor(ro, 1, (2, 8))], eps=0.0, theta=0.0, flags=0)
    a = norm_call(0x10000, 0x20000, 0x30000, 0x40000)
    b = norm_call(0x50000, 0x60000, 0x70000, 0x80000)
    assert G.calls_independent([a, b])  # disjoint, and both read one gamma
    assert G.calls_independent([a, norm_call(0x10000, 0x20000, 0x70000, 0x80000)])  # shared inputs
    assert not G.calls_independent([a, norm_call(0x40000, 0x60000, 0x70000, 0x80000)])  # reads a's r_out
    assert not G.calls_independent([norm_call(0x50000, 0x60000, 0x30000, 0x80000), a])  # both write y
    # b's x ends one byte into a's y (rows of 16 bytes; 2 rows = 32 bytes)
    assert not G.calls_independent([a, norm_call(0x30000 - 31, 0x60000, 0x70000, 0x80000)])
    assert G.calls_independent([a, norm_call(0x30000 - 32, 0x60000, 0x70000, 0x80000)])
    assert G.calls_independent([a])


def test_bind_tree_hand_cases():
    """The recipe binder on hand-made trees: structure, kinds, guarded constants, bound
    scalars, ignored leaves and the slot each consumed tensor fills."""
    a, b, c = (cases.tensor(0x1000 * k, 1, (2, 8)) for k in (1, 2, 3))
    g = cases.tensor(0x9000, 3, (8,))
    rec = cases.recipe(1, ("tuple", [("tensor", 1), ("tensor", 0)]), ("tensor", 2), ("none",),
                       ("tuple", [("tensor", 3), ("tensor", -1), ("tensor", 4)]), ("float", "eps"),
                       ("int", "const", 2), eps=0.5, theta=7.0)
    got = G.bind_tree(rec, [(a, b), g, None, (c, a, b), 1e-3, 2])
    assert [t["addr"] for t in got["tensors"]] == [b["addr"], a["addr"], g["addr"], c["addr"], b["addr"]]
    assert (got["op"], got["eps"], got["theta"], got["scalar"]) == (1, 1e-3, 7.0, 0.0)
    assert G.bind_tree(rec, [(a, b), g, None, (c, a, b), 1e-3, 3]) is None      # constant differs
    assert G.bind_tree(rec, [(a, b), g, None, (c, a, b), 1e-3, 2.0]) is None    # float, not int
    assert G.bind_tree(rec, [(a, b), g, None, (c, a, b), 1, 2]) is None         # int eps
    assert G.bind_tree(rec, [(a, b), g, a, (c, a, b), 1e-3, 2]) is None         # tensor for None
    assert G.bind_tree(rec, [(a, b, c), g, None, (c, a, b), 1e-3, 2]) is None   # tuple arity
    assert G.bind_tree(rec, [a, g, None, (c, a, b), 1e-3, 2]) is None           # tensor for tuple
    assert G.bind_tree(rec, [(a, b), g, None, (c, a, b), 1e-3]) is None         # parameter count
    assert G.bind_tree(rec, [(a, b), g, None, (c, g, b), 1e-3, 2]) is not None  # ignored leaf: any tensor
    assert G.bind_tree(rec, [(a, b), g, None, (c, 5, b), 1e-3, 2]) is None      # ... but a tensor
    # True is the int 1 (Python semantics)
    one = cases.recipe(7, ("tensor", 0), ("tensor", 1), ("tensor", 2), ("int", "const", 1))
    assert G.bind_tree(one, [a, g, b, True]) is not None


def test_bucket_definition():
    assert [G.bucket_of(t) for t in (1, 2, 3, 4, 5, 8, 9, 128, 129)] == [0, 1, 2, 2, 3, 3, 4, 7, 8]
    for b in range(10):
        lo, hi = G.bucket_range(b)
        assert all(G.bucket_of(t) == b for t in range(lo, hi + 1))


def test_parallel_oracle_build_matches_serial():
    """The OpenMP build of the C oracle (used only to time it on all host cores) computes
    exactly the serial build's values: every loop iteration writes its own outputs."""
    cfg = dict(synth.LLAMA)
    cfg.update(H=256, Hq=4, Hkv=2, D=64, S=64, I=320)
    inp = synth.layer_inputs(np.random.default_rng(5), 7, cfg)
    inp["pos"][3] = cfg["S"]  # one bad position: the reduction of the flag
    serial = L.layer_chain(inp, cfg["theta"], cfg["eps"], synth.BF16)
    try:
        L.set_parallel(True)
        par = L.layer_chain(inp, cfg["theta"], cfg["eps"], synth.BF16)
        assert L.threads() >= 1
    finally:
        L.set_parallel(False)
    assert serial.keys() == par.keys()
    for k in serial:
        a, b = np.atleast_1d(np.asarray(serial[k])), np.atleast_1d(np.asarray(par[k]))
        assert a.dtype == b.dtype and a.shape == b.shape, k
        assert np.array_equal(a.view(np.uint8), b.view(np.uint8)), k  # bitwise (NaN included)
