"""Seeded random configurations of every op against the oracle: token counts (ragged,
across the one-block-per-SM threshold), widths, dtypes, contiguous and row-strided views,
in-place calls, the generic variant, and launches with programmatic dependent launch (PDL:
L2 prefetch and, for the chain, the token-major grid on small grids). Each case is one
version, one invoke, every output compared."""
import random

import numpy as np
import pytest
import torch

from oracle import layer as L
from paper_2609_37241_gb300 import synth
from tests import parity as P
from tests.test_parity_gpu import chain_device, check_chain, check_rope, run_rope

pytestmark = pytest.mark.gpu
BF16, FP16, FP32 = 1, 2, 3
ES = {BF16: 2, FP16: 2, FP32: 4}


@pytest.fixture(scope="module")
def S(built_lib):
    from paper_2609_37241_gb300 import scm
    return scm


def stream():
    return torch.cuda.current_stream().cuda_stream


def rows(bits, dtype, pad):
    return P.padded(bits, dtype, pad) if pad else P.dev(bits, dtype)


def run_one(S, desc, op, ts, pdl, **kw):
    s = S.Scm(device=0, flags=S.OPT_PDL if pdl else 0)
    s.register(desc)
    st, sel = s.invoke(S.make_args(op, ts, **kw), stream())
    assert (st, sel) == (S.OK, 0), S.trident_scm_last_error()
    torch.cuda.synchronize()
    assert S.trident_scm_device_status(s.h, stream())[1] == 0
    s.close()


def layout_of(S, T, pad):
    return S.LAYOUT_ROWSTRIDED if pad and T > 1 else S.LAYOUT_CONTIG


@pytest.mark.parametrize("seed", range(12))
def test_fuzz_add_rmsnorm_and_rmsnorm(S, seed):
    rng = random.Random(seed)
    g = np.random.default_rng(seed)
    dtype = rng.choice([BF16, BF16, FP16, FP32])
    H = rng.choice([64, 128, 256, 1000, 2048, 4096, 8192] + ([520] if dtype != FP32 else []))
    T = rng.choice([1, 2, 7, 37, 150, 153, 300, 1024, 1100])
    es = ES[dtype]
    vec_ok = (H * es) % 16 == 0
    pad = rng.choice([0, 0, 8 * (16 // es)]) if vec_ok else 0
    generic = rng.random() < 0.2
    pdl = rng.random() < 0.5
    inplace = rng.random() < 0.3
    eps = rng.choice([1e-6, 1e-5, 0.25])
    x, r = synth.act(g, (T, H), dtype), synth.act(g, (T, H), dtype)
    gam = synth.gamma(g, H)
    gd = torch.from_numpy(gam).cuda()
    align = 16 if vec_ok and not generic else es
    variant = S.VARIANT_GENERIC if generic else S.VARIANT_AUTO
    # add + RMSNorm
    xd, rd = rows(x, dtype, pad), rows(r, dtype, pad)
    yd, rod = (xd, rd) if inplace else (rows(np.zeros_like(x), dtype, pad), rows(np.zeros_like(r), dtype, pad))
    desc = S.make_spec(S.OP_ADD_RMSNORM, dtype, [H], 1, 1 << 20, layout=layout_of(S, T, pad),
                       align_bytes=align, variant=variant)
    run_one(S, desc, S.OP_ADD_RMSNORM, [xd, rd, gd, yd, rod], pdl, eps=eps)
    y_ref, y_bits, ro_bits = L.add_rmsnorm(x, r, gam, eps, dtype)
    assert np.array_equal(P.host_bits(rod, dtype), ro_bits)
    P.check_act(P.host_bits(yd, dtype), y_ref, y_bits, dtype, f"add_rmsnorm {dtype} {H} {T}")
    # RMSNorm
    xd = rows(x, dtype, pad)
    yd = xd if inplace else rows(np.zeros_like(x), dtype, pad)
    desc = S.make_spec(S.OP_RMSNORM, dtype, [H], 1, 1 << 20, layout=layout_of(S, T, pad),
                       align_bytes=align, variant=variant)
    run_one(S, desc, S.OP_RMSNORM, [xd, gd, yd], pdl, eps=eps)
    y_ref, y_bits = L.rmsnorm(x, gam, eps, dtype)
    P.check_act(P.host_bits(yd, dtype), y_ref, y_bits, dtype, f"rmsnorm {dtype} {H} {T}")


@pytest.mark.parametrize("seed", range(6))
def test_fuzz_add_rmsnorm_bulk_rows(S, seed):
    """H 8192 with at least 1024 rows: the kernel that stages rows by bulk copies."""
    rng = random.Random(50 + seed)
    g = np.random.default_rng(50 + seed)
    dtype = rng.choice([BF16, FP16])
    T = rng.choice([1024, 1100, 2048])
    H = 8192
    pad = rng.choice([0, 64])
    pdl = rng.random() < 0.5
    inplace = rng.random() < 0.4
    x, r = synth.act(g, (T, H), dtype), synth.act(g, (T, H), dtype)
    gam = synth.gamma(g, H)
    xd, rd = rows(x, dtype, pad), rows(r, dtype, pad)
    yd, rod = (xd, rd) if inplace else (rows(np.zeros_like(x), dtype, pad), rows(np.zeros_like(r), dtype, pad))
    desc = S.make_spec(S.OP_ADD_RMSNORM, dtype, [H], 1, 1 << 20, layout=layout_of(S, T, pad))
    run_one(S, desc, S.OP_ADD_RMSNORM, [xd, rd, torch.from_numpy(gam).cuda(), yd, rod], pdl, eps=1e-6)
    y_ref, y_bits, ro_bits = L.add_rmsnorm(x, r, gam, 1e-6, dtype)
    assert np.array_equal(P.host_bits(rod, dtype), ro_bits)
    P.check_act(P.host_bits(yd, dtype), y_ref, y_bits, dtype, f"add_rmsnorm bulk {dtype} {T}")


@pytest.mark.parametrize("seed", range(12))
def test_fuzz_pointwise_and_swiglu(S, seed):
    rng = random.Random(100 + seed)
    g = np.random.default_rng(100 + seed)
    dtype = rng.choice([BF16, FP16, FP32])
    W = rng.choice([8, 64, 1000, 4096, 14336, 28672] + ([36] if dtype == FP32 else []))
    T = rng.choice([1, 3, 40, 151, 200])
    es = ES[dtype]
    vec_ok = (W * es) % 16 == 0
    pad = rng.choice([0, 16 // es * 4]) if vec_ok else 0
    generic = rng.random() < 0.2 or not vec_ok
    pdl = rng.random() < 0.5
    align = es if generic else 16
    variant = S.VARIANT_GENERIC if generic else S.VARIANT_AUTO
    lay = layout_of(S, T, pad)
    a = synth.act(g, (T, W), dtype, std=3.0)
    b = synth.act(g, (T, W), dtype)
    name = rng.choice(["silu", "add", "neg", "masked_fill", "swiglu"])
    ad, bd = rows(a, dtype, pad), rows(b, dtype, pad)
    yd = rows(np.zeros_like(a), dtype, pad)
    if name == "swiglu":
        desc = S.make_spec(S.OP_SWIGLU, dtype, [W], 1, 1 << 20, layout=lay, align_bytes=align, variant=variant)
        run_one(S, desc, S.OP_SWIGLU, [ad, bd, yd], pdl)
        ref, ref_bits = L.swiglu(a, b, dtype)
        P.check_act(P.host_bits(yd, dtype), ref, ref_bits, dtype, f"swiglu {dtype} {W} {T}")
        return
    op = {"silu": S.OP_SILU, "add": S.OP_ADD, "neg": S.OP_NEG, "masked_fill": S.OP_MASKED_FILL}[name]
    mask = (g.random((T, W)) < 0.4).astype(np.uint8)
    value = rng.choice([-1e4, 0.0, 3.5])
    if name == "masked_fill":
        mbuf = torch.zeros((T, W + (64 if pad else 0)), dtype=torch.uint8, device="cuda")
        md = mbuf[:, :W]
        md.copy_(torch.from_numpy(mask).cuda())
        ts = [ad, md, yd]
    else:
        ts = {"silu": [ad, yd], "neg": [ad, yd], "add": [ad, bd, yd]}[name]
    desc = S.make_spec(op, dtype, [W], 1, 1 << 20, layout=lay, align_bytes=align, variant=variant)
    run_one(S, desc, op, ts, pdl, scalar=value)
    got = P.host_bits(yd, dtype)
    if name == "silu":
        ref, ref_bits = L.silu(a, dtype)
        P.check_act(got, ref, ref_bits, dtype, f"silu {dtype} {W} {T}")
    else:
        ref_bits = {"add": lambda: L.add(a, b, dtype), "neg": lambda: L.neg(a, dtype),
                    "masked_fill": lambda: L.masked_fill(a, mask, value, dtype)}[name]()[1]
        assert np.array_equal(got, ref_bits), (name, dtype, W, T)


@pytest.mark.parametrize("seed", range(10))
def test_fuzz_rope_kv(S, seed):
    rng = random.Random(200 + seed)
    dtype = rng.choice([BF16, FP16])
    D = rng.choice([64, 128, 256])
    Hkv = rng.choice([1, 2, 8])
    Hq = Hkv * rng.choice([1, 2, 4])
    T = rng.choice([1, 3, 17, 64, 129])
    S_ = rng.choice([T, 300, 8192])
    theta = rng.choice([1e4, 5e5, 1e6])
    qk = rng.random() < 0.5
    variant = 1 if rng.random() < 0.2 else 0
    layout = rng.choice(["fused", "separate"]) if variant == 0 else "fused"
    ref, got, inputs = run_rope(S, T, Hq, Hkv, D, S_, theta, qk, dtype=dtype, layout=layout,
                                variant=variant, seed=200 + seed)
    check_rope(ref, got, inputs, dtype)


@pytest.mark.parametrize("seed", range(12))
def test_fuzz_layer_chain(S, seed):
    rng = random.Random(300 + seed)
    base = rng.choice([synth.LLAMA, synth.QWEN3])
    dtype = rng.choice([BF16, BF16, FP16])
    # up to 80 tokens one wave (late trigger under PDL from 5 tokens); 80, 150 and 260 tokens
    # several waves (one norm CTA per token, three head-rows per RoPE lane group)
    T = rng.choice([1, 2, 5, 16, 17, 19, 33, 64, 80, 150, 260])
    cfg = dict(base, S=rng.choice([128, 8192]) if T <= 128 else 8192)
    qk = cfg["qknorm"]
    pdl = rng.random() < 0.6
    layout = rng.choice(["fused", "separate"])
    g = np.random.default_rng(300 + seed)
    inp = synth.layer_inputs(g, T, cfg, dtype=dtype)
    ref = L.layer_chain(inp, cfg["theta"], cfg["eps"], dtype, qknorm=qk)
    ts, out = chain_device(inp, dtype, qk, layout=layout)
    op = S.OP_LAYER_CHAIN_QKNORM if qk else S.OP_LAYER_CHAIN
    fixed = [cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["S"], cfg["I"]]
    lay = S.LAYOUT_ROWSTRIDED if (layout == "fused" and T > 1) else S.LAYOUT_CONTIG
    desc = S.make_spec(op, dtype, fixed, 1, 4096, layout=lay, rope_theta=cfg["theta"])
    run_one(S, desc, op, ts, pdl, eps=cfg["eps"], rope_theta=cfg["theta"])
    check_chain(ref, out, inp, dtype)


@pytest.mark.parametrize("seed", range(6))
def test_fuzz_step_replay(S, seed):
    """invoke_step over several independent layers, four steps on the same buffers with new
    data each time (steps 3 and 4 replay the stored chunk), then a fifth step in which one layer
    reads another's output (never replayed: it runs call by call). Every step's outputs are
    checked against the oracle on that step's data."""
    rng = random.Random(400 + seed)
    base = rng.choice([synth.LLAMA, synth.QWEN3])
    dtype = rng.choice([BF16, FP16])
    T = rng.choice([1, 3, 8, 17])
    n = rng.choice([2, 3, 5])
    cfg = dict(base, S=rng.choice([128, 8192]))
    qk = cfg["qknorm"]
    layout = rng.choice(["fused", "separate"])
    op = S.OP_LAYER_CHAIN_QKNORM if qk else S.OP_LAYER_CHAIN
    fixed = [cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["S"], cfg["I"]]
    lay = S.LAYOUT_ROWSTRIDED if (layout == "fused" and T > 1) else S.LAYOUT_CONTIG
    s = S.Scm(device=0, flags=S.OPT_PDL if rng.random() < 0.7 else 0)
    s.register(S.make_spec(op, dtype, fixed, 1, 4096, layout=lay, rope_theta=cfg["theta"]))
    g = np.random.default_rng(400 + seed)
    inps = [synth.layer_inputs(g, T, cfg, dtype=dtype) for _ in range(n)]
    dev = [chain_device(inp, dtype, qk, layout=layout) for inp in inps]
    args = [S.make_args(op, ts, eps=cfg["eps"], rope_theta=cfg["theta"]) for ts, _ in dev]

    def step(a):
        st, sel = s.invoke_step((S.trident_args * n)(*a), stream())
        assert st == S.OK and sel == [0] * n, S.trident_scm_last_error()
        torch.cuda.synchronize()
        assert S.trident_scm_device_status(s.h, stream())[1] == 0

    for k in range(4):
        if k:
            for l in range(n):
                inps[l] = synth.layer_inputs(g, T, cfg, dtype=dtype)
                fresh, _ = chain_device(inps[l], dtype, qk, layout=layout)
                for dst, src in zip(dev[l][0], fresh):
                    dst.copy_(src)
        step(args)
        for inp, (_, out) in zip(inps, dev):
            check_chain(L.layer_chain(inp, cfg["theta"], cfg["eps"], dtype, qknorm=qk), out, inp, dtype)
    st = s.stats()
    assert (st.step_replays, st.fused_launches) == (2 * n, 4)
    # layer 1 now reads layer 0's second residual output: dependent, run in order
    for l in range(n):
        inps[l] = synth.layer_inputs(g, T, cfg, dtype=dtype)
        fresh, _ = chain_device(inps[l], dtype, qk, layout=layout)
        for dst, src in zip(dev[l][0], fresh):
            dst.copy_(src)
    ts1 = list(dev[1][0])
    ts1[1] = dev[0][1]["r2"]
    dep = list(args)
    dep[1] = S.make_args(op, ts1, eps=cfg["eps"], rope_theta=cfg["theta"])
    step(dep)
    st = s.stats()
    assert (st.step_replays, st.fused_launches) == (2 * n, 4)
    s.close()
    ref0 = L.layer_chain(inps[0], cfg["theta"], cfg["eps"], dtype, qknorm=qk)
    inp1 = dict(inps[1], r0=ref0["r2"])
    check_chain(ref0, dev[0][1], inps[0], dtype)
    check_chain(L.layer_chain(inp1, cfg["theta"], cfg["eps"], dtype, qknorm=qk), dev[1][1], inp1, dtype)
    for l in range(2, n):
        check_chain(L.layer_chain(inps[l], cfg["theta"], cfg["eps"], dtype, qknorm=qk), dev[l][1], inps[l], dtype)
