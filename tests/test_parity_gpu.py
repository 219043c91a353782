"""GPU parity: every kernel family through the C ABI against the CPU oracle, on seeded
inputs that span several tiles and ragged tails, every layout and variant, in-place
calls, the degenerate cases, and sampled rows at the full workload sizes."""
import numpy as np
import pytest
import torch

from oracle import layer as L
from paper_2609_37241_gb300 import synth
from tests import parity as P

pytestmark = pytest.mark.gpu
BF16, FP16, FP32 = 1, 2, 3


@pytest.fixture(scope="module")
def S(built_lib):
    from paper_2609_37241_gb300 import scm
    return scm


def stream():
    return torch.cuda.current_stream().cuda_stream


def one_version_scm(S, desc, flags=0):
    s = S.Scm(device=0, flags=flags)
    s.register(desc)
    return s


def invoke_ok(s, S, args):
    st, sel = s.invoke(args, stream())
    assert st == S.OK, S.trident_scm_last_error()
    return sel


# ---------------------------------------------------------------------------- add + RMSNorm
ADDNORM_CASES = [
    # (dtype, H, T, layout, variant, note)
    (BF16, 4096, 1, "contig", 0, "register row, one token"),
    (BF16, 4096, 37, "contig", 0, "register row, ragged token count"),
    (BF16, 4096, 13, "strided", 0, "row-strided views"),
    (BF16, 4096, 21, "rank3", 0, "[3, 7, H] flattened"),
    (BF16, 8192, 19, "contig", 0, "register row, H 8192"),
    (BF16, 8192, 1500, "contig", 0, "H 8192 persistent grid: several rows per block"),
    (FP16, 8192, 700, "strided", 0, "fp16 H 8192 persistent, row-strided"),
    (BF16, 2048, 5, "contig", 0, "register row, H 2048"),
    (BF16, 1000, 5, "contig", 0, "two-pass vector loop, ragged H"),
    (BF16, 100, 6, "contig", 0, "H*2 not a multiple of 16: generic"),
    (BF16, 4096, 9, "misaligned", 1, "generic on a misaligned base"),
    (BF16, 4096, 9, "contig", 1, "generic forced"),
    (FP16, 4096, 9, "contig", 0, "fp16 register row"),
    (FP16, 520, 3, "strided", 0, "fp16 vector loop, strided"),
    (FP32, 4096, 9, "contig", 0, "fp32 register row"),
    (FP32, 1000, 4, "contig", 0, "fp32 vector loop"),
    (FP32, 99, 4, "contig", 0, "fp32 generic"),
]


def run_addnorm(S, dtype, H, T, layout, variant, inplace=False, seed=0):
    g = np.random.default_rng(seed)
    x, r = synth.act(g, (T, H), dtype), synth.act(g, (T, H), dtype)
    gam = synth.gamma(g, H)
    eps = 1e-6
    y_ref, y_bits, ro_bits = L.add_rmsnorm(x, r, gam, eps, dtype)
    es = 4 if dtype == FP32 else 2
    if layout == "strided":
        xd, rd = P.padded(x, dtype, 8), P.padded(r, dtype, 24)
        yd, rod = P.padded(np.zeros_like(x), dtype, 8), P.padded(np.zeros_like(r), dtype, 40)
        lay = S.LAYOUT_ROWSTRIDED
    elif layout == "misaligned":
        def off(bits):
            buf = torch.zeros(T * H + 1, dtype=synth._TORCH_DT[dtype], device="cuda")
            v = buf[1:].view(T, H)
            v.copy_(P.dev(bits, dtype))
            return v
        xd, rd, yd, rod = off(x), off(r), off(np.zeros_like(x)), off(np.zeros_like(r))
        lay = S.LAYOUT_CONTIG
    else:
        xd, rd = P.dev(x, dtype), P.dev(r, dtype)
        yd, rod = torch.empty_like(xd), torch.empty_like(rd)
        lay = S.LAYOUT_CONTIG
    if layout == "rank3":
        xd, rd, yd, rod = (t.view(3, T // 3, H) for t in (xd, rd, yd, rod))
    if inplace:
        yd, rod = xd, rd
    gd = torch.from_numpy(gam).cuda()
    rows16 = (H * es) % 16 == 0  # a 16-byte-aligned version needs 16-byte rows
    align = 16 if variant != 1 and layout != "misaligned" and rows16 else es
    desc = S.make_spec(S.OP_ADD_RMSNORM, dtype, [H], 1, 1 << 20, rank=3 if layout == "rank3" else 2,
                       layout=lay, align_bytes=align, variant=variant)
    s = one_version_scm(S, desc)
    invoke_ok(s, S, S.make_args(S.OP_ADD_RMSNORM, [xd, rd, gd, yd, rod], eps=eps))
    torch.cuda.synchronize()
    s.close()
    got_y = P.host_bits(yd.reshape(T, H), dtype)
    got_r = P.host_bits(rod.reshape(T, H), dtype)
    return got_y, got_r, y_ref, y_bits, ro_bits


@pytest.mark.parametrize("dtype,H,T,layout,variant,note", ADDNORM_CASES,
                         ids=[c[-1] for c in ADDNORM_CASES])
def test_add_rmsnorm_parity(S, dtype, H, T, layout, variant, note):
    got_y, got_r, y_ref, y_bits, ro_bits = run_addnorm(S, dtype, H, T, layout, variant)
    # the residual is a rounding decision of an fp32 sum: bit-exact
    assert np.array_equal(got_r, ro_bits), note
    P.check_act(got_y, y_ref, y_bits, dtype, "y " + note, exact_frac=0.99)


def test_add_rmsnorm_unaligned_rows_miss_an_aligned_version(S):
    """H 100 bf16 rows are 200 bytes: a 16-byte-aligned version must not be selected."""
    x = torch.zeros((2, 100), dtype=torch.bfloat16, device="cuda")
    gam = torch.ones(100, device="cuda")
    s = one_version_scm(S, S.make_spec(S.OP_ADD_RMSNORM, BF16, [100], 1, 8, align_bytes=16))
    st, sel = s.invoke(S.make_args(S.OP_ADD_RMSNORM, [x, x.clone(), gam, x.clone(), x.clone()]), stream())
    assert (st, sel) == (S.MISS, -1)
    s.close()


@pytest.mark.parametrize("H,variant,T", [(4096, 0, 7), (1000, 0, 7), (100, 0, 7), (4096, 1, 7),
                                         (8192, 0, 1300)])
def test_add_rmsnorm_in_place(S, H, variant, T):
    got_y, got_r, y_ref, y_bits, ro_bits = run_addnorm(S, BF16, H, T, "contig", variant, inplace=True)
    assert np.array_equal(got_r, ro_bits)
    P.check_act(got_y, y_ref, y_bits, BF16, "y in place")


def test_add_rmsnorm_degenerate_rows(S):
    """Zero row with eps 0 is 0/0: skip; constant row: closed form; huge values."""
    T, H = 3, 4096
    x = np.zeros((T, H), np.float32)
    x[0] = 1.5
    x[1] = 3e4
    x[2] = -2.0 ** -100
    xb = synth.to_bits(x, BF16)
    rb = synth.to_bits(np.zeros_like(x), BF16)
    gam = np.ones(H, np.float32)
    y_ref, y_bits, ro_bits = L.add_rmsnorm(xb, rb, gam, 1e-6, BF16)
    s = one_version_scm(S, S.make_spec(S.OP_ADD_RMSNORM, BF16, [H], 1, 8))
    xd, rd, gd = P.dev(xb, BF16), P.dev(rb, BF16), torch.from_numpy(gam).cuda()
    yd, rod = torch.empty_like(xd), torch.empty_like(rd)
    invoke_ok(s, S, S.make_args(S.OP_ADD_RMSNORM, [xd, rd, gd, yd, rod], eps=1e-6))
    torch.cuda.synchronize()
    P.check_act(P.host_bits(yd, BF16), y_ref, y_bits, BF16, "degenerate")
    assert np.array_equal(P.host_bits(rod, BF16), ro_bits)
    s.close()


def test_add_rmsnorm_bulk_copy_wait_timeout_path(S):
    """The bulk-copy kernel's bounded wait for its two row copies, made to run out: with
    TRIDENT_OPT_TEST_WAIT_TIMEOUT the first wait gives up at once, so every block sets the
    timeout bit, drains its copies with the full bounded wait and returns without writing.
    The outputs keep their sentinel, the status word says TRIDENT_DEVERR_TIMEOUT, and a
    following normal call on the same tensors is clean and matches the oracle."""
    T, H = 1024, 8192  # H 8192 bf16 from 1024 rows: the bulk-copy kernel
    g = np.random.default_rng(21)
    x, r = synth.act(g, (T, H), BF16), synth.act(g, (T, H), BF16)
    gam = synth.gamma(g, H)
    y_ref, y_bits, ro_bits = L.add_rmsnorm(x, r, gam, 1e-6, BF16)
    sentinel = np.full((T, H), synth.CACHE_SENTINEL, dtype=x.dtype)
    xd, rd, gd = P.dev(x, BF16), P.dev(r, BF16), torch.from_numpy(gam).cuda()
    yd, rod = P.dev(sentinel, BF16), P.dev(sentinel, BF16)
    desc = S.make_spec(S.OP_ADD_RMSNORM, BF16, [H], 1, 1 << 20)
    args = S.make_args(S.OP_ADD_RMSNORM, [xd, rd, gd, yd, rod], eps=1e-6)
    s = one_version_scm(S, desc, flags=S.OPT_TEST_WAIT_TIMEOUT)
    invoke_ok(s, S, args)
    st, bits = S.trident_scm_device_status(s.h, stream(), clear=True)
    assert st == S.OK and bits == S.DEVERR_TIMEOUT
    assert np.array_equal(P.host_bits(yd, BF16), sentinel)
    assert np.array_equal(P.host_bits(rod, BF16), sentinel)
    assert np.array_equal(P.host_bits(xd, BF16), x) and np.array_equal(P.host_bits(rd, BF16), r)
    s.close()
    s = one_version_scm(S, desc)
    invoke_ok(s, S, args)
    st, bits = S.trident_scm_device_status(s.h, stream())
    assert st == S.OK and bits == 0
    assert np.array_equal(P.host_bits(rod, BF16), ro_bits)
    P.check_act(P.host_bits(yd, BF16), y_ref, y_bits, BF16, "y after the timeout", exact_frac=0.99)
    s.close()


# ---------------------------------------------------------------------------- RMSNorm
RMSNORM_CASES = [
    # (dtype, H, T, layout, variant, note)
    (BF16, 128, 1024, "contig", 0, "the paper's rms_norm shape: 16-lane groups"),
    (BF16, 128, 37, "strided", 0, "16-lane groups, strided, ragged"),
    (BF16, 64, 5, "contig", 0, "8-lane groups"),
    (BF16, 256, 9, "contig", 0, "32-lane groups"),
    (BF16, 8, 300, "contig", 0, "one lane per row"),
    (BF16, 4096, 7, "contig", 0, "register row"),
    (BF16, 1000, 5, "contig", 0, "two-pass loop"),
    (BF16, 100, 4, "contig", 0, "generic (200-byte rows)"),
    (BF16, 128, 9, "misaligned", 1, "generic on a misaligned base"),
    (FP16, 128, 33, "contig", 0, "fp16 lane groups"),
    (FP32, 128, 17, "contig", 0, "fp32 32-lane groups"),
    (FP32, 4096, 3, "contig", 0, "fp32 register row"),
]


@pytest.mark.parametrize("dtype,H,T,layout,variant,note", RMSNORM_CASES,
                         ids=[c[-1] for c in RMSNORM_CASES])
def test_rmsnorm_parity(S, dtype, H, T, layout, variant, note):
    g = np.random.default_rng(H + T)
    x = synth.act(g, (T, H), dtype)
    gam = synth.gamma(g, H)
    y_ref, y_bits = L.rmsnorm(x, gam, 1e-6, dtype)
    es = 4 if dtype == FP32 else 2
    if layout == "strided":
        xd, yd = P.padded(x, dtype, 16), P.padded(np.zeros_like(x), dtype, 40)
        lay = S.LAYOUT_ROWSTRIDED
    elif layout == "misaligned":
        buf = torch.zeros(2 * T * H + 2, dtype=synth._TORCH_DT[dtype], device="cuda")
        xd = buf[1:T * H + 1].view(T, H)
        xd.copy_(P.dev(x, dtype))
        yd = buf[T * H + 1:2 * T * H + 1].view(T, H)
        lay = S.LAYOUT_CONTIG
    else:
        xd = P.dev(x, dtype)
        yd = torch.empty_like(xd)
        lay = S.LAYOUT_CONTIG
    align = 16 if variant != 1 and layout != "misaligned" and (H * es) % 16 == 0 else es
    s = one_version_scm(S, S.make_spec(S.OP_RMSNORM, dtype, [H], 1, 1 << 20, layout=lay,
                                       align_bytes=align, variant=variant))
    invoke_ok(s, S, S.make_args(S.OP_RMSNORM, [xd, torch.from_numpy(gam).cuda(), yd], eps=1e-6))
    torch.cuda.synchronize()
    s.close()
    P.check_act(P.host_bits(yd, dtype), y_ref, y_bits, dtype, note, exact_frac=0.99)


def test_rmsnorm_in_place(S):
    g = np.random.default_rng(3)
    x = synth.act(g, (64, 128), BF16)
    gam = synth.gamma(g, 128)
    y_ref, y_bits = L.rmsnorm(x, gam, 1e-6, BF16)
    xd = P.dev(x, BF16)
    s = one_version_scm(S, S.make_spec(S.OP_RMSNORM, BF16, [128], 1, 4096))
    invoke_ok(s, S, S.make_args(S.OP_RMSNORM, [xd, torch.from_numpy(gam).cuda(), xd], eps=1e-6))
    torch.cuda.synchronize()
    s.close()
    P.check_act(P.host_bits(xd, BF16), y_ref, y_bits, BF16, "rmsnorm in place")


# ---------------------------------------------------------------------------- pointwise
POINTWISE_CASES = [
    # (op name, dtype, W, T, layout, variant)
    ("silu", BF16, 4096, 33, "contig", 0), ("silu", FP16, 14336, 3, "strided", 0),
    ("silu", FP32, 1000, 5, "contig", 0), ("silu", BF16, 100, 7, "contig", 1),
    ("add", BF16, 4096, 17, "contig", 0), ("add", FP16, 520, 9, "strided", 0),
    ("add", FP32, 4096, 4, "contig", 0), ("add", BF16, 77, 5, "contig", 1),
    ("neg", BF16, 4096, 9, "contig", 0), ("neg", FP32, 36, 3, "contig", 1),
    ("masked_fill", BF16, 4096, 21, "contig", 0), ("masked_fill", FP16, 2048, 6, "strided", 0),
    ("masked_fill", FP32, 1024, 5, "contig", 0), ("masked_fill", BF16, 50, 4, "contig", 1),
]


@pytest.mark.parametrize("name,dtype,W,T,layout,variant", POINTWISE_CASES)
def test_pointwise_parity(S, name, dtype, W, T, layout, variant):
    g = np.random.default_rng(W + T)
    op = {"silu": S.OP_SILU, "add": S.OP_ADD, "neg": S.OP_NEG, "masked_fill": S.OP_MASKED_FILL}[name]
    a = synth.act(g, (T, W), dtype, std=3.0)
    b = synth.act(g, (T, W), dtype)
    mask = (g.random((T, W)) < 0.3).astype(np.uint8)
    value = -1e4
    if name == "silu":
        ref, ref_bits = L.silu(a, dtype)
    elif name == "add":
        ref, ref_bits = L.add(a, b, dtype)
    elif name == "neg":
        ref, ref_bits = L.neg(a, dtype)
    else:
        ref, ref_bits = L.masked_fill(a, mask, value, dtype)
    pad = 32 if layout == "strided" else 0
    dev = (lambda bits: P.padded(bits, dtype, pad)) if pad else (lambda bits: P.dev(bits, dtype))
    ad, bd, yd = dev(a), dev(b), dev(np.zeros_like(a))
    if pad:
        mbuf = torch.zeros((T, W + 64), dtype=torch.uint8, device="cuda")
        md = mbuf[:, :W]
        md.copy_(torch.from_numpy(mask).cuda())
    else:
        md = torch.from_numpy(mask).cuda()
    ts = {"silu": [ad, yd], "neg": [ad, yd], "add": [ad, bd, yd], "masked_fill": [ad, md, yd]}[name]
    es = 4 if dtype == FP32 else 2
    lay = S.LAYOUT_ROWSTRIDED if pad else S.LAYOUT_CONTIG
    align = 16 if variant != 1 and (W * es) % 16 == 0 else es
    s = one_version_scm(S, S.make_spec(op, dtype, [W], 1, 1 << 20, layout=lay, align_bytes=align,
                                       variant=variant))
    invoke_ok(s, S, S.make_args(op, ts, scalar=value))
    torch.cuda.synchronize()
    s.close()
    got = P.host_bits(yd, dtype)
    if name in ("neg", "masked_fill", "add"):
        assert np.array_equal(got, ref_bits), name  # exact operations / one rounding of an fp32 sum
    else:
        P.check_act(got, ref, ref_bits, dtype, name, exact_frac=0.99)


def test_pointwise_in_place(S):
    g = np.random.default_rng(21)
    a = synth.act(g, (8, 4096), BF16)
    b = synth.act(g, (8, 4096), BF16)
    ref, ref_bits = L.add(a, b, BF16)
    ad, bd = P.dev(a, BF16), P.dev(b, BF16)
    s = one_version_scm(S, S.make_spec(S.OP_ADD, BF16, [4096], 1, 64))
    invoke_ok(s, S, S.make_args(S.OP_ADD, [ad, bd, bd]))  # y = b
    torch.cuda.synchronize()
    s.close()
    assert np.array_equal(P.host_bits(bd, BF16), ref_bits)


# ---------------------------------------------------------------------------- RoPE + KV
def rope_inputs(g, T, Hq, Hkv, D, S_, dtype):
    q, k, v = (synth.act(g, (T, h, D), dtype) for h in (Hq, Hkv, Hkv))
    return q, k, v, synth.positions(g, T, S_)


def run_rope(S, T, Hq, Hkv, D, S_, theta, qknorm, dtype=BF16, layout="fused", variant=0,
             pos_override=None, seed=1, flags=0):
    g = np.random.default_rng(seed)
    q, k, v, pos = rope_inputs(g, T, Hq, Hkv, D, S_, dtype)
    if pos_override is not None:
        pos = pos_override
    gq, gk = synth.gamma(g, D), synth.gamma(g, D)
    kc, vc = synth.cache(Hkv, S_, D), synth.cache(Hkv, S_, D)
    ref = L.rope_kv(q, k, v, pos, kc, vc, theta, dtype, qknorm=qknorm, gamma_q=gq, gamma_k=gk, eps=1e-6)
    W = (Hq + 2 * Hkv) * D
    tdt = synth._TORCH_DT[dtype]
    if layout == "fused":
        extra = 1 if variant == 1 else 0
        buf = torch.zeros(T * W + extra, dtype=tdt, device="cuda")
        qkv = buf[extra:].view(T, W)
        qkv[:, :Hq * D] = P.dev(q, dtype).view(T, Hq * D)
        qkv[:, Hq * D:(Hq + Hkv) * D] = P.dev(k, dtype).view(T, Hkv * D)
        qkv[:, (Hq + Hkv) * D:] = P.dev(v, dtype).view(T, Hkv * D)
        qd = qkv[:, :Hq * D].view(T, Hq, D)
        kd = qkv[:, Hq * D:(Hq + Hkv) * D].view(T, Hkv, D)
        vd = qkv[:, (Hq + Hkv) * D:].view(T, Hkv, D)
        lay = S.LAYOUT_ROWSTRIDED if T > 1 else S.LAYOUT_CONTIG
    else:
        qd, kd, vd = P.dev(q, dtype), P.dev(k, dtype), P.dev(v, dtype)
        lay = S.LAYOUT_CONTIG
    kcd, vcd = P.dev(kc, dtype), P.dev(vc, dtype)
    posd = torch.from_numpy(pos).cuda()
    op = S.OP_QKNORM_ROPE_KV if qknorm else S.OP_ROPE_KV
    ts = [qd, kd, vd, posd, kcd, vcd]
    if qknorm:
        ts += [torch.from_numpy(gq).cuda(), torch.from_numpy(gk).cuda()]
    desc = S.make_spec(op, dtype, [Hq, Hkv, D, S_], 1, 1 << 20, layout=lay,
                       align_bytes=2 if variant == 1 else 16, variant=variant, rope_theta=theta)
    s = one_version_scm(S, desc, flags=flags)
    invoke_ok(s, S, S.make_args(op, ts, eps=1e-6, rope_theta=theta))
    st, bits = S.trident_scm_device_status(s.h, stream())
    assert st == S.OK
    s.close()
    return ref, dict(q=P.host_bits(qd, dtype), k_cache=P.host_bits(kcd, dtype),
                     v_cache=P.host_bits(vcd, dtype), k=P.host_bits(kd, dtype),
                     v=P.host_bits(vd, dtype), status=bits), (q, k, v, pos)


check_rope = P.check_rope


@pytest.mark.parametrize("T,qknorm,theta", [(1, False, 5e5), (5, False, 5e5), (64, False, 5e5),
                                            (1, True, 1e6), (8, True, 1e6), (128, True, 1e6)])
def test_rope_kv_decode_shapes(S, T, qknorm, theta):
    ref, got, inp = run_rope(S, T, 32, 8, 128, 8192, theta, qknorm)
    assert got["status"] == 0 and ref["bad"] == 0
    check_rope(ref, got, inp)


@pytest.mark.parametrize("D,variant,dtype,layout", [(64, 0, BF16, "fused"), (256, 0, FP16, "separate"),
                                                    (128, 1, BF16, "fused"), (48, 0, FP16, "fused"),
                                                    (128, 0, FP16, "fused")])
def test_rope_kv_head_sizes_and_generic(S, D, variant, dtype, layout):
    for qk in (False, True):
        ref, got, inp = run_rope(S, 7, 4, 2, D, 512, 1e4, qk, dtype=dtype, layout=layout,
                                 variant=variant, seed=D + variant)
        check_rope(ref, got, inp, dtype)


def test_rope_bad_positions_flag_and_skip(S):
    pos = np.array([5, 511, 512, -1, 100], np.int32)  # 512 and -1 are outside [0, 512)
    for variant in (0, 1):
        ref, got, inp = run_rope(S, 5, 4, 2, 128, 512, 1e4, True, pos_override=pos, variant=variant)
        assert ref["bad"] == 1 and got["status"] == S.DEVERR_POS
        check_rope(ref, got, inp)


@pytest.mark.parametrize("T,Hq,Hkv,D,S_,qk,dtype,layout", [
    (515, 32, 8, 128, 8192, False, BF16, "fused"),     # Llama heads; the last block holds 3 tokens
    (1024, 32, 8, 128, 8192, True, FP16, "separate"),  # Qwen3-style q/k norm
    (601, 4, 2, 64, 1024, True, BF16, "fused"),
    (512, 8, 8, 256, 600, False, FP16, "separate"),
    (2050, 16, 1, 128, 4096, False, BF16, "fused")])
def test_rope_kv_many_tokens(S, T, Hq, Hkv, D, S_, qk, dtype, layout):
    """Calls of at least 512 tokens: the bulk-copy kernel (a few tokens per block, their rows
    staged in shared memory, each token's angles computed once), ragged last blocks included."""
    ref, got, inp = run_rope(S, T, Hq, Hkv, D, S_, 5e5, qk, dtype=dtype, layout=layout, seed=T + D)
    assert got["status"] == 0 and ref["bad"] == 0
    check_rope(ref, got, inp, dtype)


def test_rope_kv_many_tokens_bad_positions(S):
    T = 603
    pos = synth.positions(np.random.default_rng(5), T, 8192)
    pos[100], pos[601] = 8192, -5  # outside [0, 8192): one in a full block, one in the last
    ref, got, inp = run_rope(S, T, 32, 8, 128, 8192, 5e5, True, pos_override=pos)
    assert ref["bad"] >= 1 and got["status"] == S.DEVERR_POS
    check_rope(ref, got, inp)


def test_rope_kv_bulk_copy_wait_timeout_path(S):
    """The bulk-copy RoPE kernel's bounded wait for its row copies, made to run out
    (TRIDENT_OPT_TEST_WAIT_TIMEOUT: the first wait gives up at once): every block sets the
    timeout bit, drains its copies with the full bounded wait and returns without writing,
    so q, k, v and both caches keep their contents."""
    T, Hq, Hkv, D, S_ = 600, 32, 8, 128, 8192
    ref, got, inp = run_rope(S, T, Hq, Hkv, D, S_, 5e5, False, flags=S.OPT_TEST_WAIT_TIMEOUT)
    q, k, v, _ = inp
    assert got["status"] == S.DEVERR_TIMEOUT
    assert np.array_equal(got["q"], q) and np.array_equal(got["k"], k) and np.array_equal(got["v"], v)
    sentinel = synth.cache(Hkv, S_, D)
    assert np.array_equal(got["k_cache"], sentinel) and np.array_equal(got["v_cache"], sentinel)


# ---------------------------------------------------------------------------- SwiGLU
SWIGLU_CASES = [(BF16, 14336, 1, "halves", 0), (BF16, 14336, 7, "halves", 0), (BF16, 12288, 3, "separate", 0),
                (BF16, 28672, 2, "separate", 0), (BF16, 48, 5, "separate", 0), (BF16, 100, 5, "separate", 0),
                (BF16, 4096, 3, "separate", 1), (FP16, 14336, 3, "halves", 0), (FP32, 1000, 3, "separate", 0),
                (FP32, 77, 3, "separate", 0)]


@pytest.mark.parametrize("dtype,I,T,layout,variant", SWIGLU_CASES)
def test_swiglu_parity(S, dtype, I, T, layout, variant):
    g = np.random.default_rng(I + T)
    gb = synth.act(g, (T, I), dtype, std=3.0)  # wider range exercises the exp tails
    ub = synth.act(g, (T, I), dtype)
    ref, ref_bits = L.swiglu(gb, ub, dtype)
    if layout == "halves":
        gu = torch.cat([P.dev(gb, dtype), P.dev(ub, dtype)], dim=1)
        gd, ud = gu[:, :I], gu[:, I:]
        lay = S.LAYOUT_ROWSTRIDED if T > 1 else S.LAYOUT_CONTIG
    else:
        gd, ud = P.dev(gb, dtype), P.dev(ub, dtype)
        lay = S.LAYOUT_CONTIG
    od = torch.empty((T, I), dtype=synth._TORCH_DT[dtype], device="cuda")
    es = 4 if dtype == FP32 else 2
    rows16 = (I * es) % 16 == 0
    s = one_version_scm(S, S.make_spec(S.OP_SWIGLU, dtype, [I], 1, 1 << 20, layout=lay,
                                       align_bytes=16 if variant != 1 and rows16 else es,
                                       variant=variant))
    invoke_ok(s, S, S.make_args(S.OP_SWIGLU, [gd, ud, od]))
    torch.cuda.synchronize()
    s.close()
    P.check_act(P.host_bits(od, dtype), ref, ref_bits, dtype, "swiglu", exact_frac=0.99)


def test_swiglu_in_place_and_extremes(S):
    vals = np.array([0.0, -0.0, 1.0, -1.0, 20.0, -20.0, 80.0, -80.0, 3e4, -3e4, 1e-30, -1e-30,
                     88.0, -87.0, 5.5, -5.5], np.float32)
    gb = synth.to_bits(np.tile(vals, (2, 1)), BF16)
    ub = synth.to_bits(np.tile(vals[::-1].copy(), (2, 1)), BF16)
    ref, ref_bits = L.swiglu(gb, ub, BF16)
    gd, ud = P.dev(gb, BF16), P.dev(ub, BF16)
    s = one_version_scm(S, S.make_spec(S.OP_SWIGLU, BF16, [16], 1, 8))
    invoke_ok(s, S, S.make_args(S.OP_SWIGLU, [gd, ud, gd]))  # out = g (in place)
    torch.cuda.synchronize()
    s.close()
    P.check_act(P.host_bits(gd, BF16), ref, ref_bits, BF16, "swiglu extremes")


# ---------------------------------------------------------------------------- chains
def chain_device(inp, dtype, qknorm, layout="fused"):
    """Device tensors in slot order for LAYER_CHAIN(_QKNORM); returns (list, outputs)."""
    T = inp["h"].shape[0]
    Hq, D = inp["q"].shape[1], inp["q"].shape[2]
    Hkv = inp["k"].shape[1]
    I = inp["g"].shape[1]
    d = lambda n: P.dev(inp[n], dtype)
    if layout == "fused":
        qkv = torch.cat([d("q").view(T, -1), d("k").view(T, -1), d("v").view(T, -1)], dim=1)
        q = qkv[:, :Hq * D].view(T, Hq, D)
        k = qkv[:, Hq * D:(Hq + Hkv) * D].view(T, Hkv, D)
        v = qkv[:, (Hq + Hkv) * D:].view(T, Hkv, D)
        gu = torch.cat([d("g"), d("u")], dim=1)
        g, u = gu[:, :I], gu[:, I:]
    else:
        q, k, v, g, u = d("q"), d("k"), d("v"), d("g"), d("u")
    out = dict(x1=torch.empty_like(d("h")), r1=torch.empty_like(d("h")), x2=torch.empty_like(d("h")),
               r2=torch.empty_like(d("h")), o=torch.empty((T, I), dtype=synth._TORCH_DT[dtype], device="cuda"),
               q=q, k_cache=d("k_cache"), v_cache=d("v_cache"))
    f32 = lambda n: torch.from_numpy(inp[n]).cuda()
    ts = [d("h"), d("r0"), f32("gamma_attn"), out["x1"], out["r1"], q, k, v,
          torch.from_numpy(inp["pos"]).cuda(), out["k_cache"], out["v_cache"], d("attn_out"),
          f32("gamma_mlp"), out["x2"], out["r2"], g, u, out["o"]]
    if qknorm:
        ts += [f32("gamma_q"), f32("gamma_k")]
    return ts, out


def check_chain(ref, out, inp, dtype=BF16):
    hb = lambda n: P.host_bits(out[n], dtype)
    assert np.array_equal(hb("r1"), ref["r1"]) and np.array_equal(hb("r2"), ref["r2"])
    P.check_act(hb("x1"), ref["x1_ref"], ref["x1"], dtype, "x1", exact_frac=0.99)
    P.check_act(hb("x2"), ref["x2_ref"], ref["x2"], dtype, "x2", exact_frac=0.99)
    P.check_act(hb("q"), ref["q_ref"], ref["q"], dtype, "q", exact_frac=0.99)
    P.check_act(hb("o"), ref["o_ref"], ref["o"], dtype, "o", exact_frac=0.99)
    pos = inp["pos"]
    P.check_act(hb("k_cache")[:, pos, :].transpose(1, 0, 2), ref["k_ref"],
                ref["k_cache"][:, pos, :].transpose(1, 0, 2), dtype, "k_cache")
    written = np.zeros(ref["k_cache"].shape[1], bool)
    written[pos] = True
    assert np.all(hb("k_cache")[:, ~written, :] == synth.CACHE_SENTINEL)
    assert np.array_equal(hb("v_cache"), ref["v_cache"])


@pytest.mark.parametrize("pdl", [False, True], ids=["plain", "pdl"])
@pytest.mark.parametrize("cfg_name,T", [("LLAMA", 1), ("LLAMA", 4), ("LLAMA", 16), ("LLAMA", 64),
                                        ("QWEN3", 1), ("QWEN3", 8), ("QWEN3", 32), ("QWEN3", 128),
                                        # without PDL, either side of the token-major /
                                        # role-major boundary (two blocks per SM: 33 Llama
                                        # tokens are 297 blocks, 34 are 306) and of the one-wave
                                        # limit of two norm CTAs; under PDL 16, 33, 34 Llama and
                                        # 8, 32, 40 Qwen3 tokens take the late-trigger entry,
                                        # 1 and 4 the token-major grid, 64 and 67 neither
                                        ("LLAMA", 33), ("LLAMA", 34), ("LLAMA", 67), ("QWEN3", 40)])
def test_layer_chain_fused_matches_oracle(S, cfg_name, T, pdl):
    """The benchmarked layer configurations, with and without programmatic dependent launch
    (with it, as bench.py launches: token-major grids prefetch every block's lines, larger ones
    the norm blocks' rows and their tokens' RoPE head-rows, before the wait)."""
    cfg = getattr(synth, cfg_name)
    g = np.random.default_rng(T)
    inp = synth.layer_inputs(g, T, cfg)
    qk = cfg["qknorm"]
    ref = L.layer_chain(inp, cfg["theta"], cfg["eps"], BF16, qknorm=qk)
    op = S.OP_LAYER_CHAIN_QKNORM if qk else S.OP_LAYER_CHAIN
    fixed = [cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["S"], cfg["I"]]
    lay = S.LAYOUT_ROWSTRIDED if T > 1 else S.LAYOUT_CONTIG
    s = one_version_scm(S, S.make_spec(op, BF16, fixed, 1, 4096, layout=lay, rope_theta=cfg["theta"]),
                        flags=S.OPT_PDL if pdl else 0)
    ts, out = chain_device(inp, BF16, qk)
    invoke_ok(s, S, S.make_args(op, ts, eps=cfg["eps"], rope_theta=cfg["theta"]))
    torch.cuda.synchronize()
    s.close()
    check_chain(ref, out, inp)


def test_layer_chain_largest_bucket(S):
    """The largest token count the benchmark's chain versions accept (4096 Llama tokens: a grid
    of 16,384 blocks several waves long -- one CTA per token for the norms, three head-rows per
    RoPE lane group, SwiGLU tiles of 4 x 256 vectors -- with the norm-row prefetch under PDL),
    every output against the oracle."""
    cfg = synth.LLAMA
    T = 4096
    g = np.random.default_rng(4096)
    inp = synth.layer_inputs(g, T, cfg)
    ref = L.layer_chain(inp, cfg["theta"], cfg["eps"], BF16)
    fixed = [cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["S"], cfg["I"]]
    s = one_version_scm(S, S.make_spec(S.OP_LAYER_CHAIN, BF16, fixed, 1, 4096, layout=S.LAYOUT_ROWSTRIDED,
                                       rope_theta=cfg["theta"]), flags=S.OPT_PDL)
    ts, out = chain_device(inp, BF16, False)
    invoke_ok(s, S, S.make_args(S.OP_LAYER_CHAIN, ts, eps=cfg["eps"], rope_theta=cfg["theta"]))
    torch.cuda.synchronize()
    assert S.trident_scm_device_status(s.h, stream())[1] == 0
    s.close()
    check_chain(ref, out, inp)


@pytest.mark.parametrize("dtype,H,Hq,I,T,qk", [
    (FP16, 4096, 32, 14336, 4, False),     # fp16 chain
    (BF16, 8192, 64, 28672, 3, False),     # H 8192 instantiation (4 vectors per thread)
    (BF16, 8192, 64, 28672, 200, True),    # H 8192, grid beyond one wave: one block per token
    (FP16, 8192, 64, 28672, 5, True),
    # several waves with 36 head-rows per token: three-row RoPE lane groups whose rows belong
    # to two tokens (the H 8192 case above covers it with q/k norm, 80 head-rows per token)
    (BF16, 4096, 20, 14336, 300, False),
])
@pytest.mark.parametrize("pdl", [False, True], ids=["plain", "pdl"])  # PDL: token-major / late trigger
def test_layer_chain_other_sizes_and_dtypes(S, dtype, H, Hq, I, T, qk, pdl):
    cfg = dict(H=H, Hq=Hq, Hkv=8, D=128, S=2048, I=I, theta=1e6, qknorm=qk, eps=1e-6)
    g = np.random.default_rng(H + T)
    inp = synth.layer_inputs(g, T, cfg, dtype=dtype)
    ref = L.layer_chain(inp, cfg["theta"], cfg["eps"], dtype, qknorm=qk)
    op = S.OP_LAYER_CHAIN_QKNORM if qk else S.OP_LAYER_CHAIN
    fixed = [H, Hq, 8, 128, 2048, I]
    lay = S.LAYOUT_ROWSTRIDED if T > 1 else S.LAYOUT_CONTIG
    s = one_version_scm(S, S.make_spec(op, dtype, fixed, 1, 4096, layout=lay, rope_theta=cfg["theta"]),
                        flags=S.OPT_PDL if pdl else 0)
    ts, out = chain_device(inp, dtype, qk)
    invoke_ok(s, S, S.make_args(op, ts, eps=cfg["eps"], rope_theta=cfg["theta"]))
    torch.cuda.synchronize()
    s.close()
    check_chain(ref, out, inp, dtype)


@pytest.mark.parametrize("pdl", [False, True])
def test_layer_chain_unfused_four_invokes_match(S, pdl):
    """The same layer as four invokes (one SCM, four versions) equals the oracle."""
    cfg = synth.QWEN3
    T = 8
    g = np.random.default_rng(77)
    inp = synth.layer_inputs(g, T, cfg)
    ref = L.layer_chain(inp, cfg["theta"], cfg["eps"], BF16, qknorm=True)
    s = S.Scm(device=0, flags=S.OPT_PDL if pdl else 0)
    s.register(S.make_spec(S.OP_ADD_RMSNORM, BF16, [4096], 1, 4096))
    s.register(S.make_spec(S.OP_QKNORM_ROPE_KV, BF16, [32, 8, 128, 8192], 1, 4096,
                           layout=S.LAYOUT_ROWSTRIDED, rope_theta=cfg["theta"]))
    s.register(S.make_spec(S.OP_SWIGLU, BF16, [cfg["I"]], 1, 4096, layout=S.LAYOUT_ROWSTRIDED))
    ts, out = chain_device(inp, BF16, True)
    (h, r0, ga, x1, r1, q, k, v, pos, kc, vc, ao, gm, x2, r2, gg, u, o, gq, gk) = ts
    seq = [S.make_args(S.OP_ADD_RMSNORM, [h, r0, ga, x1, r1]),
           S.make_args(S.OP_QKNORM_ROPE_KV, [q, k, v, pos, kc, vc, gq, gk], rope_theta=cfg["theta"]),
           S.make_args(S.OP_ADD_RMSNORM, [ao, r1, gm, x2, r2]),
           S.make_args(S.OP_SWIGLU, [gg, u, o])]
    arr = (S.trident_args * 4)(*seq)
    st, sel = S.trident_scm_invoke_seq(s.h, arr, stream())
    assert (st, sel) == (S.OK, [0, 1, 0, 2]), S.trident_scm_last_error()
    torch.cuda.synchronize()
    s.close()
    check_chain(ref, out, inp)


@pytest.mark.parametrize("T", [6, 700])  # 700: several waves (three-row RoPE lane groups, wide tiles)
def test_layer_chain_in_place_and_bad_position(S, T):
    cfg = synth.LLAMA
    g = np.random.default_rng(5)
    inp = synth.layer_inputs(g, T, cfg)
    inp["pos"][3] = cfg["S"] + 7  # out of range: token 3's rope/append skipped and flagged
    ref = L.layer_chain(inp, cfg["theta"], cfg["eps"], BF16)
    assert ref["bad"] == 1
    fixed = [cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["S"], cfg["I"]]
    s = one_version_scm(S, S.make_spec(S.OP_LAYER_CHAIN, BF16, fixed, 1, 1024, layout=S.LAYOUT_CONTIG,
                                       rope_theta=cfg["theta"]))
    ts, out = chain_device(inp, BF16, False, layout="separate")
    # in place: x1 = h, r1 = r0, x2 = attn_out, r2 = r1, o = g
    ts[3], ts[4], ts[13], ts[14], ts[17] = ts[0], ts[1], ts[11], ts[1], ts[15]
    out.update(x1=ts[0], r1=None, x2=ts[11], r2=ts[1], o=ts[15])
    invoke_ok(s, S, S.make_args(S.OP_LAYER_CHAIN, ts, eps=cfg["eps"], rope_theta=cfg["theta"]))
    st, bits = S.trident_scm_device_status(s.h, stream())
    s.close()
    assert bits == S.DEVERR_POS
    hb = lambda t: P.host_bits(t, BF16)
    assert np.array_equal(hb(out["r2"]), ref["r2"])
    P.check_act(hb(out["x1"]), ref["x1_ref"], ref["x1"], BF16, "x1")
    P.check_act(hb(out["x2"]), ref["x2_ref"], ref["x2"], BF16, "x2")
    P.check_act(hb(out["o"]), ref["o_ref"], ref["o"], BF16, "o")
    ok = np.arange(T) != 3
    P.check_act(hb(out["q"])[ok], ref["q_ref"][ok], ref["q"][ok], BF16, "q")
    assert np.array_equal(hb(out["q"])[3], inp["q"][3])


# ---------------------------------------------------------------------------- full sizes
def test_full_size_sweep_sampled_rows(S):
    """Bandwidth-sweep sizes in the launch configuration the benchmark times (T 32768,
    H 8192, I 28672): sampled rows against the oracle."""
    T, H, I = 32768, 8192, 28672
    x = synth.act_device((T, H), BF16, 1)
    r = synth.act_device((T, H), BF16, 2)
    gam = synth.gamma_device(H, 3)
    y, ro = torch.empty_like(x), torch.empty_like(r)
    s = S.Scm(device=0)
    s.register(S.make_spec(S.OP_ADD_RMSNORM, BF16, [H], 1, 1 << 20))
    s.register(S.make_spec(S.OP_SWIGLU, BF16, [I], 1, 1 << 20))
    invoke_ok(s, S, S.make_args(S.OP_ADD_RMSNORM, [x, r, gam, y, ro]))
    rows = np.sort(np.random.default_rng(0).choice(T, 48, replace=False))
    rows = np.concatenate([[0, T - 1], rows])
    idx = torch.from_numpy(rows).cuda()
    hb = lambda t: P.host_bits(t.index_select(0, idx), BF16)
    y_ref, y_bits, ro_bits = L.add_rmsnorm(hb(x), hb(r), gam.cpu().numpy(), 1e-6, BF16)
    assert np.array_equal(hb(ro), ro_bits)
    P.check_act(hb(y), y_ref, y_bits, BF16, "y full size")
    del x, r, y, ro
    g = synth.act_device((T, I), BF16, 4)
    u = synth.act_device((T, I), BF16, 5)
    o = torch.empty_like(g)
    invoke_ok(s, S, S.make_args(S.OP_SWIGLU, [g, u, o]))
    ref, ref_bits = L.swiglu(hb(g), hb(u), BF16)
    P.check_act(hb(o), ref, ref_bits, BF16, "swiglu full size")
    s.close()
