"""The benchmarked workloads replayed as parity tests, in the launch configuration bench.py
times: a single add+RMSNorm call repeated 1000 times over a 4-version table; the 100k-call
dynamic-shape guard stress (static table and growth through the compile hook), selection
bit-exact against the oracle's replay and numerics sampled; and a 36-layer Qwen3-style step
through one table, every layer checked."""
import ctypes

import numpy as np
import pytest
import torch

from oracle import guards as G
from oracle import layer as L
from paper_2609_37241_gb300 import synth
from tests import parity as P

pytestmark = pytest.mark.gpu
BF16, FP16 = 1, 2


@pytest.fixture(scope="module")
def S(built_lib):
    from paper_2609_37241_gb300 import scm
    return scm


def stream():
    return torch.cuda.current_stream().cuda_stream


def test_single_addnorm_1000_invocations_hit_bf16_contig(S):
    H = 4096
    s = S.Scm(device=0)
    for dt, lay in ((FP16, S.LAYOUT_CONTIG), (FP16, S.LAYOUT_ROWSTRIDED), (BF16, S.LAYOUT_ROWSTRIDED),
                    (BF16, S.LAYOUT_CONTIG)):
        s.register(S.make_spec(S.OP_ADD_RMSNORM, dt, [H], 1, 1, layout=lay))
    g = np.random.default_rng(0)
    x, r, gam = synth.act(g, (1, H), BF16), synth.act(g, (1, H), BF16), synth.gamma(g, H)
    xd, rd, gd = P.dev(x, BF16), P.dev(r, BF16), torch.from_numpy(gam).cuda()
    yd, rod = torch.empty_like(xd), torch.empty_like(rd)
    a = S.make_args(S.OP_ADD_RMSNORM, [xd, rd, gd, yd, rod], eps=1e-6)
    sels = [s.invoke(a, stream()) for _ in range(1000)]
    torch.cuda.synchronize()
    assert all(v == (S.OK, 3) for v in sels)
    assert S.trident_scm_spec_hits(s.h)[1] == [0, 0, 0, 1000]
    y_ref, y_bits, ro_bits = L.add_rmsnorm(x, r, gam, 1e-6, BF16)
    assert np.array_equal(P.host_bits(rod, BF16), ro_bits)
    P.check_act(P.host_bits(yd, BF16), y_ref, y_bits, BF16, "y")
    s.close()


@pytest.mark.parametrize("mode", ["static", "growth"])
def test_guard_stress_100k_selection_and_sampled_numerics(S, mode):
    cfg = synth.STRESS
    H, pad = cfg["H"], cfg["pad"]
    Ts, dts, strided = synth.stress_trace(np.random.default_rng(0), cfg)
    Tmax = int(Ts.max())
    g = np.random.default_rng(1)
    data = {dt: (synth.act(g, (Tmax, H), dt), synth.act(g, (Tmax, H), dt)) for dt in (BF16, FP16)}
    gam = synth.gamma(g, H)
    gd = torch.from_numpy(gam).cuda()
    bufs = {}
    for dt in (BF16, FP16):
        tdt = synth._TORCH_DT[dt]
        xb = torch.zeros((Tmax, H + pad), dtype=tdt, device="cuda")
        rb = torch.zeros((Tmax, H + pad), dtype=tdt, device="cuda")
        xb[:, :H] = P.dev(data[dt][0], dt)
        rb[:, :H] = P.dev(data[dt][1], dt)
        bufs[dt] = (xb, rb, torch.empty((Tmax, H + pad), dtype=tdt, device="cuda"),
                    torch.empty((Tmax, H + pad), dtype=tdt, device="cuda"))

    generic = S.Scm(device=0)
    for dt in (BF16, FP16):
        generic.register(S.make_spec(S.OP_ADD_RMSNORM, dt, [H], 1, 1 << 40, layout=S.LAYOUT_ANY,
                                     align_bytes=2, variant=S.VARIANT_GENERIC))
    table = []
    if mode == "static":
        for b in range(8):
            lo, hi = G.bucket_range(b)
            for dt in (BF16, FP16):
                table.append(dict(op=1, dtype=dt, rank=2, layout=0, fixed=(H,), tok_lo=lo, tok_hi=hi,
                                  align=16, device=0, variant=0, theta=0.0))

    def hook(scm, args, st):
        if mode == "static":
            assert generic.invoke(args, st)[0] == S.OK
            return None
        T = int(args.t[0].shape[0])
        lo, hi = G.bucket_range(G.bucket_of(T))
        lay = S.LAYOUT_CONTIG if args.t[0].stride[0] == H or T == 1 else S.LAYOUT_ROWSTRIDED
        idx = scm.register(S.make_spec(S.OP_ADD_RMSNORM, int(args.t[0].dtype), [H], lo, hi, layout=lay))
        assert scm.invoke(args, st)[0] == S.OK
        return idx

    s = S.Scm(device=0, max_specs=64, hook=hook)
    for sp in table:
        s.register(S.make_spec(1, sp["dtype"], [H], sp["tok_lo"], sp["tok_hi"]))
    cache, memo = {}, {}
    sample = set(np.random.default_rng(2).choice(len(Ts), 40, replace=False).tolist())
    sel = ctypes.c_int32(-1)
    inv = S.lib().trident_scm_invoke
    mism = 0
    for i, (T, dt, st) in enumerate(zip(Ts, dts, strided)):
        T, dt, st = int(T), int(dt), bool(st)
        key = (T, dt, st)
        if key not in cache:
            xb, rb, yb, ob = bufs[dt]
            view = (lambda b: b[:T, :H]) if st else (lambda b: b.view(-1)[:T * H].view(T, H))
            full = [view(xb), view(rb), gd, view(yb), view(ob)]
            cache[key] = (S.make_args(S.OP_ADD_RMSNORM, full, eps=1e-6),
                          dict(op=1, tensors=[dict(addr=t.data_ptr(), dtype=(3 if t.dtype == torch.float32 else dt),
                                                   shape=tuple(t.shape), stride=tuple(t.stride()), device=0)
                                              for t in full], eps=1e-6, theta=0.0, flags=0), full)
        a, od, full = cache[key]
        rc = inv(s.h, ctypes.byref(a), ctypes.c_void_p(stream()), ctypes.byref(sel))
        mkey = (len(table), key)
        if mkey not in memo:
            memo[mkey] = G.select(table, od, check_overlap=False)
        ost, oidx = memo[mkey]
        if rc == S.OK:
            mism += not (ost == G.OK and oidx == sel.value)
        else:
            assert rc == S.MISS_HANDLED, (rc, S.trident_scm_last_error(), s.hook_error)
            mism += ost != G.MISS
            if mode == "growth":
                lo, hi = G.bucket_range(G.bucket_of(T))
                table.append(dict(op=1, dtype=dt, rank=2, layout=1 if (st and T > 1) else 0, fixed=(H,),
                                  tok_lo=lo, tok_hi=hi, align=16, device=0, variant=0, theta=0.0))
        if i in sample:  # this call's outputs against the oracle
            torch.cuda.synchronize()
            x, r = P.host_bits(full[0], dt), P.host_bits(full[1], dt)  # the view's contents
            y_ref, y_bits, ro_bits = L.add_rmsnorm(x, r, gam, 1e-6, dt)
            assert np.array_equal(P.host_bits(full[4], dt), ro_bits)
            P.check_act(P.host_bits(full[3], dt), y_ref, y_bits, dt, f"call {i}")
    torch.cuda.synchronize()
    assert mism == 0
    stats = s.stats()
    if mode == "static":
        assert stats.hits + stats.misses == len(Ts)
        assert 0.8 < stats.hits / len(Ts) < 0.9
    else:  # each miss registers, then re-invokes from the hook: one nested hit per miss
        assert stats.misses == stats.hook_registered == stats.num_specs
        assert stats.hits + stats.misses == len(Ts) + stats.hook_registered
    s.close()
    generic.close()


def test_qwen3_36_layers_through_one_table(S):
    cfg = synth.QWEN3
    T, layers = 8, cfg["layers"]
    fixed = [cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["S"], cfg["I"]]
    s = S.Scm(device=0, flags=S.OPT_PDL)
    s.register(S.make_spec(S.OP_LAYER_CHAIN_QKNORM, BF16, fixed, 1, 4096, layout=S.LAYOUT_CONTIG,
                           rope_theta=cfg["theta"]))
    g = np.random.default_rng(36)
    inps, outs, args = [], [], []
    for l in range(layers):
        inp = synth.layer_inputs(g, T, cfg)
        d = lambda n: P.dev(inp[n], BF16)
        f = lambda n: torch.from_numpy(inp[n]).cuda()
        o = dict(x1=torch.empty((T, cfg["H"]), dtype=torch.bfloat16, device="cuda"),
                 r1=torch.empty((T, cfg["H"]), dtype=torch.bfloat16, device="cuda"),
                 x2=torch.empty((T, cfg["H"]), dtype=torch.bfloat16, device="cuda"),
                 r2=torch.empty((T, cfg["H"]), dtype=torch.bfloat16, device="cuda"),
                 o=torch.empty((T, cfg["I"]), dtype=torch.bfloat16, device="cuda"),
                 q=d("q"), k_cache=d("k_cache"), v_cache=d("v_cache"))
        ts = [d("h"), d("r0"), f("gamma_attn"), o["x1"], o["r1"], o["q"], d("k"), d("v"),
              torch.from_numpy(inp["pos"]).cuda(), o["k_cache"], o["v_cache"], d("attn_out"),
              f("gamma_mlp"), o["x2"], o["r2"], d("g"), d("u"), o["o"], f("gamma_q"), f("gamma_k")]
        args.append(S.make_args(S.OP_LAYER_CHAIN_QKNORM, ts, eps=cfg["eps"], rope_theta=cfg["theta"]))
        inps.append(inp)
        outs.append((o, ts))
    arr = (S.trident_args * layers)(*args)
    st, sel = S.trident_scm_invoke_seq(s.h, arr, stream())
    assert st == S.OK and sel == [0] * layers, S.trident_scm_last_error()
    torch.cuda.synchronize()
    for l in range(layers):
        ref = L.layer_chain(inps[l], cfg["theta"], cfg["eps"], BF16, qknorm=True)
        o = outs[l][0]
        hb = lambda t: P.host_bits(t, BF16)
        assert np.array_equal(hb(o["r1"]), ref["r1"]) and np.array_equal(hb(o["r2"]), ref["r2"])
        P.check_act(hb(o["x2"]), ref["x2_ref"], ref["x2"], BF16, f"layer {l} x2")
        P.check_act(hb(o["q"]), ref["q_ref"], ref["q"], BF16, f"layer {l} q")
        P.check_act(hb(o["o"]), ref["o_ref"], ref["o"], BF16, f"layer {l} o")
        assert np.array_equal(hb(o["v_cache"]), ref["v_cache"])
    s.close()


@pytest.mark.parametrize("pdl", [False, True])
def test_launch_floor_probe_runs(S, pdl):
    """The latency-floor probe launches its empty kernels through the hit path's launch code
    (with and without programmatic dependent launch) and leaves the stream usable."""
    s = S.Scm(device=0, flags=S.OPT_PDL if pdl else 0)
    st = torch.cuda.current_stream().cuda_stream
    assert S.trident_launch_floor(s.h, st, 100) == S.OK, S.trident_scm_last_error()
    assert S.trident_launch_floor(s.h, st, 0) == S.OK
    torch.cuda.synchronize()
    assert S.trident_scm_device_status(s.h, st)[1] == 0
    s.close()


def test_launch_floor_records_each_launch_with_timing(S):
    """With TRIDENT_OPT_TIMING every launch of the probe leaves one host-time sample (the
    launch call alone), and no hit or miss is counted for it."""
    s = S.Scm(device=0, flags=S.OPT_PDL | S.OPT_TIMING)
    st = torch.cuda.current_stream().cuda_stream
    assert S.trident_launch_floor(s.h, st, 37) == S.OK, S.trident_scm_last_error()
    torch.cuda.synchronize()
    rc, ns = S.trident_scm_host_times(s.h, 100)
    assert rc == S.OK and len(ns) == 37 and all(0 < x < 10 ** 9 for x in ns)
    stats = s.stats()
    assert stats.hits == 0 and stats.misses == 0
    s.close()


@pytest.mark.parametrize("pdl", [False, True])
def test_copy_floor_probe_writes_the_xor_of_each_threads_reads(S, pdl):
    """The copy-floor probe: launch i reads set i % sets and writes set i % sets; each written
    vector is the XOR of the 16-byte vectors its thread read (a model in numpy, ragged grid
    shares included)."""
    blocks, sets, rb, wb = 7, 2, 16 * 1000, 16 * 333
    g = np.random.default_rng(3)
    src_h = g.integers(0, 2 ** 32, size=(sets, rb // 4), dtype=np.uint32)
    src = torch.from_numpy(src_h.view(np.int32)).cuda()
    dst = torch.zeros((sets, wb // 4), dtype=torch.int32, device="cuda")
    s = S.Scm(device=0, flags=S.OPT_PDL if pdl else 0)
    st = torch.cuda.current_stream().cuda_stream
    assert S.trident_copy_floor(s.h, st, src.data_ptr(), dst.data_ptr(), rb, wb, blocks, sets, sets) == S.OK, \
        S.trident_scm_last_error()
    torch.cuda.synchronize()
    s.close()
    got = dst.cpu().numpy().view(np.uint32).reshape(sets, -1, 4)
    nr, nw = rb // 16, wb // 16
    rpb, wpb = -(-nr // blocks), -(-nw // blocks)
    for k in range(sets):
        vec = src_h[k].reshape(-1, 4)
        want = np.zeros((nw, 4), np.uint32)
        for b in range(blocks):
            acc = np.zeros((256, 4), np.uint32)
            for i in range(rpb):
                if b * rpb + i < nr:
                    acc[i % 256] ^= vec[b * rpb + i]
            for j in range(wpb):
                if b * wpb + j < nw:
                    want[b * wpb + j] = acc[j % 256]
        assert np.array_equal(got[k], want), k
