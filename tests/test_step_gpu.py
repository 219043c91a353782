"""trident_scm_invoke_step on the GPU: a decoder step's layer chains in one launch (or
call by call when they depend on each other), every layer's outputs against the oracle.
Covers both norm splits (two CTAs per token while the step's grid fits one wave, one
otherwise), in-place calls, fp16, a step longer than one chunk, and a dependent step."""
import numpy as np
import pytest
import torch

from oracle import layer as L
from paper_2609_37241_gb300 import synth
from tests import parity as P
from tests.test_parity_gpu import chain_device, check_chain

pytestmark = pytest.mark.gpu
BF16, FP16 = 1, 2


@pytest.fixture(scope="module")
def S(built_lib):
    from paper_2609_37241_gb300 import scm
    return scm


def stream():
    return torch.cuda.current_stream().cuda_stream


def step_scm(S, cfg, dtype, lay):
    op = S.OP_LAYER_CHAIN_QKNORM if cfg["qknorm"] else S.OP_LAYER_CHAIN
    fixed = [cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["S"], cfg["I"]]
    s = S.Scm(device=0, flags=S.OPT_PDL)
    s.register(S.make_spec(op, dtype, fixed, 1, 4096, layout=lay, rope_theta=cfg["theta"]))
    return s, op


def build_layers(S, cfg, T, n, dtype=BF16, seed=0, layout="fused"):
    g = np.random.default_rng(seed)
    op = S.OP_LAYER_CHAIN_QKNORM if cfg["qknorm"] else S.OP_LAYER_CHAIN
    inps, outs, args = [], [], []
    for _ in range(n):
        inp = synth.layer_inputs(g, T, cfg, dtype=dtype)
        ts, out = chain_device(inp, dtype, cfg["qknorm"], layout=layout)
        inps.append(inp)
        outs.append((ts, out))
        args.append(S.make_args(op, ts, eps=cfg["eps"], rope_theta=cfg["theta"]))
    return inps, outs, args


def run_step(S, s, args):
    arr = (S.trident_args * len(args))(*args)
    st, sel = S.trident_scm_invoke_step(s.h, arr, stream())
    assert st == S.OK, S.trident_scm_last_error()
    assert S.trident_scm_device_status(s.h, stream())[1] == 0
    return sel


def test_step_qwen3_36_layers_one_launch(S):
    cfg = synth.QWEN3
    T = 8
    s, _ = step_scm(S, cfg, BF16, S.LAYOUT_ROWSTRIDED)
    inps, outs, args = build_layers(S, cfg, T, cfg["layers"], seed=36)
    assert run_step(S, s, args) == [0] * cfg["layers"]
    st = s.stats()
    assert (st.fused_launches, st.fused_calls) == (1, cfg["layers"])
    s.close()
    for inp, (_, out) in zip(inps, outs):
        check_chain(L.layer_chain(inp, cfg["theta"], cfg["eps"], BF16, qknorm=True), out, inp)


@pytest.mark.parametrize("T", [1, 16, 64])
def test_step_llama_layers_both_splits(S, T):
    # 4 Llama layers: 144 blocks per layer at T = 16 fit one wave together (two CTAs per
    # token); at T = 64 they do not (one CTA per token)
    cfg = synth.LLAMA
    lay = S.LAYOUT_ROWSTRIDED if T > 1 else S.LAYOUT_CONTIG
    s, _ = step_scm(S, cfg, BF16, lay)
    inps, outs, args = build_layers(S, cfg, T, 4, seed=T)
    run_step(S, s, args)
    assert s.stats().fused_launches == 1
    s.close()
    for inp, (_, out) in zip(inps, outs):
        check_chain(L.layer_chain(inp, cfg["theta"], cfg["eps"], BF16), out, inp)


def test_step_in_place_layers(S):
    cfg = synth.LLAMA
    T = 5
    s, op = step_scm(S, cfg, BF16, S.LAYOUT_CONTIG)
    inps, outs, _ = build_layers(S, cfg, T, 3, seed=9, layout="separate")
    refs, args, views = [], [], []
    for inp, (ts, out) in zip(inps, outs):
        refs.append(L.layer_chain(inp, cfg["theta"], cfg["eps"], BF16))
        # x1 = h, r1 = r0, x2 = attn_out, r2 = r1, o = g
        ts[3], ts[4], ts[13], ts[14], ts[17] = ts[0], ts[1], ts[11], ts[1], ts[15]
        views.append(dict(x1=ts[0], x2=ts[11], r2=ts[1], o=ts[15], q=out["q"], v_cache=out["v_cache"]))
        args.append(S.make_args(op, ts, eps=cfg["eps"], rope_theta=cfg["theta"]))
    run_step(S, s, args)
    assert s.stats().fused_launches == 1
    s.close()
    hb = lambda t: P.host_bits(t, BF16)
    for ref, v in zip(refs, views):
        assert np.array_equal(hb(v["r2"]), ref["r2"])
        assert np.array_equal(hb(v["v_cache"]), ref["v_cache"])
        P.check_act(hb(v["x1"]), ref["x1_ref"], ref["x1"], BF16, "x1")
        P.check_act(hb(v["x2"]), ref["x2_ref"], ref["x2"], BF16, "x2")
        P.check_act(hb(v["q"]), ref["q_ref"], ref["q"], BF16, "q")
        P.check_act(hb(v["o"]), ref["o_ref"], ref["o"], BF16, "o")


def test_step_dependent_layers_run_in_order(S):
    # layer 1 reads layer 0's second residual as its residual input: not independent, so
    # the step runs call by call and layer 1 sees layer 0's result
    cfg = synth.LLAMA
    T = 4
    s, op = step_scm(S, cfg, BF16, S.LAYOUT_ROWSTRIDED)
    inps, outs, args = build_layers(S, cfg, T, 2, seed=21)
    ts1 = outs[1][0]
    ts1[1] = outs[0][1]["r2"]
    args[1] = S.make_args(op, ts1, eps=cfg["eps"], rope_theta=cfg["theta"])
    run_step(S, s, args)
    st = s.stats()
    assert (st.fused_launches, st.hits) == (0, 2)
    s.close()
    ref0 = L.layer_chain(inps[0], cfg["theta"], cfg["eps"], BF16)
    inp1 = dict(inps[1], r0=ref0["r2"])
    check_chain(ref0, outs[0][1], inps[0])
    check_chain(L.layer_chain(inp1, cfg["theta"], cfg["eps"], BF16), outs[1][1], inp1)


def test_step_fp16_longer_than_one_chunk(S):
    # 50 layers at T = 1 (48 per launch, then 2), fp16, a short cache
    cfg = dict(synth.LLAMA, S=64)
    s, _ = step_scm(S, cfg, FP16, S.LAYOUT_CONTIG)
    inps, outs, args = build_layers(S, cfg, 1, 50, dtype=FP16, seed=50)
    run_step(S, s, args)
    st = s.stats()
    assert (st.fused_launches, st.fused_calls) == (2, 50)
    s.close()
    for inp, (_, out) in zip(inps, outs):
        check_chain(L.layer_chain(inp, cfg["theta"], cfg["eps"], FP16), out, inp, FP16)


@pytest.mark.parametrize("entry,T,model", [("invoke", 64, "LLAMA"), ("step", 64, "LLAMA"), ("invoke", 4, "LLAMA"),
                                           ("step", 4, "LLAMA"), ("invoke", 64, "QWEN3"), ("invoke", 128, "LLAMA"),
                                           ("invoke", 128, "QWEN3")])
def test_dependent_layers_back_to_back_with_pdl(S, entry, T, model):
    """Six layers where layer l+1's residual input is layer l's second residual output,
    launched back to back with programmatic dependent launch (one invoke each through the
    fast-call shim, or one invoke_step that must fall back to call-by-call order). Each
    kernel's memory accesses wait for the previous kernel, so every layer equals the oracle
    run in sequence. At 4 tokens the grid is small: it is token-major and prefetches its rows
    into L2 before the wait, while the previous layer still writes them; at 64 and 128 tokens
    the norm blocks prefetch their rows and their token's RoPE head-rows before the wait (two
    CTAs per token at 64, one at 128)."""
    import ctypes
    cfg = getattr(synth, model)
    n = 6
    s, op = step_scm(S, cfg, BF16, S.LAYOUT_ROWSTRIDED)
    inps, outs, args = build_layers(S, cfg, T, n, seed=606)
    for l in range(1, n):
        ts = outs[l][0]
        ts[1] = outs[l - 1][1]["r2"]
        args[l] = S.make_args(op, ts, eps=cfg["eps"], rope_theta=cfg["theta"])
    st = stream()
    if entry == "invoke":
        fc = S.fastcall()
        for a in args:
            rc = fc.invoke(s.h.value, ctypes.addressof(a), st) if fc else S.trident_scm_invoke(s.h, a, st)[0]
            assert rc == S.OK, S.trident_scm_last_error()
    else:
        run_step(S, s, args)
        assert s.stats().fused_launches == 0
    torch.cuda.synchronize()
    assert S.trident_scm_device_status(s.h, st)[1] == 0
    s.close()
    r0 = inps[0]["r0"]
    for l in range(n):
        inp = dict(inps[l], r0=r0)
        ref = L.layer_chain(inp, cfg["theta"], cfg["eps"], BF16, qknorm=cfg["qknorm"])
        check_chain(ref, outs[l][1], inp)
        r0 = ref["r2"]


def test_step_replays_follow_new_data(S):
    """A decode loop's pattern: the same buffers every step with new data in them. From the
    third step on the chunk is relaunched from the replay cache (only argument bytes are
    compared); each step's outputs equal the oracle on that step's data."""
    cfg = synth.QWEN3
    T, n = 4, 6
    s, _ = step_scm(S, cfg, BF16, S.LAYOUT_ROWSTRIDED)
    inps, outs, args = build_layers(S, cfg, T, n, seed=70)
    for step in range(4):
        if step:
            g = np.random.default_rng(700 + step)
            for l in range(n):
                inps[l] = synth.layer_inputs(g, T, cfg)
                fresh, _ = chain_device(inps[l], BF16, True)
                for dst, src in zip(outs[l][0], fresh):
                    dst.copy_(src)
        assert run_step(S, s, args) == [0] * n
        torch.cuda.synchronize()
        for inp, (_, out) in zip(inps, outs):
            check_chain(L.layer_chain(inp, cfg["theta"], cfg["eps"], BF16, qknorm=True), out, inp)
    st = s.stats()
    assert (st.step_replays, st.fused_launches, st.hits) == (2 * n, 4, 4 * n)
    s.close()


def test_multi_wave_steps_back_to_back(S):
    """Steps whose blocks outnumber the resident slots (several waves), 70 launches back to
    back under PDL, most of them from the replay cache, with new data in the same buffers at
    two points; every layer of every checked step equals the oracle."""
    cfg = synth.QWEN3
    T, n = 32, 6  # 6 x 288 blocks with one CTA per token: several waves
    s, _ = step_scm(S, cfg, BF16, S.LAYOUT_ROWSTRIDED)
    inps, outs, args = build_layers(S, cfg, T, n, seed=90)
    for step in range(70):
        if step in (40, 69):  # new data in the same buffers (inputs, caches and outputs)
            g = np.random.default_rng(900 + step)
            for l in range(n):
                inps[l] = synth.layer_inputs(g, T, cfg)
                fresh, _ = chain_device(inps[l], BF16, True)
                for dst, src in zip(outs[l][0], fresh):
                    dst.copy_(src)
        assert run_step(S, s, args) == [0] * n
        if step in (0, 40, 69):
            torch.cuda.synchronize()
            for inp, (_, out) in zip(inps, outs):
                check_chain(L.layer_chain(inp, cfg["theta"], cfg["eps"], BF16, qknorm=True), out, inp)
    st = s.stats()
    assert st.fused_launches == 70 and st.step_replays > 0
    s.close()
