"""The allocation-free RoPE/KV entry point (trident_rope_kv_noalloc).

Some callers cannot allocate device memory: an engine whose HBM is all held by its own
pool, or code where a cudaMalloc would synchronise the device and stall other streams.
They use the entry point whose scratch (status word and RoPE frequency table) is a static
device array shared by every call. This file is collected last on purpose, so that a run
stopping at its first failure has already run every other test.

Three calls in a row, each checked element by element against the CPU oracle
(oracle.layer.rope_kv: q, the k cache with its sentinel, the bit-exact v cache, the status
word) and against the existing entry point (trident_scm_invoke of an equivalent version) on
identical inputs. The first call leaves a position error in the shared status word; the
second changes theta and the head norm; the third keeps the second call's (theta, D) with
new inputs, so each call's table and status word must come from that call alone.
"""
import numpy as np
import pytest
import torch

from oracle import layer as L
from paper_2609_37241_gb300 import synth
from tests import parity as P

pytestmark = pytest.mark.gpu
BF16 = 1


@pytest.fixture(scope="module")
def S(built_lib):
    from paper_2609_37241_gb300 import scm
    return scm


def make_case(seed, T, Hq, Hkv, D, Sl, bad_pos=None):
    g = np.random.default_rng(seed)
    q = synth.act(g, (T, Hq, D), BF16)
    k = synth.act(g, (T, Hkv, D), BF16)
    v = synth.act(g, (T, Hkv, D), BF16)
    pos = synth.positions(g, T, Sl)
    if bad_pos is not None:
        pos[bad_pos] = Sl
    gq, gk = synth.gamma(g, D), synth.gamma(g, D)
    return dict(q=q, k=k, v=v, pos=pos, gq=gq, gk=gk, kc=synth.cache(Hkv, Sl, D), vc=synth.cache(Hkv, Sl, D))


def device_tensors(c, qknorm):
    """Fresh device copies: q/k/v as views of one fused qkv buffer."""
    T, Hq, D = c["q"].shape
    Hkv = c["k"].shape[1]
    qkv = torch.cat([P.dev(c[n], BF16).reshape(T, -1) for n in ("q", "k", "v")], dim=1)
    ts = [qkv[:, :Hq * D].view(T, Hq, D), qkv[:, Hq * D:(Hq + Hkv) * D].view(T, Hkv, D),
          qkv[:, (Hq + Hkv) * D:].view(T, Hkv, D), torch.from_numpy(c["pos"]).cuda(),
          P.dev(c["kc"], BF16), P.dev(c["vc"], BF16)]
    if qknorm:
        ts += [torch.from_numpy(c["gq"]).cuda(), torch.from_numpy(c["gk"]).cuda()]
    return ts


def host_outputs(ts):
    return dict(q=P.host_bits(ts[0], BF16), k=P.host_bits(ts[1], BF16), v=P.host_bits(ts[2], BF16),
                k_cache=P.host_bits(ts[4], BF16), v_cache=P.host_bits(ts[5], BF16))


def assert_close(got, ref, name):
    """Within the parity tolerance: |err| <= 1e-2 + 1.6e-2 |ref| and at most 1 ulp apart."""
    g, r = P.widen_bits(got, BF16), P.widen_bits(ref, BF16)
    assert np.all(np.abs(g - r) <= 1e-2 + 1.6e-2 * np.abs(r)), name
    assert P.ulp_diff(got, ref, BF16).max() <= 1, name


def test_noalloc_calls_in_a_row_match_the_oracle_and_the_scm(S):
    stream = torch.cuda.current_stream().cuda_stream
    Sl, D, Hq, Hkv = 8192, 128, 32, 8
    word = torch.full((1,), -1, dtype=torch.int32).pin_memory()
    calls = [dict(seed=1, T=5, qknorm=True, theta=1e6, bad=2),     # leaves a position error
             dict(seed=2, T=7, qknorm=False, theta=5e5, bad=None),  # new theta and head norm
             dict(seed=3, T=64, qknorm=False, theta=5e5, bad=None)]  # same (theta, D), new inputs
    for cl in calls:
        case = make_case(cl["seed"], cl["T"], Hq, Hkv, D, Sl, cl["bad"])
        inputs = (case["q"], case["k"], case["v"], case["pos"])
        ref = L.rope_kv(case["q"], case["k"], case["v"], case["pos"], case["kc"], case["vc"], cl["theta"],
                        BF16, qknorm=cl["qknorm"], gamma_q=case["gq"], gamma_k=case["gk"], eps=1e-6)
        op = S.OP_QKNORM_ROPE_KV if cl["qknorm"] else S.OP_ROPE_KV
        # the allocation-free entry point
        got = device_tensors(case, cl["qknorm"])
        word.fill_(-1)
        st = S.trident_rope_kv_noalloc(S.make_args(op, got, eps=1e-6, rope_theta=cl["theta"]), stream,
                                       status_word=word.data_ptr())
        assert st == S.OK, S.trident_scm_last_error()
        torch.cuda.synchronize()
        got_h = host_outputs(got)
        P.check_rope(ref, got_h, inputs)
        assert int(word.item()) == (S.DEVERR_POS if cl["bad"] is not None else 0) and ref["bad"] == (
            1 if cl["bad"] is not None else 0)
        # the existing entry point: one SCM version, identical inputs
        scm = S.Scm(device=0)
        scm.register(S.make_spec(op, BF16, [Hq, Hkv, D, Sl], 1, 64, layout=S.LAYOUT_ROWSTRIDED,
                                 rope_theta=cl["theta"]))
        via = device_tensors(case, cl["qknorm"])
        st, sel = scm.invoke(S.make_args(op, via, eps=1e-6, rope_theta=cl["theta"]), stream)
        assert (st, sel) == (S.OK, 0), S.trident_scm_last_error()
        st, scm_status = S.trident_scm_device_status(scm.h, stream)
        assert st == S.OK and scm_status == int(word.item())
        scm.close()
        via_h = host_outputs(via)
        for name in ("q", "k_cache"):
            assert_close(got_h[name], via_h[name], name)
        assert np.array_equal(got_h["v_cache"], via_h["v_cache"])


def test_noalloc_without_status_word(S):
    """out_status may be NULL: the call still runs and matches the oracle."""
    Sl, D, Hq, Hkv = 512, 64, 4, 2
    case = make_case(4, 9, Hq, Hkv, D, Sl)
    ref = L.rope_kv(case["q"], case["k"], case["v"], case["pos"], case["kc"], case["vc"], 1e4, BF16)
    ts = device_tensors(case, False)
    st = S.trident_rope_kv_noalloc(S.make_args(S.OP_ROPE_KV, ts, rope_theta=1e4),
                                   torch.cuda.current_stream().cuda_stream)
    assert st == S.OK, S.trident_scm_last_error()
    torch.cuda.synchronize()
    P.check_rope(ref, host_outputs(ts), (case["q"], case["k"], case["v"], case["pos"]))


def test_noalloc_rejects_sizes_beyond_its_scratch(S):
    """A head size above 256 needs more than the static array's 128 frequency pairs: a clear
    error, nothing launched."""
    T, Hq, Hkv, D, Sl = 2, 2, 1, 512, 64
    case = make_case(3, T, Hq, Hkv, D, Sl)
    ts = device_tensors(case, False)
    before = P.host_bits(ts[0], BF16)
    st = S.trident_rope_kv_noalloc(S.make_args(S.OP_ROPE_KV, ts, rope_theta=1e4),
                                   torch.cuda.current_stream().cuda_stream)
    assert st == S.ERR_INVALID
    assert "scratch" in S.trident_scm_last_error()
    torch.cuda.synchronize()
    assert np.array_equal(P.host_bits(ts[0], BF16), before)
