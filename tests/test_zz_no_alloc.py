"""The allocation-free RoPE/KV entry point (trident_rope_kv_noalloc) against the SCM path.

Callers that cannot allocate device memory -- an engine whose HBM is all held by its own
pool, or code where a cudaMalloc would synchronise the device -- use the entry point whose
scratch (status word and RoPE frequency table) is a static device array. This file is collected
last on purpose. Two calls in a row, each compared with the existing entry point
(trident_scm_invoke of an equivalent version) on identical inputs, within the parity
tolerance of the other tests: the second call changes theta (the shared table is rebuilt)
and must report a clean status although the first left a position error in the array.
"""
import numpy as np
import pytest
import torch

from paper_2609_37241_gb300 import synth
from tests import parity as P

pytestmark = pytest.mark.gpu
BF16 = 1


@pytest.fixture(scope="module")
def S(built_lib):
    from paper_2609_37241_gb300 import scm
    return scm


def make_case(seed, T, Hq, Hkv, D, Sl, qknorm, bad_pos=None):
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


def assert_close(got, ref, name):
    """Within the parity tolerance: |err| <= 1e-2 + 1.6e-2 |ref| and at most 1 ulp apart."""
    g, r = P.widen_bits(got, BF16), P.widen_bits(ref, BF16)
    assert np.all(np.abs(g - r) <= 1e-2 + 1.6e-2 * np.abs(r)), name
    assert P.ulp_diff(got, ref, BF16).max() <= 1, name


def test_noalloc_two_calls_in_a_row_match_the_scm(S):
    stream = torch.cuda.current_stream().cuda_stream
    Sl, D, Hq, Hkv = 8192, 128, 32, 8
    calls = [dict(seed=1, T=5, qknorm=True, theta=1e6, bad=2),    # leaves a position error
             dict(seed=2, T=7, qknorm=False, theta=5e5, bad=None)]  # new theta: table rebuilt
    for cl in calls:
        case = make_case(cl["seed"], cl["T"], Hq, Hkv, D, Sl, cl["qknorm"], cl["bad"])
        op = S.OP_QKNORM_ROPE_KV if cl["qknorm"] else S.OP_ROPE_KV
        # existing entry point: one SCM version
        scm = S.Scm(device=0)
        scm.register(S.make_spec(op, BF16, [Hq, Hkv, D, Sl], 1, 64, layout=S.LAYOUT_ROWSTRIDED,
                                 rope_theta=cl["theta"]))
        ref = device_tensors(case, cl["qknorm"])
        st, sel = scm.invoke(S.make_args(op, ref, eps=1e-6, rope_theta=cl["theta"]), stream)
        assert (st, sel) == (S.OK, 0), S.trident_scm_last_error()
        st, ref_status = S.trident_scm_device_status(scm.h, stream)
        assert st == S.OK
        scm.close()
        # the allocation-free entry point on identical inputs
        got = device_tensors(case, cl["qknorm"])
        st, word = S.trident_rope_kv_noalloc(S.make_args(op, got, eps=1e-6, rope_theta=cl["theta"]), stream)
        assert st == S.OK, S.trident_scm_last_error()
        torch.cuda.synchronize()
        assert word.value == ref_status == (S.DEVERR_POS if cl["bad"] is not None else 0)
        for i, name in ((0, "q"), (4, "k_cache")):
            assert_close(P.host_bits(got[i], BF16), P.host_bits(ref[i], BF16), name)
        assert np.array_equal(P.host_bits(got[5], BF16), P.host_bits(ref[5], BF16))  # v: bit copy
        assert np.array_equal(P.host_bits(got[1], BF16), case["k"])                    # k untouched


def test_noalloc_rejects_sizes_beyond_its_scratch(S):
    """A head size above 256 needs more than the static array's 128 frequency pairs: a clear
    error, nothing launched."""
    T, Hq, Hkv, D, Sl = 2, 2, 1, 512, 64
    case = make_case(3, T, Hq, Hkv, D, Sl, False)
    ts = device_tensors(case, False)
    before = P.host_bits(ts[0], BF16)
    st, _ = S.trident_rope_kv_noalloc(S.make_args(S.OP_ROPE_KV, ts, rope_theta=1e4),
                                      torch.cuda.current_stream().cuda_stream)
    assert st == S.ERR_INVALID
    assert "scratch" in S.trident_scm_last_error()
    torch.cuda.synchronize()
    assert np.array_equal(P.host_bits(ts[0], BF16), before)
