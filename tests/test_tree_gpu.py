"""Structured arguments on the GPU: one source signature dispatching to two ops by its
structure (tensors passed as descriptors and through DLPack), eps bound from the tree,
and a whole decoder-layer chain passed as a nested tree, against the oracle."""
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


def rms_scm(S, H, dtype):
    # rms_norm(x, residual, weight, out, eps): residual None -> RMSNORM, out = y;
    # residual a tensor -> ADD_RMSNORM, out = (y, r_out)
    s = S.Scm(device=0)
    s.register_tree(S.make_spec(S.OP_RMSNORM, dtype, [H], 1, 1 << 20),
                    S.Recipe(S.Slot(0), None, S.Slot(1), S.Slot(2), S.EPS))
    s.register_tree(S.make_spec(S.OP_ADD_RMSNORM, dtype, [H], 1, 1 << 20),
                    S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2), (S.Slot(3), S.Slot(4)), S.EPS))
    return s


@pytest.mark.parametrize("H,T,dtype,dl", [(4096, 7, BF16, True), (128, 1024, BF16, False),
                                          (4096, 3, FP16, True)])
def test_rms_norm_signature_on_gpu(S, H, T, dtype, dl):
    g = np.random.default_rng(H + T)
    x, r, gam = synth.act(g, (T, H), dtype), synth.act(g, (T, H), dtype), synth.gamma(g, H)
    xd, rd, gd = P.dev(x, dtype), P.dev(r, dtype), torch.from_numpy(gam).cuda()
    wrap = S.DL if dl else (lambda t: t)
    eps = 0.5  # large enough to show in the outputs, so the bound value is checked
    s = rms_scm(S, H, dtype)
    y = torch.empty_like(xd)
    assert s.invoke_tree(S.Tree(wrap(xd), None, wrap(gd), y, eps), stream()) == (S.OK, 0)
    y2, ro = torch.empty_like(xd), torch.empty_like(rd)
    assert s.invoke_tree(S.Tree(xd, wrap(rd), gd, (wrap(y2), ro), eps), stream()) == (S.OK, 1)
    torch.cuda.synchronize()
    s.close()
    y_ref, y_bits = L.rmsnorm(x, gam, eps, dtype)
    P.check_act(P.host_bits(y, dtype), y_ref, y_bits, dtype, "y")
    y2_ref, y2_bits, ro_bits = L.add_rmsnorm(x, r, gam, eps, dtype)
    assert np.array_equal(P.host_bits(ro, dtype), ro_bits)
    P.check_act(P.host_bits(y2, dtype), y2_ref, y2_bits, dtype, "y2")


def test_layer_chain_as_a_nested_tree(S):
    cfg = synth.LLAMA
    T = 4
    g = np.random.default_rng(404)
    inp = synth.layer_inputs(g, T, cfg)
    ref = L.layer_chain(inp, cfg["theta"], cfg["eps"], BF16)
    ts, out = chain_device(inp, BF16, False)
    (h, r0, ga, x1, r1, q, k, v, pos, kc, vc, ao, gm, x2, r2, gg, u, o) = ts
    fixed = [cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["D"], cfg["S"], cfg["I"]]
    s = S.Scm(device=0, flags=S.OPT_PDL)
    # layer(hidden=(h, r0), attn=((q, k, v), pos, (k_cache, v_cache)), mlp=(attn_out, (g, u)),
    #       weights=(gamma_attn, gamma_mlp), outs=(x1, r1, x2, r2, o), eps, theta)
    rec = S.Recipe((S.Slot(0), S.Slot(1)), ((S.Slot(5), S.Slot(6), S.Slot(7)), S.Slot(8), (S.Slot(9), S.Slot(10))),
                   (S.Slot(11), (S.Slot(15), S.Slot(16))), (S.Slot(2), S.Slot(12)),
                   (S.Slot(3), S.Slot(4), S.Slot(13), S.Slot(14), S.Slot(17)), S.EPS, S.THETA)
    s.register_tree(S.make_spec(S.OP_LAYER_CHAIN, BF16, fixed, 1, 64, layout=S.LAYOUT_ROWSTRIDED,
                                rope_theta=cfg["theta"]), rec)
    tree = S.Tree((h, r0), ((q, k, v), pos, (kc, vc)), (ao, (gg, u)), (ga, gm), (x1, r1, x2, r2, o),
                  float(cfg["eps"]), float(cfg["theta"]))
    assert s.invoke_tree(tree, stream()) == (S.OK, 0), S.trident_scm_last_error()
    # a different theta is another specialisation: a miss
    miss = S.Tree((h, r0), ((q, k, v), pos, (kc, vc)), (ao, (gg, u)), (ga, gm), (x1, r1, x2, r2, o),
                  float(cfg["eps"]), 1e4)
    assert s.invoke_tree(miss, stream()) == (S.MISS, -1)
    torch.cuda.synchronize()
    assert S.trident_scm_device_status(s.h, stream())[1] == 0
    s.close()
    check_chain(ref, out, inp)


def test_python_arguments_packed_by_the_shim(S):
    """Scm.call: the CPython shim packs the Python arguments per call (no prebuilt tree)."""
    H, T = 4096, 5
    g = np.random.default_rng(55)
    x, r, gam = synth.act(g, (T, H), BF16), synth.act(g, (T, H), BF16), synth.gamma(g, H)
    xd, rd, gd = P.dev(x, BF16), P.dev(r, BF16), torch.from_numpy(gam).cuda()
    s = rms_scm(S, H, BF16)
    y, ro = torch.empty_like(xd), torch.empty_like(rd)
    assert s.call(xd, rd, gd, [y, ro], 1e-6, stream=stream()) == S.OK
    y1 = torch.empty_like(xd)
    assert s.call(xd, None, gd, y1, 1e-6, stream=stream()) == S.OK
    assert s.call(xd, None, gd, y1, 1, stream=stream()) == S.MISS  # an int eps: no version
    torch.cuda.synchronize()
    s.close()
    y_ref, y_bits, ro_bits = L.add_rmsnorm(x, r, gam, 1e-6, BF16)
    assert np.array_equal(P.host_bits(ro, BF16), ro_bits)
    P.check_act(P.host_bits(y, BF16), y_ref, y_bits, BF16, "y")
    y1_ref, y1_bits = L.rmsnorm(x, gam, 1e-6, BF16)
    P.check_act(P.host_bits(y1, BF16), y1_ref, y1_bits, BF16, "y1")
