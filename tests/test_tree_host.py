"""Structured arguments on the host (dry-run SCM, no GPU): recipes bind a call's argument
tree (§3.3); selection over tree versions against the oracle's plain recursive binder;
malformed trees and recipes are errors; the tree hook; DLPack tensors."""
import ctypes
import random

import pytest

from oracle import guards as G
from tests import cases

H = 64


@pytest.fixture()
def S(built_lib):
    from paper_2609_37241_gb300 import scm
    return scm


def T(addr, shape=(4, H), dtype=1, stride=None):
    return cases.tensor(addr, dtype, shape, stride)


def rms_inputs(k=0, rows=4):
    base = 0x7F0000000000 + (k << 36)
    x, r = T(base + 0x100000, (rows, H)), T(base + 0x200000, (rows, H))
    w = T(base + 0x300000, (H,), 3)
    y, ro = T(base + 0x400000, (rows, H)), T(base + 0x500000, (rows, H))
    return x, r, w, y, ro


# The paper's running example as a source signature rms_norm(x, residual, weight, out, eps):
# residual None -> RMSNORM (out is y); residual a tensor -> ADD_RMSNORM (out is (y, r_out)).
def rms_table():
    spec_n = cases.make_spec(dict(op=7, fixed=[H], tok=[1, 1 << 20]))
    spec_a = cases.make_spec(dict(op=1, fixed=[H], tok=[1, 1 << 20]))
    rec_n = cases.recipe(7, ("tensor", 0), ("none",), ("tensor", 1), ("tensor", 2), ("float", "eps"))
    rec_a = cases.recipe(1, ("tensor", 0), ("tensor", 1), ("tensor", 2),
                         ("tuple", [("tensor", 3), ("tensor", 4)]), ("float", "eps"))
    return [(spec_n, rec_n), (spec_a, rec_a)]


def lib_run(S, table, tree_values, hook=None, flags=0, plain=()):
    s = S.Scm(device=0, flags=S.OPT_DRY_RUN | flags)
    for sp in plain:
        s.register(cases.lib_spec(sp))
    for spec, rec in table:
        s.register_tree(cases.lib_spec(spec), cases.lib_recipe(rec))
    if hook is not None:
        s.set_tree_hook(hook)
    out = s.invoke_tree(S.Tree(*tree_values))
    stats = s.stats()
    s.close()
    return out, stats


def check(S, table, tree_values, plain=()):
    want = G.select_tree(table, tree_values)
    (st, sel), _ = lib_run(S, table, tree_values, plain=plain)
    assert (cases.STATUS[st], sel) == (want[0], want[1] + len(plain) if want[1] >= 0 else -1)
    return want


def test_one_signature_two_ops_by_structure(S):
    table = rms_table()
    x, r, w, y, ro = rms_inputs()
    assert check(S, table, [x, None, w, y, 1e-6]) == (G.OK, 0)
    assert check(S, table, [x, r, w, (y, ro), 1e-6]) == (G.OK, 1)
    # structure that no recipe has: a residual with a single output, a 3-tuple, an int eps
    assert check(S, table, [x, r, w, y, 1e-6]) == (G.MISS, -1)
    assert check(S, table, [x, r, w, (y, ro, y), 1e-6]) == (G.MISS, -1)
    assert check(S, table, [x, None, w, y, 0]) == (G.MISS, -1)
    assert check(S, table, [x, None, w, y]) == (G.MISS, -1)


def test_plain_versions_are_skipped_and_counted_in_order(S):
    table = rms_table()
    x, r, w, y, ro = rms_inputs()
    plain = [cases.make_spec(dict(op=1, fixed=[H], tok=[1, 1 << 20]))]
    check(S, table, [x, r, w, (y, ro), 1e-6], plain=plain)  # selects index 2


def test_guarded_constant_and_bound_scalars(S):
    x, r, w, y, ro = rms_inputs()
    spec = cases.make_spec(dict(op=1, fixed=[H], tok=[1, 1 << 20]))
    # a version specialised for group size 2 (a source-visible constant absent from the
    # flat arguments), then a generic one that ignores it
    rec2 = cases.recipe(1, ("tuple", [("tensor", 0), ("tensor", 1)]), ("tensor", 2),
                        ("tuple", [("tensor", 3), ("tensor", 4)]), ("int", "const", 2), ("float", "eps"))
    recany = cases.recipe(1, ("tuple", [("tensor", 0), ("tensor", 1)]), ("tensor", 2),
                          ("tuple", [("tensor", 3), ("tensor", 4)]), ("int", "unused"), ("float", "eps"))
    table = [(spec, rec2), (spec, recany)]
    assert check(S, table, [(x, r), w, (y, ro), 2, 1e-5]) == (G.OK, 0)
    assert check(S, table, [(x, r), w, (y, ro), 3, 1e-5]) == (G.OK, 1)
    # eps comes from the tree: a negative one makes the bound arguments malformed
    assert check(S, table, [(x, r), w, (y, ro), 2, -1.0]) == (G.INVALID, -1)
    # theta bound from the tree is a guarded constant of RoPE versions
    rope = cases.make_args(dict(op=2, T=2, Hq=2, Hkv=1, D=64, S=8))["tensors"]
    spec_r = cases.make_spec(dict(op=2, fixed=[2, 1, 64, 8], tok=[1, 64], theta=1e4))
    rec_r = cases.recipe(2, ("tuple", [("tensor", 0), ("tensor", 1), ("tensor", 2)]), ("tensor", 3),
                         ("tuple", [("tensor", 4), ("tensor", 5)]), ("float", "theta"))
    assert check(S, [(spec_r, rec_r)], [tuple(rope[:3]), rope[3], tuple(rope[4:]), 1e4]) == (G.OK, 0)
    assert check(S, [(spec_r, rec_r)], [tuple(rope[:3]), rope[3], tuple(rope[4:]), 5e5]) == (G.MISS, -1)


def test_ignored_leaves_and_preorder_slots(S):
    # slots need not follow the source order: here the output pair comes first in the tree
    x, r, w, y, ro = rms_inputs()
    spec = cases.make_spec(dict(op=1, fixed=[H], tok=[1, 1 << 20]))
    rec = cases.recipe(1, ("tuple", [("tensor", 3), ("tensor", 4)]), ("tensor", -1),
                       ("tuple", [("tensor", 0), ("tuple", [("tensor", 1), ("tensor", 2)])]), eps=1e-6)
    junk = T(0x10, (3, 3), 3)
    assert check(S, [(spec, rec)], [(y, ro), junk, (x, (r, w))]) == (G.OK, 0)
    # swapping the output pair makes r_out the 'y' slot: still well formed, still a hit
    assert check(S, [(spec, rec)], [(ro, y), junk, (x, (r, w))]) == (G.OK, 0)
    # an aliasing mistake through the tree (y is x, not an in-place pair with r) is an error
    assert check(S, [(spec, rec)], [(r, ro), junk, (x, (r, w))]) == (G.INVALID, -1)


def _random_value(rng, x, r, w, y, ro):
    """A call of the two-op signature (either op, valid), then 0-2 perturbations of its
    structure, kinds or values."""
    vals = [x, None, w, y, 1e-6] if rng.random() < 0.5 else [x, r, w, (y, ro), 1e-5]
    for _ in range(rng.choice((0, 0, 1, 2))):
        k = rng.randrange(6)
        if k in (0, 1, 2, 5) and len(vals) < 5:
            continue
        if k == 0:
            vals[1] = rng.choice([None, r, (r,), 3])
        elif k == 1:
            vals[3] = rng.choice([(y, ro), y, (y,), (y, ro, ro), None, (ro, y)])
        elif k == 2:
            vals[4] = rng.choice([1e-6, 0, -1.0, None, 2.0])
        elif k == 3:
            vals = vals[:rng.randrange(len(vals))]
        elif k == 4:
            vals = vals + [rng.choice([None, 1, x])]
        else:
            vals[0] = rng.choice([x, r, None, 1.0, (x,)])
    return vals


@pytest.mark.parametrize("seed", range(40))
def test_random_structures_match_oracle(S, seed):
    rng = random.Random(seed)
    table = rms_table()
    rng.shuffle(table)
    for _ in range(5):
        check(S, table, _random_value(rng, *rms_inputs(rows=rng.choice([1, 3]))))


def test_malformed_trees_are_errors(S):
    table = rms_table()
    s = S.Scm(device=0, flags=S.OPT_DRY_RUN)
    for spec, rec in table:
        s.register_tree(cases.lib_spec(spec), cases.lib_recipe(rec))
    called = []
    s.set_tree_hook(lambda *a: called.append(1))
    x, r, w, y, ro = rms_inputs()

    def nodes_of(*vals):
        t = S.Tree(*vals)
        return t

    bad = []
    t = nodes_of(x, None, w, (y, ro), 1e-6)
    t.nodes[3].first = 2  # children before their tuple
    bad.append(t)
    t = nodes_of(x, None, w, (y, ro), 1e-6)
    t.nodes[3].first = t.nnodes - 1  # children past the end
    bad.append(t)
    t = nodes_of((y, ro), (x, r))
    t.nodes[1].first = t.nodes[0].first  # two tuples share children
    bad.append(t)
    t = nodes_of(x, 1.0)
    t.nodes[1].kind = 9  # unknown kind
    bad.append(t)
    t = nodes_of(x, 1.0)
    t.nodes[1].reserved = 1
    bad.append(t)
    deep = x
    for _ in range(16):
        deep = (deep,)
    bad.append(nodes_of(deep))
    t = nodes_of(x, 1.0)
    t.nodes[0].kind = S.NODE_DLTENSOR  # DLTENSOR without a DLTensor
    bad.append(t)
    for t in bad:
        st, sel = s.invoke_tree(t)
        assert (st, sel) == (S.ERR_INVALID, -1), S.trident_scm_last_error()
    # nargs > nnodes, negative nargs
    L = S.lib()
    t = nodes_of(x)
    assert L.trident_scm_invoke_tree(s.h, t.nodes, 2, 1, None, None) == S.ERR_INVALID
    assert L.trident_scm_invoke_tree(s.h, t.nodes, -1, 1, None, None) == S.ERR_INVALID
    assert not called
    assert s.stats().err_invalid == len(bad) + 2
    s.close()


def test_recipe_validation(S):
    s = S.Scm(device=0, flags=S.OPT_DRY_RUN)
    spec = cases.lib_spec(cases.make_spec(dict(op=1, fixed=[H], tok=[1, 64])))
    ok = S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2), (S.Slot(3), S.Slot(4)), S.EPS)
    s.register_tree(spec, ok)
    bad = [
        S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2), (S.Slot(3),), S.EPS),           # slot 4 unbound
        S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2), (S.Slot(3), S.Slot(3)), S.EPS),  # slot 3 twice
        S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2), (S.Slot(3), S.Slot(5)), S.EPS),  # no slot 5
        S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2), (S.Slot(3), S.Slot(4)), S.EPS, S.EPS),
        S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2), (S.Slot(3), S.Slot(4)), S.Num("float", -9)),
        S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2), (S.Slot(3), S.Slot(4)), S.const(float("nan"))),
        S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2), (S.Slot(3), S.Slot(4)), eps=-1.0),
    ]
    dl = S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2), (S.Slot(3), S.Slot(4)))
    dl._arr[0].kind = S.NODE_DLTENSOR
    bad.append(dl)
    for rec in bad:
        st, _ = S.trident_scm_register_tree_spec(s.h, spec, rec)
        assert st == S.ERR_INVALID
    assert S.lib().trident_scm_register_tree_spec(s.h, ctypes.byref(spec), None, None) == S.ERR_INVALID
    assert s.stats().num_specs == 1
    s.close()


def test_tree_hook_grows_the_table(S):
    x, r, w, y, ro = rms_inputs()
    spec_a, rec_a = rms_table()[1]

    def hook(scm, nodes, nargs, nnodes, stream):
        idx = scm.register_tree(cases.lib_spec(spec_a), cases.lib_recipe(rec_a))
        st, sel = S.trident_scm_invoke_tree(scm.h, _Raw(nodes, nargs, nnodes), stream)
        assert (st, sel) == (S.OK, idx)
        # a miss inside the hook does not call the hook again
        assert S.trident_scm_invoke_tree(scm.h, S.Tree(x, 5), stream)[0] == S.MISS
        return idx

    s = S.Scm(device=0, flags=S.OPT_DRY_RUN)
    s.set_tree_hook(hook)
    assert s.invoke_tree(S.Tree(x, r, w, (y, ro), 1e-6)) == (S.MISS_HANDLED, 0)
    assert s.invoke_tree(S.Tree(x, r, w, (y, ro), 1e-6)) == (S.OK, 0)
    st = s.stats()
    assert (st.hook_calls, st.hook_registered, st.hits, st.misses) == (1, 1, 2, 2)
    s.set_tree_hook(None)
    assert s.invoke_tree(S.Tree(x, None, w, y, 1e-6)) == (S.MISS, -1)
    s.close()


class _Raw:
    def __init__(self, nodes, nargs, nnodes):
        self.nodes, self.nargs, self.nnodes = nodes, nargs, nnodes


class DLDevice(ctypes.Structure):
    _fields_ = [("device_type", ctypes.c_int32), ("device_id", ctypes.c_int32)]


class DLDataType(ctypes.Structure):
    _fields_ = [("code", ctypes.c_uint8), ("bits", ctypes.c_uint8), ("lanes", ctypes.c_uint16)]


class DLTensor(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("device", DLDevice), ("ndim", ctypes.c_int32),
                ("dtype", DLDataType), ("shape", ctypes.POINTER(ctypes.c_int64)),
                ("strides", ctypes.POINTER(ctypes.c_int64)), ("byte_offset", ctypes.c_uint64)]


def _dl(addr, shape, code, bits, strides=None, offset=0, dev=(2, 0), keep=None):
    nd = len(shape)
    sh = (ctypes.c_int64 * nd)(*shape)
    st = (ctypes.c_int64 * nd)(*strides) if strides is not None else None
    d = DLTensor(addr, DLDevice(*dev), nd, DLDataType(code, bits, 1), sh, st, offset)
    keep.extend([sh, st, d])
    return d


def test_dlpack_tensors_bind_like_descriptors(S):
    keep = []
    x, r, w, y, ro = rms_inputs()
    table = rms_table()
    s = S.Scm(device=0, flags=S.OPT_DRY_RUN)
    for spec, rec in table:
        s.register_tree(cases.lib_spec(spec), cases.lib_recipe(rec))

    def call(x_node):
        t = S.Tree(x, None, w, y, 1e-6)
        t.nodes[0].kind = S.NODE_DLTENSOR
        t.nodes[0].dl = ctypes.addressof(x_node)
        return s.invoke_tree(t)

    # compact strides (NULL), bf16 (code 4): the same tensor as the descriptor x
    assert call(_dl(x["addr"], (4, H), 4, 16, keep=keep)) == (S.OK, 0)
    assert call(_dl(x["addr"], (4, H), 4, 16, strides=(H, 1), keep=keep)) == (S.OK, 0)
    # byte offset: 16 keeps 16-byte alignment (hit); 2 breaks it (every version misses)
    assert call(_dl(x["addr"] - 16, (4, H), 4, 16, offset=16, keep=keep)) == (S.OK, 0)
    assert call(_dl(x["addr"], (4, H), 4, 16, offset=2, keep=keep)) == (S.MISS, -1)
    # fp16 (code 2, 16 bits) is another dtype: a miss, not an error
    assert call(_dl(x["addr"], (4, H), 2, 16, keep=keep)) == (S.MISS, -1)
    # a CPU tensor (device type 1) misses the device guard
    assert call(_dl(x["addr"], (4, H), 4, 16, dev=(1, 0), keep=keep)) == (S.MISS, -1)
    # unsupported dtype (complex, code 5), 0-d, or a device type the library does not take
    for d in (_dl(x["addr"], (4, H), 5, 32, keep=keep), _dl(x["addr"], (4, H), 4, 16, dev=(13, 0), keep=keep)):
        assert call(d)[0] == S.ERR_INVALID
    z = _dl(x["addr"], (4, H), 4, 16, keep=keep)
    z.ndim = 0
    assert call(z)[0] == S.ERR_INVALID
    s.close()


def test_torch_dlpack_capsule(S):
    torch = pytest.importorskip("torch")
    t = torch.zeros((4, H), dtype=torch.bfloat16)
    tree = S.Tree(S.DL(t), None, t, t, 1e-6)
    assert tree.nodes[0].kind == S.NODE_DLTENSOR and tree.nodes[0].dl
    view = DLTensor.from_address(tree.nodes[0].dl)
    assert (view.ndim, view.dtype.code, view.dtype.bits, view.device.device_type) == (2, 4, 16, 1)
    assert view.data + view.byte_offset == t.data_ptr()


def _node_fields(nodes, n):
    out = []
    for i in range(n):
        d = nodes[i]
        t = d.t
        out.append((d.kind, d.n, d.first, d.i, d.f, (t.data or 0, t.dtype, t.ndim, t.device,
                                                      tuple(t.shape[:t.ndim]), tuple(t.stride[:t.ndim]))
                    if d.kind == 1 else None))
    return out


def test_c_packer_builds_the_same_tree_as_the_python_builder(S):
    torch = pytest.importorskip("torch")
    fc = S.fastcall()
    if fc is None:
        pytest.skip("Python headers not installed: no CPython shim")
    x = torch.zeros((4, 8), dtype=torch.bfloat16)
    m = torch.zeros((4, 8), dtype=torch.bool)
    v = torch.zeros((2, 3, 4), dtype=torch.float16)[:, 1:, ::2]  # a strided view
    seen = []

    def hook(scm, nodes, nargs, nnodes, stream):
        seen.append((nargs, _node_fields(nodes, nnodes)))
        return None

    s = S.Scm(device=0, flags=S.OPT_DRY_RUN)
    s.set_tree_hook(hook)
    calls = [
        (x, None, (m, (v, 3, [True, 2.5])), -7, 1e-6),
        tuple(range(70)),                 # more nodes than the packer's stack buffer
        ([x] * 40, [[x, v]] * 20),        # lists, nested, grown past the stack buffer
        (),
    ]
    for args in calls:
        assert fc.invoke_py(s.h.value, 0, *args) == S.MISS_HANDLED
        t = S.Tree(*args)
        assert seen[-1] == (t.nargs, _node_fields(t.nodes, t.nnodes))
    with pytest.raises(TypeError):
        fc.invoke_py(s.h.value, 0, x, "a string")
    with pytest.raises(TypeError):
        fc.invoke_py(s.h.value, 0, torch.zeros(2, dtype=torch.complex64))
    with pytest.raises(ValueError):
        fc.invoke_py(s.h.value, 0, torch.zeros((1, 1, 1, 1, 1)))
    with pytest.raises(ValueError):
        fc.invoke_py(s.h.value, 0, tuple(range(5000)))
    assert len(seen) == len(calls)
    s.close()


def test_tree_execution_error_is_raised_not_retried(S):
    """As for invoke: a failed launch of the selected version (injected on the host) returns
    ERR_CUDA at once -- no later version, no hook."""
    x, r, w, y, ro = rms_inputs()
    called = []
    s = S.Scm(device=0, flags=S.OPT_DRY_RUN | S.OPT_FAIL_LAUNCHES)
    s.set_tree_hook(lambda *a: called.append(1))
    spec_a, rec_a = rms_table()[1]
    for _ in range(2):
        s.register_tree(cases.lib_spec(spec_a), cases.lib_recipe(rec_a))
    assert s.invoke_tree(S.Tree(x, r, w, (y, ro), 1e-6)) == (S.ERR_CUDA, 0)
    assert "injected" in S.trident_scm_last_error()
    st = s.stats()
    assert (st.hits, st.misses, st.err_cuda, st.hook_calls) == (0, 0, 1, 0) and not called
    s.close()


def test_concurrent_tree_and_step_calls_with_growth(S):
    """Several threads call invoke_tree and invoke_step while another registers versions:
    every call sees a consistent table (first match stays version 0) and no error."""
    import threading
    s = S.Scm(device=0, flags=S.OPT_DRY_RUN, max_specs=400)
    spec_a, rec_a = rms_table()[1]
    s.register_tree(cases.lib_spec(spec_a), cases.lib_recipe(rec_a))
    x, r, w, y, ro = rms_inputs()
    tree = S.Tree(x, r, w, (y, ro), 1e-6)
    from tests.test_step_host import chain_call, chain_spec
    s.register(cases.lib_spec(chain_spec()))
    calls = (S.trident_args * 3)(*[cases.lib_args(chain_call(k)) for k in range(3)])
    stop = threading.Event()
    errors = []

    def tree_reader():
        while not stop.is_set():
            got = S.trident_scm_invoke_tree(s.h, tree)
            if got != (S.OK, 0):
                errors.append(("tree", got))

    def step_reader():
        while not stop.is_set():
            got = S.trident_scm_invoke_step(s.h, calls)
            if got != (S.OK, [1, 1, 1]):
                errors.append(("step", got))

    th = [threading.Thread(target=f) for f in (tree_reader, tree_reader, step_reader, step_reader)]
    for t in th:
        t.start()
    for _ in range(300):
        s.register_tree(cases.lib_spec(spec_a), cases.lib_recipe(rec_a))
    stop.set()
    for t in th:
        t.join()
    assert not errors, errors[:3]
    st = s.stats()
    assert st.num_specs == 302 and st.fused_launches > 0 and st.hits == st.invokes
    s.close()
