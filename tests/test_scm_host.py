"""Host-side tests of the SCM library that need no GPU: symbol exports and struct layout,
dry-run selection against the oracle (golden cases, brute force over small domains,
every op), registration validation, the hook lifecycle of §3.5, the overlap launch
precondition, statistics and concurrent growth."""
import itertools
import json
import os
import re
import subprocess
import threading

import numpy as np
import pytest

from oracle import guards as G
from tests import cases

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


@pytest.fixture()
def S(built_lib):
    from paper_2609_37241_gb300 import scm
    return scm


def dry(S, hook=None, flags=0, max_specs=256):
    return S.Scm(device=0, max_specs=max_specs, flags=S.OPT_DRY_RUN | flags, hook=hook)


def lib_select(S, table, args):
    s = dry(S)
    for sp in table:
        s.register(cases.lib_spec(sp))
    st, idx = s.select(cases.lib_args(args))
    s.close()
    return cases.STATUS[st], idx


# ---------------------------------------------------------------------------- ABI
def test_exports_every_declared_symbol(S):
    header = open(os.path.join(ROOT, "include", "trident_scm.h")).read()
    declared = set(re.findall(r"^\s*(?:[\w\s\*]+?)\b(trident_\w+)\s*\(", header, re.M))
    declared = {d for d in declared if not d.endswith("_t")}
    nm = subprocess.run(["nm", "-D", "--defined-only", S.LIB_PATH], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (trident_\w+)", nm))
    assert declared, "no declarations parsed"
    assert declared == exported, (declared ^ exported)
    assert S.trident_abi_version() == 4


def test_every_entry_point_cites_its_passage():
    """Each prototype's comment block names the paper passage that defines the call (a
    section or Algorithm 1); the allocation-free entry says instead that the paper has no
    counterpart."""
    header = open(os.path.join(ROOT, "include", "trident_scm.h")).read()
    entries = header.split("/* ---------------------------------------------------------------- entry points */")[1]
    blocks = re.findall(r"(/\*(?:[^*]|\*(?!/))*\*/)\s*(?:#define[^\n]*\n\s*)?[\w\s\*]+?\b(trident_\w+)\s*\(", entries)
    names = [n for _, n in blocks]
    declared = {d for d in re.findall(r"^\s*(?:[\w\s\*]+?)\b(trident_\w+)\s*\(", header, re.M)
                if not d.endswith("_t")}
    assert len(names) == len(set(names)) and set(names) == declared
    for comment, name in blocks:
        if name == "trident_rope_kv_noalloc":
            assert "no counterpart" in comment, name
        else:
            assert re.search(r"§\d|Algorithm 1", comment), name


def test_binding_constants_match_header_defines(S):
    header = open(os.path.join(ROOT, "include", "trident_scm.h")).read()
    defines = dict(re.findall(r"^#define TRIDENT_(\w+) \(?(-?(?:0x)?[0-9a-fA-F]+)u?\)?", header, re.M))
    defines.pop("ABI_VERSION")
    assert {"MAX_TENSORS", "MAX_FIXED", "STEP_MAX", "NOT_RUN", "OPT_PDL", "DEVERR_POS"} <= set(defines)
    for name, val in defines.items():
        assert getattr(S, name) == int(val, 0), name


def test_struct_layout_matches_header(S, tmp_path):
    import ctypes
    src = tmp_path / "layout.c"
    src.write_text(
        '#include <stdio.h>\n#include <stddef.h>\n#include "trident_scm.h"\n'
        "int main(void){printf(\"%zu %zu %zu %zu %zu %zu %zu %zu\\n\", sizeof(trident_tensor),"
        " sizeof(trident_args), offsetof(trident_args, t), sizeof(trident_spec_desc),"
        " offsetof(trident_spec_desc, rope_theta), sizeof(trident_scm_options),"
        " sizeof(trident_scm_stats_t), offsetof(trident_tensor, dtype)); "
        "printf(\"%zu %zu %zu %zu %zu %zu %zu\\n\", sizeof(trident_node), offsetof(trident_node, dl),"
        " offsetof(trident_node, t), sizeof(trident_recipe_node), offsetof(trident_recipe_node, f),"
        " sizeof(trident_recipe), offsetof(trident_recipe, eps)); return 0;}\n")
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    got = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True).stdout.split()]
    want = [ctypes.sizeof(S.trident_tensor), ctypes.sizeof(S.trident_args),
            S.trident_args.t.offset, ctypes.sizeof(S.trident_spec_desc),
            S.trident_spec_desc.rope_theta.offset, ctypes.sizeof(S.trident_scm_options),
            ctypes.sizeof(S.trident_scm_stats_t), S.trident_tensor.dtype.offset,
            ctypes.sizeof(S.trident_node), S.trident_node.dl.offset, S.trident_node.t.offset,
            ctypes.sizeof(S.trident_recipe_node), S.trident_recipe_node.f.offset,
            ctypes.sizeof(S.trident_recipe), S.trident_recipe.eps.offset]
    assert got == want


# ---------------------------------------------------------------------------- selection
def _golden():
    with open(os.path.join(HERE, "golden", "guard_cases.json")) as f:
        return json.load(f)["cases"]


@pytest.mark.parametrize("case", _golden(), ids=lambda c: c["cite"])
def test_golden_cases_library(S, case):
    table = [cases.make_spec(s) for s in case["table"]]
    args = cases.make_args(case["args"])
    assert list(lib_select(S, table, args)) == case["expect"]


def _small_domain():
    specs = [cases.make_spec({"op": 1, "dtype": dt, "fixed": [64], "tok": list(G.bucket_range(b)),
                              "layout": lay, "align": al})
             for dt in ("bf16", "fp16") for lay in ("contig", "strided", "any")
             for b in (0, 1, 2) for al in (2, 16)]
    argss = [cases.make_args({"op": 1, "dtype": dt, "T": T, "H": 64, "layout": lay, "misalign": mis})
             for dt in ("bf16", "fp16") for lay in ("contig", "strided", "badrows")
             for T in (0, 1, 2, 3, 4, 5) for mis in (False, True)]
    return specs, argss


def test_bruteforce_single_version_tables(S):
    specs, argss = _small_domain()
    for sp in specs:
        s = dry(S)
        s.register(cases.lib_spec(sp))
        for a in argss:
            st, idx = s.select(cases.lib_args(a))
            assert (cases.STATUS[st], idx) == G.select([sp], a)
        s.close()


def test_bruteforce_random_three_version_tables(S):
    specs, argss = _small_domain()
    g = np.random.default_rng(12)
    for _ in range(250):
        table = [specs[i] for i in g.integers(0, len(specs), int(g.integers(0, 4)))]
        s = dry(S)
        for sp in table:
            s.register(cases.lib_spec(sp))
        for a in argss:
            st, idx = s.select(cases.lib_args(a))
            assert (cases.STATUS[st], idx) == G.select(table, a), (table, a)
        s.close()


def _mutations(args, g):
    """Random single-field mutations of an argument tuple (shapes, strides, dtypes, ...)."""
    import copy
    out = [args]
    for _ in range(60):
        a = copy.deepcopy(args)
        i = int(g.integers(0, len(a["tensors"])))
        t = a["tensors"][i]
        kind = int(g.integers(0, 7))
        if kind == 0:
            t["dtype"] = int(g.choice([1, 2, 3, 4]))
        elif kind == 1:
            d = int(g.integers(0, len(t["shape"])))
            sh = list(t["shape"]); sh[d] = max(0, sh[d] + int(g.choice([-1, 1])))
            t["shape"] = tuple(sh)
        elif kind == 2:
            d = int(g.integers(0, len(t["stride"])))
            st = list(t["stride"]); st[d] = st[d] + int(g.choice([1, 8, 64]))
            t["stride"] = tuple(st)
        elif kind == 3:
            t["addr"] += int(g.choice([2, 4, 8, 16]))
        elif kind == 4:
            t["device"] = int(g.choice([-1, 1]))
        elif kind == 5:
            a["theta"] = float(g.choice([0.0, 10000.0, a["theta"]]))
        else:
            t["shape"] = t["shape"][:-1] if len(t["shape"]) > 1 else t["shape"] + (1,)
            t["stride"] = t["stride"][:len(t["shape"])] if len(t["stride"]) > len(t["shape"]) else t["stride"] + (1,)
        out.append(a)
    return out


@pytest.mark.parametrize("op", [2, 3, 4, 5, 6, 7, 8, 9, 10, 11])
def test_mutated_arguments_every_op(S, op):
    """Library and oracle agree on valid and mutated tuples of every op."""
    g = np.random.default_rng(100 + op)
    if op in (2, 3):
        base = dict(op=op, Hq=4, Hkv=2, D=16, S=64, theta=10000.0)
        fixed = [4, 2, 16, 64]
        mk = lambda **k: cases.make_args({**base, **k})
    elif op == 4:
        base = dict(op=4, I=48)
        fixed = [48]
        mk = lambda **k: cases.make_args({**base, **k})
    elif op in (7, 8, 9, 10, 11):
        base = dict(op=op, H=128)
        fixed = [128]
        mk = lambda **k: cases.make_args({**base, **k})
    else:  # a chain version needs a size with a fused kernel (H 4096, D 128)
        base = dict(op=op, H=4096, Hq=4, Hkv=2, D=128, S=64, I=48, theta=10000.0)
        fixed = [4096, 4, 2, 128, 64, 48]
        mk = lambda **k: cases.make_chain_args({**base, **k})
    chain = op in (5, 6)  # byte-set overlap brute force is too slow at H 4096: tested apart
    table = []
    for lay in ("contig", "strided", "any"):
        for lo, hi in ((1, 2), (3, 8)):
            table.append(cases.make_spec({"op": op, "fixed": fixed, "tok": [lo, hi], "layout": lay,
                                          "theta": base.get("theta", 0.0), "align": 16}))
    s = dry(S, flags=S.OPT_NO_ALIAS_CHECK if chain else 0)
    for sp in table:
        s.register(cases.lib_spec(sp))
    for T in (1, 2, 3, 5, 9):
        for lay in ("contig", "strided"):
            for a in _mutations(mk(T=T, layout=lay), g):
                st, idx = s.select(cases.lib_args(a))
                assert (cases.STATUS[st], idx) == G.select(table, a, check_overlap=not chain), a
    s.close()


def test_structurally_invalid_calls_are_errors_not_misses(S):
    s = dry(S)
    good = cases.make_args({"op": 1, "T": 2, "H": 64})
    bad = []
    import copy
    for mut in ("op", "null", "ndim", "negshape", "negstride", "dtype", "unaligned", "eps", "flags"):
        a = copy.deepcopy(good)
        if mut == "op": a["op"] = 12
        if mut == "null": a["tensors"][0]["addr"] = 0
        if mut == "ndim": a["tensors"][0]["shape"] = (2, 1, 1, 1, 64)[:4] + ()
        if mut == "negshape": a["tensors"][1]["shape"] = (-1, 64)
        if mut == "negstride": a["tensors"][1]["stride"] = (-64, 1)
        if mut == "dtype": a["tensors"][2]["dtype"] = 9
        if mut == "unaligned": a["tensors"][2]["addr"] += 2  # fp32 needs 4-byte alignment
        if mut == "eps": a["eps"] = -1.0
        if mut == "flags": a["flags"] = 1
        bad.append((mut, a))
    for mut, a in bad:
        want = G.select([], a)
        la = cases.lib_args(a)
        if mut == "flags":
            la.flags = 1
        if mut == "ndim":
            la.t[0].ndim = 5
            want = (G.INVALID, -1)
        st, idx = s.select(la)
        assert (cases.STATUS[st], idx) == want == (G.INVALID, -1), mut
    s.close()


def test_registration_validation(S):
    s = dry(S, max_specs=4)
    good = dict(op=1, dtype=1, fixed=[64], tok_lo=1, tok_hi=8)
    assert s.register(S.make_spec(**good)) == 0
    bad = [dict(good, op=12), dict(good, dtype=4), dict(good, fixed=[0]), dict(good, fixed=[64, 1]),
           dict(good, tok_lo=0), dict(good, tok_lo=5, tok_hi=4), dict(good, align_bytes=8),
           dict(good, rank=4), dict(good, layout=3), dict(good, variant=3),
           dict(good, variant=2, align_bytes=2), dict(good, rope_theta=1.0),
           dict(op=2, dtype=1, fixed=[4, 2, 16, 64], tok_lo=1, tok_hi=8),            # theta missing
           dict(op=2, dtype=1, fixed=[4, 2, 15, 64], tok_lo=1, tok_hi=8, rope_theta=1e4),  # odd D
           dict(op=2, dtype=3, fixed=[4, 2, 16, 64], tok_lo=1, tok_hi=8, rope_theta=1e4),  # fp32 RoPE
           dict(op=5, dtype=1, fixed=[64, 4, 2, 16, 64, 48], tok_lo=1, tok_hi=8, rope_theta=1e4),  # no chain kernel
           dict(good, fixed=[60], variant=2)]                                      # 120 B rows
    for b in bad:
        with pytest.raises(S.ScmError) as e:
            s.register(S.make_spec(**b))
        assert e.value.status == S.ERR_INVALID, b
    for _ in range(3):
        s.register(S.make_spec(**good))
    with pytest.raises(S.ScmError) as e:
        s.register(S.make_spec(**good))
    assert e.value.status == S.ERR_CAPACITY
    s.close()


# ---------------------------------------------------------------------------- hook (§3.5)
def test_hook_lifecycle_growth_errors_and_reentry(S):
    calls = []

    def hook(scm, args, stream):
        calls.append(args.op)
        if args.eps == 0.5:
            raise RuntimeError("capture failed")
        T = args.t[0].shape[0]
        b = G.bucket_of(T)
        lo, hi = G.bucket_range(b)
        idx = scm.register(S.make_spec(1, args.t[0].dtype, [args.t[0].shape[1]], lo, hi))
        st, sel = scm.invoke(args)          # re-entry: now a hit
        assert (st, sel) == (S.OK, idx)
        return idx

    s = dry(S, hook=hook)
    a4 = cases.lib_args(cases.make_args({"op": 1, "T": 4, "H": 64}))
    assert s.invoke(a4) == (S.MISS_HANDLED, 0)        # empty SCM: miss path first
    assert s.invoke(a4) == (S.OK, 0)                  # later compatible call: hit
    assert s.invoke(cases.lib_args(cases.make_args({"op": 1, "T": 3, "H": 64}))) == (S.OK, 0)
    a5 = cases.lib_args(cases.make_args({"op": 1, "T": 5, "H": 64}))
    assert s.invoke(a5) == (S.MISS_HANDLED, 1)        # growth: next bucket
    assert len(calls) == 2
    bad = cases.lib_args(cases.make_args({"op": 1, "T": 4, "H": 64, "ntensors_delta": -1}))
    assert s.invoke(bad)[0] == S.ERR_INVALID          # error: hook not called
    assert len(calls) == 2
    err = cases.lib_args(cases.make_args({"op": 1, "T": 64, "H": 64}))
    err.eps = 0.5
    assert s.invoke(err)[0] == S.ERR_HOOK             # hook failure: error, nothing registered
    st = s.stats()
    assert (st.num_specs, st.hits, st.misses, st.hook_calls, st.hook_failures, st.hook_registered,
            st.err_invalid) == (2, 4, 3, 3, 1, 2, 1)  # hits: 2 re-entries + 2 direct
    s.close()


def test_miss_inside_hook_does_not_recurse(S):
    depth = []

    def hook(scm, args, stream):
        depth.append(1)
        return None if scm.invoke(args)[0] == S.MISS else -5

    s = dry(S, hook=hook)
    a = cases.lib_args(cases.make_args({"op": 1, "T": 4, "H": 64}))
    assert s.invoke(a) == (S.MISS_HANDLED, -1)
    assert len(depth) == 1
    s.close()


def test_no_hook_returns_miss(S):
    s = dry(S)
    assert s.invoke(cases.lib_args(cases.make_args({"op": 1, "T": 4, "H": 64}))) == (S.MISS, -1)
    s.close()


def test_invoke_seq_stops_at_first_miss(S):
    s = dry(S)
    s.register(S.make_spec(1, 1, [64], 1, 8))
    hit = cases.lib_args(cases.make_args({"op": 1, "T": 4, "H": 64}))
    miss = cases.lib_args(cases.make_args({"op": 1, "T": 40, "H": 64}))
    arr = (S.trident_args * 3)(hit, miss, hit)
    assert S.trident_scm_invoke_seq(s.h, arr) == (S.MISS, [0, -1, S.NOT_RUN])
    arr = (S.trident_args * 2)(hit, hit)
    assert S.trident_scm_invoke_seq(s.h, arr) == (S.OK, [0, 0])
    s.close()


# ---------------------------------------------------------------------------- overlap
def test_overlap_precondition_matches_bruteforce(S):
    """Outputs placed at random offsets inside the inputs' buffers (same row stride):
    the library's O(1) row test equals the oracle's byte-set brute force."""
    g = np.random.default_rng(13)
    s = dry(S)
    s.register(S.make_spec(1, 1, [8], 1, 8, layout=S.LAYOUT_ANY, align_bytes=2))
    base = cases.BASE
    for _ in range(400):
        T = int(g.integers(1, 5))
        rs = int(g.choice([8, 12, 16, 24]))
        x = cases.tensor(base, 1, (T, 8), (rs, 1))
        r = cases.tensor(base + (1 << 20), 1, (T, 8), (rs, 1))
        gam = cases.tensor(base + (2 << 20), 3, (8,))
        y = cases.tensor(base + 2 * int(g.integers(-40, 40)), 1, (T, 8), (rs, 1))
        ro = cases.tensor(base + (1 << 20) + 2 * int(g.integers(-40, 40)), 1, (T, 8), (rs, 1))
        if g.random() < 0.2:
            y = dict(x)
        if g.random() < 0.2:
            ro = dict(r)
        a = dict(op=1, tensors=[x, r, gam, y, ro], eps=1e-6, theta=0.0, flags=0)
        st, idx = s.select(cases.lib_args(a))
        assert (cases.STATUS[st], idx) == G.select([cases.make_spec(
            {"op": 1, "fixed": [8], "tok": [1, 8], "layout": "any", "align": 2})], a), a
    s.close()


def test_overlap_conservative_for_different_row_strides(S):
    """Interleaved rows with different strides that share no byte: the oracle accepts,
    the library (exact only for equal strides) conservatively reports an error."""
    s = dry(S)
    s.register(S.make_spec(1, 1, [4], 1, 8, layout=S.LAYOUT_ANY, align_bytes=2))
    base = cases.BASE
    x = cases.tensor(base, 1, (2, 4), (16, 1))             # bytes [0,8) and [32,40)
    y = cases.tensor(base + 8, 1, (2, 4), (12, 1))         # bytes [8,16) and [32+..): [8,16),[32,40)?
    y = cases.tensor(base + 10, 1, (2, 4), (8, 1))         # bytes [10,18) and [26,34)? overlaps [32,40)
    y = cases.tensor(base + 8, 1, (2, 4), (4, 1))          # bytes [8,16) and [16,24): disjoint from x
    r = cases.tensor(base + (1 << 20), 1, (2, 4))
    gam = cases.tensor(base + (2 << 20), 3, (4,))
    ro = cases.tensor(base + (3 << 20), 1, (2, 4))
    a = dict(op=1, tensors=[x, r, gam, y, ro], eps=1e-6, theta=0.0, flags=0)
    assert G.launch_precondition(a)
    assert s.select(cases.lib_args(a))[0] == S.ERR_INVALID
    s.close()
    s = dry(S, flags=S.OPT_NO_ALIAS_CHECK)
    s.register(S.make_spec(1, 1, [4], 1, 8, layout=S.LAYOUT_ANY, align_bytes=2))
    assert s.select(cases.lib_args(a)) == (S.OK, 0)
    s.close()


# ---------------------------------------------------------------------------- concurrency
def test_concurrent_growth_and_invoke(S):
    """A reader never sees a half-written version while another thread registers."""
    s = dry(S, max_specs=600)
    stop = threading.Event()
    errors = []
    argss = [cases.lib_args(cases.make_args({"op": 1, "T": T, "H": 64})) for T in (1, 2, 3, 4)]

    def reader():
        while not stop.is_set():
            for a in argss:
                st, idx = s.select(a)
                if st not in (S.OK, S.MISS):
                    errors.append((st, idx))
                if st == S.OK and idx != 0:
                    errors.append(("first match", idx))

    th = [threading.Thread(target=reader) for _ in range(3)]
    for t in th:
        t.start()
    for i in range(500):
        s.register(S.make_spec(1, 1, [64], 1, 1 << 20))
    stop.set()
    for t in th:
        t.join()
    assert not errors
    assert s.stats().num_specs == 500
    s.close()


def test_fastcall_shim_matches_ctypes(S):
    """The CPython fast-call shim calls the same entry points (dry run, NULL stream = 0)."""
    import ctypes
    fc = S.fastcall()
    if fc is None:
        pytest.skip("Python headers not installed: the binding uses ctypes only")
    s = dry(S)
    s.register(S.make_spec(1, 1, [64], 1, 8))
    hit = cases.lib_args(cases.make_args({"op": 1, "T": 4, "H": 64}))
    miss = cases.lib_args(cases.make_args({"op": 1, "T": 40, "H": 64}))
    bad = cases.lib_args(cases.make_args({"op": 1, "T": 4, "H": 64, "ntensors_delta": -1}))
    h = s.h.value
    assert fc.invoke(h, ctypes.addressof(hit), 0) == S.OK
    assert fc.invoke(h, ctypes.addressof(miss), 0) == S.MISS
    assert fc.invoke(h, ctypes.addressof(bad), 0) == S.ERR_INVALID
    arr = (S.trident_args * 3)(hit, hit, miss)
    assert fc.invoke_seq(h, ctypes.addressof(arr), 3, 0) == S.MISS
    st = s.stats()
    assert (st.hits, st.misses, st.err_invalid) == (3, 2, 1)
    with pytest.raises(TypeError):
        fc.invoke(h, ctypes.addressof(hit), None)
    # invoke_step and invoke_tree through the shim
    assert fc.invoke_step(h, ctypes.addressof(arr), 2, 0) == S.OK
    s.register_tree(S.make_spec(1, 1, [64], 1, 8), S.Recipe(S.Slot(0), S.Slot(1), S.Slot(2),
                                                             (S.Slot(3), S.Slot(4)), S.EPS))
    x, r, w, y, ro = cases.make_args({"op": 1, "T": 4, "H": 64})["tensors"]
    tree = S.Tree(x, r, w, (y, ro), 1e-6)
    assert fc.invoke_tree(h, ctypes.addressof(tree.nodes), tree.nargs, tree.nnodes, 0) == S.OK
    assert fc.invoke_tree(h, ctypes.addressof(tree.nodes), tree.nargs, tree.nnodes - 1, 0) == S.ERR_INVALID
    with pytest.raises(ValueError):
        fc.invoke_tree(h, ctypes.addressof(tree.nodes), -1, tree.nnodes, 0)
    assert s.stats().hits == 6
    s.close()


def test_execution_error_is_raised_not_retried(S):
    """Algorithm 1 (§3.2): when the selected P_i fails, the error propagates at once -- no
    later version is tried, the compile hook is not called, nothing is registered (§3.5).
    The failure is injected on the host (no GPU fault)."""
    calls = []
    s = dry(S, hook=lambda scm, args, stream: calls.append(1), flags=S.OPT_FAIL_LAUNCHES)
    s.register(S.make_spec(1, 1, [64], 1, 8))
    s.register(S.make_spec(1, 1, [64], 1, 8))  # a second matching version is never reached
    a = cases.lib_args(cases.make_args({"op": 1, "T": 4, "H": 64}))
    st, sel = s.invoke(a)
    assert st == S.ERR_CUDA and sel == 0
    assert "injected" in S.trident_scm_last_error()
    stt = s.stats()
    assert (stt.hits, stt.misses, stt.err_cuda, stt.hook_calls, stt.num_specs) == (0, 0, 1, 0, 2)
    assert not calls
    # a miss still takes the hook path, and an error inside a sequence stops it
    miss = cases.lib_args(cases.make_args({"op": 1, "T": 40, "H": 64}))
    assert s.invoke(miss) == (S.MISS_HANDLED, -1) and len(calls) == 1
    arr = (S.trident_args * 3)(miss, a, miss)
    st, sels = S.trident_scm_invoke_seq(s.h, arr)
    assert st == S.ERR_CUDA and sels == [-1, 0, S.NOT_RUN] and len(calls) == 2
    s.close()


def test_launch_floor_probe_rejects_dry_runs_and_bad_counts(S):
    s = S.Scm(device=0, flags=S.OPT_DRY_RUN)
    assert S.trident_launch_floor(s.h, None, 1) == S.ERR_STATE
    assert S.trident_launch_floor(s.h, None, -1) == S.ERR_INVALID
    assert S.trident_launch_floor(None, None, 1) == S.ERR_INVALID
    s.close()


def test_nvtx_ranges_build_only_with_the_flag(S, tmp_path):
    """NVTX ranges around the boundary calls are compiled in only with -DTRIDENT_NVTX: the
    default library references no NVTX symbol, and the flagged host core still compiles."""
    from paper_2609_37241_gb300 import build as B
    nm = subprocess.run(["nm", "-D", S.LIB_PATH], capture_output=True, text=True).stdout
    assert "nvtx" not in nm.lower()
    src = os.path.join(B.CSRC, "scm.cpp")
    obj = tmp_path / "scm_nvtx.o"
    subprocess.run([B.nvcc(), *B.ARCH, *B.FLAGS, "-DTRIDENT_NVTX", "-c", src, "-o", str(obj)], check=True)
    syms = subprocess.run(["nm", str(obj)], capture_output=True, text=True).stdout
    assert "nvtx" in syms.lower()


def test_noalloc_rejects_calls_without_heads(S):
    """The allocation-free RoPE entry validates its tuple on the host before any CUDA call: a
    call whose q and k have no heads (nothing to map a unit to) is ERR_INVALID, as is a
    malformed one, and neither needs a GPU."""
    args = cases.make_args({"op": 2, "T": 4, "Hq": 0, "Hkv": 0, "D": 128, "S": 64})
    st = S.trident_rope_kv_noalloc(cases.lib_args(dict(args, theta=1e4)), None)
    assert st == S.ERR_INVALID and "no heads" in S.trident_scm_last_error()
    args = cases.make_args({"op": 2, "T": 4, "Hq": 4, "Hkv": 2, "D": 128, "S": 64})
    args["tensors"][3] = dict(args["tensors"][3], dtype=cases.DT["fp32"])  # positions must be int32
    st = S.trident_rope_kv_noalloc(cases.lib_args(dict(args, theta=1e4)), None)
    assert st == S.ERR_INVALID


def test_copy_floor_probe_rejects_dry_runs_and_bad_arguments(S):
    s = S.Scm(device=0, flags=S.OPT_DRY_RUN)
    a, b = 1 << 20, 2 << 20  # never dereferenced: every call below is refused first
    assert S.trident_copy_floor(s.h, None, a, b, 4096, 1024, 8, 2, 1) == S.ERR_STATE
    for args in ((a, b, 4095, 1024, 8, 2, 1), (a, b, 4096, 0, 8, 2, 1), (a + 8, b, 4096, 1024, 8, 2, 1),
                 (a, b, 4096, 1024, 0, 2, 1), (a, b, 4096, 1024, 8, 0, 1), (a, b, 4096, 1024, 8, 2, -1),
                 (None, b, 4096, 1024, 8, 2, 1)):
        assert S.trident_copy_floor(s.h, None, *args) == S.ERR_INVALID, args
    assert S.trident_copy_floor(None, None, a, b, 4096, 1024, 8, 2, 1) == S.ERR_INVALID
    s.close()
