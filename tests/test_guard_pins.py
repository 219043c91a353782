"""Pins of the guard oracle (`oracle.guards`) against definitions written apart from it.

Algorithm 1 (§3.2) selects the first version, in creation order, whose guard holds, and
misses when none does. Over a tiny domain the selected index therefore has a plain
set-based definition, min{i : every guarded field of version i matches the call}, which
this file writes out from the generating parameters of each call (dtype, layout, token
count, alignment) -- not from the oracle's tensor-level predicates. Every table of at most
three versions drawn from {bf16, fp16} x {contiguous, row-strided} x token buckets
{1}, {2}, {3,4} x {16-byte, natural} alignment is checked against every call of the same
domain, so a dropped term, a wrong bucket edge or a swapped field anywhere in the oracle's
guard or in its ordering fails here.

The second half pins, by hand, the three guard branches the brute force does not reach:
the cache-stride clause of the auxiliary layouts, the collapse of rank-3 activations whose
batch or sequence size is 1, and the head-packing test of q/k/v views. Each expected
result is decided from the reading it cites (guard readings 1, 3 and 5: caches dense
[Hkv, S, D]; one-row tensors count as contiguous, ROWSTRIDED needs every row stride >= the
width, no class when inner dims are not packed; rank-3 [B, S, W] collapses to B*S rows).
The same hand cases run through the library's selection when it is built."""
import itertools

import pytest

from oracle import guards as G
from tests import cases

H = 64
DTYPES = ("bf16", "fp16")
SPEC_LAYOUTS = ("contig", "strided")
BUCKETS = {1: (1, 1), 2: (2, 2), 4: (3, 4)}  # named by their upper edge
SPEC_ALIGNS = {"ok": 16, "bad": 2}            # 16-byte alignment required, or natural only
CALL_LAYOUTS = ("contig", "strided", "badrows")
CALL_T = (0, 1, 2, 3, 4, 5)


# ----------------------------------------------------------------------------- independent definition
def _spec_params():
    return [dict(dtype=dt, layout=lay, bucket=b, align=al)
            for dt in DTYPES for lay in SPEC_LAYOUTS for b in BUCKETS for al in SPEC_ALIGNS]


def _call_params():
    return [dict(dtype=dt, layout=lay, T=T, misaligned=mis)
            for dt in DTYPES for lay in CALL_LAYOUTS for T in CALL_T for mis in (False, True)]


def _row_class(call):
    """Layout class of the call's rows: a call of at most one row is contiguous whatever its
    row stride; otherwise contiguous rows, padded rows (stride > width) or no class
    (stride < width, rows overlap)."""
    if call["T"] <= 1:
        return "contig"
    return {"contig": "contig", "strided": "strided", "badrows": None}[call["layout"]]


def _fields_match(spec, call):
    """Every guarded field of one version against one call, field by field."""
    lo, hi = BUCKETS[spec["bucket"]]
    return (spec["dtype"] == call["dtype"]
            and lo <= call["T"] <= hi
            and _row_class(call) == spec["layout"]
            and (spec["align"] == "bad" or not call["misaligned"]))


def _expected(table, call):
    hits = {i for i, spec in enumerate(table) if _fields_match(spec, call)}
    return (G.OK, min(hits)) if hits else (G.MISS, -1)


def _oracle_spec(p):
    return cases.make_spec({"op": 1, "dtype": p["dtype"], "fixed": [H], "tok": list(BUCKETS[p["bucket"]]),
                            "layout": p["layout"], "align": SPEC_ALIGNS[p["align"]]})


def _oracle_args(c):
    return cases.make_args({"op": 1, "dtype": c["dtype"], "T": c["T"], "H": H, "layout": c["layout"],
                            "misalign": c["misaligned"]})


def test_domain_is_what_the_definition_assumes():
    """The descriptors the oracle sees have the properties the definition reads off the
    generating parameters: misaligned calls start off a 16-byte boundary, aligned calls have
    16-byte-multiple row strides, padded rows are wider than the row, bad rows narrower."""
    for c in _call_params():
        a = _oracle_args(c)
        x = a["tensors"][0]
        assert (x["addr"] % 16 != 0) == c["misaligned"]
        if c["T"] >= 1:
            rs = x["stride"][0]
            assert (rs * 2) % 16 == 0
            assert {"contig": rs == H, "strided": rs > H, "badrows": rs < H}[c["layout"]]


def test_every_table_of_at_most_three_versions():
    """G.select equals min{i : fields match} for all 1 + 24 + 24^2 + 24^3 tables and all
    72 calls of the domain (the empty table misses everything)."""
    sps = _spec_params()
    calls = _call_params()
    oracle_specs = [_oracle_spec(p) for p in sps]
    oracle_args = [_oracle_args(c) for c in calls]
    n = 0
    for size in range(4):
        for idx in itertools.product(range(len(sps)), repeat=size):
            table = [sps[i] for i in idx]
            otable = [oracle_specs[i] for i in idx]
            for c, a in zip(calls, oracle_args):
                got = G.select(otable, a, check_overlap=False)
                assert got == _expected(table, c), (table, c, got)
                n += 1
    assert n == (1 + 24 + 24 ** 2 + 24 ** 3) * 72


def test_overlap_check_does_not_change_the_domain():
    """The calls of the domain use disjoint buffers, so the launch precondition holds on
    every hit and selection with it equals selection without it."""
    sps = _spec_params()
    otable = [_oracle_spec(p) for p in sps]
    for c in _call_params():
        a = _oracle_args(c)
        assert G.select(otable, a) == G.select(otable, a, check_overlap=False) == _expected(sps, c)


def test_definition_has_every_outcome():
    """The domain reaches hits at index 0, 1 and 2 and misses for every reason the
    definition has (dtype, bucket, layout class, no class, alignment, T = 0)."""
    sps = _spec_params()
    seen = set()
    for t in itertools.product(range(len(sps)), repeat=3):
        for c in _call_params():
            seen.add(_expected([sps[i] for i in t], c)[1])
        if seen >= {-1, 0, 1, 2}:
            break
    assert seen >= {-1, 0, 1, 2}
    assert _expected(sps, dict(dtype="bf16", layout="contig", T=0, misaligned=False)) == (G.MISS, -1)
    assert _expected(sps, dict(dtype="bf16", layout="badrows", T=3, misaligned=False)) == (G.MISS, -1)
    assert _expected(sps, dict(dtype="bf16", layout="badrows", T=1, misaligned=False))[0] == G.OK


# ----------------------------------------------------------------------------- hand pins
def _rope_spec(layout="any"):
    return cases.make_spec({"op": 2, "dtype": "bf16", "fixed": [4, 2, 8, 16], "tok": [1, 64],
                            "layout": layout, "theta": 10000.0})


def _rope_args(T=3, layout="contig"):
    return cases.make_args({"op": 2, "dtype": "bf16", "T": T, "Hq": 4, "Hkv": 2, "D": 8, "S": 16,
                            "layout": layout, "theta": 10000.0})


def _cache_cases():
    """Reading 1: the caches are dense [Hkv, S, D] arrays, strides (S*D, D, 1)."""
    Hkv, S, D = 2, 16, 8
    out = []
    a = _rope_args()
    out.append(("dense cache [Hkv,S,D]", a, (G.OK, 0)))
    for slot in (4, 5):
        # the same shape viewed out of an [S, Hkv, D] buffer: strides (D, Hkv*D, 1)
        a = _rope_args()
        a["tensors"][slot]["stride"] = (D, Hkv * D, 1)
        out.append((f"slot {slot}: cache transposed from [S,Hkv,D]", a, (G.MISS, -1)))
        # padded slots: a slot stride above D (rows still 16-byte aligned)
        a = _rope_args()
        a["tensors"][slot]["stride"] = (S * 2 * D, 2 * D, 1)
        out.append((f"slot {slot}: cache with padded slots", a, (G.MISS, -1)))
        # padded heads: a head stride above S*D
        a = _rope_args()
        a["tensors"][slot]["stride"] = (S * D + 8, D, 1)
        out.append((f"slot {slot}: cache with padded heads", a, (G.MISS, -1)))
    return out


def _rank3_norm(B, S, stride_of, layout_spec):
    """ADD_RMSNORM over [B, S, H] activations, every activation with strides stride_of."""
    spec = cases.make_spec({"op": 1, "dtype": "bf16", "rank": 3, "fixed": [H], "tok": [1, 64],
                            "layout": layout_spec})
    a = cases.make_args({"op": 1, "dtype": "bf16", "rank": 3, "B": B, "T": B * S, "H": H})
    for k in (0, 1, 3, 4):
        a["tensors"][k]["stride"] = stride_of
    return spec, a


def _rank3_cases():
    """Reading 5 (rank-3 [B, S, W] collapses to B*S rows) with reading 3's classes: the row
    stride of a collapsed view is the stride of the dimension that still has size > 1, and
    a dimension of size 1 contributes no stride (its stride is never used)."""
    out = []
    odd = 4096 * 3 + 8  # a stride nobody would read as a row stride (16-byte multiple)
    # [1, S, W]: rows are the S dim; the batch stride is arbitrary
    for lay, want in (("contig", (G.OK, 0)), ("strided", (G.MISS, -1))):
        spec, a = _rank3_norm(1, 4, (odd, H, 1), lay)
        out.append((f"[1,4,W] batch stride {odd}, spec {lay}", spec, a, want))
    for lay, want in (("contig", (G.MISS, -1)), ("strided", (G.OK, 0))):
        spec, a = _rank3_norm(1, 4, (odd, H + 8, 1), lay)
        out.append((f"[1,4,W] padded rows, batch stride {odd}, spec {lay}", spec, a, want))
    # [B, 1, W]: rows are the B dim; the sequence stride is arbitrary
    for lay, want in (("contig", (G.OK, 0)), ("strided", (G.MISS, -1))):
        spec, a = _rank3_norm(4, 1, (H, odd, 1), lay)
        out.append((f"[4,1,W] seq stride {odd}, spec {lay}", spec, a, want))
    for lay, want in (("contig", (G.MISS, -1)), ("strided", (G.OK, 0))):
        spec, a = _rank3_norm(4, 1, (H + 8, odd, 1), lay)
        out.append((f"[4,1,W] padded rows, seq stride {odd}, spec {lay}", spec, a, want))
    # [B, S, W] with B, S > 1: the two outer dims collapse only when stride[0] == S*stride[1]
    spec, a = _rank3_norm(2, 2, (2 * H, H, 1), "any")
    out.append(("[2,2,W] dense", spec, a, (G.OK, 0)))
    spec, a = _rank3_norm(2, 2, (2 * (H + 8), H + 8, 1), "strided")
    out.append(("[2,2,W] uniformly padded rows", spec, a, (G.OK, 0)))
    spec, a = _rank3_norm(2, 2, (4 * H, H, 1), "any")
    out.append(("[2,2,W] batch stride breaks the row sequence", spec, a, (G.MISS, -1)))
    spec, a = _rank3_norm(2, 2, (H, 2 * H, 1), "any")
    out.append(("[2,2,W] outer dims transposed", spec, a, (G.MISS, -1)))
    return out


def _heads_cases():
    """Reading 3 (no class when the inner dims are not packed): a [T, Hn, D] view is packed
    when its elements are unit-stride and its heads are D apart (or there is one head); its
    rows are then T rows of Hn*D elements, contiguous or row-strided by the token stride."""
    D, Hq, Hkv = 8, 4, 2
    out = []
    a = _rope_args(layout="strided")  # q/k/v as views of one fused qkv buffer
    out.append(("qkv views of one buffer", a, (G.OK, 0)))
    a = _rope_args()
    a["tensors"][0]["stride"] = (Hq * 2 * D, 2 * D, 1)  # q heads 2D apart
    out.append(("q head stride 2D", a, (G.MISS, -1)))
    a = _rope_args()
    a["tensors"][1]["stride"] = (Hkv * 2 * D, 2 * D, 1)  # k heads 2D apart
    out.append(("k head stride 2D", a, (G.MISS, -1)))
    a = _rope_args()
    a["tensors"][2]["stride"] = (Hq * D, D, 2)  # v elements 2 apart (and head stride D)
    out.append(("v element stride 2", a, (G.MISS, -1)))
    a = _rope_args()
    a["tensors"][0]["stride"] = (D, Hq * D, 1)  # q as [T, Hq, D] transposed from [Hq, T, D]
    out.append(("q token and head dims transposed", a, (G.MISS, -1)))
    return out


def _heads_one_head_cases():
    """One kv head: the head stride is never used, any value is packed."""
    spec = cases.make_spec({"op": 2, "dtype": "bf16", "fixed": [4, 1, 8, 16], "tok": [1, 64],
                            "layout": "any", "theta": 10000.0})
    a = cases.make_args({"op": 2, "dtype": "bf16", "T": 3, "Hq": 4, "Hkv": 1, "D": 8, "S": 16,
                         "theta": 10000.0})
    a["tensors"][1]["stride"] = (8, 4096, 1)
    a["tensors"][2]["stride"] = (8, 8, 1)
    return [("one kv head, arbitrary head stride", spec, a, (G.OK, 0))]


def _all_hand_cases():
    out = [(n, _rope_spec(), a, w) for n, a, w in _cache_cases()]
    out += _rank3_cases()
    out += [(n, _rope_spec(), a, w) for n, a, w in _heads_cases()]
    out += _heads_one_head_cases()
    return out


@pytest.mark.parametrize("name,spec,args,want", _all_hand_cases(), ids=lambda v: v if isinstance(v, str) else "")
def test_hand_pins_oracle(name, spec, args, want):
    assert G.validate(args), name
    assert G.select([spec], args) == want, name


@pytest.mark.parametrize("name,spec,args,want", _all_hand_cases(), ids=lambda v: v if isinstance(v, str) else "")
def test_hand_pins_library(built_lib, name, spec, args, want):
    from paper_2609_37241_gb300 import scm
    s = scm.Scm(device=0, max_specs=4, flags=scm.OPT_DRY_RUN)
    try:
        s.register(cases.lib_spec(spec))
        st, idx = s.select(cases.lib_args(args))
    finally:
        s.close()
    assert (cases.STATUS[st], idx) == want, name
