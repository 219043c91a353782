"""Oracle for guarded specialisation selection -- TEST INFRASTRUCTURE ONLY.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may import this
module. The product path (the C-ABI library and its binding) never calls it.

It restates, as plainly as possible, what the SCM dispatcher must decide:

* Algorithm 1 (§3.2): versions are tried in creation order; the first version whose
  guard G_i holds is selected; if every G_i fails the result is MISS.
* The guard G_i is a short-circuit conjunction of checks over the source-level
  arguments (§3.2 and Fig. 4: a rank check, then shape checks; any failure is a miss).
  The guard kinds follow §2.2.1 (dtype, device, shape-related metadata, and bounds such
  as a size upper bound); the concrete field list -- op, device, dtype, rank, fixed
  sizes, token-count bucket, layout class, 16-byte alignment, and the specialised RoPE
  base -- is this library's choice of guarded metadata.
* Malformed arguments are neither a hit nor a miss but an error (§3.4: a miss keeps its
  own tag so it is never confused with a failure; §3.5: an error never triggers growth).
* A selected version checks its launch preconditions just before the launch (§3.3, §3.4):
  here, that no output shares a byte with another argument except the documented
  in-place pairs. This module decides overlap by brute force over element byte sets,
  so it is only meant for small test tensors.

Everything is plain Python over plain dicts:
  tensor = dict(addr, dtype, shape, stride, device)     (shape/stride tuples, elements)
  args   = dict(op, tensors, eps, theta, flags)
  spec   = dict(op, dtype, rank, layout, fixed, tok_lo, tok_hi, align, device, variant, theta)
"""

OK, MISS, INVALID = "OK", "MISS", "INVALID"

BF16, FP16, FP32, I32, I64, U8 = 1, 2, 3, 4, 5, 6
ELEM_SIZE = {BF16: 2, FP16: 2, FP32: 4, I32: 4, I64: 8, U8: 1}

ADD_RMSNORM, ROPE_KV, QKNORM_ROPE_KV, SWIGLU, LAYER_CHAIN, LAYER_CHAIN_QKNORM, RMSNORM = 1, 2, 3, 4, 5, 6, 7
SILU, ADD, NEG, MASKED_FILL = 8, 9, 10, 11

CONTIG, ROWSTRIDED, ANY = 0, 1, 2
LAYOUT_NONE = -1

# Slot tables. Each slot: (name, kind, is_output). Kinds:
#   "act_H" [T,H] activation; "act_I" [T,I] activation; "gamma_H" [H] fp32;
#   "gamma_D" [D] fp32; "heads_q" [T,Hq,D]; "heads_kv" [T,Hkv,D]; "pos" [T] i32;
#   "cache" [Hkv,S,D] activation dtype.
SLOTS = {
    ADD_RMSNORM: [("x", "act_H", False), ("r", "act_H", False), ("gamma", "gamma_H", False),
                  ("y", "act_H", True), ("r_out", "act_H", True)],
    ROPE_KV: [("q", "heads_q", True), ("k", "heads_kv", False), ("v", "heads_kv", False),
              ("pos", "pos", False), ("k_cache", "cache", True), ("v_cache", "cache", True)],
    SWIGLU: [("g", "act_I", False), ("u", "act_I", False), ("out", "act_I", True)],
    LAYER_CHAIN: [("h", "act_H", False), ("r0", "act_H", False), ("gamma_attn", "gamma_H", False),
                  ("x1", "act_H", True), ("r1", "act_H", True),
                  ("q", "heads_q", True), ("k", "heads_kv", False), ("v", "heads_kv", False),
                  ("pos", "pos", False), ("k_cache", "cache", True), ("v_cache", "cache", True),
                  ("attn_out", "act_H", False), ("gamma_mlp", "gamma_H", False),
                  ("x2", "act_H", True), ("r2", "act_H", True),
                  ("g", "act_I", False), ("u", "act_I", False), ("o", "act_I", True)],
}
SLOTS[RMSNORM] = [("x", "act_H", False), ("gamma", "gamma_H", False), ("y", "act_H", True)]
# pointwise operators over [T, W] rows (W is the version's fixed size, named "H" here)
SLOTS[SILU] = [("x", "act_H", False), ("y", "act_H", True)]
SLOTS[NEG] = [("x", "act_H", False), ("y", "act_H", True)]
SLOTS[ADD] = [("a", "act_H", False), ("b", "act_H", False), ("y", "act_H", True)]
SLOTS[MASKED_FILL] = [("x", "act_H", False), ("mask", "mask_H", False), ("y", "act_H", True)]
SLOTS[QKNORM_ROPE_KV] = SLOTS[ROPE_KV] + [("gamma_q", "gamma_D", False), ("gamma_k", "gamma_D", False)]
SLOTS[LAYER_CHAIN_QKNORM] = SLOTS[LAYER_CHAIN] + [("gamma_q", "gamma_D", False),
                                                  ("gamma_k", "gamma_D", False)]

# Groups of slots that may be the very same tensor (in-place operation).
INPLACE_GROUPS = {
    ADD_RMSNORM: [{"x", "y"}, {"r", "r_out"}],
    ROPE_KV: [],
    QKNORM_ROPE_KV: [],
    SWIGLU: [{"g", "u", "out"}],
    LAYER_CHAIN: [{"h", "x1"}, {"r0", "r1", "r2"}, {"attn_out", "x2"}, {"g", "u", "o"}],
}
INPLACE_GROUPS[LAYER_CHAIN_QKNORM] = INPLACE_GROUPS[LAYER_CHAIN]
INPLACE_GROUPS[RMSNORM] = [{"x", "y"}]
INPLACE_GROUPS[SILU] = [{"x", "y"}]
INPLACE_GROUPS[NEG] = [{"x", "y"}]
INPLACE_GROUPS[ADD] = [{"a", "b", "y"}]
INPLACE_GROUPS[MASKED_FILL] = [{"x", "y"}]

# Names of the fixed sizes of each op, in spec["fixed"] order.
FIXED_NAMES = {
    ADD_RMSNORM: ("H",), SWIGLU: ("I",), RMSNORM: ("H",),
    SILU: ("H",), NEG: ("H",), ADD: ("H",), MASKED_FILL: ("H",),
    ROPE_KV: ("Hq", "Hkv", "D", "S"), QKNORM_ROPE_KV: ("Hq", "Hkv", "D", "S"),
    LAYER_CHAIN: ("H", "Hq", "Hkv", "D", "S", "I"),
    LAYER_CHAIN_QKNORM: ("H", "Hq", "Hkv", "D", "S", "I"),
}
ROPE_OPS = (ROPE_KV, QKNORM_ROPE_KV, LAYER_CHAIN, LAYER_CHAIN_QKNORM)
FLATTENING_OPS = (ADD_RMSNORM, SWIGLU, RMSNORM, SILU, ADD, NEG, MASKED_FILL)  # rank 2 or 3


def numel(t):
    n = 1
    for s in t["shape"]:
        n *= s
    return n


# ----------------------------------------------------------------------------- validation
def validate(args):
    """Structural validation: True if the tuple is well formed (else the call is an error)."""
    op = args["op"]
    if op not in SLOTS:
        return False
    if len(args["tensors"]) != len(SLOTS[op]):
        return False
    if args.get("flags", 0) != 0:
        return False
    eps = args["eps"]
    if not (eps >= 0.0):  # also rejects NaN
        return False
    for t in args["tensors"]:
        if t["dtype"] not in ELEM_SIZE:
            return False
        nd = len(t["shape"])
        if nd < 1 or nd > 4 or len(t["stride"]) != nd:
            return False
        if any(s < 0 for s in t["shape"]) or any(s < 0 for s in t["stride"]):
            return False
        if t["device"] < -1:
            return False
        if numel(t) > 0 and t["addr"] == 0:
            return False
        if t["addr"] % ELEM_SIZE[t["dtype"]] != 0:
            return False
    return True


# ----------------------------------------------------------------------------- the guard
def token_count(op, slot0):
    """T: rows of the primary activation (leading dims flattened for rank-3 activations)."""
    if op in FLATTENING_OPS and len(slot0["shape"]) == 3:
        return slot0["shape"][0] * slot0["shape"][1]
    return slot0["shape"][0]


def expected_rank(op, kind, spec_rank):
    if kind in ("act_H", "act_I", "mask_H"):
        return spec_rank if op in FLATTENING_OPS else 2
    return {"gamma_H": 1, "gamma_D": 1, "pos": 1, "heads_q": 3, "heads_kv": 3, "cache": 3}[kind]


def expected_dtype(kind, spec_dtype):
    if kind in ("gamma_H", "gamma_D"):
        return FP32
    if kind == "pos":
        return I32
    if kind == "mask_H":
        return U8
    return spec_dtype


def shape_ok(kind, shape, lead, fx):
    """Does `shape` equal what slot `kind` must have, given the leading dims `lead` of slot 0
    (one entry for rank 2, two for rank 3) and the version's fixed sizes `fx`?"""
    if kind in ("act_H", "mask_H"):
        return list(shape) == list(lead) + [fx["H"]]
    if kind == "act_I":
        return list(shape) == list(lead) + [fx["I"]]
    if kind == "gamma_H":
        return list(shape) == [fx["H"]]
    if kind == "gamma_D":
        return list(shape) == [fx["D"]]
    if kind == "heads_q":
        return list(shape) == [lead[0], fx["Hq"], fx["D"]]
    if kind == "heads_kv":
        return list(shape) == [lead[0], fx["Hkv"], fx["D"]]
    if kind == "pos":
        return list(shape) == [lead[0]]
    if kind == "cache":
        return list(shape) == [fx["Hkv"], fx["S"], fx["D"]]
    raise AssertionError(kind)


def rows_of(t, kind):
    """(rows, row_width, row_stride, packed) of an activation tensor viewed as rows."""
    shape, stride = t["shape"], t["stride"]
    if kind in ("heads_q", "heads_kv"):
        n, hn, d = shape
        packed = stride[2] == 1 and (hn <= 1 or stride[1] == d)
        return n, hn * d, stride[0], packed
    if len(shape) == 2:
        return shape[0], shape[1], stride[0], stride[1] == 1
    b, s, w = shape
    packed = stride[2] == 1
    if s == 1:
        return b, w, stride[0], packed
    if b == 1:
        return s, w, stride[1], packed
    return b * s, w, stride[1], packed and stride[0] == s * stride[1]


def layout_class(args):
    op = args["op"]
    all_contig = True
    for (name, kind, _), t in zip(SLOTS[op], args["tensors"]):
        if kind not in ("act_H", "act_I", "mask_H", "heads_q", "heads_kv"):
            continue
        rows, width, rstride, packed = rows_of(t, kind)
        if not packed:
            return LAYOUT_NONE
        if rows <= 1:
            continue
        if rstride < width:
            return LAYOUT_NONE
        if rstride != width:
            all_contig = False
    return CONTIG if all_contig else ROWSTRIDED


def aux_layout_ok(args, fx):
    """gamma and pos must be dense vectors, the caches dense [Hkv,S,D] arrays."""
    op = args["op"]
    for (name, kind, _), t in zip(SLOTS[op], args["tensors"]):
        if kind in ("gamma_H", "gamma_D", "pos"):
            if t["shape"][0] > 1 and t["stride"][0] != 1:
                return False
        if kind == "cache":
            if tuple(t["stride"]) != (fx["S"] * fx["D"], fx["D"], 1):
                return False
    return True


def aligned16(args):
    """Every tensor the kernels move in 16-byte units -- all but the positions, which are
    read one element at a time -- starts on a multiple of 16 bytes, and so does every
    stride (in bytes) of every dimension except the innermost, among dimensions of
    size > 1."""
    for (name, kind, _), t in zip(SLOTS[args["op"]], args["tensors"]):
        if kind == "pos":
            continue
        es = ELEM_SIZE[t["dtype"]]
        if t["addr"] % 16 != 0:
            return False
        for d in range(len(t["shape"]) - 1):
            if t["shape"][d] > 1 and (t["stride"][d] * es) % 16 != 0:
                return False
    return True


def guard(spec, args):
    """G_i(args): the short-circuit conjunction, cheapest and most basic checks first
    (a check that reads shape[k] only runs after the rank check that makes it exist)."""
    op = args["op"]
    ts = args["tensors"]
    if spec["op"] != op:
        return False
    if any(t["device"] != spec["device"] for t in ts):
        return False
    for (name, kind, _), t in zip(SLOTS[op], ts):
        if t["dtype"] != expected_dtype(kind, spec["dtype"]):
            return False
    for (name, kind, _), t in zip(SLOTS[op], ts):
        if len(t["shape"]) != expected_rank(op, kind, spec["rank"]):
            return False
    fx = dict(zip(FIXED_NAMES[op], spec["fixed"]))
    slot0 = ts[0]
    lead = list(slot0["shape"][:-1]) if op in FLATTENING_OPS else [slot0["shape"][0]]
    for (name, kind, _), t in zip(SLOTS[op], ts):
        if not shape_ok(kind, t["shape"], lead, fx):
            return False
    if op in ROPE_OPS and args["theta"] != spec["theta"]:
        return False
    T = token_count(op, slot0)
    if not (spec["tok_lo"] <= T <= spec["tok_hi"]):
        return False
    lc = layout_class(args)
    if lc == LAYOUT_NONE:
        return False
    if spec["layout"] == ANY:
        pass
    elif spec["layout"] != lc:
        return False
    if not aux_layout_ok(args, fx):
        return False
    if spec["align"] == 16 and not aligned16(args):
        return False
    return True


# ----------------------------------------------------------------------------- overlap
def byte_set(t):
    """Every byte address the tensor's elements occupy (brute force)."""
    es = ELEM_SIZE[t["dtype"]]
    out = set()
    shape, stride = t["shape"], t["stride"]
    if numel(t) == 0:
        return out

    def rec(dim, off):
        if dim == len(shape):
            base = t["addr"] + off * es
            out.update(range(base, base + es))
            return
        for i in range(shape[dim]):
            rec(dim + 1, off + i * stride[dim])

    rec(0, 0)
    return out


def same_tensor(a, b):
    return (a["addr"] == b["addr"] and a["dtype"] == b["dtype"]
            and tuple(a["shape"]) == tuple(b["shape"]) and tuple(a["stride"]) == tuple(b["stride"]))


def launch_precondition(args):
    """No output may share a byte with another slot, unless both slots are the same
    tensor and belong to one of the op's in-place groups."""
    op = args["op"]
    slots = SLOTS[op]
    ts = args["tensors"]
    sets = [byte_set(t) for t in ts]
    for i, (ni, _, out_i) in enumerate(slots):
        if not out_i:
            continue
        for j, (nj, _, _) in enumerate(slots):
            if j == i:
                continue
            if not (sets[i] & sets[j]):
                continue
            grouped = any(ni in g and nj in g for g in INPLACE_GROUPS[op])
            if grouped and same_tensor(ts[i], ts[j]):
                continue
            return False
    return True


def calls_independent(calls):
    """Several argument tuples may run in any order -- and so in one launch -- iff no
    output byte of one call is a byte of any tensor of another call (brute force over
    byte sets, as launch_precondition does within one call)."""
    sets = [[byte_set(t) for t in c["tensors"]] for c in calls]
    for i, ci in enumerate(calls):
        for j in range(len(calls)):
            if j == i:
                continue
            for si, (_, _, out_i) in enumerate(SLOTS[ci["op"]]):
                if out_i and any(sets[i][si] & other for other in sets[j]):
                    return False
    return True


# ----------------------------------------------------------------------------- Algorithm 1
def select(table, args, check_overlap=True):
    """Algorithm 1 over `table` (list of specs in creation order).
    Returns (OK, i), (MISS, -1) or (INVALID, -1)."""
    if not validate(args):
        return INVALID, -1
    for i, spec in enumerate(table):
        if not guard(spec, args):
            continue
        if check_overlap and not launch_precondition(args):
            return INVALID, -1
        return OK, i
    return MISS, -1


# ----------------------------------------------------------------------------- structured arguments
def bind_tree(recipe, args_tree):
    """§3.3: bind a call's structured arguments to a version's recipe, or None.

    args_tree: the top-level parameters, each a tensor dict, None, an int, a float, or a
    tuple/list of such values. recipe: dict(op, params, eps, theta, scalar) where params
    holds one pattern per top-level parameter, a pattern being
      ("tensor", k)          a tensor, filling op slot k (k = -1: not consumed)
      ("none",)              None
      ("tuple", [patterns])  a tuple of exactly that many elements
      ("int" | "float", bind, value)   bind: "const" (must equal value), "eps", "theta",
                             "scalar" (the value becomes that argument), "unused".
    A mismatch of structure, kind or guarded constant is this version's miss (None). The
    consumed tensors fill the op's slots; scalars not bound keep the recipe's values."""
    params = recipe["params"]
    if len(args_tree) != len(params):
        return None
    slots = [None] * len(SLOTS[recipe["op"]])
    scal = dict(eps=recipe["eps"], theta=recipe["theta"], scalar=recipe["scalar"])

    def match(p, v):
        kind = p[0]
        if kind == "none":
            return v is None
        if kind == "tensor":
            if not isinstance(v, dict):
                return False
            if p[1] >= 0:
                slots[p[1]] = v
            return True
        if kind == "tuple":
            if not isinstance(v, (tuple, list)) or len(v) != len(p[1]):
                return False
            for pc, vc in zip(p[1], v):
                if not match(pc, vc):
                    return False
            return True
        is_int = isinstance(v, int)  # bool counts as int, as in Python
        if kind == "int" and not is_int:
            return False
        if kind == "float" and not isinstance(v, float):
            return False
        bind = p[1]
        if bind == "const":
            return v == p[2]
        if bind in scal:
            scal[bind] = float(v)
        return True

    for p, v in zip(params, args_tree):
        if not match(p, v):
            return None
    return dict(op=recipe["op"], tensors=slots, eps=scal["eps"], theta=scal["theta"],
                scalar=scal["scalar"], flags=0)


def select_tree(table, args_tree, check_overlap=True):
    """Algorithm 1 over versions with recipes: table = [(spec, recipe)] in creation order.
    The first version whose recipe binds and whose guard holds is selected; bound
    arguments that are malformed are an error, not a miss."""
    for i, (spec, recipe) in enumerate(table):
        args = bind_tree(recipe, args_tree)
        if args is None:
            continue
        if not validate(args):
            return INVALID, -1
        if not guard(spec, args):
            continue
        if check_overlap and not launch_precondition(args):
            return INVALID, -1
        return OK, i
    return MISS, -1


def bucket_of(T):
    """Token-count bucket b: b = 0 holds T = 1; b >= 1 holds 2^(b-1) < T <= 2^b."""
    b = 0
    while (1 << b) < T:
        b += 1
    return b


def bucket_range(b):
    return (1, 1) if b == 0 else ((1 << (b - 1)) + 1, 1 << b)
