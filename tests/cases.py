"""Test helpers: expand compact case descriptions into argument tuples and versions.

Tensors here are descriptors only (fake addresses), for host-side selection tests.
The same dicts are handed to the oracle (`oracle.guards`) and, converted field by
field, to the library (`paper_2609_37241_gb300.scm`).
"""
DT = {"bf16": 1, "fp16": 2, "fp32": 3, "i32": 4, "i64": 5, "u8": 6}
ES = {1: 2, 2: 2, 3: 4, 4: 4, 5: 8, 6: 1}
LAYOUT = {"contig": 0, "strided": 1, "any": 2}
BASE = 0x7F0000000000
SPAN = 1 << 32  # address distance between buffers


def tensor(addr, dtype, shape, stride=None, device=0):
    shape = tuple(int(s) for s in shape)
    if stride is None:
        stride, acc = [], 1
        for s in reversed(shape):
            stride.append(acc)
            acc *= max(s, 1)
        stride = tuple(reversed(stride))
    return dict(addr=int(addr), dtype=dtype, shape=shape, stride=tuple(int(s) for s in stride),
                device=device)


def make_spec(d):
    op = d["op"]
    rank = d.get("rank", 3 if op in (2, 3) else 2)
    lo, hi = d.get("tok", [1, 1 << 20])
    return dict(op=op, dtype=DT[d.get("dtype", "bf16")], rank=rank,
                layout=LAYOUT[d.get("layout", "contig")], fixed=tuple(d["fixed"]),
                tok_lo=lo, tok_hi=hi, align=d.get("align", 16), device=d.get("device", 0),
                variant=d.get("variant", 0), theta=float(d.get("theta", 0.0)))


class _Alloc:
    def __init__(self):
        self.n = 0

    def __call__(self):
        self.n += 1
        return BASE + self.n * SPAN


def _rows(alloc, dt, lead, width, layout, device, misalign=False):
    """An activation [*lead, width] in the requested row layout."""
    es = ES[dt]
    if layout == "contig":
        rs = width
    elif layout == "strided":
        rs = width + 64
    elif layout == "badrows":
        rs = max(width // 2, 1)
    else:
        raise ValueError(layout)
    addr = alloc() + (es if misalign else 0)
    if len(lead) == 1:
        return tensor(addr, dt, (lead[0], width), (rs, 1), device)
    b, s = lead
    return tensor(addr, dt, (b, s, width), (s * rs, rs, 1), device)


def make_args(d):
    """Argument tuple for ops 1 (ADD_RMSNORM), 2/3 (ROPE ops) and 4 (SWIGLU)."""
    op = d["op"]
    dt = DT[d.get("dtype", "bf16")]
    dev = d.get("device", 0)
    layout = d.get("layout", "contig")
    mis = d.get("misalign", False)
    alloc = _Alloc()
    T = d["T"]
    if op == 7:
        lead = (T,) if d.get("rank", 2) == 2 else (d["B"], T // d["B"])
        W = d["H"]
        ts = [_rows(alloc, dt, lead, W, layout, dev, mis), tensor(alloc(), 3, (W,), device=dev),
              _rows(alloc, dt, lead, W, layout, dev)]
    elif op in (8, 9, 10, 11):
        lead = (T,) if d.get("rank", 2) == 2 else (d["B"], T // d["B"])
        W = d["H"]
        ts = [_rows(alloc, dt, lead, W, layout, dev, mis)]
        if op == 9:
            ts.append(_rows(alloc, dt, lead, W, layout, dev))
        if op == 11:
            ts.append(_rows(alloc, 6, lead, W, layout, dev))
        ts.append(_rows(alloc, dt, lead, W, layout, dev))
    elif op in (1, 4):
        if d.get("rank", 2) == 3:
            B = d["B"]
            lead = (B, T // B)
        else:
            lead = (T,)
        W = d["H"] if op == 1 else d["I"]
        if op == 1:
            ts = [_rows(alloc, dt, lead, W, layout, dev, mis), _rows(alloc, dt, lead, W, layout, dev),
                  tensor(alloc(), 3, (W,), device=dev),
                  _rows(alloc, dt, lead, W, layout, dev), _rows(alloc, dt, lead, W, layout, dev)]
        else:
            ts = [_rows(alloc, dt, lead, W, layout, dev, mis), _rows(alloc, dt, lead, W, layout, dev),
                  _rows(alloc, dt, lead, W, layout, dev)]
    elif op in (2, 3):
        Hq, Hkv, D, S = d["Hq"], d["Hkv"], d["D"], d["S"]
        es = ES[dt]
        if layout == "contig":
            q = tensor(alloc() + (es if mis else 0), dt, (T, Hq, D), device=dev)
            k = tensor(alloc(), dt, (T, Hkv, D), device=dev)
            v = tensor(alloc(), dt, (T, Hkv, D), device=dev)
        else:  # views into one fused qkv buffer [T, (Hq + 2 Hkv) D]
            W = (Hq + 2 * Hkv) * D
            base = alloc() + (es if mis else 0)
            q = tensor(base, dt, (T, Hq, D), (W, D, 1), dev)
            k = tensor(base + Hq * D * es, dt, (T, Hkv, D), (W, D, 1), dev)
            v = tensor(base + (Hq + Hkv) * D * es, dt, (T, Hkv, D), (W, D, 1), dev)
        ts = [q, k, v, tensor(alloc(), 4, (T,), device=dev),
              tensor(alloc(), dt, (Hkv, S, D), device=dev), tensor(alloc(), dt, (Hkv, S, D), device=dev)]
        if op == 3:
            ts += [tensor(alloc(), 3, (D,), device=dev), tensor(alloc(), 3, (D,), device=dev)]
    else:
        raise ValueError(op)
    delta = d.get("ntensors_delta", 0)
    if delta < 0:
        ts = ts[:delta]
    elif delta > 0:
        ts = ts + [tensor(alloc(), 3, (1,), device=dev)] * delta
    return dict(op=op, tensors=ts, eps=float(d.get("eps", 1e-6)),
                theta=float(d.get("theta", 0.0)), flags=0, scalar=float(d.get("scalar", 0.0)))


def make_chain_args(d):
    """Argument tuple for ops 5/6 (layer chains). layout 'contig': separate dense
    buffers; 'strided': q/k/v views of one qkv buffer and g/u halves of one [T, 2I]."""
    op = d["op"]
    dt = DT[d.get("dtype", "bf16")]
    dev = d.get("device", 0)
    alloc = _Alloc()
    T, H, Hq, Hkv, D, S, I = (d[k] for k in ("T", "H", "Hq", "Hkv", "D", "S", "I"))
    es = ES[dt]
    act = lambda w: tensor(alloc(), dt, (T, w), device=dev)
    ts = [act(H), act(H), tensor(alloc(), 3, (H,), device=dev), act(H), act(H)]
    if d.get("layout", "contig") == "contig":
        q = tensor(alloc(), dt, (T, Hq, D), device=dev)
        k = tensor(alloc(), dt, (T, Hkv, D), device=dev)
        v = tensor(alloc(), dt, (T, Hkv, D), device=dev)
        g, u = act(I), act(I)
    else:
        W = (Hq + 2 * Hkv) * D
        base = alloc()
        q = tensor(base, dt, (T, Hq, D), (W, D, 1), dev)
        k = tensor(base + Hq * D * es, dt, (T, Hkv, D), (W, D, 1), dev)
        v = tensor(base + (Hq + Hkv) * D * es, dt, (T, Hkv, D), (W, D, 1), dev)
        gu = alloc()
        g = tensor(gu, dt, (T, I), (2 * I, 1), dev)
        u = tensor(gu + I * es, dt, (T, I), (2 * I, 1), dev)
    ts += [q, k, v, tensor(alloc(), 4, (T,), device=dev),
           tensor(alloc(), dt, (Hkv, S, D), device=dev), tensor(alloc(), dt, (Hkv, S, D), device=dev),
           act(H), tensor(alloc(), 3, (H,), device=dev), act(H), act(H), g, u, act(I)]
    if op == 6:
        ts += [tensor(alloc(), 3, (D,), device=dev), tensor(alloc(), 3, (D,), device=dev)]
    return dict(op=op, tensors=ts, eps=float(d.get("eps", 1e-6)), theta=float(d.get("theta", 0.0)),
                flags=0)


def lib_spec(spec):
    """Library descriptor (ctypes) from an oracle-style spec dict."""
    from paper_2609_37241_gb300 import scm
    return scm.make_spec(spec["op"], spec["dtype"], spec["fixed"], spec["tok_lo"], spec["tok_hi"],
                         rank=spec["rank"], layout=spec["layout"], align_bytes=spec["align"],
                         device=spec["device"], variant=spec["variant"], rope_theta=spec["theta"])


def lib_args(args):
    """Library argument tuple (ctypes) from an oracle-style args dict."""
    from paper_2609_37241_gb300 import scm
    return scm.make_args(args["op"], args["tensors"], eps=args["eps"], rope_theta=args["theta"],
                         scalar=args.get("scalar", 0.0))


STATUS = {0: "OK", 2: "MISS", -1: "INVALID"}


def lib_recipe(recipe):
    """Library recipe (scm.Recipe) from an oracle-style recipe dict (oracle.guards.bind_tree)."""
    from paper_2609_37241_gb300 import scm
    binds = {"const": scm.BIND_CONST, "eps": scm.BIND_EPS, "theta": scm.BIND_THETA,
             "scalar": scm.BIND_SCALAR, "unused": scm.BIND_UNUSED}

    def conv(p):
        if p[0] == "none":
            return None
        if p[0] == "tensor":
            return scm.Slot(p[1])
        if p[0] == "tuple":
            return tuple(conv(c) for c in p[1])
        return scm.Num(p[0], binds[p[1]], p[2] if len(p) > 2 else 0)

    return scm.Recipe(*[conv(p) for p in recipe["params"]], eps=recipe["eps"],
                      rope_theta=recipe["theta"], scalar=recipe["scalar"])


def recipe(op, *params, eps=0.0, theta=0.0, scalar=0.0):
    return dict(op=op, params=list(params), eps=eps, theta=theta, scalar=scalar)
