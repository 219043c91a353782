"""Test helpers: expand compact case descriptions into argument tuples and versions.

Tensors here are descriptors only (fake addresses), for host-side selection tests.
The same dicts are handed to the oracle (`oracle.guards`) and, converted field by
field, to the library (`paper_2609_37241_gb300.scm`).
"""
DT = {"bf16": 1, "fp16": 2, "fp32": 3, "i32": 4, "i64": 5}
ES = {1: 2, 2: 2, 3: 4, 4: 4, 5: 8}
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
    if op in (1, 4):
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
                theta=float(d.get("theta", 0.0)), flags=0)
