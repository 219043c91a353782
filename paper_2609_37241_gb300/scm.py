"""Thin Python binding of the SCM C ABI (include/trident_scm.h).

Argument marshalling only: every step of a call -- validation, guard evaluation,
parameter packing and the launch -- runs in libtrident_scm.so. The functions keep the C
names; `Scm` is a small convenience wrapper. There is no fallback: if the library is
missing, importing it raises.
"""
import ctypes
import os

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "_lib", "libtrident_scm.so")

# ---------------------------------------------------------------- constants (trident_scm.h)
OK, MISS_HANDLED, MISS = 0, 1, 2
ERR_INVALID, ERR_CUDA, ERR_HOOK, ERR_CAPACITY, ERR_STATE = -1, -2, -3, -4, -5
NOT_RUN = -2
BF16, FP16, FP32, I32, I64, U8 = 1, 2, 3, 4, 5, 6
OP_ADD_RMSNORM, OP_ROPE_KV, OP_QKNORM_ROPE_KV, OP_SWIGLU, OP_LAYER_CHAIN, OP_LAYER_CHAIN_QKNORM = 1, 2, 3, 4, 5, 6
OP_RMSNORM = 7
OP_SILU, OP_ADD, OP_NEG, OP_MASKED_FILL = 8, 9, 10, 11
LAYOUT_CONTIG, LAYOUT_ROWSTRIDED, LAYOUT_ANY = 0, 1, 2
VARIANT_AUTO, VARIANT_GENERIC, VARIANT_VECTOR = 0, 1, 2
OPT_DRY_RUN, OPT_NO_ALIAS_CHECK, OPT_PDL, OPT_TIMING, OPT_FAIL_LAUNCHES = 0x1, 0x2, 0x4, 0x8, 0x10
OPT_NO_STEP_REPLAY = 0x20
OPT_TEST_WAIT_TIMEOUT = 0x40
DEVERR_POS, DEVERR_TIMEOUT = 0x1, 0x2
MAX_TENSORS, MAX_FIXED = 20, 8
STEP_MAX = 48  # calls per launch of trident_scm_invoke_step
TREE_MAX_NODES, TREE_MAX_DEPTH = 4096, 16
NODE_NONE, NODE_TENSOR, NODE_DLTENSOR, NODE_TUPLE, NODE_INT, NODE_FLOAT = 0, 1, 2, 3, 4, 5
BIND_UNUSED, BIND_CONST, BIND_EPS, BIND_THETA, BIND_SCALAR = -1, -2, -3, -4, -5
OP_NTENSORS = {1: 5, 2: 6, 3: 8, 4: 3, 5: 18, 6: 20, 7: 3, 8: 2, 9: 3, 10: 2, 11: 3}

c_i32, c_i64, c_u32, c_u64, c_dbl, c_vp = (ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32,
                                           ctypes.c_uint64, ctypes.c_double, ctypes.c_void_p)


class trident_tensor(ctypes.Structure):
    _fields_ = [("data", c_vp), ("shape", c_i64 * 4), ("stride", c_i64 * 4), ("dtype", c_i32),
                ("ndim", c_i32), ("device", c_i32), ("reserved", c_i32)]


class trident_args(ctypes.Structure):
    _fields_ = [("op", c_i32), ("ntensors", c_i32), ("eps", c_dbl), ("rope_theta", c_dbl),
                ("scalar", c_dbl), ("flags", c_i32), ("reserved", c_i32),
                ("t", trident_tensor * MAX_TENSORS)]


class trident_spec_desc(ctypes.Structure):
    _fields_ = [("op", c_i32), ("dtype", c_i32), ("rank", c_i32), ("layout", c_i32),
                ("fixed", c_i64 * MAX_FIXED), ("tok_lo", c_i64), ("tok_hi", c_i64),
                ("align_bytes", c_i32), ("device", c_i32), ("variant", c_i32),
                ("reserved", c_i32), ("rope_theta", c_dbl)]


class trident_scm_options(ctypes.Structure):
    _fields_ = [("device", c_i32), ("max_specs", c_i32), ("flags", c_i32), ("timing_ring", c_i32)]


class trident_scm_stats_t(ctypes.Structure):
    _fields_ = [("invokes", c_u64), ("hits", c_u64), ("misses", c_u64), ("hook_calls", c_u64),
                ("hook_failures", c_u64), ("hook_registered", c_u64), ("err_invalid", c_u64),
                ("err_cuda", c_u64), ("guard_evals", c_u64), ("num_specs", c_i32),
                ("reserved", c_i32), ("fused_launches", c_u64), ("fused_calls", c_u64),
                ("step_replays", c_u64)]


class trident_node(ctypes.Structure):
    _fields_ = [("kind", c_i32), ("n", c_i32), ("first", c_i32), ("reserved", c_i32),
                ("i", c_i64), ("f", c_dbl), ("dl", c_vp), ("t", trident_tensor)]


class trident_recipe_node(ctypes.Structure):
    _fields_ = [("kind", c_i32), ("n", c_i32), ("first", c_i32), ("bind", c_i32),
                ("i", c_i64), ("f", c_dbl)]


class trident_recipe(ctypes.Structure):
    _fields_ = [("nargs", c_i32), ("nnodes", c_i32), ("nodes", ctypes.POINTER(trident_recipe_node)),
                ("eps", c_dbl), ("rope_theta", c_dbl), ("scalar", c_dbl)]


HOOK = ctypes.CFUNCTYPE(c_i32, c_vp, c_vp, ctypes.POINTER(trident_args), c_vp, ctypes.POINTER(c_i32))
TREE_HOOK = ctypes.CFUNCTYPE(c_i32, c_vp, c_vp, ctypes.POINTER(trident_node), c_i32, c_i32, c_vp,
                             ctypes.POINTER(c_i32))

_lib = None


def lib():
    """The loaded C library. Raises if it has not been built (no fallback path exists)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        P = ctypes.POINTER
        sig = {
            "trident_abi_version": (c_i32, []),
            "trident_scm_create": (c_i32, [P(trident_scm_options), HOOK, c_vp, P(c_vp)]),
            "trident_scm_register_spec": (c_i32, [c_vp, P(trident_spec_desc), P(c_i32)]),
            "trident_scm_invoke": (c_i32, [c_vp, P(trident_args), c_vp, P(c_i32)]),
            "trident_scm_invoke_seq": (c_i32, [c_vp, P(trident_args), c_i32, c_vp, P(c_i32)]),
            "trident_scm_invoke_step": (c_i32, [c_vp, P(trident_args), c_i32, c_vp, P(c_i32)]),
            "trident_scm_select": (c_i32, [c_vp, P(trident_args), P(c_i32)]),
            "trident_scm_register_tree_spec": (c_i32, [c_vp, P(trident_spec_desc), P(trident_recipe),
                                                       P(c_i32)]),
            "trident_scm_invoke_tree": (c_i32, [c_vp, P(trident_node), c_i32, c_i32, c_vp, P(c_i32)]),
            "trident_scm_set_tree_hook": (c_i32, [c_vp, TREE_HOOK, c_vp]),
            "trident_scm_stats": (c_i32, [c_vp, P(trident_scm_stats_t)]),
            "trident_scm_spec_hits": (c_i32, [c_vp, P(c_u64), c_i32, P(c_i32)]),
            "trident_scm_host_times": (c_i32, [c_vp, P(c_u32), c_i32, P(c_i32)]),
            "trident_scm_device_status": (c_i32, [c_vp, c_vp, P(c_u32), c_i32]),
            "trident_launch_floor": (c_i32, [c_vp, c_vp, c_i32]),
            "trident_copy_floor": (c_i32, [c_vp, c_vp, c_vp, c_vp, c_i64, c_i64, c_i32, c_i32, c_i32]),
            "trident_scm_destroy": (None, [c_vp]),
            "trident_rope_kv_noalloc": (c_i32, [P(trident_args), c_vp, P(c_u32)]),
            "trident_scm_last_error": (ctypes.c_char_p, []),
            "trident_status_name": (ctypes.c_char_p, [c_i32]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def fastcall():
    """The CPython fast-call shim (`invoke(scm, args_address, stream)`,
    `invoke_seq(scm, args_address, n, stream)` and `invoke_step(...)`, same arguments, on raw
    integer addresses; the default stream is 0), or None if it was not built. Same C calls
    as trident_scm_invoke / _seq / _step, without ctypes' per-call cost."""
    try:
        lib()
        from . import _fastcall
        return _fastcall
    except ImportError:
        return None


class ScmError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        L = lib()
        msg = L.trident_scm_last_error().decode()
        super().__init__(f"{where}: {L.trident_status_name(status).decode()} ({status}): {msg}")


# ---------------------------------------------------------------- C names
def trident_abi_version():
    return lib().trident_abi_version()


def trident_scm_create(options=None, hook=None, user=None):
    """Returns (status, handle)."""
    h = c_vp()
    st = lib().trident_scm_create(ctypes.byref(options) if options is not None else None,
                                  hook if hook is not None else HOOK(), user, ctypes.byref(h))
    return st, h


def trident_scm_register_spec(scm, desc):
    idx = c_i32(-1)
    st = lib().trident_scm_register_spec(scm, ctypes.byref(desc), ctypes.byref(idx))
    return st, idx.value


def trident_scm_invoke(scm, args, stream=None):
    sel = c_i32(-1)
    st = lib().trident_scm_invoke(scm, ctypes.byref(args), stream, ctypes.byref(sel))
    return st, sel.value


def trident_scm_invoke_seq(scm, args_array, stream=None):
    n = len(args_array)
    sel = (c_i32 * max(n, 1))()
    st = lib().trident_scm_invoke_seq(scm, args_array, n, stream, sel)
    return st, list(sel)[:n]


def trident_scm_invoke_step(scm, args_array, stream=None):
    """Like trident_scm_invoke_seq; independent layer-chain calls share one launch."""
    n = len(args_array)
    sel = (c_i32 * max(n, 1))()
    st = lib().trident_scm_invoke_step(scm, args_array, n, stream, sel)
    return st, list(sel)[:n]


def trident_scm_register_tree_spec(scm, desc, recipe):
    idx = c_i32(-1)
    st = lib().trident_scm_register_tree_spec(scm, ctypes.byref(desc), ctypes.byref(recipe.c),
                                              ctypes.byref(idx))
    return st, idx.value


def trident_scm_invoke_tree(scm, tree, stream=None):
    sel = c_i32(-1)
    st = lib().trident_scm_invoke_tree(scm, tree.nodes, tree.nargs, tree.nnodes, stream,
                                       ctypes.byref(sel))
    return st, sel.value


def trident_scm_select(scm, args):
    sel = c_i32(-1)
    st = lib().trident_scm_select(scm, ctypes.byref(args), ctypes.byref(sel))
    return st, sel.value


def trident_scm_stats(scm):
    s = trident_scm_stats_t()
    st = lib().trident_scm_stats(scm, ctypes.byref(s))
    return st, s


def trident_scm_spec_hits(scm, cap=4096):
    buf = (c_u64 * cap)()
    n = c_i32(0)
    st = lib().trident_scm_spec_hits(scm, buf, cap, ctypes.byref(n))
    return st, list(buf)[:min(n.value, cap)]


def trident_scm_host_times(scm, cap=1 << 16):
    buf = (c_u32 * cap)()
    n = c_i32(0)
    st = lib().trident_scm_host_times(scm, buf, cap, ctypes.byref(n))
    return st, list(buf)[:n.value]


def trident_scm_device_status(scm, stream=None, clear=True):
    bits = c_u32(0)
    st = lib().trident_scm_device_status(scm, stream, ctypes.byref(bits), 1 if clear else 0)
    return st, bits.value


def trident_launch_floor(scm, stream=None, n=1):
    """Latency-floor probe: n empty kernels launched back to back as a hit launches."""
    return lib().trident_launch_floor(scm, stream, n)


def trident_copy_floor(scm, stream, src, dst, read_bytes, write_bytes, blocks, sets, n):
    """Copy-floor probe: n launches of a chain-shaped copy (src/dst: device addresses)."""
    return lib().trident_copy_floor(scm, stream, src, dst, read_bytes, write_bytes, blocks, sets, n)


def trident_rope_kv_noalloc(args, stream=None, status_word=None):
    """RoPE + KV append with no allocation (static scratch). Returns the status code.
    status_word: None (the device status word is not copied out), or the address of a
    4-byte host word -- page-locked for the copy to stay asynchronous -- that receives the
    TRIDENT_DEVERR_* bits once the stream has been synchronised."""
    out = None if status_word is None else ctypes.cast(ctypes.c_void_p(status_word), ctypes.POINTER(c_u32))
    return lib().trident_rope_kv_noalloc(ctypes.byref(args), stream, out)


def trident_scm_destroy(scm):
    lib().trident_scm_destroy(scm)


def trident_scm_last_error():
    return lib().trident_scm_last_error().decode()


def trident_status_name(status):
    return lib().trident_status_name(status).decode()


# ---------------------------------------------------------------- marshalling helpers
_TORCH_DT = None


def _torch_dtypes():
    global _TORCH_DT
    if _TORCH_DT is None:
        import torch
        _TORCH_DT = {torch.bfloat16: BF16, torch.float16: FP16, torch.float32: FP32,
                     torch.int32: I32, torch.int64: I64, torch.uint8: U8, torch.bool: U8}
    return _TORCH_DT


def fill_tensor(dst, t):
    """Fills a trident_tensor from a torch.Tensor (no copy of data)."""
    dst.data = t.data_ptr()
    nd = t.dim()
    dst.ndim = nd
    sh, st = t.shape, t.stride()
    for i in range(nd):
        dst.shape[i] = sh[i]
        dst.stride[i] = st[i]
    dst.dtype = _torch_dtypes()[t.dtype]
    dst.device = t.device.index if t.is_cuda else -1
    return dst


def fill_tensor_dict(dst, d):
    """Fills a trident_tensor from a plain dict(addr, dtype, shape, stride, device)."""
    dst.data = d["addr"] or None
    dst.ndim = len(d["shape"])
    for i, (s, r) in enumerate(zip(d["shape"], d["stride"])):
        dst.shape[i] = s
        dst.stride[i] = r
    dst.dtype = d["dtype"]
    dst.device = d["device"]
    return dst


def make_args(op, tensors, eps=1e-6, rope_theta=0.0, scalar=0.0):
    """trident_args from torch tensors (or plain dicts) in the op's slot order."""
    a = trident_args()
    a.op = op
    a.ntensors = len(tensors)
    a.eps = eps
    a.rope_theta = rope_theta
    a.scalar = scalar
    for i, t in enumerate(tensors):
        if isinstance(t, dict):
            fill_tensor_dict(a.t[i], t)
        else:
            fill_tensor(a.t[i], t)
    return a


def make_spec(op, dtype, fixed, tok_lo, tok_hi, rank=None, layout=LAYOUT_CONTIG, align_bytes=16,
              device=0, variant=VARIANT_AUTO, rope_theta=0.0):
    d = trident_spec_desc()
    d.op, d.dtype = op, dtype
    d.rank = rank if rank is not None else (3 if op in (OP_ROPE_KV, OP_QKNORM_ROPE_KV) else 2)
    d.layout = layout
    for i, f in enumerate(fixed):
        d.fixed[i] = f
    d.tok_lo, d.tok_hi = tok_lo, tok_hi
    d.align_bytes, d.device, d.variant = align_bytes, device, variant
    d.rope_theta = rope_theta
    return d


# ---------------------------------------------------------------- structured arguments
class DL:
    """Marks a tensor to be passed through DLPack (a DLTENSOR node) instead of as a
    descriptor; the capsule is kept alive by the tree."""

    def __init__(self, tensor):
        self.tensor = tensor


_capsule_ptr = None


def _dltensor_address(capsule):
    global _capsule_ptr
    if _capsule_ptr is None:
        f = ctypes.pythonapi.PyCapsule_GetPointer
        f.restype = c_vp
        f.argtypes = [ctypes.py_object, ctypes.c_char_p]
        _capsule_ptr = f
    return _capsule_ptr(capsule, b"dltensor")  # DLManagedTensor: its DLTensor comes first


class Tree:
    """A call's structured arguments as a trident_node array: the top-level parameters
    first, each tuple's children contiguous after it (breadth-first)."""

    def __init__(self, *args):
        import torch
        values = list(args)
        self._keep = []
        queue = list(range(len(values)))
        nodes = [None] * len(values)
        q = 0
        while q < len(queue):
            i = queue[q]
            q += 1
            v = values[i]
            if isinstance(v, (tuple, list)):
                first = len(values)
                values.extend(v)
                nodes.extend([None] * len(v))
                queue.extend(range(first, first + len(v)))
                nodes[i] = ("tuple", len(v), first)
            else:
                nodes[i] = ("leaf",)
        arr = (trident_node * max(len(values), 1))()
        for i, v in enumerate(values):
            nd = arr[i]
            if nodes[i][0] == "tuple":
                nd.kind, nd.n, nd.first = NODE_TUPLE, nodes[i][1], nodes[i][2]
            elif v is None:
                nd.kind = NODE_NONE
            elif isinstance(v, DL):
                cap = torch.utils.dlpack.to_dlpack(v.tensor)
                self._keep.append(cap)
                nd.kind, nd.dl = NODE_DLTENSOR, _dltensor_address(cap)
            elif isinstance(v, torch.Tensor) or isinstance(v, dict):
                nd.kind = NODE_TENSOR
                (fill_tensor_dict if isinstance(v, dict) else fill_tensor)(nd.t, v)
            elif isinstance(v, bool) or isinstance(v, int):
                nd.kind, nd.i = NODE_INT, int(v)
            elif isinstance(v, float):
                nd.kind, nd.f = NODE_FLOAT, v
            else:
                raise TypeError(f"unsupported argument type {type(v).__name__}")
        self.nodes, self.nargs, self.nnodes = arr, len(args), len(values)


class Slot:
    """Recipe leaf: a tensor that fills op slot k (k = -1: a tensor the version ignores)."""

    def __init__(self, k):
        self.k = k


class Num:
    """Recipe leaf for an int or float argument: kind 'int' | 'float', bind BIND_*, value
    for BIND_CONST."""

    def __init__(self, kind, bind, value=0):
        self.kind, self.bind, self.value = kind, bind, value


IGNORED = Slot(-1)
EPS = Num("float", BIND_EPS)
THETA = Num("float", BIND_THETA)
SCALAR_ARG = Num("float", BIND_SCALAR)
ANY_INT, ANY_FLOAT = Num("int", BIND_UNUSED), Num("float", BIND_UNUSED)


def const(v):
    """A guarded constant (int or float)."""
    return Num("int" if isinstance(v, int) else "float", BIND_CONST, v)


class Recipe:
    """A version's recipe (trident_recipe) from a pattern over the top-level parameters:
    Slot / IGNORED for tensors, None, tuples, Num (EPS, THETA, SCALAR_ARG, const(v),
    ANY_INT, ANY_FLOAT)."""

    def __init__(self, *pattern, eps=0.0, rope_theta=0.0, scalar=0.0):
        values = list(pattern)
        spans = [None] * len(values)
        q = 0
        while q < len(values):
            v = values[q]
            if isinstance(v, (tuple, list)):
                spans[q] = (len(v), len(values))
                values.extend(v)
                spans.extend([None] * len(v))
            q += 1
        arr = (trident_recipe_node * max(len(values), 1))()
        for i, v in enumerate(values):
            nd = arr[i]
            if spans[i] is not None:
                nd.kind, nd.n, nd.first = NODE_TUPLE, spans[i][0], spans[i][1]
            elif v is None:
                nd.kind = NODE_NONE
            elif isinstance(v, Slot):
                nd.kind, nd.bind = NODE_TENSOR, v.k
            elif isinstance(v, Num):
                nd.kind = NODE_INT if v.kind == "int" else NODE_FLOAT
                nd.bind = v.bind
                if v.kind == "int":
                    nd.i = int(v.value)
                else:
                    nd.f = float(v.value)
            else:
                raise TypeError(f"unsupported recipe element {v!r}")
        self._arr = arr
        self.c = trident_recipe(len(pattern), len(values), ctypes.cast(arr, ctypes.POINTER(trident_recipe_node)),
                                eps, rope_theta, scalar)


class Scm:
    """Owning wrapper: create on construction, destroy on close/GC."""

    def __init__(self, device=0, max_specs=256, flags=0, timing_ring=0, hook=None):
        self._hook_fn = hook
        self._cb = HOOK(self._trampoline) if hook is not None else None
        opt = trident_scm_options(device, max_specs, flags, timing_ring)
        st, h = trident_scm_create(opt, self._cb, None)
        if st != OK:
            raise ScmError(st, "trident_scm_create")
        self.h = h
        self.hook_error = None

    def _trampoline(self, user, scm, args, stream, out_registered):
        try:
            reg = self._hook_fn(self, args.contents, stream)
            out_registered[0] = -1 if reg is None else int(reg)
            return 0
        except Exception as e:  # reported through ERR_HOOK
            self.hook_error = e
            out_registered[0] = -1
            return 1

    def register(self, desc):
        st, idx = trident_scm_register_spec(self.h, desc)
        if st != OK:
            raise ScmError(st, "trident_scm_register_spec")
        return idx

    def invoke(self, args, stream=None):
        return trident_scm_invoke(self.h, args, stream)

    def register_tree(self, desc, recipe):
        st, idx = trident_scm_register_tree_spec(self.h, desc, recipe)
        if st != OK:
            raise ScmError(st, "trident_scm_register_tree_spec")
        return idx

    def invoke_tree(self, tree, stream=None):
        return trident_scm_invoke_tree(self.h, tree, stream)

    def call(self, *args, stream=None):
        """invoke_tree on Python arguments (tensors, tuples, lists, ints, floats, None),
        packed by the CPython shim when it is built, else by Tree. Returns the status."""
        fc = fastcall()
        if fc is not None:
            return fc.invoke_py(self.h.value, stream or 0, *args)
        return trident_scm_invoke_tree(self.h, Tree(*args), stream)[0]

    def set_tree_hook(self, fn):
        """fn(scm, nodes_pointer, nargs, nnodes, stream) -> registered index or None."""
        def tramp(user, scm, nodes, nargs, nnodes, stream, out_registered):
            try:
                reg = fn(self, nodes, nargs, nnodes, stream)
                out_registered[0] = -1 if reg is None else int(reg)
                return 0
            except Exception as e:
                self.hook_error = e
                out_registered[0] = -1
                return 1
        self._tree_cb = TREE_HOOK(tramp) if fn is not None else TREE_HOOK()
        st = lib().trident_scm_set_tree_hook(self.h, self._tree_cb, None)
        if st != OK:
            raise ScmError(st, "trident_scm_set_tree_hook")

    def invoke_seq(self, args_array, stream=None):
        return trident_scm_invoke_seq(self.h, args_array, stream)

    def invoke_step(self, args_array, stream=None):
        return trident_scm_invoke_step(self.h, args_array, stream)

    def select(self, args):
        return trident_scm_select(self.h, args)

    def stats(self):
        return trident_scm_stats(self.h)[1]

    def close(self):
        if getattr(self, "h", None):
            trident_scm_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
