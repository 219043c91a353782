/* fastcall.c -- CPython entry points for the per-call hot path of the Python binding.
 *
 * Argument marshalling only: each function converts Python ints (the SCM handle, the
 * address of a trident_args array built once with ctypes, a cudaStream_t) and calls the
 * C ABI. It exists because a ctypes foreign call costs about a microsecond, comparable to
 * the whole dispatch it wraps; a METH_FASTCALL call costs a few tens of nanoseconds. */
#define PY_SSIZE_T_CLEAN
#include <Python.h>
#include <stdint.h>
#include <string.h>

#include "trident_scm.h"

/* invoke(scm, args_address, stream) -> status */
static PyObject* fc_invoke(PyObject* self, PyObject* const* args, Py_ssize_t nargs) {
  (void)self;
  if (nargs != 3) {
    PyErr_SetString(PyExc_TypeError, "invoke(scm, args_address, stream)");
    return NULL;
  }
  void* scm = PyLong_AsVoidPtr(args[0]);
  void* a = PyLong_AsVoidPtr(args[1]);
  void* stream = PyLong_AsVoidPtr(args[2]);
  if (PyErr_Occurred()) return NULL;
  return PyLong_FromLong(trident_scm_invoke((trident_scm_t*)scm, (const trident_args*)a, stream, NULL));
}

typedef int32_t (*seq_fn)(trident_scm_t*, const trident_args*, int32_t, void*, int32_t*);

/* (scm, args_address, n, stream) -> status of fn */
static PyObject* call_seq(seq_fn fn, const char* usage, PyObject* const* args, Py_ssize_t nargs) {
  if (nargs != 4) {
    PyErr_SetString(PyExc_TypeError, usage);
    return NULL;
  }
  void* scm = PyLong_AsVoidPtr(args[0]);
  void* a = PyLong_AsVoidPtr(args[1]);
  long n = PyLong_AsLong(args[2]);
  void* stream = PyLong_AsVoidPtr(args[3]);
  if (PyErr_Occurred()) return NULL;
  if (n < 0 || n > INT32_MAX) {
    PyErr_SetString(PyExc_ValueError, "n out of range");
    return NULL;
  }
  return PyLong_FromLong(fn((trident_scm_t*)scm, (const trident_args*)a, (int32_t)n, stream, NULL));
}

/* invoke_seq(scm, args_address, n, stream) -> status */
static PyObject* fc_invoke_seq(PyObject* self, PyObject* const* args, Py_ssize_t nargs) {
  (void)self;
  return call_seq(trident_scm_invoke_seq, "invoke_seq(scm, args_address, n, stream)", args, nargs);
}

/* invoke_step(scm, args_address, n, stream) -> status */
static PyObject* fc_invoke_step(PyObject* self, PyObject* const* args, Py_ssize_t nargs) {
  (void)self;
  return call_seq(trident_scm_invoke_step, "invoke_step(scm, args_address, n, stream)", args, nargs);
}

/* invoke_tree(scm, nodes_address, nargs, nnodes, stream) -> status */
static PyObject* fc_invoke_tree(PyObject* self, PyObject* const* args, Py_ssize_t nargs) {
  (void)self;
  if (nargs != 5) {
    PyErr_SetString(PyExc_TypeError, "invoke_tree(scm, nodes_address, nargs, nnodes, stream)");
    return NULL;
  }
  void* scm = PyLong_AsVoidPtr(args[0]);
  void* nodes = PyLong_AsVoidPtr(args[1]);
  long na = PyLong_AsLong(args[2]);
  long nn = PyLong_AsLong(args[3]);
  void* stream = PyLong_AsVoidPtr(args[4]);
  if (PyErr_Occurred()) return NULL;
  if (na < 0 || na > INT32_MAX || nn < 0 || nn > INT32_MAX) {
    PyErr_SetString(PyExc_ValueError, "nargs or nnodes out of range");
    return NULL;
  }
  return PyLong_FromLong(trident_scm_invoke_tree((trident_scm_t*)scm, (const trident_node*)nodes,
                                                 (int32_t)na, (int32_t)nn, stream, NULL));
}

/* ---------------------------------------------------------------- structured arguments
 * invoke_py(scm, stream, *args): packs the Python arguments -- torch tensors, tuples and
 * lists, ints (bool included), floats, None -- into a trident_node array (top-level
 * arguments first, each tuple's children contiguous after it) and calls
 * trident_scm_invoke_tree. Tensor metadata is read through the tensor's Python attributes
 * (data_ptr, shape, stride, dtype, get_device); nothing is copied. */
typedef struct {
  PyObject* tensor_type;
  PyObject* dtypes[7]; /* bfloat16, float16, float32, int32, int64, uint8, bool */
  int32_t codes[7];
  PyObject *s_data_ptr, *s_shape, *s_stride, *s_dtype, *s_get_device;
} TorchNames;
static TorchNames tn;

static int torch_names(void) {
  if (tn.tensor_type) return 0;
  PyObject* torch = PyImport_ImportModule("torch");
  if (!torch) return -1;
  static const char* names[7] = {"bfloat16", "float16", "float32", "int32", "int64", "uint8", "bool"};
  static const int32_t codes[7] = {TRIDENT_BF16, TRIDENT_FP16, TRIDENT_FP32, TRIDENT_I32, TRIDENT_I64,
                                   TRIDENT_U8, TRIDENT_U8};
  PyObject* tt = PyObject_GetAttrString(torch, "Tensor");
  int ok = tt != NULL;
  for (int k = 0; ok && k < 7; ++k) {
    tn.dtypes[k] = PyObject_GetAttrString(torch, names[k]);
    tn.codes[k] = codes[k];
    ok = tn.dtypes[k] != NULL;
  }
  Py_DECREF(torch);
  if (!ok) return -1;
  tn.s_data_ptr = PyUnicode_InternFromString("data_ptr");
  tn.s_shape = PyUnicode_InternFromString("shape");
  tn.s_stride = PyUnicode_InternFromString("stride");
  tn.s_dtype = PyUnicode_InternFromString("dtype");
  tn.s_get_device = PyUnicode_InternFromString("get_device");
  if (!tn.s_data_ptr || !tn.s_shape || !tn.s_stride || !tn.s_dtype || !tn.s_get_device) return -1;
  tn.tensor_type = tt;
  return 0;
}

/* Fills a TENSOR node from a torch.Tensor. 0 on success, -1 with a Python error. */
static int fill_from_torch(PyObject* t, trident_node* nd) {
  memset(&nd->t, 0, sizeof(nd->t));
  nd->kind = TRIDENT_NODE_TENSOR;
  PyObject* dp = PyObject_CallMethodNoArgs(t, tn.s_data_ptr);
  PyObject* shape = dp ? PyObject_GetAttr(t, tn.s_shape) : NULL;
  PyObject* stride = shape ? PyObject_CallMethodNoArgs(t, tn.s_stride) : NULL;
  PyObject* dt = stride ? PyObject_GetAttr(t, tn.s_dtype) : NULL;
  PyObject* dev = dt ? PyObject_CallMethodNoArgs(t, tn.s_get_device) : NULL;
  int rc = -1;
  if (dev) {
    const Py_ssize_t nd_ = PyTuple_Check(shape) ? PyTuple_GET_SIZE(shape) : -1;
    if (nd_ < 1 || nd_ > 4 || !PyTuple_Check(stride) || PyTuple_GET_SIZE(stride) != nd_) {
      PyErr_SetString(PyExc_ValueError, "tensors must have 1 to 4 dimensions");
    } else {
      nd->t.data = PyLong_AsVoidPtr(dp);
      nd->t.ndim = (int32_t)nd_;
      for (Py_ssize_t k = 0; k < nd_; ++k) {
        nd->t.shape[k] = PyLong_AsLongLong(PyTuple_GET_ITEM(shape, k));
        nd->t.stride[k] = PyLong_AsLongLong(PyTuple_GET_ITEM(stride, k));
      }
      nd->t.dtype = 0;
      for (int k = 0; k < 7; ++k)
        if (dt == tn.dtypes[k]) nd->t.dtype = tn.codes[k];
      const long d = PyLong_AsLong(dev);
      nd->t.device = d >= 0 ? (int32_t)d : -1;
      if (!PyErr_Occurred()) {
        if (nd->t.dtype == 0) PyErr_SetString(PyExc_TypeError, "unsupported tensor dtype");
        else rc = 0;
      }
    }
  }
  Py_XDECREF(dp);
  Py_XDECREF(shape);
  Py_XDECREF(stride);
  Py_XDECREF(dt);
  Py_XDECREF(dev);
  return rc;
}

#define FC_STACK_NODES 64

static PyObject* fc_invoke_py(PyObject* self, PyObject* const* args, Py_ssize_t nargs) {
  (void)self;
  if (nargs < 2) {
    PyErr_SetString(PyExc_TypeError, "invoke_py(scm, stream, *args)");
    return NULL;
  }
  void* scm = PyLong_AsVoidPtr(args[0]);
  void* stream = PyLong_AsVoidPtr(args[1]);
  if (PyErr_Occurred() || torch_names() != 0) return NULL;
  trident_node stack_nodes[FC_STACK_NODES];
  PyObject* stack_vals[FC_STACK_NODES];
  trident_node* nodes = stack_nodes;
  PyObject** vals = stack_vals;
  Py_ssize_t cap = FC_STACK_NODES, n = nargs - 2;
  PyObject* result = NULL;
  if (n > TRIDENT_TREE_MAX_NODES) {
    PyErr_SetString(PyExc_ValueError, "too many arguments");
    return NULL;
  }
  if (n > cap) {
    cap = n;
    nodes = (trident_node*)PyMem_Malloc(sizeof(trident_node) * (size_t)cap);
    vals = (PyObject**)PyMem_Malloc(sizeof(PyObject*) * (size_t)cap);
    if (!nodes || !vals) {
      PyErr_NoMemory();
      goto done;
    }
  }
  for (Py_ssize_t i = 0; i < n; ++i) vals[i] = args[i + 2];
  for (Py_ssize_t q = 0; q < n; ++q) { /* breadth first: children appended after their tuple */
    PyObject* v = vals[q];
    trident_node* nd = &nodes[q];
    nd->kind = TRIDENT_NODE_NONE;
    nd->n = nd->first = nd->reserved = 0;
    nd->i = 0;
    nd->f = 0.0;
    nd->dl = NULL;
    if (v == Py_None) continue;
    if (PyTuple_Check(v) || PyList_Check(v)) {
      const Py_ssize_t k = PySequence_Fast_GET_SIZE(v);
      if (n + k > TRIDENT_TREE_MAX_NODES) {
        PyErr_SetString(PyExc_ValueError, "argument tree too large");
        goto done;
      }
      if (n + k > cap) {
        Py_ssize_t ncap = cap * 2 > n + k ? cap * 2 : n + k;
        trident_node* nn = (trident_node*)PyMem_Malloc(sizeof(trident_node) * (size_t)ncap);
        PyObject** nv = (PyObject**)PyMem_Malloc(sizeof(PyObject*) * (size_t)ncap);
        if (!nn || !nv) {
          PyMem_Free(nn);
          PyMem_Free(nv);
          PyErr_NoMemory();
          goto done;
        }
        memcpy(nn, nodes, sizeof(trident_node) * (size_t)n);
        memcpy(nv, vals, sizeof(PyObject*) * (size_t)n);
        if (nodes != stack_nodes) {
          PyMem_Free(nodes);
          PyMem_Free(vals);
        }
        nodes = nn;
        vals = nv;
        cap = ncap;
        nd = &nodes[q];
      }
      PyObject** items = PySequence_Fast_ITEMS(v);
      nd->kind = TRIDENT_NODE_TUPLE;
      nd->n = (int32_t)k;
      nd->first = (int32_t)n;
      for (Py_ssize_t c = 0; c < k; ++c) vals[n + c] = items[c];
      n += k;
    } else if (PyLong_Check(v)) {
      nd->kind = TRIDENT_NODE_INT;
      nd->i = PyLong_AsLongLong(v);
      if (PyErr_Occurred()) goto done;
    } else if (PyFloat_Check(v)) {
      nd->kind = TRIDENT_NODE_FLOAT;
      nd->f = PyFloat_AS_DOUBLE(v);
    } else {
      const int is_t = PyObject_IsInstance(v, tn.tensor_type);
      if (is_t < 0) goto done;
      if (!is_t) {
        PyErr_Format(PyExc_TypeError, "unsupported argument type %s", Py_TYPE(v)->tp_name);
        goto done;
      }
      if (fill_from_torch(v, nd) != 0) goto done;
    }
  }
  {
    const int32_t st = trident_scm_invoke_tree((trident_scm_t*)scm, nodes, (int32_t)(nargs - 2), (int32_t)n,
                                               stream, NULL);
    result = PyLong_FromLong(st);
  }
done:
  if (nodes != stack_nodes) {
    PyMem_Free(nodes);
    PyMem_Free(vals);
  }
  return result;
}

static PyMethodDef methods[] = {
    {"invoke", (PyCFunction)(void (*)(void))fc_invoke, METH_FASTCALL, "trident_scm_invoke"},
    {"invoke_seq", (PyCFunction)(void (*)(void))fc_invoke_seq, METH_FASTCALL, "trident_scm_invoke_seq"},
    {"invoke_step", (PyCFunction)(void (*)(void))fc_invoke_step, METH_FASTCALL, "trident_scm_invoke_step"},
    {"invoke_tree", (PyCFunction)(void (*)(void))fc_invoke_tree, METH_FASTCALL, "trident_scm_invoke_tree"},
    {"invoke_py", (PyCFunction)(void (*)(void))fc_invoke_py, METH_FASTCALL,
     "invoke_py(scm, stream, *args): trident_scm_invoke_tree on Python arguments"},
    {NULL, NULL, 0, NULL}};

static struct PyModuleDef module = {PyModuleDef_HEAD_INIT, "_fastcall", NULL, -1, methods,
                                    NULL, NULL, NULL, NULL};

PyMODINIT_FUNC PyInit__fastcall(void) { return PyModule_Create(&module); }
