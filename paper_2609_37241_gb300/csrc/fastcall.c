/* fastcall.c -- CPython entry points for the per-call hot path of the Python binding.
 *
 * Argument marshalling only: each function converts Python ints (the SCM handle, the
 * address of a trident_args array built once with ctypes, a cudaStream_t) and calls the
 * C ABI. It exists because a ctypes foreign call costs about a microsecond, comparable to
 * the whole dispatch it wraps; a METH_FASTCALL call costs a few tens of nanoseconds. */
#define PY_SSIZE_T_CLEAN
#include <Python.h>
#include <stdint.h>

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

static PyMethodDef methods[] = {
    {"invoke", (PyCFunction)(void (*)(void))fc_invoke, METH_FASTCALL, "trident_scm_invoke"},
    {"invoke_seq", (PyCFunction)(void (*)(void))fc_invoke_seq, METH_FASTCALL, "trident_scm_invoke_seq"},
    {"invoke_step", (PyCFunction)(void (*)(void))fc_invoke_step, METH_FASTCALL, "trident_scm_invoke_step"},
    {"invoke_tree", (PyCFunction)(void (*)(void))fc_invoke_tree, METH_FASTCALL, "trident_scm_invoke_tree"},
    {NULL, NULL, 0, NULL}};

static struct PyModuleDef module = {PyModuleDef_HEAD_INIT, "_fastcall", NULL, -1, methods,
                                    NULL, NULL, NULL, NULL};

PyMODINIT_FUNC PyInit__fastcall(void) { return PyModule_Create(&module); }
