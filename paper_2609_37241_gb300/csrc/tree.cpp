// tree.cpp -- structured arguments (§3.3): tree validation, recipes, binding.
#include "tree.h"

#include <cuda_runtime.h>

#include <cstring>
#include <new>

#include "internal.h"

namespace trident {
namespace {

// DLPack's DLTensor, restated field for field from the public DLPack specification (the
// layout is the same from DLPack 0.6 to 1.x); only read here.
struct DLDeviceView {
  int32_t device_type;
  int32_t device_id;
};
struct DLDataTypeView {
  uint8_t code;
  uint8_t bits;
  uint16_t lanes;
};
struct DLTensorView {
  void* data;
  DLDeviceView device;
  int32_t ndim;
  DLDataTypeView dtype;
  int64_t* shape;
  int64_t* strides;
  uint64_t byte_offset;
};
enum : int32_t { kDLCPU = 1, kDLCUDA = 2 };
enum : uint8_t { kDLInt = 0, kDLUInt = 1, kDLFloat = 2, kDLBfloat = 4, kDLBool = 6 };

// trident dtype of a DLPack dtype, or 0.
int32_t dl_dtype(const DLDataTypeView& d) {
  if (d.lanes != 1) return 0;
  if (d.code == kDLBfloat && d.bits == 16) return TRIDENT_BF16;
  if (d.code == kDLFloat && d.bits == 16) return TRIDENT_FP16;
  if (d.code == kDLFloat && d.bits == 32) return TRIDENT_FP32;
  if (d.code == kDLInt && d.bits == 32) return TRIDENT_I32;
  if (d.code == kDLInt && d.bits == 64) return TRIDENT_I64;
  if ((d.code == kDLUInt || d.code == kDLBool) && d.bits == 8) return TRIDENT_U8;
  return 0;
}

int32_t check_dl(const void* p, int32_t idx) {
  if (!p) return internal_fail(TRIDENT_ERR_INVALID, "DLTENSOR node without a DLTensor");
  const DLTensorView& d = *static_cast<const DLTensorView*>(p);
  (void)idx;
  if (d.ndim < 1 || d.ndim > 4) return internal_fail(TRIDENT_ERR_INVALID, "DLTensor ndim must be 1..4");
  if (!d.shape) return internal_fail(TRIDENT_ERR_INVALID, "DLTensor without a shape");
  if (!dl_dtype(d.dtype)) return internal_fail(TRIDENT_ERR_INVALID, "DLTensor dtype not supported");
  if (d.device.device_type != kDLCUDA && d.device.device_type != kDLCPU)
    return internal_fail(TRIDENT_ERR_INVALID, "DLTensor device must be CUDA or CPU");
  return TRIDENT_OK;
}

void from_dl(const void* p, trident_tensor* t) {
  const DLTensorView& d = *static_cast<const DLTensorView*>(p);
  std::memset(t, 0, sizeof(*t));
  t->data = d.data ? static_cast<char*>(d.data) + d.byte_offset : nullptr;
  t->ndim = d.ndim;
  t->dtype = dl_dtype(d.dtype);
  t->device = d.device.device_type == kDLCUDA ? d.device.device_id : -1;
  int64_t acc = 1;
  for (int k = d.ndim - 1; k >= 0; --k) {
    t->shape[k] = d.shape[k];
    t->stride[k] = d.strides ? d.strides[k] : acc;  // NULL strides: compact row-major
    acc *= d.shape[k] > 0 ? d.shape[k] : 1;
  }
}

// Shared walk for trees and recipes (both node types have kind, n, first): every node
// reached at most once, children after their parent and inside the array, depth bounded;
// visit(node, index) checks each node.
template <class N, class Visit>
int32_t walk(const N* nodes, int32_t nargs, int32_t nnodes, Visit visit) {
  if (nargs < 0 || nnodes < nargs || nnodes > TRIDENT_TREE_MAX_NODES)
    return internal_fail(TRIDENT_ERR_INVALID, "tree size (nargs <= nnodes <= 4096)");
  if (nnodes > 0 && !nodes) return internal_fail(TRIDENT_ERR_INVALID, "tree nodes are NULL");
  uint8_t seen[TRIDENT_TREE_MAX_NODES];
  std::memset(seen, 0, (size_t)nnodes);
  int32_t stack[TRIDENT_TREE_MAX_NODES], depth[TRIDENT_TREE_MAX_NODES];
  int32_t top = 0;
  for (int32_t i = nargs - 1; i >= 0; --i) {
    stack[top] = i;
    depth[top++] = 1;
  }
  while (top > 0) {
    --top;
    const int32_t i = stack[top], dep = depth[top];
    if (seen[i]) return internal_fail(TRIDENT_ERR_INVALID, "a tree node is reached twice");
    seen[i] = 1;
    if (dep > TRIDENT_TREE_MAX_DEPTH) return internal_fail(TRIDENT_ERR_INVALID, "tree deeper than 16");
    const N& x = nodes[i];
    int32_t st = visit(x, i);
    if (st != TRIDENT_OK) return st;
    if (x.kind == TRIDENT_NODE_TUPLE) {
      if (x.n < 0) return internal_fail(TRIDENT_ERR_INVALID, "negative tuple size");
      if (x.n > 0 && (x.first <= i || x.first > nnodes - x.n))
        return internal_fail(TRIDENT_ERR_INVALID, "tuple children must follow the tuple inside the array");
      for (int32_t c = x.n - 1; c >= 0; --c) {  // top - 1 + n <= nnodes: each node pushed once
        if (top >= TRIDENT_TREE_MAX_NODES) return internal_fail(TRIDENT_ERR_INVALID, "tree too large");
        stack[top] = x.first + c;
        depth[top++] = dep + 1;
      }
    }
  }
  return TRIDENT_OK;
}

bool match(const Recipe& r, int32_t ri, const trident_node* nodes, int32_t ni, trident_args* a) {
  const trident_recipe_node& p = r.nodes[ri];
  const trident_node& x = nodes[ni];
  switch (p.kind) {
    case TRIDENT_NODE_NONE:
      return x.kind == TRIDENT_NODE_NONE;
    case TRIDENT_NODE_TENSOR:
      if (x.kind == TRIDENT_NODE_TENSOR) {
        if (p.bind >= 0) a->t[p.bind] = x.t;
        return true;
      }
      if (x.kind == TRIDENT_NODE_DLTENSOR) {
        if (p.bind >= 0) from_dl(x.dl, &a->t[p.bind]);
        return true;
      }
      return false;
    case TRIDENT_NODE_TUPLE:
      if (x.kind != TRIDENT_NODE_TUPLE || x.n != p.n) return false;
      for (int32_t c = 0; c < p.n; ++c)
        if (!match(r, p.first + c, nodes, x.first + c, a)) return false;
      return true;
    case TRIDENT_NODE_INT:
    case TRIDENT_NODE_FLOAT: {
      if (x.kind != p.kind) return false;
      const double v = p.kind == TRIDENT_NODE_INT ? (double)x.i : x.f;
      switch (p.bind) {
        case TRIDENT_BIND_CONST:
          return p.kind == TRIDENT_NODE_INT ? x.i == p.i : x.f == p.f;
        case TRIDENT_BIND_EPS: a->eps = v; return true;
        case TRIDENT_BIND_THETA: a->rope_theta = v; return true;
        case TRIDENT_BIND_SCALAR: a->scalar = v; return true;
        default: return true;  // UNUSED
      }
    }
    default:
      return false;
  }
}

}  // namespace

int32_t validate_tree(const trident_node* nodes, int32_t nargs, int32_t nnodes) {
  return walk(nodes, nargs, nnodes, [](const trident_node& x, int32_t i) -> int32_t {
    if (x.reserved != 0) return internal_fail(TRIDENT_ERR_INVALID, "tree node reserved field must be 0");
    switch (x.kind) {
      case TRIDENT_NODE_NONE:
      case TRIDENT_NODE_TENSOR:  // its fields are validated with the bound argument tuple
      case TRIDENT_NODE_TUPLE:
      case TRIDENT_NODE_INT:
      case TRIDENT_NODE_FLOAT:
        return TRIDENT_OK;
      case TRIDENT_NODE_DLTENSOR:
        return check_dl(x.dl, i);
      default:
        return internal_fail(TRIDENT_ERR_INVALID, "unknown tree node kind");
    }
  });
}

int32_t make_recipe(const trident_recipe* r, int32_t op, int32_t nslots, Recipe* out) {
  if (!r) return internal_fail(TRIDENT_ERR_INVALID, "recipe is NULL");
  if (!(r->eps >= 0.0) || !(r->rope_theta >= 0.0) || r->scalar != r->scalar)
    return internal_fail(TRIDENT_ERR_INVALID, "recipe scalars (eps, theta >= 0; scalar not NaN)");
  int32_t slot_uses[TRIDENT_MAX_TENSORS] = {0};
  int32_t scalar_uses[3] = {0, 0, 0};
  int32_t st = walk(r->nodes, r->nargs, r->nnodes, [&](const trident_recipe_node& p, int32_t) -> int32_t {
    switch (p.kind) {
      case TRIDENT_NODE_NONE:
      case TRIDENT_NODE_TUPLE:
        return TRIDENT_OK;
      case TRIDENT_NODE_TENSOR:
        if (p.bind == TRIDENT_BIND_UNUSED) return TRIDENT_OK;
        if (p.bind < 0 || p.bind >= nslots)
          return internal_fail(TRIDENT_ERR_INVALID, "recipe tensor bound to a slot the op does not have");
        ++slot_uses[p.bind];
        return TRIDENT_OK;
      case TRIDENT_NODE_INT:
      case TRIDENT_NODE_FLOAT:
        if (p.bind == TRIDENT_BIND_CONST) {
          if (p.kind == TRIDENT_NODE_FLOAT && p.f != p.f)
            return internal_fail(TRIDENT_ERR_INVALID, "recipe constant is NaN");
          return TRIDENT_OK;
        }
        if (p.bind == TRIDENT_BIND_UNUSED) return TRIDENT_OK;
        if (p.bind > TRIDENT_BIND_EPS || p.bind < TRIDENT_BIND_SCALAR)
          return internal_fail(TRIDENT_ERR_INVALID, "recipe scalar bind code");
        ++scalar_uses[TRIDENT_BIND_EPS - p.bind];
        return TRIDENT_OK;
      default:
        return internal_fail(TRIDENT_ERR_INVALID, "recipe node kind");
    }
  });
  if (st != TRIDENT_OK) return st;
  for (int32_t k = 0; k < nslots; ++k)
    if (slot_uses[k] != 1) return internal_fail(TRIDENT_ERR_INVALID, "every op slot must be bound exactly once");
  for (int32_t k = 0; k < 3; ++k)
    if (scalar_uses[k] > 1) return internal_fail(TRIDENT_ERR_INVALID, "eps, theta and scalar are bound at most once");
  out->nodes = new (std::nothrow) trident_recipe_node[(size_t)(r->nnodes > 0 ? r->nnodes : 1)];
  if (!out->nodes) return internal_fail(TRIDENT_ERR_INVALID, "out of host memory");
  if (r->nnodes > 0) std::memcpy(out->nodes, r->nodes, sizeof(trident_recipe_node) * (size_t)r->nnodes);
  out->nargs = r->nargs;
  out->nnodes = r->nnodes;
  out->eps = r->eps;
  out->rope_theta = r->rope_theta;
  out->scalar = r->scalar;
  out->op = op;
  out->nslots = nslots;
  return TRIDENT_OK;
}

void free_recipe(Recipe* r) {
  delete[] r->nodes;
  r->nodes = nullptr;
}

bool bind_tree(const Recipe& r, const trident_node* nodes, int32_t nargs, trident_args* a) {
  if (nargs != r.nargs) return false;
  a->op = r.op;
  a->ntensors = r.nslots;
  a->eps = r.eps;
  a->rope_theta = r.rope_theta;
  a->scalar = r.scalar;
  a->flags = 0;
  a->reserved = 0;
  for (int32_t i = 0; i < nargs; ++i)
    if (!match(r, i, nodes, i, a)) return false;
  return true;
}

}  // namespace trident
