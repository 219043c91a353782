// scm.cpp -- the Specialization Cache Module: version table, guards, dispatch, launch.
//
// The paper's SCM (§3.1, Fig. 1c) compiles, for several guarded specialisations, the
// guard evaluation, the argument/environment preparation and the host execution into one
// native module, so a cache hit never returns to Python (§3.2). Here that module is this
// file: trident_scm_invoke validates the argument tuple, evaluates the versions' guards
// in creation order (Algorithm 1), packs the selected kernel's parameters and launches it
// on the caller's stream. Only a miss leaves native code, through the compile hook
// (§3.5); an error is returned at once and never falls through to another version.
//
// Guards are evaluated in two halves. The argument tuple's guarded properties (common
// device, dtypes, ranks, sizes, token count, layout class, alignment) are computed once
// per call into a Sig; each version's G_i then compares its fields against the Sig, so
// checks shared by every version run once (§3.2: redundant checks are removed and the
// rest ordered by their data dependencies). The result equals evaluating each G_i on
// its own, field by field.
//
// Table publication is append-only: slots never move and are written before the count
// that exposes them is released, so a reader needs one acquire load and no lock, and a
// registration from inside a hook is visible to every later call (§3.5: growth).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <initializer_list>
#include <mutex>
#include <tuple>
#include <new>
#include <vector>

#include "internal.h"
#include "measure.h"
#include "tree.h"
#include "trident_scm.h"

#define TRIDENT_API extern "C" __attribute__((visibility("default")))

// NVTX ranges around the boundary calls, for profilers' timelines. Compiled in only with
// -DTRIDENT_NVTX (build.py --nvtx); off by default, the calls then contain no trace of them.
#ifdef TRIDENT_NVTX
#include <nvtx3/nvToolsExt.h>
namespace {
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
};
}  // namespace
#define TRIDENT_RANGE(name) NvtxRange trident_nvtx_range_(name)
#else
#define TRIDENT_RANGE(name) ((void)0)
#endif

using namespace trident;

namespace {

// ------------------------------------------------------------------ errors
thread_local char tl_err[512] = "";
thread_local int tl_hook_depth = 0;

int32_t fail(int32_t status, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(tl_err, sizeof(tl_err), fmt, ap);
  va_end(ap);
  return status;
}

// ------------------------------------------------------------------ driver entry points
// The launch goes straight to the driver (cuLaunchKernelEx) with the CUfunction resolved
// at registration. The driver is reached through the runtime's entry-point query, so the
// library has no link-time dependency on libcuda and loads on machines without a GPU.
struct Driver {
  CUresult (*launch_ex)(const CUlaunchConfig*, CUfunction, void**, void**) = nullptr;
  CUresult (*ctx_get)(CUcontext*) = nullptr;
  CUresult (*ctx_push)(CUcontext) = nullptr;
  CUresult (*ctx_pop)(CUcontext*) = nullptr;
  bool ok = false;
};
Driver g_drv;
std::once_flag g_drv_once;

bool driver() {
  std::call_once(g_drv_once, [] {
    cudaDriverEntryPointQueryResult q;
    void* f = nullptr;
    bool ok = true;
    auto get = [&](const char* name) -> void* {
      f = nullptr;
      if (cudaGetDriverEntryPointByVersion(name, &f, 12000, cudaEnableDefault, &q) != cudaSuccess ||
          q != cudaDriverEntryPointSuccess)
        ok = false;
      return f;
    };
    g_drv.launch_ex = reinterpret_cast<decltype(g_drv.launch_ex)>(get("cuLaunchKernelEx"));
    g_drv.ctx_get = reinterpret_cast<decltype(g_drv.ctx_get)>(get("cuCtxGetCurrent"));
    g_drv.ctx_push = reinterpret_cast<decltype(g_drv.ctx_push)>(get("cuCtxPushCurrent"));
    g_drv.ctx_pop = reinterpret_cast<decltype(g_drv.ctx_pop)>(get("cuCtxPopCurrent"));
    g_drv.ok = ok && g_drv.launch_ex && g_drv.ctx_get && g_drv.ctx_push && g_drv.ctx_pop;
  });
  return g_drv.ok;
}

// ------------------------------------------------------------------ op tables
enum Kind : uint8_t { K_ACT_H, K_ACT_I, K_GAMMA_H, K_GAMMA_D, K_HEADS_Q, K_HEADS_KV, K_POS, K_CACHE,
                     K_MASK_H };

struct OpInfo {
  int32_t nslots;
  int32_t nfixed;
  bool flattening;  // activations may be rank 2 [T,W] or rank 3 [B,S,W]
  bool rope;        // guarded RoPE base
  Kind kind[TRIDENT_MAX_TENSORS];
  bool out[TRIDENT_MAX_TENSORS];
  uint8_t group[TRIDENT_MAX_TENSORS];  // in-place group id (0: none)
};

constexpr int kMaxOp = 11;
OpInfo g_ops[kMaxOp + 1];

// slot index constants of the chains
enum { C_H = 0, C_R0, C_GA, C_X1, C_R1, C_Q, C_K, C_V, C_POS, C_KC, C_VC, C_AO, C_GM, C_X2, C_R2,
       C_G, C_U, C_O, C_GQ, C_GK };

struct OpInit {
  OpInit() {
    auto set = [](int op, int nfixed, bool flat, bool rope,
                  std::initializer_list<std::tuple<Kind, bool, int>> slots) {
      OpInfo& o = g_ops[op];
      o.nslots = (int32_t)slots.size();
      o.nfixed = nfixed;
      o.flattening = flat;
      o.rope = rope;
      int i = 0;
      for (auto& s : slots) {
        o.kind[i] = std::get<0>(s);
        o.out[i] = std::get<1>(s);
        o.group[i] = (uint8_t)std::get<2>(s);
        ++i;
      }
    };
    set(TRIDENT_OP_ADD_RMSNORM, 1, true, false,
        {{K_ACT_H, false, 1}, {K_ACT_H, false, 2}, {K_GAMMA_H, false, 0}, {K_ACT_H, true, 1},
         {K_ACT_H, true, 2}});
    set(TRIDENT_OP_ROPE_KV, 4, false, true,
        {{K_HEADS_Q, true, 0}, {K_HEADS_KV, false, 0}, {K_HEADS_KV, false, 0}, {K_POS, false, 0},
         {K_CACHE, true, 0}, {K_CACHE, true, 0}});
    set(TRIDENT_OP_QKNORM_ROPE_KV, 4, false, true,
        {{K_HEADS_Q, true, 0}, {K_HEADS_KV, false, 0}, {K_HEADS_KV, false, 0}, {K_POS, false, 0},
         {K_CACHE, true, 0}, {K_CACHE, true, 0}, {K_GAMMA_D, false, 0}, {K_GAMMA_D, false, 0}});
    set(TRIDENT_OP_SWIGLU, 1, true, false, {{K_ACT_I, false, 1}, {K_ACT_I, false, 1}, {K_ACT_I, true, 1}});
    set(TRIDENT_OP_RMSNORM, 1, true, false, {{K_ACT_H, false, 1}, {K_GAMMA_H, false, 0}, {K_ACT_H, true, 1}});
    set(TRIDENT_OP_SILU, 1, true, false, {{K_ACT_H, false, 1}, {K_ACT_H, true, 1}});
    set(TRIDENT_OP_NEG, 1, true, false, {{K_ACT_H, false, 1}, {K_ACT_H, true, 1}});
    set(TRIDENT_OP_ADD, 1, true, false, {{K_ACT_H, false, 1}, {K_ACT_H, false, 1}, {K_ACT_H, true, 1}});
    set(TRIDENT_OP_MASKED_FILL, 1, true, false, {{K_ACT_H, false, 1}, {K_MASK_H, false, 0}, {K_ACT_H, true, 1}});
    const std::initializer_list<std::tuple<Kind, bool, int>> chain = {
        {K_ACT_H, false, 1},  {K_ACT_H, false, 2},    {K_GAMMA_H, false, 0}, {K_ACT_H, true, 1},
        {K_ACT_H, true, 2},   {K_HEADS_Q, true, 0},   {K_HEADS_KV, false, 0}, {K_HEADS_KV, false, 0},
        {K_POS, false, 0},    {K_CACHE, true, 0},     {K_CACHE, true, 0},     {K_ACT_H, false, 3},
        {K_GAMMA_H, false, 0}, {K_ACT_H, true, 3},    {K_ACT_H, true, 2},     {K_ACT_I, false, 4},
        {K_ACT_I, false, 4},  {K_ACT_I, true, 4}};
    set(TRIDENT_OP_LAYER_CHAIN, 6, false, true, chain);
    OpInfo& o = g_ops[TRIDENT_OP_LAYER_CHAIN_QKNORM];
    o = g_ops[TRIDENT_OP_LAYER_CHAIN];
    o.nslots = 20;
    o.kind[18] = o.kind[19] = K_GAMMA_D;
    o.out[18] = o.out[19] = false;
    o.group[18] = o.group[19] = 0;
  }
} g_op_init;

inline int elem_size(int32_t dt) {
  switch (dt) {
    case TRIDENT_BF16: case TRIDENT_FP16: return 2;
    case TRIDENT_FP32: case TRIDENT_I32: return 4;
    case TRIDENT_I64: return 8;
    case TRIDENT_U8: return 1;
    default: return 0;
  }
}
inline bool is_act(Kind k) { return k == K_ACT_H || k == K_ACT_I || k == K_HEADS_Q || k == K_HEADS_KV; }
// Tensors with activation-like rows (they take part in the layout class): activations and masks.
inline bool is_rowlike(Kind k) { return is_act(k) || k == K_MASK_H; }

// Rows view of a tensor: (rows, row width in elements, row stride in elements, packed).
struct Rows {
  int64_t n, width, stride;
  bool packed;
};

inline Rows rows_of(const trident_tensor& t, Kind k) {
  const int64_t* sh = t.shape;
  const int64_t* st = t.stride;
  if (k == K_HEADS_Q || k == K_HEADS_KV)
    return {sh[0], sh[1] * sh[2], st[0], st[2] == 1 && (sh[1] <= 1 || st[1] == sh[2])};
  if (k == K_ACT_H || k == K_ACT_I || k == K_MASK_H) {
    if (t.ndim == 2) return {sh[0], sh[1], st[0], st[1] == 1};
    const bool inner = st[2] == 1;
    if (sh[1] == 1) return {sh[0], sh[2], st[0], inner};
    if (sh[0] == 1) return {sh[1], sh[2], st[1], inner};
    return {sh[0] * sh[1], sh[2], st[1], inner && st[0] == sh[1] * st[1]};
  }
  // gamma, pos, cache: one dense row
  int64_t n = 1;
  for (int d = 0; d < t.ndim; ++d) n *= sh[d];
  return {1, n, n, true};
}

// ------------------------------------------------------------------ argument signature
constexpr int32_t kMixed = INT32_MIN;

struct Sig {
  int32_t device;
  int32_t act_dtype;
  int32_t rank;
  int32_t layout;  // trident_layout class, or -1
  bool aux_dtype_ok, ranks_ok, shapes_ok, aux_layout_ok, aligned16;
  int64_t T;
  int64_t lead[2];
  int32_t nlead;
  int64_t fixed[TRIDENT_MAX_FIXED];
};

inline bool shape_is(const trident_tensor& t, std::initializer_list<int64_t> want) {
  int d = 0;
  for (int64_t w : want) {
    if (t.shape[d] != w) return false;
    ++d;
  }
  return true;
}

// Structural validation -- everything that makes a call malformed rather than a miss --
// fused with the per-tensor guarded properties (common device, dtypes, ranks, 16-byte
// alignment) in one pass over the tensors; a second pass checks shapes and layouts against
// the sizes read off the arguments. Returns ERR_INVALID for a malformed tuple.
int32_t analyze(const trident_args* a, const OpInfo** info, Sig* s) {
  if (!a) return fail(TRIDENT_ERR_INVALID, "args is NULL");
  if (a->op < 1 || a->op > kMaxOp) return fail(TRIDENT_ERR_INVALID, "unknown op %d", a->op);
  const OpInfo& oi = g_ops[a->op];
  if (a->ntensors != oi.nslots)
    return fail(TRIDENT_ERR_INVALID, "op %d takes %d tensors, got %d", a->op, oi.nslots, a->ntensors);
  if (a->flags != 0) return fail(TRIDENT_ERR_INVALID, "args.flags must be 0");
  if (!(a->eps >= 0.0)) return fail(TRIDENT_ERR_INVALID, "eps must be >= 0");
  const trident_tensor* t = a->t;
  const int n = oi.nslots;
  s->device = t[0].device;
  s->act_dtype = -1;
  s->aux_dtype_ok = true;
  s->rank = t[0].ndim;
  const int act_rank = oi.flattening ? s->rank : 2;
  s->ranks_ok = !oi.flattening || s->rank == 2 || s->rank == 3;
  s->aligned16 = true;
  for (int i = 0; i < n; ++i) {  // pass 1: validation and per-tensor properties
    const trident_tensor& x = t[i];
    const int es = elem_size(x.dtype);
    if (es == 0) return fail(TRIDENT_ERR_INVALID, "tensor %d: unknown dtype %d", i, x.dtype);
    if (x.ndim < 1 || x.ndim > 4) return fail(TRIDENT_ERR_INVALID, "tensor %d: ndim %d", i, x.ndim);
    if (x.device < -1) return fail(TRIDENT_ERR_INVALID, "tensor %d: device %d", i, x.device);
    bool empty = false;
    for (int d = 0; d < x.ndim; ++d) {
      if (x.shape[d] < 0 || x.stride[d] < 0)
        return fail(TRIDENT_ERR_INVALID, "tensor %d: negative shape or stride", i);
      if (x.shape[d] == 0) empty = true;
    }
    const uintptr_t ptr = reinterpret_cast<uintptr_t>(x.data);
    if (!ptr && !empty) return fail(TRIDENT_ERR_INVALID, "tensor %d: NULL data", i);
    if (ptr % (uintptr_t)es != 0) return fail(TRIDENT_ERR_INVALID, "tensor %d: not element-aligned", i);
    if (x.device != t[0].device) s->device = kMixed;
    const Kind k = oi.kind[i];
    if (is_act(k) || k == K_CACHE) {
      if (s->act_dtype == -1) s->act_dtype = x.dtype;
      else if (s->act_dtype != x.dtype) s->act_dtype = kMixed;
    } else if (k == K_POS) {
      s->aux_dtype_ok &= x.dtype == TRIDENT_I32;
    } else if (k == K_MASK_H) {
      s->aux_dtype_ok &= x.dtype == TRIDENT_U8;
    } else {
      s->aux_dtype_ok &= x.dtype == TRIDENT_FP32;
    }
    const int want = (k == K_ACT_H || k == K_ACT_I || k == K_MASK_H) ? act_rank
                   : (k == K_HEADS_Q || k == K_HEADS_KV || k == K_CACHE) ? 3 : 1;
    s->ranks_ok &= x.ndim == want;
    // 16-byte alignment of every tensor the kernels move in 16-byte units (positions are
    // read one element at a time and only need their natural alignment)
    if (k != K_POS && s->aligned16) {
      if (ptr % 16 != 0) s->aligned16 = false;
      for (int d = 0; d + 1 < x.ndim; ++d)
        if (x.shape[d] > 1 && (x.stride[d] * es) % 16 != 0) s->aligned16 = false;
    }
  }
  *info = &oi;
  s->shapes_ok = false;
  s->layout = -1;
  s->aux_layout_ok = false;
  for (int i = 0; i < TRIDENT_MAX_FIXED; ++i) s->fixed[i] = -1;
  s->T = -1;
  if (!s->ranks_ok) return TRIDENT_OK;
  // leading dims, T and the fixed sizes read off the arguments
  if (oi.flattening && s->rank == 3) {
    s->nlead = 2;
    s->lead[0] = t[0].shape[0];
    s->lead[1] = t[0].shape[1];
    s->T = s->lead[0] * s->lead[1];
  } else {
    s->nlead = 1;
    s->lead[0] = t[0].shape[0];
    s->T = s->lead[0];
  }
  int64_t H = -1, I = -1, Hq = -1, Hkv = -1, D = -1, S = -1;
  const int op = a->op;
  if (op == TRIDENT_OP_ADD_RMSNORM || op == TRIDENT_OP_RMSNORM || op >= TRIDENT_OP_SILU) {
    H = t[0].shape[s->rank - 1];
    s->fixed[0] = H;
  } else if (op == TRIDENT_OP_SWIGLU) {
    I = t[0].shape[s->rank - 1];
    s->fixed[0] = I;
  } else {
    const int qs = (op == TRIDENT_OP_ROPE_KV || op == TRIDENT_OP_QKNORM_ROPE_KV) ? 0 : C_Q;
    Hq = t[qs].shape[1];
    D = t[qs].shape[2];
    Hkv = t[qs + 1].shape[1];
    S = t[qs + 4].shape[1];
    if (qs == 0) {
      s->fixed[0] = Hq; s->fixed[1] = Hkv; s->fixed[2] = D; s->fixed[3] = S;
    } else {
      H = t[C_H].shape[1];
      I = t[C_G].shape[1];
      s->fixed[0] = H; s->fixed[1] = Hq; s->fixed[2] = Hkv; s->fixed[3] = D; s->fixed[4] = S;
      s->fixed[5] = I;
    }
  }
  // pass 2: shapes, the layout class over the activation-like rows, and the auxiliary
  // layouts (gamma and pos dense, caches dense [Hkv, S, D])
  const int64_t T0 = s->lead[0];
  bool shapes = true, all_contig = true, none = false, aux = true;
  for (int i = 0; i < n; ++i) {
    const trident_tensor& x = t[i];
    const Kind k = oi.kind[i];
    switch (k) {
      case K_ACT_H: case K_ACT_I: case K_MASK_H: {
        const int64_t w = k == K_ACT_I ? I : H;
        shapes &= s->nlead == 2 ? shape_is(x, {s->lead[0], s->lead[1], w}) : shape_is(x, {T0, w});
        break;
      }
      case K_GAMMA_H: shapes &= shape_is(x, {H}); break;
      case K_GAMMA_D: shapes &= shape_is(x, {D}); break;
      case K_HEADS_Q: shapes &= shape_is(x, {T0, Hq, D}); break;
      case K_HEADS_KV: shapes &= shape_is(x, {T0, Hkv, D}); break;
      case K_POS: shapes &= shape_is(x, {T0}); break;
      case K_CACHE: shapes &= shape_is(x, {Hkv, S, D}); break;
    }
    if (is_rowlike(k)) {
      const Rows r = rows_of(x, k);
      if (!r.packed) none = true;
      else if (r.n > 1) {
        if (r.stride < r.width) none = true;
        else if (r.stride != r.width) all_contig = false;
      }
    } else if (k == K_GAMMA_H || k == K_GAMMA_D || k == K_POS) {
      aux &= x.shape[0] <= 1 || x.stride[0] == 1;
    } else if (k == K_CACHE) {
      aux &= x.stride[0] == S * D && x.stride[1] == D && x.stride[2] == 1;
    }
  }
  s->shapes_ok = shapes;
  s->layout = none ? -1 : (all_contig ? TRIDENT_LAYOUT_CONTIG : TRIDENT_LAYOUT_ROWSTRIDED);
  s->aux_layout_ok = aux;
  return TRIDENT_OK;
}

// ------------------------------------------------------------------ versions
struct RopeTable {  // theta^(-2i/D) = hi + lo for i < D/2, split from fp64
  double theta;
  int32_t D;
  float2* dev;
};

struct Version {
  trident_spec_desc d;
  int32_t nfixed;
  bool rope;
  KernelEntry ke;
  CUfunction fn;
  CUfunction fn_inplace;  // layer chain: one block per token when outputs alias inputs
  CUfunction fn_late;     // layer chain: `fn` with the late launch trigger
  CUfunction fn_wide;     // layer chain: `fn_inplace` with kChainWideSwigluUnroll tiles
  int32_t wave_blocks;    // layer chain: blocks of `fn` resident at once on the whole GPU
  CUfunction fn_large;          // add+RMSNorm: entry for calls of >= ke.large_rows rows
  CUfunction step_fn;           // layer chain: several calls per launch (two blocks per token)
  CUfunction step_fn_inplace;   // ... one block per token
  CUfunction step_fn_role;      // ... one block per token, role-major order over the step
  int32_t step_wave_blocks;     // blocks of `step_fn` resident at once
  const float2* inv_freq;
  Recipe* recipe;               // structured-argument binding (register_tree_spec), or NULL
};

// Step replay cache of invoke_step. A fused chunk's outcome is a function of its argument
// bytes alone: selection reads the arguments and a table that only grows (a call's first
// match stays its first match), the byte rules read only the arguments, and the packed
// parameter block reads the arguments, the selected versions and state fixed at creation.
// So a chunk whose argument bytes equal a stored one relaunches the stored block. Entries
// are stored only for chunks whose fingerprint was seen before (a decode loop passing the
// same buffers step after step), so chunks that never repeat pay one fingerprint.
constexpr int kMemoEntries = 4;
constexpr int kSeenRing = 8;

struct StepMemo {
  uint64_t fp;     // fingerprint; 0 marks an empty entry
  uint64_t used;   // clock of the last store or replay (least recently used is replaced)
  int32_t m;       // calls
  int32_t ndist;   // distinct selected versions
  unsigned grid;
  CUfunction fn;
  int32_t sel[kStepMax];
  int32_t dist_idx[kStepMax], dist_cnt[kStepMax];
  trident_args args[kStepMax];
  ChainStepParams P;
};

}  // namespace

struct trident_scm {
  trident_scm_options opt{};
  trident_compile_hook hook = nullptr;
  void* user = nullptr;
  trident_tree_hook tree_hook = nullptr;
  void* tree_user = nullptr;
  bool dry = false;
  Version* versions = nullptr;
  std::atomic<int32_t> count{0};
  std::mutex reg_mu;
  std::atomic<uint64_t>* hits_per = nullptr;
  std::atomic<uint64_t> invokes{0}, hits{0}, misses{0}, hook_calls{0}, hook_failures{0},
      hook_registered{0}, err_invalid{0}, err_cuda{0}, guard_evals{0}, fused_launches{0},
      fused_calls{0};
  // device state
  int32_t device = 0;
  CUcontext ctx = nullptr;
  uint32_t* d_err = nullptr;
  int32_t sm_count = 0;  // grids of at most this many blocks prefetch before the PDL wait
  std::vector<RopeTable> tables;
  // host timing of hits
  uint32_t* ring = nullptr;
  int32_t ring_cap = 0;
  std::atomic<uint64_t> ring_n{0};
  // step replay cache (invoke_step); memo, seen and memo_clock are used only while
  // memo_lock is held (a thread that finds it held takes the full path)
  StepMemo* memo = nullptr;  // kMemoEntries entries, allocated by the first store
  uint64_t seen[kSeenRing] = {};
  uint32_t seen_next = 0;
  uint64_t memo_clock = 0;
  std::atomic_flag memo_lock = ATOMIC_FLAG_INIT;
  std::atomic<uint64_t> step_replays{0};
};

namespace {

bool guard_holds(const Version& v, const Sig& s, const trident_args* a) {
  const trident_spec_desc& d = v.d;
  if (d.device != s.device || d.dtype != s.act_dtype || !s.aux_dtype_ok) return false;
  if (d.rank != s.rank || !s.ranks_ok || !s.shapes_ok) return false;
  for (int i = 0; i < v.nfixed; ++i)
    if (d.fixed[i] != s.fixed[i]) return false;
  if (v.rope && !(d.rope_theta == a->rope_theta)) return false;
  if (s.T < d.tok_lo || s.T > d.tok_hi) return false;
  if (s.layout < 0 || (d.layout != TRIDENT_LAYOUT_ANY && d.layout != s.layout)) return false;
  if (!s.aux_layout_ok) return false;
  if (d.align_bytes == 16 && !s.aligned16) return false;
  return true;
}

// floor division for int64 with positive divisor
inline int64_t fdiv(int64_t a, int64_t b) { return a >= 0 ? a / b : -((-a + b - 1) / b); }

// Do two row sets share a byte? Rows are byte intervals [base + i*rs, base + i*rs + w).
// Exact when one set has one row or both have the same row stride; otherwise the
// answer is "yes" (conservative) once their overall extents intersect.
bool rows_overlap(int64_t a, int64_t na, int64_t wa, int64_t rsa, int64_t b, int64_t nb,
                  int64_t wb, int64_t rsb) {
  if (na <= 0 || nb <= 0 || wa <= 0 || wb <= 0) return false;
  const int64_t ea = a + (na - 1) * rsa + wa, eb = b + (nb - 1) * rsb + wb;
  if (ea <= b || eb <= a) return false;
  if (na == 1 && nb == 1) return true;  // extents are the rows
  if (na == 1 || nb == 1) {
    // single interval [p, p+w) against rows q + j*rs, j in [0, n)
    const bool a1 = na == 1;
    const int64_t p = a1 ? a : b, w = a1 ? wa : wb;
    const int64_t q = a1 ? b : a, wq = a1 ? wb : wa, rs = a1 ? rsb : rsa, n = a1 ? nb : na;
    // need q + j rs < p + w and p < q + j rs + wq  <=>  (p - wq - q) < j rs < (p + w - q)
    const int64_t jmin = fdiv(p - wq - q, rs) + 1;
    const int64_t jmax = -fdiv(-(p + w - q), rs) - 1;  // ceil(x/rs) - 1
    const int64_t lo = jmin > 0 ? jmin : 0, hi = jmax < n - 1 ? jmax : n - 1;
    return lo <= hi;
  }
  if (rsa != rsb) return true;
  const int64_t rs = rsa, d = a - b;
  // rows i of A and j of B overlap iff -wa < d + k rs < wb with k = i - j
  const int64_t kmin = fdiv(-wa - d, rs) + 1;
  const int64_t kmax = -fdiv(-(wb - d), rs) - 1;
  const int64_t lo = kmin > -(nb - 1) ? kmin : -(nb - 1);
  const int64_t hi = kmax < na - 1 ? kmax : na - 1;
  return lo <= hi;
}

bool same_desc(const trident_tensor& x, const trident_tensor& y) {
  if (x.data != y.data || x.dtype != y.dtype || x.ndim != y.ndim) return false;
  for (int d = 0; d < x.ndim; ++d)
    if (x.shape[d] != y.shape[d] || x.stride[d] != y.stride[d]) return false;
  return true;
}

// Launch precondition (checked after a hit, before the launch): no output shares a byte
// with another slot unless the two are the same tensor in one of the op's in-place groups.
// Slots are sorted by the start of their byte extent and swept once, so only pairs whose
// extents intersect (views into one buffer, in practice) reach the exact row test.
int32_t check_overlap(const trident_args* a, const OpInfo& oi) {
  const int n = oi.nslots;
  int64_t base[TRIDENT_MAX_TENSORS], nr[TRIDENT_MAX_TENSORS], w[TRIDENT_MAX_TENSORS],
      rs[TRIDENT_MAX_TENSORS], end[TRIDENT_MAX_TENSORS];
  int order[TRIDENT_MAX_TENSORS];
  int m = 0;
  for (int i = 0; i < n; ++i) {
    const Rows r = rows_of(a->t[i], oi.kind[i]);
    const int es = elem_size(a->t[i].dtype);
    base[i] = (int64_t)reinterpret_cast<uintptr_t>(a->t[i].data);
    nr[i] = r.n;
    w[i] = r.width * es;
    rs[i] = r.stride * es;
    if (nr[i] <= 0 || w[i] <= 0) continue;  // no bytes: overlaps nothing
    end[i] = base[i] + (nr[i] - 1) * rs[i] + w[i];
    int k = m++;  // insertion sort by extent start
    while (k > 0 && base[order[k - 1]] > base[i]) {
      order[k] = order[k - 1];
      --k;
    }
    order[k] = i;
  }
  for (int x = 0; x < m; ++x) {
    const int i = order[x];
    for (int y = x + 1; y < m && base[order[y]] < end[i]; ++y) {  // extents intersect
      const int j = order[y];
      if (!oi.out[i] && !oi.out[j]) continue;  // inputs may share bytes
      if (!rows_overlap(base[i], nr[i], w[i], rs[i], base[j], nr[j], w[j], rs[j])) continue;
      if (oi.group[i] != 0 && oi.group[i] == oi.group[j] && same_desc(a->t[i], a->t[j])) continue;
      const int o = oi.out[i] ? i : j;
      return fail(TRIDENT_ERR_INVALID, "output tensor %d overlaps tensor %d", o, o == i ? j : i);
    }
  }
  return TRIDENT_OK;
}

// ------------------------------------------------------------------ parameter packing
inline int64_t row_stride(const trident_tensor& t, Kind k) { return rows_of(t, k).stride; }

void pack_addnorm(const trident_args* a, int x, int r, int g, int y, int ro, const Sig& s,
                  Kind kind, AddNormParams* p) {
  const trident_tensor* t = a->t;
  p->x = t[x].data; p->r = t[r].data; p->gamma = (const float*)t[g].data;
  p->y = t[y].data; p->r_out = t[ro].data;
  p->T = s.T;
  p->H = t[g].shape[0];
  p->x_rs = row_stride(t[x], kind); p->r_rs = row_stride(t[r], kind);
  p->y_rs = row_stride(t[y], kind); p->ro_rs = row_stride(t[ro], kind);
  p->eps = (float)a->eps;
  p->inv_H = (float)(1.0 / (double)p->H);
  p->prefetch = 0;
  p->first_wait_polls = kBulkWaitPolls;
  p->err = nullptr;
}

void pack_rmsnorm(const trident_args* a, const Sig& s, RmsNormParams* p) {
  const trident_tensor* t = a->t;
  p->x = t[0].data; p->gamma = (const float*)t[1].data; p->y = t[2].data;
  p->T = s.T;
  p->H = t[1].shape[0];
  p->x_rs = row_stride(t[0], K_ACT_H); p->y_rs = row_stride(t[2], K_ACT_H);
  p->eps = (float)a->eps;
  p->inv_H = (float)(1.0 / (double)p->H);
  p->prefetch = 0;
}

void pack_pointwise(const trident_args* a, const Sig& s, PointwiseParams* p) {
  const trident_tensor* t = a->t;
  const int op = a->op;
  const int yi = (op == TRIDENT_OP_SILU || op == TRIDENT_OP_NEG) ? 1 : 2;
  p->a = t[0].data;
  p->b = op == TRIDENT_OP_ADD ? t[1].data : nullptr;
  p->mask = op == TRIDENT_OP_MASKED_FILL ? (const uint8_t*)t[1].data : nullptr;
  p->y = t[yi].data;
  p->T = s.T;
  p->W = s.fixed[0];
  p->a_rs = row_stride(t[0], K_ACT_H);
  p->b_rs = op == TRIDENT_OP_ADD ? row_stride(t[1], K_ACT_H) : 0;
  p->m_rs = op == TRIDENT_OP_MASKED_FILL ? row_stride(t[1], K_MASK_H) : 0;
  p->y_rs = row_stride(t[yi], K_ACT_H);
  p->scalar = (float)a->scalar;
  p->prefetch = 0;
}

// Round-up multiplier and shift for dividing 32-bit unsigned integers by d (1 <= d < 2^31):
// l = ceil(log2 d), m = floor(2^32 (2^l - d) / d) + 1; the kernels take the quotient as
// (h + ((n - h) >> 1)) >> (l - 1) with h = umulhi(n, m) (fast_div; Granlund and Montgomery,
// 1994), and l = 0 (d = 1) as n itself.
void div_magic(uint32_t d, uint32_t* m, int32_t* l) {
  if (d == 0) {  // no divisor: callers reject such calls first; stay defined regardless
    *m = 0;
    *l = 0;
    return;
  }
  int32_t s = 0;
  while ((1ull << s) < d) ++s;
  *m = (uint32_t)(((1ull << 32) * ((1ull << s) - d)) / d + 1);
  *l = s;
}

void pack_rope(const trident_args* a, int base, int gq, const Version& v, uint32_t* err,
               RopeParams* p) {
  const trident_tensor* t = a->t;
  p->q = t[base].data; p->k = t[base + 1].data; p->v = t[base + 2].data;
  p->pos = (const int32_t*)t[base + 3].data;
  p->k_cache = t[base + 4].data; p->v_cache = t[base + 5].data;
  p->gamma_q = gq >= 0 ? (const float*)t[gq].data : nullptr;
  p->gamma_k = gq >= 0 ? (const float*)t[gq + 1].data : nullptr;
  p->inv_freq = v.inv_freq;
  p->err = err;
  p->T = t[base].shape[0];
  p->S = t[base + 4].shape[1];
  p->q_rs = t[base].stride[0]; p->k_rs = t[base + 1].stride[0]; p->v_rs = t[base + 2].stride[0];
  p->Hq = (int32_t)t[base].shape[1];
  p->Hkv = (int32_t)t[base + 1].shape[1];
  p->D = (int32_t)t[base].shape[2];
  p->NH = p->Hq + 2 * p->Hkv;
  div_magic((uint32_t)p->NH, &p->nh_magic, &p->nh_shift);
  p->eps = (float)a->eps;
  p->inv_D = (float)(1.0 / (double)p->D);
  p->prefetch = 0;
}

void pack_swiglu(const trident_args* a, int g, int u, int o, int64_t T, SwigluParams* p) {
  const trident_tensor* t = a->t;
  p->g = t[g].data; p->u = t[u].data; p->out = t[o].data;
  p->T = T;
  p->I = t[g].shape[t[g].ndim - 1];
  p->g_rs = row_stride(t[g], K_ACT_I); p->u_rs = row_stride(t[u], K_ACT_I);
  p->o_rs = row_stride(t[o], K_ACT_I);
  p->prefetch = 0;
}

// Launches fn with the SCM's context current on this thread.
int32_t launch_on(trident_scm* scm, CUlaunchConfig* cfg, CUfunction fn, void** kp) {
  CUcontext cur = nullptr;
  g_drv.ctx_get(&cur);
  const bool swap = cur != scm->ctx;
  if (swap && g_drv.ctx_push(scm->ctx) != CUDA_SUCCESS)
    return fail(TRIDENT_ERR_CUDA, "cannot make the SCM's context current");
  const CUresult rc = g_drv.launch_ex(cfg, fn, kp, nullptr);
  if (swap) {
    CUcontext dummy;
    g_drv.ctx_pop(&dummy);
  }
  if (rc != CUDA_SUCCESS) return fail(TRIDENT_ERR_CUDA, "cuLaunchKernelEx failed (%d)", (int)rc);
  return TRIDENT_OK;
}

// Launch configuration with the block size and, with TRIDENT_OPT_PDL, programmatic
// stream serialisation (attr must outlive the launch).
void base_config(const trident_scm* scm, void* stream, CUlaunchConfig* cfg, CUlaunchAttribute* attr) {
  std::memset(cfg, 0, sizeof(*cfg));
  std::memset(attr, 0, sizeof(*attr));
  cfg->blockDimX = kThreads; cfg->blockDimY = 1; cfg->blockDimZ = 1;
  cfg->gridDimY = 1; cfg->gridDimZ = 1;
  cfg->hStream = (CUstream)stream;
  cfg->attrs = attr;
  cfg->numAttrs = 0;
  if (scm->opt.flags & TRIDENT_OPT_PDL) {
    attr->id = CU_LAUNCH_ATTRIBUTE_PROGRAMMATIC_STREAM_SERIALIZATION;
    attr->value.programmaticStreamSerializationAllowed = 1;
    cfg->numAttrs = 1;
  }
}

// Packs one layer-chain call: both norms, RoPE/KV, SwiGLU and the RoPE and SwiGLU block
// counts, for SwiGLU tiles of `unroll` x 256 vectors (kChainSwigluUnroll in a call's own
// launch, kChainStepSwigluUnroll in a whole-step launch). The norm split (set_chain_split)
// is decided by the caller.
// SwiGLU tiles of `unroll` x 256 vectors per row: their count, nC, and the row multiplier.
void set_chain_tiles(ChainParams* c, int64_t T, int32_t unroll, int32_t vec) {
  const int64_t per = (int64_t)unroll * kThreads * vec;
  const int64_t tiles = (c->sw.I + per - 1) / per;
  c->nC = (int32_t)(T * tiles);
  c->sw_tiles_per_row = (int32_t)tiles;
  div_magic((uint32_t)tiles, &c->sw_magic, &c->sw_shift);
  c->sw_tiles = T * tiles;
}

int32_t pack_chain(trident_scm* scm, const Version& v, const trident_args* a, const Sig& s,
                   int32_t unroll, ChainParams* c) {
  pack_addnorm(a, C_H, C_R0, C_GA, C_X1, C_R1, s, K_ACT_H, &c->n1);
  pack_addnorm(a, C_AO, C_R1, C_GM, C_X2, C_R2, s, K_ACT_H, &c->n2);
  pack_rope(a, C_Q, a->op == TRIDENT_OP_LAYER_CHAIN_QKNORM ? C_GQ : -1, v, scm->d_err, &c->rope);
  pack_swiglu(a, C_G, C_U, C_O, s.T, &c->sw);
  const int64_t per = (int64_t)unroll * kThreads * v.ke.vec;
  const int64_t tiles = (c->sw.I + per - 1) / per;
  const int64_t upb = rope_units_per_block(c->rope.D, 2);
  const int64_t nB = (s.T * c->rope.NH + upb - 1) / upb, nC = s.T * tiles;
  if (2 * s.T + nB + nC > 0x7fffffff) return fail(TRIDENT_ERR_INVALID, "layer chain too large for one launch");
  c->nB = (int32_t)nB;
  set_chain_tiles(c, s.T, unroll, v.ke.vec);
  c->prefetch = 0;
  c->tok_grid = 0;
  c->rope_per_tok = 0;
  c->rope_k = 1;
  return TRIDENT_OK;
}

// Does a chain call write an output over an input? Then the norms keep one CTA per
// token: with two, a CTA could overwrite row bytes its partner has not read yet.
bool chain_inplace(const trident_args* a) {
  const trident_tensor* t = a->t;
  return t[C_X1].data == t[C_H].data || t[C_R1].data == t[C_R0].data ||
         t[C_R2].data == t[C_R0].data || t[C_X2].data == t[C_AO].data;
}

// Sets the norm CTAs per token (split) and the RoPE head-rows per lane group (rope_k), and
// with them nA, nB and the grid's block count.
int32_t set_chain_split(ChainParams* c, int64_t T, int32_t split, int32_t rope_k, int64_t* blocks) {
  c->a_split = split;
  c->nA = (int32_t)(T * split);
  c->rope_k = rope_k;
  const int64_t upb = (int64_t)rope_units_per_block(c->rope.D, 2) * rope_k;
  c->nB = (int32_t)((T * c->rope.NH + upb - 1) / upb);
  *blocks = (int64_t)c->nA + c->nB + c->nC;
  return TRIDENT_OK;
}

// Three head-rows per RoPE lane group (rope_rows) on grids several waves long: a grid whose
// one-CTA-per-token form with one head-row per lane group (`one` blocks) exceeds the resident
// slots. There blocks queue for slots and a RoPE block that moves three rows for the same
// fixed costs pays; within one wave a block's own latency is the step (a single-wave grid of
// such blocks measured slower: 64 tokens 3.52 -> 4.46 us). Same-box A/B: Llama layer steps
// at 128 tokens 5.61 -> 5.12 us, 256 tokens 9.37 -> 8.39 us; 36 Qwen3-style layers in one
// launch at 32 / 64 / 128 / 256 tokens 36.7 / 70.5 / 142.9 / 281.0 -> 35.2 / 65.6 / 128.6 /
// 252.7 us.
inline int32_t chain_rope_k(int64_t one, int64_t wave_blocks) { return one > wave_blocks ? 3 : 1; }

// Layer-chain prefetch before the PDL wait: every block's first lines for grids of at most
// one block per SM (small_grid); otherwise, when norm_rows, only the norm blocks prefetch:
// their rows -- the first loads of the longest blocks, which then come from L2 while every
// other block's loads stream from DRAM -- and their token's RoPE head-rows. Measured: one
// call at 64 tokens (one wave) 3.80 -> 3.53 us per layer step with the rows (4.02 -> 3.78 us
// in a timeline probe with the head-rows too), at 128 tokens (two waves) 6.1 -> 5.8 us;
// prefetching every block's own lines there was slower (4.26 -> 4.68 us at 64 tokens).
// Whole-step launches take it only with two norm CTAs per token (one wave): on multi-wave
// steps it measured 1-2 % slower.
inline int32_t chain_prefetch_mode(bool pdl, bool small_grid, bool norm_rows) {
  if (!pdl) return 0;
  return small_grid ? 1 : (norm_rows ? 2 : 0);
}

inline unsigned cap_grid(int64_t n) { return (unsigned)(n < 1 ? 1 : (n > 0x7fffffff ? 0x7fffffff : n)); }

int32_t do_launch(trident_scm* scm, const Version& v, const trident_args* a, const Sig& s,
                  void* stream) {
  const int op = a->op;
  CUlaunchConfig cfg;
  CUlaunchAttribute attr;
  base_config(scm, stream, &cfg, &attr);
  union {
    AddNormParams an;
    RmsNormParams rn;
    PointwiseParams pw;
    RopeParams rp;
    RopeBulkParams rb;  // rb.rp is rp
    SwigluParams sw;
    ChainParams ch;
  } P;
  void* kp[1] = {&P};
  bool late = false;  // layer chain: launch fn_late (the late launch trigger)
  bool wide = false;  // layer chain: launch fn_wide (wider SwiGLU tiles)
  switch (op) {
    case TRIDENT_OP_ADD_RMSNORM:
      pack_addnorm(a, 0, 1, 2, 3, 4, s, K_ACT_H, &P.an);
      P.an.err = scm->d_err;
      if (scm->opt.flags & TRIDENT_OPT_TEST_WAIT_TIMEOUT) P.an.first_wait_polls = 0;
      cfg.gridDimX = cap_grid(s.T);
      break;
    case TRIDENT_OP_RMSNORM:
      pack_rmsnorm(a, s, &P.rn);
      cfg.gridDimX = v.ke.kind == KK_NORM_ROWS ? cap_grid((s.T + v.ke.rows - 1) / v.ke.rows) : cap_grid(s.T);
      break;
    case TRIDENT_OP_ROPE_KV:
    case TRIDENT_OP_QKNORM_ROPE_KV: {
      pack_rope(a, 0, op == TRIDENT_OP_QKNORM_ROPE_KV ? 6 : -1, v, scm->d_err, &P.rp);
      const int64_t units = P.rp.T * P.rp.NH;
      if (v.fn_large && s.T >= v.ke.large_rows) {  // bulk-copy kernel: ke.rows tokens per block,
        const int64_t tpb = v.ke.rows;            // their head-rows staged in shared memory
        cfg.gridDimX = cap_grid((P.rp.T + tpb - 1) / tpb);
        cfg.sharedMemBytes = (unsigned)(tpb * P.rp.NH * P.rp.D * 2);
        P.rb.first_wait_polls = (scm->opt.flags & TRIDENT_OPT_TEST_WAIT_TIMEOUT) ? 0u : kBulkWaitPolls;
        break;
      }
      const int64_t upb = v.ke.kind == KK_ROPE_HALFWARP ? rope_units_per_block(P.rp.D, 2) : kThreads / 32;
      cfg.gridDimX = cap_grid((units + upb - 1) / upb);
      break;
    }
    case TRIDENT_OP_SWIGLU:
    case TRIDENT_OP_SILU:
    case TRIDENT_OP_ADD:
    case TRIDENT_OP_NEG:
    case TRIDENT_OP_MASKED_FILL: {
      int64_t W;
      if (op == TRIDENT_OP_SWIGLU) {
        pack_swiglu(a, 0, 1, 2, s.T, &P.sw);
        W = P.sw.I;
      } else {
        pack_pointwise(a, s, &P.pw);
        W = P.pw.W;
      }
      if (v.ke.kind == KK_SWIGLU_TILE) {  // (column tiles, rows)
        const int64_t per = (int64_t)v.ke.unroll * kThreads * v.ke.vec;
        cfg.gridDimX = cap_grid((W + per - 1) / per);
        cfg.gridDimY = (unsigned)(s.T < 65535 ? (s.T < 1 ? 1 : s.T) : 65535);
      } else {  // flat grid-stride
        const int64_t blocks = (s.T * W + kThreads - 1) / kThreads;
        cfg.gridDimX = cap_grid(blocks < 152 * 64 ? blocks : 152 * 64);
      }
      break;
    }
    case TRIDENT_OP_LAYER_CHAIN:
    case TRIDENT_OP_LAYER_CHAIN_QKNORM: {
      ChainParams& c = P.ch;
      int32_t st = pack_chain(scm, v, a, s, v.ke.unroll, &c);
      if (st != TRIDENT_OK) return st;
      // Two CTAs per token for the norms -- so no SM carries a whole token's norm traffic --
      // while the grid still fits in one wave, and unless an output is written over an
      // input the partner CTA still reads (in-place calls keep one CTA per token).
      const int32_t split = (!chain_inplace(a) && 2 * s.T + c.nB + c.nC <= v.wave_blocks) ? 2 : 1;
      const int64_t one = s.T + c.nB + c.nC;  // one CTA per token, one head-row per lane group
      const int32_t rope_k = split == 1 ? chain_rope_k(one, v.wave_blocks) : 1;
      // Wider SwiGLU tiles (fn_wide) on grids of more than four waves: same-box probe, one
      // Llama layer at 1024 / 4096 tokens 34.2 / 122.8 -> 31.3 / 112.6 us; at 256 tokens
      // (3.4 waves) 9.81 -> 9.75 us, at 128 tokens (1.7 waves) 4.72 -> 5.11 us.
      wide = split == 1 && v.fn_wide && one > 4 * (int64_t)v.wave_blocks;
      if (wide) set_chain_tiles(&c, s.T, kChainWideSwigluUnroll, v.ke.vec);
      int64_t blocks = 0;
      st = set_chain_split(&c, s.T, split, rope_k, &blocks);
      if (st != TRIDENT_OK) return st;
      cfg.gridDimX = (unsigned)blocks;
      // Under PDL, a role-major grid of more than a quarter block per SM whose blocks, with
      // its own norm blocks, fit the resident slots give or take an eighth of them launches
      // fn_late: its RoPE and SwiGLU blocks trigger the next launch at their exit, so the
      // next grid is placed whole while this one's norm blocks finish, one norm block per SM
      // instead of up to four. Same-box A/B of Llama layer steps against the grids below: 6
      // tokens 2.22 -> 2.12 us, 8 tokens 2.33 -> 2.14, 16 tokens 2.58 -> 2.29, 24 tokens
      // 3.19 -> 2.44, 32 tokens 2.98 -> 2.57, 48 tokens 3.21 -> 2.99, 56 tokens 3.31 ->
      // 3.19; equal at 2 and 4 tokens and at 1 token 1.5-2 % slower (nothing to place, and
      // the next launch starts later), hence the lower bound; a few dozen blocks placed late
      // cost less than stacked norm blocks (36 Qwen3-style launches at 64 tokens 125.9 ->
      // 122.3 us, 62 Llama tokens equal), but at 64 Llama tokens, with 96 blocks placed late,
      // the probe measured 3.51 -> 3.69 us, hence the upper bound.
      // Otherwise a token-major grid (chain_block_tok) for grids of at most two blocks per SM,
      // when every token has the same number of RoPE blocks: consecutive blocks then mix
      // roles, so the blocks that land together on one SM are not all norm blocks (measured
      // against role-major grids without the late trigger: 16 tokens 3.55 -> 2.85 us per
      // layer step, 1 token 2.20 -> 2.04 us). Larger grids are role-major, which starts the
      // longest (norm) blocks first (64 tokens: 3.98 us role-major, 4.05 us token-major; 48
      // and 64 tokens in other interleaved orders were slower as well).
      const int64_t upb = rope_units_per_block(c.rope.D, 2);
      if ((scm->opt.flags & TRIDENT_OPT_PDL) && split == 2 && v.fn_late && 4 * blocks > scm->sm_count &&
          blocks + c.nA <= v.wave_blocks + v.wave_blocks / 8) {
        late = true;
      } else if (c.rope.NH % upb == 0 && s.T >= 1 && s.T <= 65535 && blocks <= 2 * scm->sm_count) {
        c.tok_grid = 1;
        c.rope_per_tok = (int32_t)(c.rope.NH / upb);
        cfg.gridDimX = (unsigned)(split + c.rope_per_tok + c.sw_tiles_per_row);
        cfg.gridDimY = (unsigned)s.T;
      }
      break;
    }
    default:
      return fail(TRIDENT_ERR_INVALID, "op");
  }
  // L2 prefetch before the PDL wait (prefetch_l2 in device_common.cuh): only for grids of
  // at most one block per SM launched with programmatic serialisation (measured: ~10%
  // faster layer steps at 1-4 tokens; slower once the grid fills the GPU, where a layer
  // chain prefetches only its norm rows -- see chain_prefetch_mode)
  const bool pdl = (scm->opt.flags & TRIDENT_OPT_PDL) != 0;
  const int32_t pf = pdl && (int64_t)cfg.gridDimX * cfg.gridDimY <= scm->sm_count ? 1 : 0;
  switch (op) {
    case TRIDENT_OP_ADD_RMSNORM: P.an.prefetch = pf; break;
    case TRIDENT_OP_RMSNORM: P.rn.prefetch = pf; break;
    case TRIDENT_OP_ROPE_KV:
    case TRIDENT_OP_QKNORM_ROPE_KV: P.rp.prefetch = pf; break;
    case TRIDENT_OP_SWIGLU: P.sw.prefetch = pf; break;
    case TRIDENT_OP_LAYER_CHAIN:
    case TRIDENT_OP_LAYER_CHAIN_QKNORM: P.ch.prefetch = chain_prefetch_mode(pdl, pf != 0 && !late, true); break;
    default: P.pw.prefetch = pf; break;
  }
  CUfunction fn = v.fn;
  if ((op == TRIDENT_OP_LAYER_CHAIN || op == TRIDENT_OP_LAYER_CHAIN_QKNORM) && P.ch.a_split == 1)
    fn = wide ? v.fn_wide : v.fn_inplace;
  else if (late && v.fn_late)
    fn = v.fn_late;
  if (v.fn_large && s.T >= v.ke.large_rows) fn = v.fn_large;  // many rows: add+RMSNorm's bulk-copy
                                                              // kernel, RoPE's several rows per lane
  return launch_on(scm, &cfg, fn, kp);
}

// Can calls a[0..m-1] run in one launch, as far as their bytes go? Two rules from one
// sweep over every slot's extent, sorted by start (only pairs whose extents intersect --
// views into one buffer, in practice -- reach the exact row test):
//  - within a call, its launch precondition (check_overlap), when check_own is set;
//  - between calls, independence: no output byte of one call is a byte of another call's
//    tensor, so running them together equals running them in order.
bool step_bytes_ok(const trident_args* a, int32_t m, bool check_own) {
  struct Ext {
    int64_t base, end, nr, w, rs;
    int32_t call, slot;
    bool out;
  };
  constexpr int kMaxExt = kStepMax * TRIDENT_MAX_TENSORS;  // on the stack: no allocation
  Ext ext[kMaxExt];
  uint64_t keys[kMaxExt], keys2[kMaxExt];
  uint32_t order[kMaxExt];
  size_t n = 0;
  int64_t lo = INT64_MAX, hi = INT64_MIN;
  // Slot-major: one slot of every call, then the next slot. When each slot's tensors sit in
  // one arena in call order (a serving engine's per-layer buffers, or views into one
  // buffer), every slot then contributes an ascending run of starts.
  int32_t nslots = 0;
  for (int32_t c = 0; c < m; ++c) nslots = g_ops[a[c].op].nslots > nslots ? g_ops[a[c].op].nslots : nslots;
  for (int i = 0; i < nslots; ++i) {
    for (int32_t c = 0; c < m; ++c) {
      const OpInfo& oi = g_ops[a[c].op];
      if (i >= oi.nslots) continue;
      const trident_tensor& t = a[c].t[i];
      const Rows r = rows_of(t, oi.kind[i]);
      const int es = elem_size(t.dtype);
      Ext& e = ext[n];
      e.base = (int64_t)reinterpret_cast<uintptr_t>(t.data);
      e.nr = r.n;
      e.w = r.width * es;
      e.rs = r.stride * es;
      if (e.nr <= 0 || e.w <= 0) continue;  // no bytes: overlaps nothing
      e.end = e.base + (e.nr - 1) * e.rs + e.w;
      e.call = c;
      e.slot = i;
      e.out = oi.out[i];
      lo = e.base < lo ? e.base : lo;
      hi = e.base > hi ? e.base : hi;
      ++n;
    }
  }
  // Sort by start. One 64-bit key per extent -- the start relative to the lowest one,
  // shifted past an 11-bit extent index. With few ascending runs (see above) a natural
  // merge sort merges them pairwise in a few linear passes (on the Grace host: 0.3 us for
  // sorted input, 3.0 us for 20 interleaved runs, against 2.9 and 3.6 us for std::sort);
  // otherwise std::sort (random layouts: 3.6 us against 6.9). Spans beyond 2^53 bytes fall
  // back to sorting indices by start.
  if (n > 0 && (uint64_t)(hi - lo) < (1ull << 53)) {
    uint64_t* src = keys;
    uint64_t* dst = keys2;
    size_t runs = 1;
    for (size_t i = 0; i < n; ++i) {
      src[i] = ((uint64_t)(ext[i].base - lo) << 11) | (uint64_t)i;
      runs += i > 0 && src[i] < src[i - 1];
    }
    if (runs > 24) {  // little run structure to use: an ordinary sort
      std::sort(src, src + n);
      runs = 1;
    }
    while (runs > 1) {  // one pass merges each pair of consecutive ascending runs of src into dst
      size_t merged = 0, i = 0;
      while (i < n) {
        size_t j = i + 1;
        while (j < n && src[j - 1] < src[j]) ++j;  // first run [i, j)
        size_t k = j;
        if (j < n) {
          k = j + 1;
          while (k < n && src[k - 1] < src[k]) ++k;  // second run [j, k)
        }
        std::merge(src + i, src + j, src + j, src + k, dst + i);
        ++merged;
        i = k;
      }
      std::swap(src, dst);
      if (merged == 1) break;  // the whole array was at most two runs: now sorted
    }
    for (size_t i = 0; i < n; ++i) order[i] = (uint32_t)(src[i] & 2047u);
  } else {
    for (size_t i = 0; i < n; ++i) order[i] = (uint32_t)i;
    std::sort(order, order + n, [&](uint32_t x, uint32_t y) { return ext[x].base < ext[y].base; });
  }
  for (size_t x = 0; x < n; ++x) {
    const Ext& p = ext[order[x]];
    for (size_t y = x + 1; y < n && ext[order[y]].base < p.end; ++y) {
      const Ext& q = ext[order[y]];
      if (!p.out && !q.out) continue;  // inputs may share bytes
      if (q.call == p.call && !check_own) continue;
      if (!rows_overlap(p.base, p.nr, p.w, p.rs, q.base, q.nr, q.w, q.rs)) continue;
      if (q.call != p.call) return false;  // dependent calls
      const OpInfo& oi = g_ops[a[p.call].op];
      const trident_tensor* t = a[p.call].t;
      if (oi.group[p.slot] != 0 && oi.group[p.slot] == oi.group[q.slot] && same_desc(t[p.slot], t[q.slot]))
        continue;  // an in-place pair
      return false;  // the call's own precondition fails (reported by the call-by-call path)
    }
  }
  return true;
}

// Algorithm 1 over the current table snapshot. Returns OK with *sel, MISS, or an error.
int32_t dispatch(const trident_scm* scm, const trident_args* a, const OpInfo** oi_out, Sig* s,
                 int32_t* sel, bool check_alias) {
  const OpInfo* oi = nullptr;
  int32_t st = analyze(a, &oi, s);
  if (st != TRIDENT_OK) return st;
  *oi_out = oi;
  const int32_t n = scm->count.load(std::memory_order_acquire);
  for (int32_t i = 0; i < n; ++i) {
    const Version& v = scm->versions[i];
    if (v.d.op != a->op) continue;
    if (!guard_holds(v, *s, a)) continue;
    if (check_alias) {
      st = check_overlap(a, *oi);
      if (st != TRIDENT_OK) return st;
    }
    *sel = i;
    return TRIDENT_OK;
  }
  *sel = -1;
  return TRIDENT_MISS;
}

inline uint64_t now_ns() {
  return (uint64_t)std::chrono::duration_cast<std::chrono::nanoseconds>(
             std::chrono::steady_clock::now().time_since_epoch()).count();
}

// One host-time sample (ns since t0) into the SCM's ring (TRIDENT_OPT_TIMING).
void record_host_time(trident_scm* scm, uint64_t t0) {
  const uint64_t k = scm->ring_n.fetch_add(1, std::memory_order_relaxed);
  const uint64_t dt = now_ns() - t0;
  scm->ring[k % (uint64_t)scm->ring_cap] = dt > 0xffffffffull ? 0xffffffffu : (uint32_t)dt;
}

int32_t count_error(trident_scm* scm, int32_t st) {
  if (st == TRIDENT_ERR_INVALID) scm->err_invalid.fetch_add(1, std::memory_order_relaxed);
  else if (st == TRIDENT_ERR_CUDA) scm->err_cuda.fetch_add(1, std::memory_order_relaxed);
  return st;
}

// Runs `fn` with the SCM's device current on this thread, restoring the previous one.
template <class F>
int32_t on_device(trident_scm* scm, F fn) {
  int prev = -1;
  if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
  if (prev != scm->device && cudaSetDevice(scm->device) != cudaSuccess)
    return fail(TRIDENT_ERR_CUDA, "cudaSetDevice(%d) failed", scm->device);
  const int32_t st = fn();
  if (prev >= 0 && prev != scm->device) cudaSetDevice(prev);
  return st;
}

// Frequency table of RoPE base theta: f_i = theta^(-2i/D) in fp64, stored as the fp32
// pair (hi, lo) with hi = fp32(f_i) and lo = fp32(f_i - hi), so the kernel can form the
// angle pos * f_i to about 2^-48 relative before reducing it.
int32_t get_rope_table(trident_scm* scm, double theta, int32_t D, const float2** out) {
  for (const RopeTable& rt : scm->tables)
    if (rt.theta == theta && rt.D == D) { *out = rt.dev; return TRIDENT_OK; }
  const int64_t half = D / 2;
  std::vector<float2> host((size_t)half);
  for (int64_t i = 0; i < half; ++i) {
    const double f = std::pow(theta, -2.0 * (double)i / (double)D);
    const float hi = (float)f;
    host[(size_t)i] = make_float2(hi, (float)(f - (double)hi));
  }
  float2* dev = nullptr;
  if (cudaMalloc(&dev, host.size() * sizeof(float2)) != cudaSuccess)
    return fail(TRIDENT_ERR_CUDA, "cudaMalloc of the RoPE frequency table failed");
  // The copy must have landed before this registration returns: kernels read the table
  // before their programmatic-launch wait, on any stream. A copy from pageable memory may
  // return while its DMA is still in flight on the legacy default stream, so that stream
  // (and only it: other streams' work does not hold the registration up) is synchronised.
  if (cudaMemcpy(dev, host.data(), host.size() * sizeof(float2), cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaStreamSynchronize(cudaStreamLegacy) != cudaSuccess) {
    cudaFree(dev);
    return fail(TRIDENT_ERR_CUDA, "upload of the RoPE frequency table failed");
  }
  scm->tables.push_back({theta, D, dev});
  *out = dev;
  return TRIDENT_OK;
}

int32_t validate_desc(const trident_scm* scm, const trident_spec_desc* d, int32_t* nfixed) {
  if (!d) return fail(TRIDENT_ERR_INVALID, "descriptor is NULL");
  if (d->op < 1 || d->op > kMaxOp) return fail(TRIDENT_ERR_INVALID, "unknown op %d", d->op);
  const OpInfo& oi = g_ops[d->op];
  const bool chain = d->op == TRIDENT_OP_LAYER_CHAIN || d->op == TRIDENT_OP_LAYER_CHAIN_QKNORM;
  if (d->dtype != TRIDENT_BF16 && d->dtype != TRIDENT_FP16 && d->dtype != TRIDENT_FP32)
    return fail(TRIDENT_ERR_INVALID, "activation dtype %d", d->dtype);
  if (d->dtype == TRIDENT_FP32 && (oi.rope))
    return fail(TRIDENT_ERR_INVALID, "RoPE ops and chains take bf16 or fp16");
  if (oi.flattening ? (d->rank != 2 && d->rank != 3) : (d->rank != (chain ? 2 : 3)))
    return fail(TRIDENT_ERR_INVALID, "rank %d is not valid for op %d", d->rank, d->op);
  if (d->layout < TRIDENT_LAYOUT_CONTIG || d->layout > TRIDENT_LAYOUT_ANY)
    return fail(TRIDENT_ERR_INVALID, "layout %d", d->layout);
  for (int i = 0; i < oi.nfixed; ++i)
    if (d->fixed[i] < 1) return fail(TRIDENT_ERR_INVALID, "fixed[%d] must be >= 1", i);
  for (int i = oi.nfixed; i < TRIDENT_MAX_FIXED; ++i)
    if (d->fixed[i] != 0) return fail(TRIDENT_ERR_INVALID, "fixed[%d] must be 0 for op %d", i, d->op);
  if (d->tok_lo < 1 || d->tok_hi < d->tok_lo) return fail(TRIDENT_ERR_INVALID, "token bucket");
  const int es = elem_size(d->dtype);
  if (d->align_bytes != 16 && d->align_bytes != es)
    return fail(TRIDENT_ERR_INVALID, "align_bytes must be 16 or the element size");
  if (!scm->dry && d->device != scm->device)
    return fail(TRIDENT_ERR_INVALID, "version device %d differs from the SCM's %d", d->device, scm->device);
  if (d->device < 0) return fail(TRIDENT_ERR_INVALID, "device");
  if (d->variant < TRIDENT_VARIANT_AUTO || d->variant > TRIDENT_VARIANT_VECTOR)
    return fail(TRIDENT_ERR_INVALID, "variant %d", d->variant);
  if (d->variant == TRIDENT_VARIANT_VECTOR && d->align_bytes != 16)
    return fail(TRIDENT_ERR_INVALID, "the vector variant needs align_bytes 16");
  if (oi.rope && !(d->rope_theta > 0.0 && std::isfinite(d->rope_theta)))
    return fail(TRIDENT_ERR_INVALID, "rope_theta must be positive");
  if (!oi.rope && d->rope_theta != 0.0) return fail(TRIDENT_ERR_INVALID, "rope_theta must be 0");
  if (d->reserved != 0) return fail(TRIDENT_ERR_INVALID, "reserved must be 0");
  if (oi.rope) {
    const int64_t D = chain ? d->fixed[3] : d->fixed[2];
    if (D % 2 != 0 || D > 1024) return fail(TRIDENT_ERR_INVALID, "head size D must be even and <= 1024");
  }
  *nfixed = oi.nfixed;
  return TRIDENT_OK;
}

// Chooses the kernel of a version (AUTO -> VECTOR when the version guarantees 16-byte
// alignment and the sizes have a vector kernel, else GENERIC).
int32_t resolve_kernel(const trident_spec_desc& d, KernelEntry* ke) {
  const char* why = "";
  const bool chain = d.op == TRIDENT_OP_LAYER_CHAIN || d.op == TRIDENT_OP_LAYER_CHAIN_QKNORM;
  auto try_variant = [&](int32_t var) -> bool {
    switch (d.op) {
      case TRIDENT_OP_ADD_RMSNORM: return addnorm_kernel(d.dtype, var, d.fixed[0], ke, &why);
      case TRIDENT_OP_RMSNORM: return rmsnorm_kernel(d.dtype, var, d.fixed[0], ke, &why);
      case TRIDENT_OP_SILU:
      case TRIDENT_OP_ADD:
      case TRIDENT_OP_NEG:
      case TRIDENT_OP_MASKED_FILL: return pointwise_kernel(d.op, d.dtype, var, d.fixed[0], ke, &why);
      case TRIDENT_OP_SWIGLU: return swiglu_kernel(d.dtype, var, d.fixed[0], ke, &why);
      case TRIDENT_OP_ROPE_KV:
      case TRIDENT_OP_QKNORM_ROPE_KV:
        return rope_kernel(d.dtype, var, (int32_t)d.fixed[2], d.op == TRIDENT_OP_QKNORM_ROPE_KV, ke, &why);
      default:
        if (var == TRIDENT_VARIANT_GENERIC) { why = "the layer chain has no generic variant"; return false; }
        return chain_kernel(d.dtype, d.fixed[0], (int32_t)d.fixed[3], d.op == TRIDENT_OP_LAYER_CHAIN_QKNORM, ke, &why);
    }
  };
  if (d.variant == TRIDENT_VARIANT_AUTO) {
    if (d.align_bytes == 16 && try_variant(TRIDENT_VARIANT_VECTOR)) return TRIDENT_OK;
    if (!chain && try_variant(TRIDENT_VARIANT_GENERIC)) return TRIDENT_OK;
    return fail(TRIDENT_ERR_INVALID, "no kernel for this version: %s", why);
  }
  if (!try_variant(d.variant)) return fail(TRIDENT_ERR_INVALID, "no kernel for this version: %s", why);
  return TRIDENT_OK;
}

}  // namespace

// ====================================================================== internal
int32_t trident::prepare_rope_args(const void* args_ptr, RopeParams* p, int32_t* dtype, bool* qknorm) {
  const trident_args* a = static_cast<const trident_args*>(args_ptr);
  const OpInfo* oi = nullptr;
  Sig s;
  int32_t st = analyze(a, &oi, &s);
  if (st != TRIDENT_OK) return st;
  if (a->op != TRIDENT_OP_ROPE_KV && a->op != TRIDENT_OP_QKNORM_ROPE_KV)
    return fail(TRIDENT_ERR_INVALID, "op %d is not a RoPE op", a->op);
  if (s.device == kMixed || s.device < 0) return fail(TRIDENT_ERR_INVALID, "tensors must share one CUDA device");
  if (s.act_dtype != TRIDENT_BF16 && s.act_dtype != TRIDENT_FP16)
    return fail(TRIDENT_ERR_INVALID, "activations must all be bf16 or all fp16");
  if (!s.aux_dtype_ok) return fail(TRIDENT_ERR_INVALID, "gamma must be fp32 and pos int32");
  if (!s.ranks_ok || !s.shapes_ok) return fail(TRIDENT_ERR_INVALID, "inconsistent ranks or shapes");
  if (s.T < 1) return fail(TRIDENT_ERR_INVALID, "no tokens");
  if (a->t[0].shape[1] < 1 || a->t[1].shape[1] < 1 || a->t[0].shape[2] < 1)
    return fail(TRIDENT_ERR_INVALID, "no heads: q and k need at least one head of at least one element");
  if (s.layout < 0 || !s.aux_layout_ok) return fail(TRIDENT_ERR_INVALID, "unsupported layout");
  if (!s.aligned16) return fail(TRIDENT_ERR_INVALID, "tensors must be 16-byte aligned");
  if (!(a->rope_theta > 0.0 && std::isfinite(a->rope_theta)))
    return fail(TRIDENT_ERR_INVALID, "rope_theta must be positive");
  st = check_overlap(a, *oi);
  if (st != TRIDENT_OK) return st;
  Version v;
  std::memset(&v, 0, sizeof(v));
  pack_rope(a, 0, a->op == TRIDENT_OP_QKNORM_ROPE_KV ? 6 : -1, v, nullptr, p);
  *dtype = s.act_dtype;
  *qknorm = a->op == TRIDENT_OP_QKNORM_ROPE_KV;
  return TRIDENT_OK;
}

int32_t trident::internal_fail(int32_t status, const char* msg) { return fail(status, "%s", msg); }

// ====================================================================== C ABI
TRIDENT_API int32_t trident_abi_version(void) { return TRIDENT_ABI_VERSION; }

TRIDENT_API const char* trident_scm_last_error(void) { return tl_err; }

TRIDENT_API const char* trident_status_name(int32_t s) {
  switch (s) {
    case TRIDENT_OK: return "OK";
    case TRIDENT_MISS_HANDLED: return "MISS_HANDLED";
    case TRIDENT_MISS: return "MISS";
    case TRIDENT_ERR_INVALID: return "ERR_INVALID";
    case TRIDENT_ERR_CUDA: return "ERR_CUDA";
    case TRIDENT_ERR_HOOK: return "ERR_HOOK";
    case TRIDENT_ERR_CAPACITY: return "ERR_CAPACITY";
    case TRIDENT_ERR_STATE: return "ERR_STATE";
    default: return "UNKNOWN";
  }
}

TRIDENT_API int32_t trident_scm_create(const trident_scm_options* opt, trident_compile_hook hook,
                                       void* user, trident_scm_t** out) {
  if (!out) return fail(TRIDENT_ERR_INVALID, "out is NULL");
  *out = nullptr;
  trident_scm_options o{};
  if (opt) o = *opt;
  if (o.max_specs == 0) o.max_specs = 256;
  if (o.max_specs < 1 || o.max_specs > 4096) return fail(TRIDENT_ERR_INVALID, "max_specs must be 1..4096");
  if (o.timing_ring == 0) o.timing_ring = 65536;
  if (o.timing_ring < 1 || o.timing_ring > (1 << 24)) return fail(TRIDENT_ERR_INVALID, "timing_ring");
  if (o.flags & ~(TRIDENT_OPT_DRY_RUN | TRIDENT_OPT_NO_ALIAS_CHECK | TRIDENT_OPT_PDL | TRIDENT_OPT_TIMING |
                  TRIDENT_OPT_FAIL_LAUNCHES | TRIDENT_OPT_NO_STEP_REPLAY | TRIDENT_OPT_TEST_WAIT_TIMEOUT))
    return fail(TRIDENT_ERR_INVALID, "unknown option flags");
  if (o.device < 0) return fail(TRIDENT_ERR_INVALID, "device");
  trident_scm* s = new (std::nothrow) trident_scm();
  if (!s) return fail(TRIDENT_ERR_INVALID, "out of host memory");
  s->opt = o;
  s->hook = hook;
  s->user = user;
  s->dry = (o.flags & TRIDENT_OPT_DRY_RUN) != 0;
  s->device = o.device;
  s->versions = static_cast<Version*>(std::calloc((size_t)o.max_specs, sizeof(Version)));
  s->hits_per = new (std::nothrow) std::atomic<uint64_t>[(size_t)o.max_specs];
  if (o.flags & TRIDENT_OPT_TIMING) {
    s->ring_cap = o.timing_ring;
    s->ring = static_cast<uint32_t*>(std::calloc((size_t)o.timing_ring, sizeof(uint32_t)));
  }
  if (!s->versions || !s->hits_per || ((o.flags & TRIDENT_OPT_TIMING) && !s->ring)) {
    trident_scm_destroy(s);
    return fail(TRIDENT_ERR_INVALID, "out of host memory");
  }
  for (int i = 0; i < o.max_specs; ++i) s->hits_per[i].store(0);
  if (!s->dry) {
    if (!driver()) {
      trident_scm_destroy(s);
      return fail(TRIDENT_ERR_CUDA, "CUDA driver entry points unavailable");
    }
    const int32_t st = on_device(s, [&]() -> int32_t {
      if (cudaFree(nullptr) != cudaSuccess) return fail(TRIDENT_ERR_CUDA, "CUDA init failed");
      if (g_drv.ctx_get(&s->ctx) != CUDA_SUCCESS || !s->ctx)
        return fail(TRIDENT_ERR_CUDA, "no current CUDA context");
      if (cudaDeviceGetAttribute(&s->sm_count, cudaDevAttrMultiProcessorCount, s->device) != cudaSuccess)
        return fail(TRIDENT_ERR_CUDA, "cannot read the SM count");
      if (cudaMalloc(&s->d_err, sizeof(uint32_t)) != cudaSuccess)
        return fail(TRIDENT_ERR_CUDA, "cudaMalloc of the status word failed");
      if (cudaMemset(s->d_err, 0, sizeof(uint32_t)) != cudaSuccess)
        return fail(TRIDENT_ERR_CUDA, "cudaMemset failed");
      return TRIDENT_OK;
    });
    if (st != TRIDENT_OK) {
      trident_scm_destroy(s);
      return st;
    }
  }
  *out = s;
  return TRIDENT_OK;
}

namespace {

// Resolves the version's kernels and tables and publishes it (copy, then release the count).
int32_t append_version(trident_scm_t* scm, const trident_spec_desc* desc, int32_t nfixed, Version* vp,
                       int32_t* out_index) {
  Version& v = *vp;
  int32_t st = TRIDENT_OK;
  v.d = *desc;
  v.nfixed = nfixed;
  v.rope = g_ops[desc->op].rope;
  st = resolve_kernel(v.d, &v.ke);
  if (st != TRIDENT_OK) return st;
  std::lock_guard<std::mutex> lk(scm->reg_mu);
  const int32_t n = scm->count.load(std::memory_order_relaxed);
  if (n >= scm->opt.max_specs) return fail(TRIDENT_ERR_CAPACITY, "version table full (%d)", n);
  if (!scm->dry) {
    st = on_device(scm, [&]() -> int32_t {
      cudaFunction_t f = nullptr;
      if (cudaGetFuncBySymbol(&f, v.ke.fn) != cudaSuccess || !f)
        return fail(TRIDENT_ERR_CUDA, "cannot resolve the kernel entry");
      v.fn = reinterpret_cast<CUfunction>(f);
      if (v.ke.fn_large) {
        cudaFunction_t h = nullptr;
        if (cudaGetFuncBySymbol(&h, v.ke.fn_large) != cudaSuccess || !h)
          return fail(TRIDENT_ERR_CUDA, "cannot resolve the large-call kernel entry");
        v.fn_large = reinterpret_cast<CUfunction>(h);
        if (v.ke.kind == KK_ROPE_HALFWARP) {
          // the bulk-copy RoPE kernel stages ke.rows tokens' head-rows in dynamic shared memory:
          // allow up to what the device gives a block (one setting for every version), or
          // leave such calls to the vector kernel when a version's rows do not fit
          const int64_t need = (int64_t)v.ke.rows * (v.d.fixed[0] + 2 * v.d.fixed[1]) * v.d.fixed[2] * 2;
          int dev = 0, optin = 0;
          cudaFuncAttributes fa;
          if (cudaGetDevice(&dev) != cudaSuccess ||
              cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
              cudaFuncGetAttributes(&fa, v.ke.fn_large) != cudaSuccess)
            return fail(TRIDENT_ERR_CUDA, "cannot read the shared-memory limits");
          const int64_t room = (int64_t)optin - (int64_t)fa.sharedSizeBytes;
          if (need > room) {
            v.fn_large = nullptr;
          } else if (cudaFuncSetAttribute(v.ke.fn_large, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)room) !=
                         cudaSuccess ||
                     cudaFuncSetAttribute(v.ke.fn_large, cudaFuncAttributePreferredSharedMemoryCarveout,
                                          (int)cudaSharedmemCarveoutMaxShared) != cudaSuccess) {
            return fail(TRIDENT_ERR_CUDA, "cannot set the RoPE kernel's shared-memory size");
          }
        }
      }
      if (v.ke.fn_inplace) {
        cudaFunction_t g = nullptr;
        if (cudaGetFuncBySymbol(&g, v.ke.fn_inplace) != cudaSuccess || !g)
          return fail(TRIDENT_ERR_CUDA, "cannot resolve the in-place kernel entry");
        v.fn_inplace = reinterpret_cast<CUfunction>(g);
        if (v.ke.fn_late) {
          cudaFunction_t l = nullptr;
          if (cudaGetFuncBySymbol(&l, v.ke.fn_late) != cudaSuccess || !l)
            return fail(TRIDENT_ERR_CUDA, "cannot resolve the late-trigger kernel entry");
          v.fn_late = reinterpret_cast<CUfunction>(l);
        }
        if (v.ke.fn_wide) {
          cudaFunction_t w = nullptr;
          if (cudaGetFuncBySymbol(&w, v.ke.fn_wide) != cudaSuccess || !w)
            return fail(TRIDENT_ERR_CUDA, "cannot resolve the wide-tile kernel entry");
          v.fn_wide = reinterpret_cast<CUfunction>(w);
        }
        cudaFunction_t h = nullptr, k = nullptr;
        if (cudaGetFuncBySymbol(&h, v.ke.fn_step) != cudaSuccess || !h ||
            cudaGetFuncBySymbol(&k, v.ke.fn_step_inplace) != cudaSuccess || !k)
          return fail(TRIDENT_ERR_CUDA, "cannot resolve the multi-call kernel entries");
        v.step_fn = reinterpret_cast<CUfunction>(h);
        v.step_fn_inplace = reinterpret_cast<CUfunction>(k);
        if (v.ke.fn_step_role) {
          cudaFunction_t q = nullptr;
          if (cudaGetFuncBySymbol(&q, v.ke.fn_step_role) != cudaSuccess || !q)
            return fail(TRIDENT_ERR_CUDA, "cannot resolve the role-major multi-call kernel entry");
          v.step_fn_role = reinterpret_cast<CUfunction>(q);
        }
        int per_sm = 0, step_per_sm = 0, sms = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, v.ke.fn, kThreads, 0) != cudaSuccess ||
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&step_per_sm, v.ke.fn_step, kThreads, 0) != cudaSuccess ||
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, scm->device) != cudaSuccess)
          return fail(TRIDENT_ERR_CUDA, "occupancy query failed");
        v.wave_blocks = per_sm * sms;
        v.step_wave_blocks = step_per_sm * sms;
      }
      if (v.rope) {
        const bool chain = desc->op == TRIDENT_OP_LAYER_CHAIN || desc->op == TRIDENT_OP_LAYER_CHAIN_QKNORM;
        const int32_t D = (int32_t)(chain ? desc->fixed[3] : desc->fixed[2]);
        return get_rope_table(scm, desc->rope_theta, D, &v.inv_freq);
      }
      return TRIDENT_OK;
    });
    if (st != TRIDENT_OK) return st;
  }
  scm->versions[n] = v;
  scm->hits_per[n].store(0, std::memory_order_relaxed);
  scm->count.store(n + 1, std::memory_order_release);
  if (tl_hook_depth > 0) scm->hook_registered.fetch_add(1, std::memory_order_relaxed);
  if (out_index) *out_index = n;
  return TRIDENT_OK;
}

// Appends a version (with its recipe, or none); shared by register_spec and
// register_tree_spec. On failure the recipe is freed.
int32_t register_version(trident_scm_t* scm, const trident_spec_desc* desc, const trident_recipe* recipe,
                         int32_t* out_index) {
  if (!scm) return fail(TRIDENT_ERR_INVALID, "scm is NULL");
  int32_t nfixed = 0;
  int32_t st = validate_desc(scm, desc, &nfixed);
  if (st != TRIDENT_OK) return st;
  Version v;
  std::memset(&v, 0, sizeof(v));
  if (recipe) {
    Recipe* r = new (std::nothrow) Recipe();
    if (!r) return fail(TRIDENT_ERR_INVALID, "out of host memory");
    st = make_recipe(recipe, desc->op, g_ops[desc->op].nslots, r);
    if (st != TRIDENT_OK) {
      delete r;
      return st;
    }
    v.recipe = r;
  }
  st = append_version(scm, desc, nfixed, &v, out_index);
  if (st != TRIDENT_OK && v.recipe) {
    free_recipe(v.recipe);
    delete v.recipe;
  }
  return st;
}

}  // namespace

TRIDENT_API int32_t trident_scm_register_spec(trident_scm_t* scm, const trident_spec_desc* desc,
                                              int32_t* out_index) {
  return register_version(scm, desc, nullptr, out_index);
}

TRIDENT_API int32_t trident_scm_register_tree_spec(trident_scm_t* scm, const trident_spec_desc* desc,
                                                   const trident_recipe* recipe, int32_t* out_index) {
  if (!recipe) return fail(TRIDENT_ERR_INVALID, "recipe is NULL");
  return register_version(scm, desc, recipe, out_index);
}

TRIDENT_API int32_t trident_scm_select(const trident_scm_t* scm, const trident_args* args,
                                       int32_t* out_selected) {
  if (out_selected) *out_selected = -1;
  if (!scm) return fail(TRIDENT_ERR_INVALID, "scm is NULL");
  const OpInfo* oi = nullptr;
  Sig s;
  int32_t sel = -1;
  const int32_t st = dispatch(scm, args, &oi, &s, &sel, !(scm->opt.flags & TRIDENT_OPT_NO_ALIAS_CHECK));
  if (out_selected) *out_selected = sel;
  return st;
}

namespace {

// A guard hit on version `sel`: launch (unless dry-run), count, record host time.
int32_t run_hit(trident_scm* scm, int32_t sel, const trident_args* args, const Sig& s, void* stream,
                uint64_t t0, int32_t* out_selected) {
  const Version& v = scm->versions[sel];
  if (out_selected) *out_selected = sel;
  if (scm->opt.flags & TRIDENT_OPT_FAIL_LAUNCHES)  // injected failure of P_i
    return count_error(scm, fail(TRIDENT_ERR_CUDA, "launch failure injected (TRIDENT_OPT_FAIL_LAUNCHES)"));
  if (!scm->dry) {
    const int32_t st = do_launch(scm, v, args, s, stream);
    if (st != TRIDENT_OK) return count_error(scm, st);  // Algorithm 1: raise, no next version
  }
  scm->hits.fetch_add(1, std::memory_order_relaxed);
  scm->hits_per[sel].fetch_add(1, std::memory_order_relaxed);
  scm->guard_evals.fetch_add((uint64_t)sel + 1, std::memory_order_relaxed);
  if (scm->ring) record_host_time(scm, t0);
  return TRIDENT_OK;
}

// Every guard failed: a specialisation miss (§3.5). `call_hook` runs the hook (if the
// call is not already inside one) and returns its status.
template <class Hook>
int32_t run_miss(trident_scm* scm, bool have_hook, Hook call_hook, int32_t* out_selected) {
  scm->misses.fetch_add(1, std::memory_order_relaxed);
  scm->guard_evals.fetch_add((uint64_t)scm->count.load(std::memory_order_relaxed),
                             std::memory_order_relaxed);
  if (!have_hook || tl_hook_depth > 0) return TRIDENT_MISS;
  scm->hook_calls.fetch_add(1, std::memory_order_relaxed);
  int32_t reg = -1;
  ++tl_hook_depth;
  const int32_t hr = call_hook(&reg);
  --tl_hook_depth;
  if (hr != 0) {
    scm->hook_failures.fetch_add(1, std::memory_order_relaxed);
    return fail(TRIDENT_ERR_HOOK, "compile hook returned %d", hr);
  }
  if (out_selected) *out_selected = reg;
  return TRIDENT_MISS_HANDLED;
}

}  // namespace

TRIDENT_API int32_t trident_scm_invoke(trident_scm_t* scm, const trident_args* args, void* stream,
                                       int32_t* out_selected) {
  TRIDENT_RANGE("trident_scm_invoke");
  if (out_selected) *out_selected = -1;
  if (!scm) return fail(TRIDENT_ERR_INVALID, "scm is NULL");
  const uint64_t t0 = scm->ring ? now_ns() : 0;
  scm->invokes.fetch_add(1, std::memory_order_relaxed);
  const OpInfo* oi = nullptr;
  Sig s;
  int32_t sel = -1;
  const int32_t st = dispatch(scm, args, &oi, &s, &sel, !(scm->opt.flags & TRIDENT_OPT_NO_ALIAS_CHECK));
  if (st == TRIDENT_OK) return run_hit(scm, sel, args, s, stream, t0, out_selected);
  if (st != TRIDENT_MISS) return count_error(scm, st);
  return run_miss(scm, scm->hook != nullptr, [&](int32_t* reg) {
    return scm->hook(scm->user, scm, args, stream, reg);
  }, out_selected);
}

TRIDENT_API int32_t trident_scm_invoke_tree(trident_scm_t* scm, const trident_node* nodes, int32_t nargs,
                                            int32_t nnodes, void* stream, int32_t* out_selected) {
  TRIDENT_RANGE("trident_scm_invoke_tree");
  if (out_selected) *out_selected = -1;
  if (!scm) return fail(TRIDENT_ERR_INVALID, "scm is NULL");
  const uint64_t t0 = scm->ring ? now_ns() : 0;
  scm->invokes.fetch_add(1, std::memory_order_relaxed);
  int32_t st = validate_tree(nodes, nargs, nnodes);
  if (st != TRIDENT_OK) return count_error(scm, st);
  const bool check_alias = !(scm->opt.flags & TRIDENT_OPT_NO_ALIAS_CHECK);
  const int32_t n = scm->count.load(std::memory_order_acquire);
  trident_args a;
  for (int32_t i = 0; i < n; ++i) {
    const Version& v = scm->versions[i];
    if (!v.recipe) continue;
    if (!bind_tree(*v.recipe, nodes, nargs, &a)) continue;  // structure or a guarded constant differs
    const OpInfo* oi = nullptr;
    Sig s;
    st = analyze(&a, &oi, &s);
    if (st != TRIDENT_OK) return count_error(scm, st);  // the bound arguments are malformed
    if (!guard_holds(v, s, &a)) continue;
    if (check_alias) {
      st = check_overlap(&a, *oi);
      if (st != TRIDENT_OK) return count_error(scm, st);
    }
    return run_hit(scm, i, &a, s, stream, t0, out_selected);
  }
  return run_miss(scm, scm->tree_hook != nullptr, [&](int32_t* reg) {
    return scm->tree_hook(scm->tree_user, scm, nodes, nargs, nnodes, stream, reg);
  }, out_selected);
}

TRIDENT_API int32_t trident_scm_set_tree_hook(trident_scm_t* scm, trident_tree_hook hook, void* user) {
  if (!scm) return fail(TRIDENT_ERR_INVALID, "scm is NULL");
  scm->tree_hook = hook;
  scm->tree_user = user;
  return TRIDENT_OK;
}

TRIDENT_API int32_t trident_scm_invoke_seq(trident_scm_t* scm, const trident_args* args, int32_t n,
                                           void* stream, int32_t* out_selected) {
  TRIDENT_RANGE("trident_scm_invoke_seq");
  if (!scm || (!args && n > 0) || n < 0) return fail(TRIDENT_ERR_INVALID, "bad sequence");
  int32_t result = TRIDENT_OK;
  for (int32_t i = 0; i < n; ++i) {
    int32_t sel = -1;
    const int32_t st = trident_scm_invoke(scm, args + i, stream, &sel);
    if (out_selected) out_selected[i] = sel;
    if (st < 0 || st == TRIDENT_MISS) {
      if (out_selected)
        for (int32_t j = i + 1; j < n; ++j) out_selected[j] = TRIDENT_NOT_RUN;
      return st;
    }
    if (st == TRIDENT_MISS_HANDLED) result = TRIDENT_MISS_HANDLED;
  }
  return result;
}

namespace {

constexpr int32_t kNotFused = 100;  // step_chunk: run the chunk call by call
static_assert(kStepMax == TRIDENT_STEP_MAX, "step chunk size");
static_assert(kStepMax * TRIDENT_MAX_TENSORS <= 2048, "extent index fits the sort key");
static_assert(sizeof(ChainStepParams) <= 32764, "kernel parameter limit");

// Fingerprint of a chunk for the replay cache: a few words from its first, middle and last
// calls (collisions only cost a failed byte comparison or one unneeded store).
uint64_t step_fingerprint(const trident_args* a, int32_t m) {
  uint64_t h = 0x9e3779b97f4a7c15ull ^ (uint64_t)m;
  auto mix = [&h](uint64_t v) {
    h ^= v + 0x9e3779b97f4a7c15ull + (h << 6) + (h >> 2);
    h *= 0xff51afd7ed558ccdull;
  };
  const int32_t pick[3] = {0, m / 2, m - 1};
  for (int32_t k : pick) {
    const trident_args& c = a[k];
    mix((uint64_t)(uint32_t)c.op | ((uint64_t)(uint32_t)c.ntensors << 32));
    mix((uint64_t)reinterpret_cast<uintptr_t>(c.t[0].data));
    mix((uint64_t)reinterpret_cast<uintptr_t>(c.t[1].data));
    mix((uint64_t)c.t[0].shape[0]);
  }
  return h | 1;  // never 0 (the empty-entry mark)
}

// Under memo_lock. Looks the chunk up; on a match relaunches it (or, in a dry run, only
// counts it) and returns its status. Otherwise returns kNotFused and sets *repeat when
// the fingerprint was seen before (the full path then stores the chunk).
int32_t replay_chunk(trident_scm* scm, const trident_args* a, int32_t m, uint64_t fp, void* stream,
                     int32_t* out_selected, bool* repeat) {
  StepMemo* e = nullptr;
  if (scm->memo)
    for (int k = 0; k < kMemoEntries && !e; ++k) {
      StepMemo& x = scm->memo[k];
      if (x.fp == fp && x.m == m && std::memcmp(x.args, a, (size_t)m * sizeof(trident_args)) == 0) e = &x;
    }
  if (!e) {
    for (int k = 0; k < kSeenRing; ++k)
      if (scm->seen[k] == fp) *repeat = true;
    if (!*repeat) scm->seen[scm->seen_next++ % kSeenRing] = fp;
    return kNotFused;
  }
  e->used = ++scm->memo_clock;
  scm->invokes.fetch_add((uint64_t)m, std::memory_order_relaxed);
  if (out_selected)
    for (int32_t i = 0; i < m; ++i) out_selected[i] = e->sel[i];
  if (scm->opt.flags & TRIDENT_OPT_FAIL_LAUNCHES)
    return count_error(scm, fail(TRIDENT_ERR_CUDA, "launch failure injected (TRIDENT_OPT_FAIL_LAUNCHES)"));
  if (!scm->dry) {
    CUlaunchConfig cfg;
    CUlaunchAttribute attr;
    base_config(scm, stream, &cfg, &attr);
    cfg.gridDimX = e->grid;
    void* kp[1] = {&e->P};
    const int32_t st = launch_on(scm, &cfg, e->fn, kp);
    if (st != TRIDENT_OK) return count_error(scm, st);
  }
  for (int32_t k = 0; k < e->ndist; ++k)
    scm->hits_per[e->dist_idx[k]].fetch_add((uint64_t)e->dist_cnt[k], std::memory_order_relaxed);
  scm->hits.fetch_add((uint64_t)m, std::memory_order_relaxed);
  scm->fused_launches.fetch_add(1, std::memory_order_relaxed);
  scm->fused_calls.fetch_add((uint64_t)m, std::memory_order_relaxed);
  scm->step_replays.fetch_add((uint64_t)m, std::memory_order_relaxed);
  return TRIDENT_OK;
}

// Under memo_lock: stores a fused chunk over the least recently used entry.
void store_chunk(trident_scm* scm, const trident_args* a, int32_t m, uint64_t fp, const int32_t* sel,
                 const ChainStepParams* P, unsigned grid, CUfunction fn) {
  if (!scm->memo) {
    scm->memo = static_cast<StepMemo*>(std::calloc(kMemoEntries, sizeof(StepMemo)));
    if (!scm->memo) return;  // no cache: every chunk takes the full path
  }
  StepMemo* e = &scm->memo[0];
  for (int k = 1; k < kMemoEntries; ++k)
    if (scm->memo[k].used < e->used) e = &scm->memo[k];
  e->fp = fp;
  e->used = ++scm->memo_clock;
  e->m = m;
  e->grid = grid;
  e->fn = fn;
  e->ndist = 0;
  for (int32_t i = 0; i < m; ++i) {
    e->sel[i] = sel[i];
    int32_t k = 0;
    while (k < e->ndist && e->dist_idx[k] != sel[i]) ++k;
    if (k == e->ndist) {
      e->dist_idx[k] = sel[i];
      e->dist_cnt[k] = 0;
      ++e->ndist;
    }
    ++e->dist_cnt[k];
  }
  std::memcpy(e->args, a, (size_t)m * sizeof(trident_args));
  if (P) std::memcpy(&e->P, P, sizeof(ChainStepParams));
}

// One chunk of trident_scm_invoke_step: select every call; if all hit layer-chain
// versions with one kernel and the calls are independent, pack them into one launch.
// A chunk stored in the replay cache is relaunched without re-running these steps.
int32_t step_chunk(trident_scm* scm, const trident_args* a, int32_t m, void* stream,
                   int32_t* out_selected) {
  if (m < 2) return kNotFused;
  const bool memo_on = !(scm->opt.flags & TRIDENT_OPT_NO_STEP_REPLAY);
  uint64_t fp = 0;
  bool repeat = false;
  if (memo_on) {
    fp = step_fingerprint(a, m);
    if (!scm->memo_lock.test_and_set(std::memory_order_acquire)) {
      const int32_t st = replay_chunk(scm, a, m, fp, stream, out_selected, &repeat);
      scm->memo_lock.clear(std::memory_order_release);
      if (st != kNotFused) return st;
    }
  }
  Sig sig[kStepMax];
  int32_t sel[kStepMax];
  const Version* v0 = nullptr;
  for (int32_t i = 0; i < m; ++i) {  // guards only: the byte rules follow for all calls at once
    const OpInfo* oi = nullptr;
    if (dispatch(scm, a + i, &oi, &sig[i], &sel[i], false) != TRIDENT_OK) return kNotFused;
    const Version& v = scm->versions[sel[i]];
    if (v.ke.kind != KK_CHAIN) return kNotFused;
    if (!v0) v0 = &v;
    else if (v.ke.fn != v0->ke.fn) return kNotFused;
  }
  if (!step_bytes_ok(a, m, !(scm->opt.flags & TRIDENT_OPT_NO_ALIAS_CHECK))) return kNotFused;
  scm->invokes.fetch_add((uint64_t)m, std::memory_order_relaxed);
  if (out_selected)
    for (int32_t i = 0; i < m; ++i) out_selected[i] = sel[i];
  if (scm->opt.flags & TRIDENT_OPT_FAIL_LAUNCHES)
    return count_error(scm, fail(TRIDENT_ERR_CUDA, "launch failure injected (TRIDENT_OPT_FAIL_LAUNCHES)"));
  thread_local ChainStepParams P;
  unsigned grid = 0;
  CUfunction fn = nullptr;
  if (!scm->dry) {
    bool inplace = false;
    int64_t two = 0, one = 0;  // blocks with two / one CTAs per token (one head-row per lane group)
    for (int32_t i = 0; i < m; ++i) {
      ChainParams& c = P.c[i];
      const int32_t st = pack_chain(scm, scm->versions[sel[i]], a + i, sig[i], kChainStepSwigluUnroll, &c);
      if (st != TRIDENT_OK) return count_error(scm, st);
      inplace = inplace || chain_inplace(a + i);
      two += 2 * sig[i].T + c.nB + c.nC;
      one += sig[i].T + c.nB + c.nC;
    }
    const int32_t split = (!inplace && two <= v0->step_wave_blocks) ? 2 : 1;
    const int32_t rope_k = split == 1 ? chain_rope_k(one, v0->step_wave_blocks) : 1;
    int64_t first = 0;
    for (int32_t i = 0; i < m; ++i) {
      int64_t blocks = 0;
      set_chain_split(&P.c[i], sig[i].T, split, rope_k, &blocks);
      P.first[i] = (int32_t)first;
      first += blocks;
      if (first > 0x7fffffff)
        return count_error(scm, fail(TRIDENT_ERR_INVALID, "step too large for one launch"));
    }
    P.first[m] = (int32_t)first;
    P.n = m;
    // One-CTA-per-token steps of one to two waves run role-major over the whole step (every
    // call's norm blocks, then every call's RoPE blocks, then every call's SwiGLU tiles), so
    // the longer blocks fill the first wave and the second is short tiles: 36 Qwen3-style
    // layers replayed, 6 / 8 tokens 9.15 / 10.83 -> 8.59 / 10.32 us; at 12 tokens (2.8 waves)
    // +0.9 %, at 32 and 128 tokens +9 % and +7 %, so not there.
    const bool role_major = split == 1 && v0->step_fn_role && first > v0->step_wave_blocks &&
                            first <= 2 * (int64_t)v0->step_wave_blocks;
    if (role_major) {
      int64_t at = 0;
      for (int r = 0; r < 3; ++r) {
        for (int32_t i = 0; i < m; ++i) {
          P.role_first[r][i] = (int32_t)at;
          at += r == 0 ? P.c[i].nA : (r == 1 ? P.c[i].nB : P.c[i].nC);
        }
        P.role_first[r][m] = (int32_t)at;
      }
    }
    // L2 prefetch before the PDL wait under the same rule as single calls (do_launch)
    const int32_t pf = chain_prefetch_mode((scm->opt.flags & TRIDENT_OPT_PDL) != 0,
                                           first <= scm->sm_count, split == 2);
    for (int32_t i = 0; i < m; ++i) P.c[i].prefetch = pf;
    CUlaunchConfig cfg;
    CUlaunchAttribute attr;
    base_config(scm, stream, &cfg, &attr);
    grid = (unsigned)first;
    fn = split == 2 ? v0->step_fn : (role_major ? v0->step_fn_role : v0->step_fn_inplace);
    cfg.gridDimX = grid;
    void* kp[1] = {&P};
    const int32_t st = launch_on(scm, &cfg, fn, kp);
    if (st != TRIDENT_OK) return count_error(scm, st);
  }
  uint64_t evals = 0;
  for (int32_t i = 0; i < m; ++i) {
    scm->hits_per[sel[i]].fetch_add(1, std::memory_order_relaxed);
    evals += (uint64_t)sel[i] + 1;
  }
  scm->hits.fetch_add((uint64_t)m, std::memory_order_relaxed);
  scm->guard_evals.fetch_add(evals, std::memory_order_relaxed);
  scm->fused_launches.fetch_add(1, std::memory_order_relaxed);
  scm->fused_calls.fetch_add((uint64_t)m, std::memory_order_relaxed);
  if (repeat && !scm->memo_lock.test_and_set(std::memory_order_acquire)) {
    store_chunk(scm, a, m, fp, sel, scm->dry ? nullptr : &P, grid, fn);
    scm->memo_lock.clear(std::memory_order_release);
  }
  return TRIDENT_OK;
}

}  // namespace

TRIDENT_API int32_t trident_scm_invoke_step(trident_scm_t* scm, const trident_args* args, int32_t n,
                                            void* stream, int32_t* out_selected) {
  TRIDENT_RANGE("trident_scm_invoke_step");
  if (!scm || (!args && n > 0) || n < 0) return fail(TRIDENT_ERR_INVALID, "bad sequence");
  int32_t result = TRIDENT_OK;
  for (int32_t c0 = 0; c0 < n; c0 += kStepMax) {
    const int32_t m = n - c0 < kStepMax ? n - c0 : kStepMax;
    int32_t* sel = out_selected ? out_selected + c0 : nullptr;
    int32_t st = step_chunk(scm, args + c0, m, stream, sel);
    if (st == kNotFused) st = trident_scm_invoke_seq(scm, args + c0, m, stream, sel);
    if (st < 0 || st == TRIDENT_MISS) {
      if (out_selected)
        for (int32_t j = c0 + m; j < n; ++j) out_selected[j] = TRIDENT_NOT_RUN;
      return st;
    }
    if (st == TRIDENT_MISS_HANDLED) result = TRIDENT_MISS_HANDLED;
  }
  return result;
}

TRIDENT_API int32_t trident_scm_stats(const trident_scm_t* scm, trident_scm_stats_t* out) {
  if (!scm || !out) return fail(TRIDENT_ERR_INVALID, "NULL argument");
  std::memset(out, 0, sizeof(*out));
  out->invokes = scm->invokes.load();
  out->hits = scm->hits.load();
  out->misses = scm->misses.load();
  out->hook_calls = scm->hook_calls.load();
  out->hook_failures = scm->hook_failures.load();
  out->hook_registered = scm->hook_registered.load();
  out->err_invalid = scm->err_invalid.load();
  out->err_cuda = scm->err_cuda.load();
  out->guard_evals = scm->guard_evals.load();
  out->num_specs = scm->count.load();
  out->fused_launches = scm->fused_launches.load();
  out->fused_calls = scm->fused_calls.load();
  out->step_replays = scm->step_replays.load();
  return TRIDENT_OK;
}

TRIDENT_API int32_t trident_scm_spec_hits(const trident_scm_t* scm, uint64_t* out, int32_t cap,
                                          int32_t* n) {
  if (!scm || (cap > 0 && !out) || cap < 0) return fail(TRIDENT_ERR_INVALID, "bad arguments");
  const int32_t cnt = scm->count.load(std::memory_order_acquire);
  const int32_t m = cnt < cap ? cnt : cap;
  for (int32_t i = 0; i < m; ++i) out[i] = scm->hits_per[i].load(std::memory_order_relaxed);
  if (n) *n = cnt;
  return TRIDENT_OK;
}

TRIDENT_API int32_t trident_scm_host_times(const trident_scm_t* scm, uint32_t* out, int32_t cap,
                                           int32_t* n) {
  if (!scm || (cap > 0 && !out) || cap < 0) return fail(TRIDENT_ERR_INVALID, "bad arguments");
  if (!scm->ring) return fail(TRIDENT_ERR_STATE, "TRIDENT_OPT_TIMING is off");
  const uint64_t total = scm->ring_n.load(std::memory_order_relaxed);
  const uint64_t have = total < (uint64_t)scm->ring_cap ? total : (uint64_t)scm->ring_cap;
  const uint64_t m = have < (uint64_t)cap ? have : (uint64_t)cap;
  const uint64_t first = total - m;
  for (uint64_t i = 0; i < m; ++i) out[i] = scm->ring[(first + i) % (uint64_t)scm->ring_cap];
  if (n) *n = (int32_t)m;
  return TRIDENT_OK;
}

TRIDENT_API int32_t trident_scm_device_status(trident_scm_t* scm, void* stream, uint32_t* out_bits,
                                              int32_t clear) {
  if (!scm || !out_bits) return fail(TRIDENT_ERR_INVALID, "NULL argument");
  if (scm->dry) return fail(TRIDENT_ERR_STATE, "dry-run SCM has no device state");
  return on_device(scm, [&]() -> int32_t {
    if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess)
      return fail(TRIDENT_ERR_CUDA, "stream synchronize failed: %s", cudaGetErrorString(cudaGetLastError()));
    if (cudaMemcpy(out_bits, scm->d_err, sizeof(uint32_t), cudaMemcpyDeviceToHost) != cudaSuccess)
      return fail(TRIDENT_ERR_CUDA, "status read failed");
    if (clear && cudaMemset(scm->d_err, 0, sizeof(uint32_t)) != cudaSuccess)
      return fail(TRIDENT_ERR_CUDA, "status clear failed");
    return TRIDENT_OK;
  });
}

TRIDENT_API int32_t trident_launch_floor(trident_scm_t* scm, void* stream, int32_t n) {
  if (!scm || n < 0) return fail(TRIDENT_ERR_INVALID, "bad arguments");
  if (scm->dry) return fail(TRIDENT_ERR_STATE, "dry-run SCM launches nothing");
  CUfunction fn = nullptr;  // resolved in the SCM's own context (a handle is per context)
  const int32_t rs = on_device(scm, [&]() -> int32_t {
    cudaFunction_t f = nullptr;
    if (cudaGetFuncBySymbol(&f, empty_kernel_entry()) != cudaSuccess || !f)
      return fail(TRIDENT_ERR_CUDA, "cannot resolve the empty kernel");
    fn = reinterpret_cast<CUfunction>(f);
    return TRIDENT_OK;
  });
  if (rs != TRIDENT_OK) return rs;
  CUlaunchConfig cfg;
  CUlaunchAttribute attr;
  base_config(scm, stream, &cfg, &attr);
  cfg.blockDimX = 32;
  cfg.gridDimX = 1;
  for (int32_t i = 0; i < n; ++i) {
    const uint64_t t0 = scm->ring ? now_ns() : 0;
    const int32_t st = launch_on(scm, &cfg, fn, nullptr);
    if (st != TRIDENT_OK) return st;
    if (scm->ring) record_host_time(scm, t0);
  }
  return TRIDENT_OK;
}

TRIDENT_API int32_t trident_copy_floor(trident_scm_t* scm, void* stream, const void* src, void* dst,
                                       int64_t read_bytes, int64_t write_bytes, int32_t blocks,
                                       int32_t sets, int32_t n) {
  if (!scm || !src || !dst || n < 0 || blocks < 1 || sets < 1 || read_bytes < 16 || write_bytes < 16 ||
      read_bytes % 16 != 0 || write_bytes % 16 != 0 || reinterpret_cast<uintptr_t>(src) % 16 != 0 ||
      reinterpret_cast<uintptr_t>(dst) % 16 != 0)
    return fail(TRIDENT_ERR_INVALID, "bad arguments");
  if (scm->dry) return fail(TRIDENT_ERR_STATE, "dry-run SCM launches nothing");
  CUfunction fn = nullptr;
  const int32_t rs = on_device(scm, [&]() -> int32_t {
    cudaFunction_t f = nullptr;
    if (cudaGetFuncBySymbol(&f, copy_floor_entry()) != cudaSuccess || !f)
      return fail(TRIDENT_ERR_CUDA, "cannot resolve the copy kernel");
    fn = reinterpret_cast<CUfunction>(f);
    return TRIDENT_OK;
  });
  if (rs != TRIDENT_OK) return rs;
  CUlaunchConfig cfg;
  CUlaunchAttribute attr;
  base_config(scm, stream, &cfg, &attr);
  cfg.gridDimX = (unsigned)blocks;
  CopyFloorParams P;
  P.nr = read_bytes / 16;
  P.nw = write_bytes / 16;
  P.prefetch = (scm->opt.flags & TRIDENT_OPT_PDL) ? 1 : 0;
  void* kp[1] = {&P};
  for (int32_t i = 0; i < n; ++i) {
    const int64_t k = i % sets;
    P.src = static_cast<const char*>(src) + k * read_bytes;
    P.dst = static_cast<char*>(dst) + k * write_bytes;
    const int32_t st = launch_on(scm, &cfg, fn, kp);
    if (st != TRIDENT_OK) return st;
  }
  return TRIDENT_OK;
}

TRIDENT_API void trident_scm_destroy(trident_scm_t* scm) {
  if (!scm) return;
  if (!scm->dry && (scm->d_err || !scm->tables.empty())) {
    on_device(scm, [&]() -> int32_t {
      for (RopeTable& rt : scm->tables) cudaFree(rt.dev);
      if (scm->d_err) cudaFree(scm->d_err);
      return TRIDENT_OK;
    });
  }
  if (scm->versions) {
    const int32_t n = scm->count.load();
    for (int32_t i = 0; i < n; ++i)
      if (scm->versions[i].recipe) {
        free_recipe(scm->versions[i].recipe);
        delete scm->versions[i].recipe;
      }
  }
  std::free(scm->versions);
  delete[] scm->hits_per;
  std::free(scm->ring);
  std::free(scm->memo);
  delete scm;
}
