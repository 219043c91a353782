// internal.h -- interface between the SCM host core (scm.cpp) and the kernels (*.cu).
//
// Each kernel takes one parameter struct by value. The host core packs it on the hit
// path (argument preparation, §3.2 and §3.5 of the paper: graph operands are rebuilt
// only after every guard passed) and launches the kernel entry that was resolved when
// the version was registered (§3.3).
#pragma once
#include <stdint.h>

namespace trident {

// Activation element types (values equal trident_dtype).
enum : int32_t { DT_BF16 = 1, DT_FP16 = 2, DT_FP32 = 3 };

constexpr int kThreads = 256;  // block size of every kernel in this library

// add + RMSNorm over T rows of H elements. Row strides in elements.
struct AddNormParams {
  const void* x;
  const void* r;
  const float* gamma;
  void* y;
  void* r_out;
  int64_t T, H;
  int64_t x_rs, r_rs, y_rs, ro_rs;
  float eps, inv_H;
  int32_t prefetch;  // 1: prefetch this block's first lines into L2 before the PDL wait
  uint32_t first_wait_polls;  // bulk-copy kernel: polls of its first wait for the copies
                              // (kBulkWaitPolls; 0 under TRIDENT_OPT_TEST_WAIT_TIMEOUT)
  uint32_t* err;     // device status word (the bulk-copy kernel reports a timed-out wait)
};

// Bound of every mbarrier wait of the bulk-copy kernel (try_wait polls, each itself bounded
// by the hardware's suspend time).
constexpr uint32_t kBulkWaitPolls = 1u << 20;

// RMSNorm over T rows of H elements (no residual). Row strides in elements.
struct RmsNormParams {
  const void* x;
  const float* gamma;
  void* y;
  int64_t T, H;
  int64_t x_rs, y_rs;
  float eps, inv_H;
  int32_t prefetch;
};

// Pointwise operators over T rows of W elements (a: x or the first addend; b: the second
// addend; mask: u8 for MASKED_FILL). Row strides in elements.
enum PointwiseOp : int32_t { PW_SILU = 8, PW_ADD = 9, PW_NEG = 10, PW_MASKED_FILL = 11 };
struct PointwiseParams {
  const void* a;
  const void* b;
  const uint8_t* mask;
  void* y;
  int64_t T, W;
  int64_t a_rs, b_rs, m_rs, y_rs;
  float scalar;
  int32_t prefetch;
};

// RoPE on q/k (optionally after per-head RMSNorm) plus KV-cache append.
// q/k/v rows: token stride *_rs, head stride D, element stride 1. Caches dense [Hkv][S][D].
// inv_freq: [D/2] pairs (hi, lo), theta^(-2i/D) = hi + lo, split from fp64 on the host.
struct RopeParams {
  void* q;
  const void* k;
  const void* v;
  const int32_t* pos;
  void* k_cache;
  void* v_cache;
  const float* gamma_q;
  const float* gamma_k;
  const float2* inv_freq;
  uint32_t* err;
  int64_t T, S;
  int64_t q_rs, k_rs, v_rs;
  int32_t Hq, Hkv, D, NH;  // NH = Hq + 2 Hkv head-rows per token
  float eps, inv_D;
  int32_t prefetch;
  uint32_t nh_magic;  // unit / NH for units below 2^32 by fast_div
  int32_t nh_shift;
};

// RoPE with the block's rows staged by bulk copies (rope_bulk_kernel, calls of many tokens).
struct RopeBulkParams {
  RopeParams rp;
  uint32_t first_wait_polls;  // polls of the wait for the copies (kBulkWaitPolls; 0 under
                              // TRIDENT_OPT_TEST_WAIT_TIMEOUT)
};

// out = silu(g) * u over T rows of I elements.
struct SwigluParams {
  const void* g;
  const void* u;
  void* out;
  int64_t T, I;
  int64_t g_rs, u_rs, o_rs;
  int32_t prefetch;
};

// One decoder layer's chain in one launch. Blocks [0, nA) run the two add+RMSNorm steps
// of one token each, [nA, nA+nB) the RoPE/KV head-rows, the rest SwiGLU tiles.
struct ChainParams {
  AddNormParams n1;   // h, r0 -> x1, r1
  AddNormParams n2;   // attn_out, (r1 from registers) -> x2, r2; n2.r is unused
  RopeParams rope;
  SwigluParams sw;
  int32_t nA, nB, nC, sw_tiles_per_row;
  int32_t a_split;   // CTAs per token for the norms (2, or 1 for in-place calls)
  int32_t prefetch;  // before the PDL wait, into L2: 1 every block's first input lines,
                     // 2 only the norm blocks' rows, 0 none
  int32_t tok_grid;  // 1: grid (a_split + rope_per_tok + sw_tiles_per_row, T), token-major
  int32_t rope_per_tok;  // RoPE blocks per token (token-major grid: nB = T * rope_per_tok)
  int32_t rope_k;    // head-rows per RoPE lane group: 1, or 3 on grids several waves long
  uint32_t sw_magic;  // tile / sw_tiles_per_row by fast_div
  int32_t sw_shift;
  int64_t sw_tiles;  // T * sw_tiles_per_row (valid SwiGLU tiles)
};

// Several independent layer-chain calls in one launch (a decoder step's chains). Call i
// owns blocks [first[i], first[i+1]); inside its range a block plays the same role as in
// the single-call kernel. The struct is passed as the kernel parameter (about 25 KB, under
// the 32 KB parameter limit), so no device buffer is written before the launch.
constexpr int kStepMax = 48;
// SwiGLU tile width of the layer chain's blocks, in 256-thread rounds of 16-byte vectors of
// g and of u: one call's grid keeps tiles small (more blocks for small token counts); a whole
// step's grid, several waves long, does better with fewer, larger tiles (measured on 36 Qwen3
// layers: 8 tokens 11.7 -> 11.4 us, 32 tokens 39.1 -> 37.2 us, 128 tokens 155 -> 150 us;
// the same change on single calls made them slower, 64 tokens 3.56 -> 4.09 us).
constexpr int kChainSwigluUnroll = 2;
constexpr int kChainStepSwigluUnroll = 4;
// A single call's grid of many waves (one CTA per token) takes the wider tiles too: blocks
// queue for slots there, and a tile that moves twice the bytes for the same fixed costs pays.
constexpr int kChainWideSwigluUnroll = 4;
struct ChainStepParams {
  int32_t n;
  int32_t first[kStepMax + 1];  // call-major: call i owns blocks [first[i], first[i+1])
  int32_t role_first[3][kStepMax + 1];  // role-major: call i's norm / RoPE / SwiGLU blocks
                                        // start at role_first[r][i]; [r][n] ends role r
  ChainParams c[kStepMax];
};

// Kernel entry (host stub address) plus its launch shape rule.
struct KernelEntry {
  const void* fn = nullptr;
  const void* fn_inplace = nullptr;  // chain only: the entry for calls that write in place
  const void* fn_late = nullptr;     // chain only: fn with the late launch trigger (LATE)
  const void* fn_wide = nullptr;     // chain only: fn_inplace with kChainWideSwigluUnroll tiles
  const void* fn_step_role = nullptr;  // chain only: fn_step_inplace, role-major block order
  const void* fn_step = nullptr;          // chain only: several calls per launch (ChainStepParams)
  const void* fn_step_inplace = nullptr;  // ... one block per token for the norms
  const void* fn_large = nullptr;  // add+RMSNorm / RoPE: the entry for calls of >= large_rows rows
                                   // (tokens)
  int32_t large_rows = 0;
  int32_t kind = 0;      // which grid rule the host applies (KernelKind)
  int32_t vec = 0;       // elements per vector (VE), or tile width for SwiGLU
  int32_t unroll = 1;    // vectors per thread per tile (SwiGLU, chain)
  int32_t rows = 1;      // rows per block (KK_NORM_ROWS; RoPE's fn_large: tokens per block)
};

enum KernelKind : int32_t {
  KK_ADDNORM_ROW = 1,   // grid = T rows, one block per row
  KK_ROPE_HALFWARP = 2, // grid = ceil(T*NH / units_per_block)
  KK_ROPE_WARP = 3,     // generic: one warp per head-row
  KK_SWIGLU_TILE = 4,   // grid = (tiles per row, rows)
  KK_SWIGLU_FLAT = 5,   // generic: flat grid-stride
  KK_CHAIN = 6,
  KK_NORM_ROWS = 7      // grid = ceil(T / rows): several rows per block
};

// Lookup of compiled kernels. Return false (with a reason) if no kernel fits.
bool addnorm_kernel(int32_t dtype, int32_t variant, int64_t H, KernelEntry* out, const char** why);
bool rmsnorm_kernel(int32_t dtype, int32_t variant, int64_t H, KernelEntry* out, const char** why);
bool pointwise_kernel(int32_t op, int32_t dtype, int32_t variant, int64_t W, KernelEntry* out,
                      const char** why);
bool rope_kernel(int32_t dtype, int32_t variant, int32_t D, bool qknorm, KernelEntry* out,
                 const char** why);
bool swiglu_kernel(int32_t dtype, int32_t variant, int64_t I, KernelEntry* out, const char** why);
bool chain_kernel(int32_t dtype, int64_t H, int32_t D, bool qknorm, KernelEntry* out,
                  const char** why);
const void* empty_kernel_entry();  // the latency-floor probe's kernel (does nothing)

// Validation, guard-equivalent checks (sizes, layouts, 16-byte alignment, overlap) and
// parameter packing of a ROPE_KV / QKNORM_ROPE_KV argument tuple without an SCM. Leaves
// p->cs and p->err NULL. Returns a trident_status (message in trident_scm_last_error).
int32_t prepare_rope_args(const void* trident_args_ptr, RopeParams* p, int32_t* dtype,
                          bool* qknorm);

// Sets the thread-local last-error message and returns `status`.
int32_t internal_fail(int32_t status, const char* msg);

// Units (head-rows) handled by one block of the vector RoPE kernel for head size D.
inline int32_t rope_units_per_block(int32_t D, int32_t elem_bytes) {
  int32_t lanes_per_head = D * elem_bytes / 16;
  return kThreads / lanes_per_head;
}

}  // namespace trident
