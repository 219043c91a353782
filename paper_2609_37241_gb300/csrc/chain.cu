// chain.cu -- one decoder layer's non-GEMM chain in a single launch.
//
//   add+RMSNorm(h, r0) -> x1, r1;  [q/k RMSNorm +] RoPE(q, k) + KV append;
//   add+RMSNorm(attn_out, r1) -> x2, r2;  SwiGLU(g, u) -> o
//
// The only data dependency inside the chain is r1 feeding the second norm, and it is
// row-local: the block that produces row t of r1 keeps it in registers and runs the
// second norm of row t itself. So no grid-wide barrier is needed; the launch is a
// horizontal fusion where block ranges take different roles:
//   [0, nA)            two add+RMSNorm steps of token b (the longest per-block work,
//                      so these blocks are scheduled first)
//   [nA, nA + nB)      RoPE/KV head-rows, (256 / (D/8)) per block
//   [nA + nB, end)     SwiGLU tiles of one row each
// One launch replaces four, which is what matters at decode sizes, where each step
// moves well under a microsecond of HBM traffic.
#include "device_common.cuh"

namespace trident {

constexpr int kChainSwigluUnroll = 2;

template <int DT, int VPT, int D, bool QKNORM>
__global__ void __launch_bounds__(kThreads) chain_kernel(const ChainParams c) {
  pdl_prologue();
  constexpr int EB = Act<DT>::BYTES;
  constexpr int VE = Act<DT>::VE;
  const int tid = threadIdx.x;
  const int b = blockIdx.x;
  if (b < c.nA) {
    __shared__ float red[2][kThreads / 32];
    const int64_t row = b;
    const AddNormParams& n1 = c.n1;
    const AddNormParams& n2 = c.n2;
    AddNormRegs<DT, VPT> A, B;
    // every load of both norms is issued before the first reduction
    A.load(row_ptr(n1.x, row, n1.x_rs, EB), row_ptr(n1.r, row, n1.r_rs, EB), n1.gamma, tid);
    B.load_x_gamma(row_ptr(n2.x, row, n2.x_rs, EB), n2.gamma, tid);
    float s[VPT][VE];
    float ss = A.residual(row_ptr(n1.r_out, row, n1.ro_rs, EB), tid, s);
    float tot = block_sum(ss, red[0]);
    A.normalize(row_ptr(n1.y, row, n1.y_rs, EB), tid, s, rsqrtf(tot * n1.inv_H + n1.eps));
    // the second residual input is r1 as stored (rounded), taken from registers
#pragma unroll
    for (int v = 0; v < VPT; ++v) B.rv[v] = A.rv[v];
    ss = B.residual(row_ptr(n2.r_out, row, n2.ro_rs, EB), tid, s);
    tot = block_sum(ss, red[1]);
    B.normalize(row_ptr(n2.y, row, n2.y_rs, EB), tid, s, rsqrtf(tot * n2.inv_H + n2.eps));
  } else if (b < c.nA + c.nB) {
    constexpr int LPH = D / VE;
    constexpr int UPB = kThreads / LPH;
    const int64_t unit = (int64_t)(b - c.nA) * UPB + tid / LPH;
    if (unit < c.rope.T * c.rope.NH) rope_head_row<DT, D, QKNORM>(c.rope, unit, tid % LPH);
  } else {
    const int tile = b - c.nA - c.nB;
    const int64_t row = tile / c.sw_tiles_per_row;
    const int64_t col_tile = tile - row * c.sw_tiles_per_row;
    swiglu_tile<DT, kChainSwigluUnroll>(c.sw, row, col_tile * kChainSwigluUnroll * kThreads, tid);
  }
}

template <int DT, bool QK>
static const void* pick(int64_t H) {
  constexpr int per = kThreads * Act<DT>::VE;
  if (H == per * 2) return (const void*)chain_kernel<DT, 2, 128, QK>;
  if (H == per * 4) return (const void*)chain_kernel<DT, 4, 128, QK>;
  return nullptr;
}

bool chain_kernel(int32_t dtype, int64_t H, int32_t D, bool qknorm, KernelEntry* out,
                  const char** why) {
  if (dtype != DT_BF16 && dtype != DT_FP16) { *why = "layer chain supports bf16 and fp16"; return false; }
  if (D != 128) { *why = "layer chain supports D = 128"; return false; }
  out->kind = KK_CHAIN;
  out->vec = 8;
  out->unroll = kChainSwigluUnroll;
  if (dtype == DT_BF16) out->fn = qknorm ? pick<DT_BF16, true>(H) : pick<DT_BF16, false>(H);
  else out->fn = qknorm ? pick<DT_FP16, true>(H) : pick<DT_FP16, false>(H);
  if (!out->fn) { *why = "layer chain supports H in {4096, 8192}"; return false; }
  return true;
}

}  // namespace trident
