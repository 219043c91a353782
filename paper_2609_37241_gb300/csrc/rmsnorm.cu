// rmsnorm.cu -- RMSNorm kernels (no residual): y = round(x * rsqrt(mean(x^2) + eps) * gamma).
//
// rms_norm is the paper's running example (Fig. 1, §2.3; its motivation experiment uses
// x (1024, 128)), where the host side picks between a one-shot kernel for short rows and a
// looping kernel for long ones. The same choice is made here, once, when a version is
// registered:
//   rmsnorm_rows_kernel<DT, LPR>  H = LPR * VE <= 256 bf16: a group of LPR lanes per row,
//                                 256 / LPR rows per block, reduced by xor-shuffles
//   rmsnorm_vec_kernel<DT, VPT>   H = VPT * 256 * VE: one block per row, row in registers
//   rmsnorm_loop_kernel<DT>       any H with 16-byte rows (two passes, the second from L2)
//   rmsnorm_generic_kernel<DT>    any H, any element-aligned pointer (scalar accesses)
#include "device_common.cuh"

namespace trident {

template <int DT, int LPR>
__global__ void __launch_bounds__(kThreads) rmsnorm_rows_kernel(const RmsNormParams p) {
  pdl_trigger();
  constexpr int VE = Act<DT>::VE;
  constexpr int EB = Act<DT>::BYTES;
  constexpr int RPB = kThreads / LPR;
  const int lane = threadIdx.x % LPR;
  if (p.prefetch && (lane & 7) == 0) {  // the first row's lines (prefetch_l2)
    const int64_t row0 = (int64_t)blockIdx.x * RPB + threadIdx.x / LPR;
    if (row0 < p.T) prefetch_l2(row_ptr(p.x, row0, p.x_rs, EB) + (int64_t)lane * 16);
  }
  pdl_wait();
  const unsigned mask =
      (LPR == 32) ? 0xffffffffu : (((1u << LPR) - 1u) << ((threadIdx.x & 31) & ~(LPR - 1)));
  for (int64_t row = (int64_t)blockIdx.x * RPB + threadIdx.x / LPR; row < p.T;
       row += (int64_t)gridDim.x * RPB) {
    const uint4 xv = ldg16(row_ptr(p.x, row, p.x_rs, EB) + (int64_t)lane * 16);
    float g[VE];
#pragma unroll
    for (int q = 0; q < VE / 4; ++q) {
      const float4 g4 = ldg_f4(p.gamma + lane * VE + 4 * q);
      g[4 * q] = g4.x; g[4 * q + 1] = g4.y; g[4 * q + 2] = g4.z; g[4 * q + 3] = g4.w;
    }
    float x[VE];
    unpack<DT>(xv, x);
    float ss = 0.f;
#pragma unroll
    for (int e = 0; e < VE; ++e) ss = fmaf(x[e], x[e], ss);
#pragma unroll
    for (int o = LPR / 2; o > 0; o >>= 1) ss += __shfl_xor_sync(mask, ss, o, LPR);
    const float inv = rsqrtf(ss * p.inv_H + p.eps);
#pragma unroll
    for (int e = 0; e < VE; ++e) x[e] = x[e] * inv * g[e];
    st16(row_ptr(p.y, row, p.y_rs, EB) + (int64_t)lane * 16, pack<DT>(x));
  }
}

template <int DT, int VPT>
__global__ void __launch_bounds__(kThreads) rmsnorm_vec_kernel(const RmsNormParams p) {
  pdl_trigger();
  __shared__ float red[kThreads / 32];
  constexpr int VE = Act<DT>::VE;
  constexpr int EB = Act<DT>::BYTES;
  const int tid = threadIdx.x;
  if (p.prefetch && (tid & 7) == 0 && blockIdx.x < p.T) {  // the first row's lines (prefetch_l2)
#pragma unroll
    for (int v = 0; v < VPT; ++v)
      prefetch_l2(reinterpret_cast<const uint4*>(row_ptr(p.x, blockIdx.x, p.x_rs, EB)) +
                  (int64_t)v * kThreads + tid);
  }
  pdl_wait();
  for (int64_t row = blockIdx.x; row < p.T; row += gridDim.x) {
    const uint4* xr = reinterpret_cast<const uint4*>(row_ptr(p.x, row, p.x_rs, EB));
    uint4 xv[VPT];
    float g[VPT][VE];
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      const int64_t vi = (int64_t)v * kThreads + tid;
      xv[v] = ldg16(xr + vi);
#pragma unroll
      for (int q = 0; q < VE / 4; ++q) {
        const float4 g4 = ldg_f4(p.gamma + vi * VE + 4 * q);
        g[v][4 * q] = g4.x; g[v][4 * q + 1] = g4.y; g[v][4 * q + 2] = g4.z; g[v][4 * q + 3] = g4.w;
      }
    }
    float ss = 0.f;
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      float x[VE];
      unpack<DT>(xv[v], x);
#pragma unroll
      for (int e = 0; e < VE; ++e) ss = fmaf(x[e], x[e], ss);
    }
    const float inv = rsqrtf(block_sum(ss, red) * p.inv_H + p.eps);
    uint4* yr = reinterpret_cast<uint4*>(row_ptr(p.y, row, p.y_rs, EB));
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      float x[VE];
      unpack<DT>(xv[v], x);
#pragma unroll
      for (int e = 0; e < VE; ++e) x[e] = x[e] * inv * g[v][e];
      st16(yr + (int64_t)v * kThreads + tid, pack<DT>(x));
    }
    __syncthreads();  // `red` is reused by the next row
  }
}

// Two passes: the first reduces, the second rescales; in place (y = x) each thread rewrites
// only the vectors it read.
template <int DT>
__global__ void __launch_bounds__(kThreads) rmsnorm_loop_kernel(const RmsNormParams p) {
  pdl_prologue();
  __shared__ float red[kThreads / 32];
  constexpr int VE = Act<DT>::VE;
  constexpr int EB = Act<DT>::BYTES;
  const int tid = threadIdx.x;
  const int64_t nvec = p.H / VE;
  for (int64_t row = blockIdx.x; row < p.T; row += gridDim.x) {
    const uint4* xr = reinterpret_cast<const uint4*>(row_ptr(p.x, row, p.x_rs, EB));
    float ss = 0.f;
    for (int64_t vi = tid; vi < nvec; vi += kThreads) {
      float x[VE];
      unpack<DT>(ld16(xr + vi), x);
#pragma unroll
      for (int e = 0; e < VE; ++e) ss = fmaf(x[e], x[e], ss);
    }
    const float inv = rsqrtf(block_sum(ss, red) * p.inv_H + p.eps);
    uint4* yr = reinterpret_cast<uint4*>(row_ptr(p.y, row, p.y_rs, EB));
    for (int64_t vi = tid; vi < nvec; vi += kThreads) {
      float x[VE], g[VE];
      unpack<DT>(ld16(xr + vi), x);
#pragma unroll
      for (int q = 0; q < VE / 4; ++q) {
        const float4 g4 = ldg_f4(p.gamma + vi * VE + 4 * q);
        g[4 * q] = g4.x; g[4 * q + 1] = g4.y; g[4 * q + 2] = g4.z; g[4 * q + 3] = g4.w;
      }
#pragma unroll
      for (int e = 0; e < VE; ++e) x[e] = x[e] * inv * g[e];
      st16(yr + vi, pack<DT>(x));
    }
    __syncthreads();
  }
}

template <int DT>
__global__ void __launch_bounds__(kThreads) rmsnorm_generic_kernel(const RmsNormParams p) {
  pdl_prologue();
  __shared__ float red[kThreads / 32];
  const int tid = threadIdx.x;
  for (int64_t row = blockIdx.x; row < p.T; row += gridDim.x) {
    const int64_t xo = row * p.x_rs;
    float ss = 0.f;
    for (int64_t j = tid; j < p.H; j += kThreads) {
      const float v = load_elem<DT>(p.x, xo + j);
      ss = fmaf(v, v, ss);
    }
    const float inv = rsqrtf(block_sum(ss, red) * p.inv_H + p.eps);
    for (int64_t j = tid; j < p.H; j += kThreads)
      store_elem<DT>(p.y, row * p.y_rs + j, load_elem<DT>(p.x, xo + j) * inv * p.gamma[j]);
    __syncthreads();
  }
}

template <int DT>
static void pick_vec(int64_t H, KernelEntry* out) {
  constexpr int VE = Act<DT>::VE;
  out->kind = KK_NORM_ROWS;
  const int64_t lanes = H / VE;
  switch (lanes) {  // one-shot: a lane group per row
    case 1: out->fn = (const void*)rmsnorm_rows_kernel<DT, 1>; out->rows = kThreads; return;
    case 2: out->fn = (const void*)rmsnorm_rows_kernel<DT, 2>; out->rows = kThreads / 2; return;
    case 4: out->fn = (const void*)rmsnorm_rows_kernel<DT, 4>; out->rows = kThreads / 4; return;
    case 8: out->fn = (const void*)rmsnorm_rows_kernel<DT, 8>; out->rows = kThreads / 8; return;
    case 16: out->fn = (const void*)rmsnorm_rows_kernel<DT, 16>; out->rows = kThreads / 16; return;
    case 32: out->fn = (const void*)rmsnorm_rows_kernel<DT, 32>; out->rows = kThreads / 32; return;
    default: break;
  }
  out->kind = KK_ADDNORM_ROW;
  out->rows = 1;
  const int64_t per = (int64_t)kThreads * VE;
  if (H == per * 1) { out->fn = (const void*)rmsnorm_vec_kernel<DT, 1>; return; }
  if (H == per * 2) { out->fn = (const void*)rmsnorm_vec_kernel<DT, 2>; return; }
  if (H == per * 4) { out->fn = (const void*)rmsnorm_vec_kernel<DT, 4>; return; }
  if (H == per * 8) { out->fn = (const void*)rmsnorm_vec_kernel<DT, 8>; return; }
  out->fn = (const void*)rmsnorm_loop_kernel<DT>;  // looping kernel for other long rows
}

bool rmsnorm_kernel(int32_t dtype, int32_t variant, int64_t H, KernelEntry* out, const char** why) {
  if (dtype != DT_BF16 && dtype != DT_FP16 && dtype != DT_FP32) { *why = "dtype"; return false; }
  if (H < 1) { *why = "H must be >= 1"; return false; }
  const int eb = dtype == DT_FP32 ? 4 : 2;
  out->unroll = 1;
  if (variant == 1) {  // GENERIC
    out->kind = KK_ADDNORM_ROW;
    out->vec = 1;
    out->rows = 1;
    out->fn = dtype == DT_BF16 ? (const void*)rmsnorm_generic_kernel<DT_BF16>
            : dtype == DT_FP16 ? (const void*)rmsnorm_generic_kernel<DT_FP16>
                               : (const void*)rmsnorm_generic_kernel<DT_FP32>;
    return true;
  }
  if ((H * eb) % 16 != 0) { *why = "vector RMSNorm needs H * elem_size % 16 == 0"; return false; }
  out->vec = 16 / eb;
  if (dtype == DT_BF16) pick_vec<DT_BF16>(H, out);
  else if (dtype == DT_FP16) pick_vec<DT_FP16>(H, out);
  else pick_vec<DT_FP32>(H, out);
  return true;
}

}  // namespace trident
