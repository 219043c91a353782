// addnorm.cu -- fused residual add + RMSNorm kernels (sm_103a).
//
//   s = x + r (fp32);  r_out = round(s);  y = round(s * rsqrt(mean(s^2) + eps) * gamma)
//
// rms_norm is the paper's running example (Fig. 1, §2.3); the residual add fused in front
// of it is how decoder layers call it. One block owns one row: the row's bytes are
// loaded once with 16-byte accesses, the sum of squares is reduced with warp shuffles and
// one barrier, and both outputs are written with 16-byte stores. Three families:
//   addnorm_vec_kernel<DT, VPT>   H = VPT * 256 * VE, row held in registers (one pass)
//   addnorm_bulk_kernel<DT>       H = 8192 bf16/fp16, >= 1024 rows: rows staged by bulk copies
//   addnorm_loop_kernel<DT>       any H with 16-byte rows (two passes, the second from L2)
//   addnorm_generic_kernel<DT>    any H, any element-aligned pointer (scalar accesses)
#include "device_common.cuh"

namespace trident {

// The row in registers: x and r as packed 16-byte vectors, gamma and the fp32 sum
// s = x + r as floats (thread `tid` owns vectors v*256 + tid, v < VPT: coalesced).
template <int DT, int VPT>
__global__ void __launch_bounds__(kThreads) addnorm_vec_kernel(const AddNormParams p) {
  pdl_trigger();
  __shared__ float red[kThreads / 32];
  constexpr int EB = Act<DT>::BYTES;
  constexpr int VE = Act<DT>::VE;
  const int tid = threadIdx.x;
  if (p.prefetch && (tid & 7) == 0 && blockIdx.x < p.T) {  // the first row's lines (prefetch_l2)
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      const int64_t vi = (int64_t)v * kThreads + tid;
      prefetch_l2(reinterpret_cast<const uint4*>(row_ptr(p.x, blockIdx.x, p.x_rs, EB)) + vi);
      prefetch_l2(reinterpret_cast<const uint4*>(row_ptr(p.r, blockIdx.x, p.r_rs, EB)) + vi);
    }
  }
  pdl_wait();
  for (int64_t row = blockIdx.x; row < p.T; row += gridDim.x) {
    const uint4* xp = reinterpret_cast<const uint4*>(row_ptr(p.x, row, p.x_rs, EB));
    const uint4* rp = reinterpret_cast<const uint4*>(row_ptr(p.r, row, p.r_rs, EB));
    uint4 xv[VPT], rv[VPT];
    float g[VPT][VE], s[VPT][VE];
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      const int64_t vi = (int64_t)v * kThreads + tid;
      xv[v] = ldg16(xp + vi);
      rv[v] = ldg16(rp + vi);
#pragma unroll
      for (int q = 0; q < VE / 4; ++q) {
        const float4 gg = ldg_f4(p.gamma + vi * VE + 4 * q);
        g[v][4 * q] = gg.x; g[v][4 * q + 1] = gg.y; g[v][4 * q + 2] = gg.z; g[v][4 * q + 3] = gg.w;
      }
    }
    uint4* rop = reinterpret_cast<uint4*>(row_ptr(p.r_out, row, p.ro_rs, EB));
    float ss = 0.f;
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      float xf[VE], rf[VE];
      unpack<DT>(xv[v], xf);
      unpack<DT>(rv[v], rf);
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        s[v][e] = xf[e] + rf[e];
        ss = fmaf(s[v][e], s[v][e], ss);
      }
      st16(rop + (int64_t)v * kThreads + tid, pack<DT>(s[v]));
    }
    const float inv = rsqrtf(block_sum(ss, red) * p.inv_H + p.eps);
    uint4* yp = reinterpret_cast<uint4*>(row_ptr(p.y, row, p.y_rs, EB));
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      float y[VE];
#pragma unroll
      for (int e = 0; e < VE; ++e) y[e] = s[v][e] * inv * g[v][e];
      st16(yp + (int64_t)v * kThreads + tid, pack<DT>(y));
    }
    __syncthreads();  // `red` is reused by the next row
  }
}

// H = 8192 in bf16/fp16 for calls of many rows: the row's x and r (16 KB each) are staged
// in shared memory by two bulk copies (cp.async.bulk, completion counted on an mbarrier)
// issued by one thread, while every thread loads its gamma vectors; s = x + r is formed
// from shared memory twice (the same fp32 addition both times). With the rows out of the
// registers four blocks fit per SM instead of two, which pays once a call has enough rows to
// keep them busy (measured: 2-4 % faster from 1024 rows, slower at 256). The wait is bounded:
// if it runs out, the block sets TRIDENT_DEVERR_TIMEOUT, waits again (bounded) for its copies
// and returns without writing.
template <int DT>
__global__ void __launch_bounds__(kThreads, 4) addnorm_bulk_kernel(const AddNormParams p) {
  constexpr int VPT = 4;
  constexpr int VE = Act<DT>::VE;
  constexpr int EB = Act<DT>::BYTES;
  constexpr uint32_t kRowBytes = VPT * kThreads * 16;
  static_assert(VE == 8, "bf16 / fp16 rows");
  __shared__ __align__(128) uint4 xs[VPT * kThreads];
  __shared__ __align__(128) uint4 rs[VPT * kThreads];
  __shared__ __align__(8) unsigned long long bar;
  __shared__ float red[kThreads / 32];
  const int tid = threadIdx.x;
  const int64_t row = blockIdx.x;
  const uint32_t bar_a = (uint32_t)__cvta_generic_to_shared(&bar);
  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" :: "r"(bar_a) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  pdl_trigger();
  pdl_wait();
  __syncthreads();  // the barrier is initialised before anyone waits on it
  if (tid == 0) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
                 :: "r"(bar_a), "r"(2 * kRowBytes) : "memory");
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 :: "r"((uint32_t)__cvta_generic_to_shared(xs)), "l"(row_ptr(p.x, row, p.x_rs, EB)),
                    "r"(kRowBytes), "r"(bar_a) : "memory");
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 :: "r"((uint32_t)__cvta_generic_to_shared(rs)), "l"(row_ptr(p.r, row, p.r_rs, EB)),
                    "r"(kRowBytes), "r"(bar_a) : "memory");
  }
  float g[VPT][VE];
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
    const int64_t vi = (int64_t)v * kThreads + tid;
#pragma unroll
    for (int q = 0; q < VE / 4; ++q) {
      const float4 gg = ldg_f4(p.gamma + vi * VE + 4 * q);
      g[v][4 * q] = gg.x; g[v][4 * q + 1] = gg.y; g[v][4 * q + 2] = gg.z; g[v][4 * q + 3] = gg.w;
    }
  }
  auto landed = [&](uint32_t polls) -> bool {
    uint32_t done = 0;
    for (uint32_t it = 0; it < polls && !done; ++it)
      asm volatile("{ .reg .pred q; mbarrier.try_wait.parity.shared::cta.b64 q, [%1], 0; selp.u32 %0, 1, 0, q; }"
                   : "=r"(done) : "r"(bar_a) : "memory");
    return done != 0;
  };
  const bool ok = landed(p.first_wait_polls);
  if (__syncthreads_or(!ok)) {  // one decision for the whole block
    if (tid == 0 && p.err) atomicOr(p.err, kErrTimeout);
    if (!ok) landed(kBulkWaitPolls);  // a second bounded wait for the copies before the block exits
    return;
  }
  uint4* rop = reinterpret_cast<uint4*>(row_ptr(p.r_out, row, p.ro_rs, EB));
  float ss = 0.f;
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
    const int vi = v * kThreads + tid;
    float xf[VE], rf[VE], sv[VE];
    unpack<DT>(xs[vi], xf);
    unpack<DT>(rs[vi], rf);
#pragma unroll
    for (int e = 0; e < VE; ++e) {
      sv[e] = xf[e] + rf[e];
      ss = fmaf(sv[e], sv[e], ss);
    }
    st16(rop + vi, pack<DT>(sv));
  }
  const float inv = rsqrtf(block_sum(ss, red) * p.inv_H + p.eps);
  uint4* yp = reinterpret_cast<uint4*>(row_ptr(p.y, row, p.y_rs, EB));
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
    const int vi = v * kThreads + tid;
    float xf[VE], rf[VE], y[VE];
    unpack<DT>(xs[vi], xf);
    unpack<DT>(rs[vi], rf);
#pragma unroll
    for (int e = 0; e < VE; ++e) y[e] = (xf[e] + rf[e]) * inv * g[v][e];
    st16(yp + vi, pack<DT>(y));
  }
}

// Two passes: the first only reduces, the second recomputes s and writes both outputs,
// so that in-place calls (r_out = r, y = x) never read a value they already overwrote.
template <int DT>
__global__ void __launch_bounds__(kThreads) addnorm_loop_kernel(const AddNormParams p) {
  pdl_prologue();
  __shared__ float red[kThreads / 32];
  constexpr int EB = Act<DT>::BYTES;
  constexpr int VE = Act<DT>::VE;
  const int tid = threadIdx.x;
  const int64_t nvec = p.H / VE;
  for (int64_t row = blockIdx.x; row < p.T; row += gridDim.x) {
    const uint4* x = reinterpret_cast<const uint4*>(row_ptr(p.x, row, p.x_rs, EB));
    const uint4* r = reinterpret_cast<const uint4*>(row_ptr(p.r, row, p.r_rs, EB));
    float ss = 0.f;
    for (int64_t vi = tid; vi < nvec; vi += kThreads) {
      float xf[VE], rf[VE];
      unpack<DT>(ld16(x + vi), xf);
      unpack<DT>(ld16(r + vi), rf);
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        const float s = xf[e] + rf[e];
        ss = fmaf(s, s, ss);
      }
    }
    const float inv = rsqrtf(block_sum(ss, red) * p.inv_H + p.eps);
    uint4* y = reinterpret_cast<uint4*>(row_ptr(p.y, row, p.y_rs, EB));
    uint4* ro = reinterpret_cast<uint4*>(row_ptr(p.r_out, row, p.ro_rs, EB));
    for (int64_t vi = tid; vi < nvec; vi += kThreads) {
      float xf[VE], rf[VE], s[VE], yf[VE], g[VE];
      unpack<DT>(ld16(x + vi), xf);
      unpack<DT>(ld16(r + vi), rf);
#pragma unroll
      for (int q = 0; q < VE / 4; ++q) {
        const float4 g4 = ldg_f4(p.gamma + vi * VE + 4 * q);
        g[4 * q] = g4.x; g[4 * q + 1] = g4.y; g[4 * q + 2] = g4.z; g[4 * q + 3] = g4.w;
      }
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        s[e] = xf[e] + rf[e];
        yf[e] = s[e] * inv * g[e];
      }
      st16(ro + vi, pack<DT>(s));
      st16(y + vi, pack<DT>(yf));
    }
    __syncthreads();
  }
}

template <int DT>
__global__ void __launch_bounds__(kThreads) addnorm_generic_kernel(const AddNormParams p) {
  pdl_prologue();
  __shared__ float red[kThreads / 32];
  const int tid = threadIdx.x;
  for (int64_t row = blockIdx.x; row < p.T; row += gridDim.x) {
    const int64_t xo = row * p.x_rs, ro = row * p.r_rs;
    float ss = 0.f;
    for (int64_t j = tid; j < p.H; j += kThreads) {
      const float s = load_elem<DT>(p.x, xo + j) + load_elem<DT>(p.r, ro + j);
      ss = fmaf(s, s, ss);
    }
    const float inv = rsqrtf(block_sum(ss, red) * p.inv_H + p.eps);
    for (int64_t j = tid; j < p.H; j += kThreads) {
      const float s = load_elem<DT>(p.x, xo + j) + load_elem<DT>(p.r, ro + j);
      store_elem<DT>(p.r_out, row * p.ro_rs + j, s);
      store_elem<DT>(p.y, row * p.y_rs + j, s * inv * p.gamma[j]);
    }
    __syncthreads();
  }
}

template <int DT>
static bool pick_vec(int64_t H, KernelEntry* out) {
  constexpr int VE = Act<DT>::VE;
  const int64_t per = (int64_t)kThreads * VE;
  if (H == per * 1) { out->fn = (const void*)addnorm_vec_kernel<DT, 1>; return true; }
  if (H == per * 2) { out->fn = (const void*)addnorm_vec_kernel<DT, 2>; return true; }
  if (H == per * 4) {
    out->fn = (const void*)addnorm_vec_kernel<DT, 4>;
    if constexpr (VE == 8) {  // bf16 / fp16 H 8192: rows staged by bulk copies for long calls
      out->fn_large = (const void*)addnorm_bulk_kernel<DT>;
      out->large_rows = 1024;
    }
    return true;
  }
  if (H == per * 8) { out->fn = (const void*)addnorm_vec_kernel<DT, 8>; return true; }
  out->fn = (const void*)addnorm_loop_kernel<DT>;
  return true;
}

bool addnorm_kernel(int32_t dtype, int32_t variant, int64_t H, KernelEntry* out, const char** why) {
  out->kind = KK_ADDNORM_ROW;
  out->unroll = 1;
  const int eb = dtype == DT_FP32 ? 4 : 2;
  if (dtype != DT_BF16 && dtype != DT_FP16 && dtype != DT_FP32) { *why = "dtype"; return false; }
  if (H < 1) { *why = "H must be >= 1"; return false; }
  if (variant == 1) {  // GENERIC
    out->vec = 1;
    out->fn = dtype == DT_BF16 ? (const void*)addnorm_generic_kernel<DT_BF16>
            : dtype == DT_FP16 ? (const void*)addnorm_generic_kernel<DT_FP16>
                               : (const void*)addnorm_generic_kernel<DT_FP32>;
    return true;
  }
  if ((H * eb) % 16 != 0) { *why = "vector add+RMSNorm needs H * elem_size % 16 == 0"; return false; }
  out->vec = 16 / eb;
  if (dtype == DT_BF16) return pick_vec<DT_BF16>(H, out);
  if (dtype == DT_FP16) return pick_vec<DT_FP16>(H, out);
  return pick_vec<DT_FP32>(H, out);
}

}  // namespace trident
