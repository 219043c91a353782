// rope.cu -- RoPE on q/k with KV-cache append, optionally after per-head q/k RMSNorm.
//
// Work unit: one head-row (token t, head hh) of D elements; per token there are
// NH = Hq + 2*Hkv of them (q heads, k heads, v heads). The vector kernel gives each unit
// D/VE lanes (16 lanes for D = 128 in bf16) so that a unit is one 256-byte coalesced
// access, and exchanges the rotate-half partner with one xor-shuffle per element.
// The generic kernel gives each unit one warp and scalar accesses (any alignment, any
// even D). Both compute (cos, sin) of pos * theta^(-2i/D) in the kernel from the version's
// double-float frequency table [D/2], which the host splits from fp64 at registration.
#include "device_common.cuh"

namespace trident {

template <int DT, int D, bool QKNORM>
__global__ void __launch_bounds__(kThreads) rope_vec_kernel(const RopeParams p) {
  pdl_trigger();
  constexpr int LPH = D / Act<DT>::VE;
  constexpr int UPB = kThreads / LPH;
  const int64_t total = p.T * p.NH;
  const int lane = threadIdx.x % LPH;
  if (p.prefetch) rope_prefetch<DT, D>(p, (int64_t)blockIdx.x * UPB + threadIdx.x / LPH, lane);
  float fq[2 * Act<DT>::VE];
  rope_lane_freqs<DT, D>(p.inv_freq, lane, fq);  // the version's table: readable before the wait
  pdl_wait();
  for (int64_t unit = (int64_t)blockIdx.x * UPB + threadIdx.x / LPH; unit < total;
       unit += (int64_t)gridDim.x * UPB) {
    rope_head_row<DT, D, QKNORM>(p, unit, lane, fq);
  }
}

template <int DT, bool QKNORM>
__global__ void __launch_bounds__(kThreads) rope_generic_kernel(const RopeParams p) {
  pdl_prologue();
  const int lane = threadIdx.x & 31;
  const int64_t total = p.T * p.NH;
  const int64_t nwarps = (int64_t)gridDim.x * (kThreads / 32);
  const int half = p.D / 2;
  for (int64_t unit = ((int64_t)blockIdx.x * kThreads + threadIdx.x) / 32; unit < total;
       unit += nwarps) {
    const int64_t t = unit / p.NH;
    const int hh = (int)(unit - t * p.NH);
    const int32_t pos = p.pos[t];
    if (pos < 0 || (int64_t)pos >= p.S) {
      if (lane == 0) atomicOr(p.err, kErrPos);
      continue;
    }
    if (hh >= p.Hq + p.Hkv) {
      const int h = hh - p.Hq - p.Hkv;
      const int64_t so = t * p.v_rs + (int64_t)h * p.D;
      const int64_t dst = ((int64_t)h * p.S + pos) * p.D;
      const uint16_t* vs = reinterpret_cast<const uint16_t*>(p.v);  // bit copy (2-byte types)
      uint16_t* vd = reinterpret_cast<uint16_t*>(p.v_cache);
      for (int j = lane; j < p.D; j += 32) vd[dst + j] = vs[so + j];
      continue;
    }
    const bool is_q = hh < p.Hq;
    const int h = is_q ? hh : hh - p.Hq;
    const void* src = is_q ? (const void*)p.q : p.k;
    const int64_t so = t * (is_q ? p.q_rs : p.k_rs) + (int64_t)h * p.D;
    const float* gam = is_q ? p.gamma_q : p.gamma_k;
    float inv = 1.f;
    if (QKNORM) {
      float ss = 0.f;
      for (int j = lane; j < p.D; j += 32) {
        const float v = load_elem<DT>(src, so + j);
        ss = fmaf(v, v, ss);
      }
      inv = rsqrtf(warp_sum(ss) * p.inv_D + p.eps);
    }
    for (int i = lane; i < half; i += 32) {
      float lo = load_elem<DT>(src, so + i), hi = load_elem<DT>(src, so + i + half);
      if (QKNORM) {
        lo = lo * inv * gam[i];
        hi = hi * inv * gam[i + half];
      }
      const float2 f = p.inv_freq[i];
      float sn, cs;
      rope_sincos((float)pos, f.x, f.y, &sn, &cs);
      const float ylo = fmaf(lo, cs, -hi * sn);
      const float yhi = fmaf(hi, cs, lo * sn);
      if (is_q) {
        store_elem<DT>(p.q, so + i, ylo);
        store_elem<DT>(p.q, so + i + half, yhi);
      } else {
        const int64_t dst = ((int64_t)h * p.S + pos) * p.D;
        store_elem<DT>(p.k_cache, dst + i, ylo);
        store_elem<DT>(p.k_cache, dst + i + half, yhi);
      }
    }
  }
}

template <int DT, bool QK>
static const void* pick_vec(int32_t D) {
  if (D == 64) return (const void*)rope_vec_kernel<DT, 64, QK>;
  if (D == 128) return (const void*)rope_vec_kernel<DT, 128, QK>;
  if (D == 256) return (const void*)rope_vec_kernel<DT, 256, QK>;
  return nullptr;
}

bool rope_kernel(int32_t dtype, int32_t variant, int32_t D, bool qknorm, KernelEntry* out,
                 const char** why) {
  if (dtype != DT_BF16 && dtype != DT_FP16) { *why = "RoPE supports bf16 and fp16"; return false; }
  if (D < 2 || D % 2 != 0) { *why = "head size D must be even"; return false; }
  out->unroll = 1;
  if (variant == 1) {  // GENERIC
    out->kind = KK_ROPE_WARP;
    out->vec = 1;
    if (dtype == DT_BF16) out->fn = qknorm ? (const void*)rope_generic_kernel<DT_BF16, true>
                                           : (const void*)rope_generic_kernel<DT_BF16, false>;
    else out->fn = qknorm ? (const void*)rope_generic_kernel<DT_FP16, true>
                          : (const void*)rope_generic_kernel<DT_FP16, false>;
    return true;
  }
  out->kind = KK_ROPE_HALFWARP;
  out->vec = 8;
  if (dtype == DT_BF16) out->fn = qknorm ? pick_vec<DT_BF16, true>(D) : pick_vec<DT_BF16, false>(D);
  else out->fn = qknorm ? pick_vec<DT_FP16, true>(D) : pick_vec<DT_FP16, false>(D);
  if (!out->fn) { *why = "vector RoPE supports D in {64, 128, 256}"; return false; }
  return true;
}

}  // namespace trident
