// rope.cu -- RoPE on q/k with KV-cache append, optionally after per-head q/k RMSNorm.
//
// Work unit: one head-row (token t, head hh) of D elements; per token there are
// NH = Hq + 2*Hkv of them (q heads, k heads, v heads). The vector kernel gives each unit
// D/VE lanes (16 lanes for D = 128 in bf16) so that a unit is one 256-byte coalesced
// access, and exchanges the rotate-half partner with one xor-shuffle per element.
// The generic kernel gives each unit one warp and scalar accesses (any alignment, any
// even D). Calls of many tokens take the bulk-copy kernel (rope_bulk_kernel): a few tokens
// per block, their rows staged in shared memory by cp.async.bulk on an mbarrier, each
// token's angles computed once. All compute (cos, sin) of pos * theta^(-2i/D) in the kernel
// from the version's double-float frequency table [D/2], which the host splits from fp64 at
// registration.
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

// Calls of many tokens (the vector kernel's grid several waves long): a block takes up to
// kRopeBulkTokens tokens. One thread issues, per token, three bulk copies (cp.async.bulk: a
// token's q, k and v head-rows are each contiguous, D elements per head) into shared memory,
// completing on one mbarrier, while the block's threads compute the tokens' D/2 pairs
// (sin, cos) of pos * theta^(-2i/D) once into shared memory (rope_sincos: the values the vector
// kernel's lanes compute for each of their elements, so outputs are bit-identical); lanes then
// rotate head-rows out of shared memory and store them.
//
// Why not the vector kernel: each of a token's 2 (Hq + Hkv) q/k head-rows recomputes all of
// its elements' angles there, about half of its instructions, and its register-resident rows
// (64 registers, four blocks per SM of 4 KB of reads each) keep too few bytes in flight: at
// 4096 Llama tokens it reaches 0.35 of the measured copy bandwidth, this kernel 0.58 (8192:
// 0.37 and 0.71). Measured and dropped: lane groups of three register-resident head-rows with
// the angles in shared memory (0.51 / 0.57), and four or eight tokens per block (0.51 / 0.64,
// 0.46 / 0.51: a block copies, then computes, so heavier blocks idle the memory longer).
//
// The wait is bounded (bp.first_wait_polls try_wait polls, kBulkWaitPolls by default): a
// block whose copies have not landed by then sets TRIDENT_DEVERR_TIMEOUT, waits (again
// bounded) for them and returns without writing.
#ifndef TRIDENT_ROPE_BULK_TOKENS
#define TRIDENT_ROPE_BULK_TOKENS 2
#endif
constexpr int kRopeBulkTokens = TRIDENT_ROPE_BULK_TOKENS;

template <int DT, int D, bool QKNORM>
__global__ void __launch_bounds__(kThreads) rope_bulk_kernel(const RopeBulkParams bp) {
  const RopeParams& p = bp.rp;
  constexpr int TB = kRopeBulkTokens;
  constexpr int VE = Act<DT>::VE;
  constexpr int LPH = D / VE;
  constexpr int HALF = LPH / 2;
  constexpr int EB = Act<DT>::BYTES;
  constexpr int G = kThreads / LPH;
  constexpr int NF = D / 2;
  static_assert(LPH >= 2 && LPH <= 32 && (LPH & (LPH - 1)) == 0, "head size");
  extern __shared__ __align__(128) unsigned char s_rows[];  // [TB][NH][D] elements
  __shared__ __align__(16) float s_sin[TB][NF];
  __shared__ __align__(16) float s_cos[TB][NF];
  __shared__ int32_t s_pos[TB];
  __shared__ __align__(8) unsigned long long bar;
  const int tid = threadIdx.x;
  const int lane = tid % LPH;
  const int g = tid / LPH;
  const unsigned group_mask =
      (LPH == 32) ? 0xffffffffu : (((1u << LPH) - 1u) << ((tid & 31) & ~(LPH - 1)));
  const bool low = lane < HALF;
  const int f0 = (lane % HALF) * VE;
  const int64_t tb = (int64_t)blockIdx.x * TB;
  const int ntok = (int)(p.T - tb < TB ? p.T - tb : TB);
  const uint32_t qb = (uint32_t)(p.Hq * D * EB), kb = (uint32_t)(p.Hkv * D * EB);
  const uint32_t tok_bytes = qb + 2 * kb;
  const uint32_t bar_a = (uint32_t)__cvta_generic_to_shared(&bar);
  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" :: "r"(bar_a) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  pdl_trigger();
  if (p.prefetch) {  // the block's row lines into L2 while the previous kernel finishes
    const int lines = (int)(tok_bytes / 128);
    for (int i = tid; i < ntok * lines; i += kThreads) {
      const int tk = i / lines, l = i - tk * lines;
      const uint32_t off = (uint32_t)l * 128;
      const int64_t t = tb + tk;
      const char* src = off < qb ? row_ptr(p.q, t, p.q_rs, EB) + off
                                 : off < qb + kb ? row_ptr(p.k, t, p.k_rs, EB) + (off - qb)
                                                 : row_ptr(p.v, t, p.v_rs, EB) + (off - qb - kb);
      prefetch_l2(src);
    }
  }
  pdl_wait();
  __syncthreads();  // the barrier is initialised before anyone waits on it
  if (tid == 0) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
                 :: "r"(bar_a), "r"((uint32_t)ntok * tok_bytes) : "memory");
    for (int tk = 0; tk < ntok; ++tk) {
      const int64_t t = tb + tk;
      const uint32_t dst = (uint32_t)__cvta_generic_to_shared(s_rows + (size_t)tk * tok_bytes);
      asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                   :: "r"(dst), "l"(row_ptr(p.q, t, p.q_rs, EB)), "r"(qb), "r"(bar_a) : "memory");
      asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                   :: "r"(dst + qb), "l"(row_ptr(p.k, t, p.k_rs, EB)), "r"(kb), "r"(bar_a) : "memory");
      asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                   :: "r"(dst + qb + kb), "l"(row_ptr(p.v, t, p.v_rs, EB)), "r"(kb), "r"(bar_a) : "memory");
    }
  }
  for (int idx = tid; idx < ntok * NF; idx += kThreads) {  // the tokens' angles, once each
    const int tk = idx / NF, i = idx % NF;
    const int32_t pos = __ldg(p.pos + tb + tk);
    if (i == 0) s_pos[tk] = pos;
    float sn = 0.f, cs = 1.f;
    if (pos >= 0 && (int64_t)pos < p.S) {
      const float2 f = __ldg(p.inv_freq + i);
      rope_sincos((float)pos, f.x, f.y, &sn, &cs);
    }
    s_sin[tk][i] = sn;
    s_cos[tk][i] = cs;
  }
  auto landed = [&](uint32_t polls) -> bool {
    uint32_t done = 0;
    for (uint32_t it = 0; it < polls && !done; ++it)
      asm volatile("{ .reg .pred q; mbarrier.try_wait.parity.shared::cta.b64 q, [%1], 0; selp.u32 %0, 1, 0, q; }"
                   : "=r"(done) : "r"(bar_a) : "memory");
    return done != 0;
  };
  const bool ok = landed(bp.first_wait_polls);
  if (__syncthreads_or(!ok)) {  // one decision for the whole block (also publishes the angles)
    if (tid == 0 && p.err) atomicOr(p.err, kErrTimeout);
    if (!ok) landed(kBulkWaitPolls);  // a second bounded wait for the copies before the block exits
    return;
  }
  // head-rows u = g + G * i of the block: token tk = u / NH, head-row hh = u % NH, by stepping
  int tk = 0, hh = g;
  while (hh >= p.NH) { hh -= p.NH; ++tk; }
  for (int u = g; u < ntok * p.NH; u += G) {
    if (u != g) {
      hh += G;
      while (hh >= p.NH) { hh -= p.NH; ++tk; }
    }
    const int64_t t = tb + tk;
    const int32_t pos = s_pos[tk];
    if (pos < 0 || (int64_t)pos >= p.S) {
      if (lane == 0) atomicOr(p.err, kErrPos);
      continue;
    }
    const uint4 raw = *reinterpret_cast<const uint4*>(s_rows + ((size_t)tk * p.NH + hh) * (D * EB) + lane * 16);
    int h;
    bool is_q, is_v;
    rope_head_of(p, hh, &h, &is_q, &is_v);
    if (is_v) {  // bit copy into the cache
      st16(reinterpret_cast<char*>(p.v_cache) + (((int64_t)h * p.S + pos) * D + lane * VE) * EB, raw);
      continue;
    }
    float x[VE];
    unpack<DT>(raw, x);
    if (QKNORM) {
      const float* gam = (is_q ? p.gamma_q : p.gamma_k) + lane * VE;
      float gg[VE];
#pragma unroll
      for (int q = 0; q < VE / 4; ++q) {
        const float4 g4 = ldg_f4(gam + 4 * q);
        gg[4 * q] = g4.x; gg[4 * q + 1] = g4.y; gg[4 * q + 2] = g4.z; gg[4 * q + 3] = g4.w;
      }
      float ss = 0.f;
#pragma unroll
      for (int e = 0; e < VE; ++e) ss = fmaf(x[e], x[e], ss);
#pragma unroll
      for (int o = LPH / 2; o > 0; o >>= 1) ss += __shfl_xor_sync(group_mask, ss, o, LPH);
      const float inv = rsqrtf(ss * p.inv_D + p.eps);
#pragma unroll
      for (int e = 0; e < VE; ++e) x[e] = x[e] * inv * gg[e];
    }
    float other[VE];
#pragma unroll
    for (int e = 0; e < VE; ++e) other[e] = __shfl_xor_sync(group_mask, x[e], HALF, LPH);
    float sn[VE], cs[VE];
#pragma unroll
    for (int q = 0; q < VE / 4; ++q) {
      const float4 a = *reinterpret_cast<const float4*>(&s_sin[tk][f0 + 4 * q]);
      const float4 b = *reinterpret_cast<const float4*>(&s_cos[tk][f0 + 4 * q]);
      sn[4 * q] = a.x; sn[4 * q + 1] = a.y; sn[4 * q + 2] = a.z; sn[4 * q + 3] = a.w;
      cs[4 * q] = b.x; cs[4 * q + 1] = b.y; cs[4 * q + 2] = b.z; cs[4 * q + 3] = b.w;
    }
    float y[VE];
#pragma unroll
    for (int e = 0; e < VE; ++e)
      y[e] = low ? fmaf(x[e], cs[e], -other[e] * sn[e]) : fmaf(x[e], cs[e], other[e] * sn[e]);
    if (is_q) {
      st16(row_ptr(p.q, t, p.q_rs, EB) + ((int64_t)h * D + lane * VE) * EB, pack<DT>(y));
    } else {
      st16(reinterpret_cast<char*>(p.k_cache) + (((int64_t)h * p.S + pos) * D + lane * VE) * EB,
           pack<DT>(y));
    }
  }
}

// Calls of at least this many tokens take rope_bulk_kernel (Llama heads: 512 tokens 8.3
// against 9.5 us; from 256 tokens down the vector kernel is as fast or faster).
#ifndef TRIDENT_ROPE_BULK_MIN_TOKENS
#define TRIDENT_ROPE_BULK_MIN_TOKENS 512
#endif

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

template <int DT, bool QK>
static const void* pick_bulk(int32_t D) {
  if (D == 64) return (const void*)rope_bulk_kernel<DT, 64, QK>;
  if (D == 128) return (const void*)rope_bulk_kernel<DT, 128, QK>;
  if (D == 256) return (const void*)rope_bulk_kernel<DT, 256, QK>;
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
  if (dtype == DT_BF16) out->fn_large = qknorm ? pick_bulk<DT_BF16, true>(D) : pick_bulk<DT_BF16, false>(D);
  else out->fn_large = qknorm ? pick_bulk<DT_FP16, true>(D) : pick_bulk<DT_FP16, false>(D);
  out->large_rows = TRIDENT_ROPE_BULK_MIN_TOKENS;
  out->rows = kRopeBulkTokens;  // tokens per block
  return true;
}

}  // namespace trident
