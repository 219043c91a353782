// device_common.cuh -- device-side building blocks shared by the kernels of this library.
//
// Every kernel is memory bound (a few flops per byte), so the building blocks are about
// moving bytes: 16-byte vector loads and stores per thread, fp32 math in registers,
// warp-shuffle reductions. Each kernel starts with the programmatic-dependent-launch
// pair (trigger, then wait) so that, when launched with programmatic stream
// serialisation, the next kernel's launch overlaps this one while every global memory
// access still waits for the previous kernel to finish; between the two, small grids
// prefetch their first lines into L2 (prefetch_l2).
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "internal.h"

namespace trident {

constexpr uint32_t kErrPos = 0x1u;  // TRIDENT_DEVERR_POS
constexpr uint32_t kErrTimeout = 0x2u;  // TRIDENT_DEVERR_TIMEOUT

__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_prologue() {
  pdl_trigger();
  pdl_wait();
}

// L2 prefetch of one line. Kernels issue prefetches of the lines they read first between
// pdl_trigger and pdl_wait, while the previous kernel of the stream may still run: a
// prefetch changes no value that a later load returns (the loads come after the wait), it
// only lets the DRAM fetch overlap the previous kernel's tail and the launch handoff. The
// host enables it (params.prefetch) for grids of at most one block per SM launched with
// programmatic stream serialisation: a grid that fills the GPU becomes resident only as the
// previous kernel's blocks retire, and its prefetches then compete with that kernel.
__device__ __forceinline__ void prefetch_l2(const void* p) { asm volatile("prefetch.L2 [%0];" :: "l"(p)); }

template <int DT> struct Act;
template <> struct Act<DT_BF16> { static constexpr int VE = 8; static constexpr int BYTES = 2; };
template <> struct Act<DT_FP16> { static constexpr int VE = 8; static constexpr int BYTES = 2; };
template <> struct Act<DT_FP32> { static constexpr int VE = 4; static constexpr int BYTES = 4; };

// ---------------------------------------------------------------- 16-byte vectors
__device__ __forceinline__ uint4 ldg16(const void* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }
__device__ __forceinline__ uint4 ld16(const void* p) { return *reinterpret_cast<const uint4*>(p); }
__device__ __forceinline__ void st16(void* p, uint4 v) { *reinterpret_cast<uint4*>(p) = v; }
__device__ __forceinline__ float4 ldg_f4(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }

template <int DT> __device__ __forceinline__ void unpack(const uint4& v, float* f);
template <> __device__ __forceinline__ void unpack<DT_BF16>(const uint4& v, float* f) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}
template <> __device__ __forceinline__ void unpack<DT_FP16>(const uint4& v, float* f) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    __half2 h;
    memcpy(&h, &w[i], 4);
    float2 ff = __half22float2(h);
    f[2 * i] = ff.x;
    f[2 * i + 1] = ff.y;
  }
}
template <> __device__ __forceinline__ void unpack<DT_FP32>(const uint4& v, float* f) {
  f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
  f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
}

template <int DT> __device__ __forceinline__ uint4 pack(const float* f);
template <> __device__ __forceinline__ uint4 pack<DT_BF16>(const float* f) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    __nv_bfloat162 b = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
    memcpy(&w[i], &b, 4);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}
template <> __device__ __forceinline__ uint4 pack<DT_FP16>(const float* f) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    __half2 h = __floats2half2_rn(f[2 * i], f[2 * i + 1]);
    memcpy(&w[i], &h, 4);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}
template <> __device__ __forceinline__ uint4 pack<DT_FP32>(const float* f) {
  return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]),
                    __float_as_uint(f[3]));
}

// ---------------------------------------------------------------- scalar elements
template <int DT> __device__ __forceinline__ float load_elem(const void* p, int64_t i);
template <> __device__ __forceinline__ float load_elem<DT_BF16>(const void* p, int64_t i) {
  return __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(p)[i]);
}
template <> __device__ __forceinline__ float load_elem<DT_FP16>(const void* p, int64_t i) {
  return __half2float(reinterpret_cast<const __half*>(p)[i]);
}
template <> __device__ __forceinline__ float load_elem<DT_FP32>(const void* p, int64_t i) {
  return reinterpret_cast<const float*>(p)[i];
}
template <int DT> __device__ __forceinline__ void store_elem(void* p, int64_t i, float v);
template <> __device__ __forceinline__ void store_elem<DT_BF16>(void* p, int64_t i, float v) {
  reinterpret_cast<__nv_bfloat16*>(p)[i] = __float2bfloat16_rn(v);
}
template <> __device__ __forceinline__ void store_elem<DT_FP16>(void* p, int64_t i, float v) {
  reinterpret_cast<__half*>(p)[i] = __float2half_rn(v);
}
template <> __device__ __forceinline__ void store_elem<DT_FP32>(void* p, int64_t i, float v) {
  reinterpret_cast<float*>(p)[i] = v;
}
// Rounds v to the activation type and back (the value a store would hold).
template <int DT> __device__ __forceinline__ float round_act(float v);
template <> __device__ __forceinline__ float round_act<DT_BF16>(float v) {
  return __bfloat162float(__float2bfloat16_rn(v));
}
template <> __device__ __forceinline__ float round_act<DT_FP16>(float v) {
  return __half2float(__float2half_rn(v));
}
template <> __device__ __forceinline__ float round_act<DT_FP32>(float v) { return v; }

__device__ __forceinline__ const char* row_ptr(const void* base, int64_t row, int64_t rs, int eb) {
  return reinterpret_cast<const char*>(base) + row * rs * eb;
}
__device__ __forceinline__ char* row_ptr(void* base, int64_t row, int64_t rs, int eb) {
  return reinterpret_cast<char*>(base) + row * rs * eb;
}

// ---------------------------------------------------------------- reductions
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Sum over the block; every thread gets the same total (same summation order).
// `red` holds kThreads/32 floats and must not be reused until after a barrier.
__device__ __forceinline__ float block_sum(float v, float* red) {
  constexpr int NW = kThreads / 32;
  v = warp_sum(v);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  float t = 0.f;
#pragma unroll
  for (int i = 0; i < NW; ++i) t += red[i];
  return t;
}

// ---------------------------------------------------------------- RoPE angles
// sin and cos of the angle pos * f, with f = fhi + flo (a double-float split of
// theta^(-2i/D) made in fp64 on the host). The product is kept as ah + al (al holds the
// exact rounding error of pos * fhi, from one fma, plus pos * flo); ah is reduced modulo
// 2 pi with the Cody-Waite method (Cody and Waite, "Software Manual for the Elementary
// Functions", 1980) using 2 pi = A + B + C, A with 12 significant bits so that k * A is
// exact for k < 4096, i.e. angles up to about 25700 rad; the reduced angle, within about
// [-pi, pi], goes to the hardware sine/cosine (absolute error about 2^-21).
constexpr float kInv2Pi = 0.159154936671257019f;     // 1 / (2 pi), rounded to fp32
constexpr float k2PiA = 6.283203125f;                // 2 pi to 12 significant bits (3217/512)
constexpr float k2PiB = -1.78178197529632598e-05f;   // fp32(2 pi - A)
constexpr float k2PiC = -6.60559822986128669e-13f;   // fp32(2 pi - A - B)

__device__ __forceinline__ void rope_sincos(float pos, float fhi, float flo, float* s, float* c) {
  const float ah = pos * fhi;
  const float al = fmaf(pos, fhi, -ah) + pos * flo;
  const float k = rintf(ah * kInv2Pi);
  float r = fmaf(-k, k2PiA, ah);
  r = fmaf(-k, k2PiB, r);
  r = fmaf(-k, k2PiC, r);
  __sincosf(r + al, s, c);
}

// ---------------------------------------------------------------- RoPE head-row
// n / d for a 32-bit n and a divisor d known per launch, from the host's round-up multiplier
// m and shift l for d (div_magic; Granlund and Montgomery, "Division by invariant integers
// using multiplication", 1994): (h + ((n - h) >> 1)) >> (l - 1) with h = umulhi(n, m), exact
// for every 32-bit n; l = 0 stands for d = 1. A division by a runtime divisor is otherwise a
// long instruction sequence (64-bit: several times longer).
__device__ __forceinline__ uint32_t fast_div(uint32_t n, uint32_t m, int32_t l) {
  if (l == 0) return n;
  const uint32_t h = __umulhi(n, m);
  return (h + ((n - h) >> 1)) >> (l - 1);
}

// Token and head-row of a unit: unit = t * NH + hh (units below 2^32, every grid in practice,
// by fast_div).
__device__ __forceinline__ void rope_unit_split(const RopeParams& p, int64_t unit, int64_t* t, int* hh) {
  if (unit <= 0xffffffffll) {
    const uint32_t u = (uint32_t)unit;
    const uint32_t q = fast_div(u, p.nh_magic, p.nh_shift);
    *t = q;
    *hh = (int)(u - q * (uint32_t)p.NH);
  } else {
    *t = unit / p.NH;
    *hh = (int)(unit - *t * p.NH);
  }
}

// q, k or v head of head-row hh of a token.
__device__ __forceinline__ void rope_head_of(const RopeParams& p, int hh, int* h, bool* is_q, bool* is_v) {
  *is_v = hh >= p.Hq + p.Hkv;
  *is_q = hh < p.Hq;
  *h = *is_q ? hh : (*is_v ? hh - p.Hq - p.Hkv : hh - p.Hq);
}

// L2 prefetch of head-row `unit`'s source line(s) and position (lanes on a line boundary).
template <int DT, int D>
__device__ __forceinline__ void rope_prefetch(const RopeParams& p, int64_t unit, int lane) {
  constexpr int VE = Act<DT>::VE;
  constexpr int EB = Act<DT>::BYTES;
  if (unit >= p.T * p.NH || (lane * VE * EB) % 128 != 0) return;
  int64_t t;
  int hh, h;
  bool is_q, is_v;
  rope_unit_split(p, unit, &t, &hh);
  rope_head_of(p, hh, &h, &is_q, &is_v);
  const char* src = is_q ? row_ptr(p.q, t, p.q_rs, EB) : is_v ? row_ptr(p.v, t, p.v_rs, EB)
                                                             : row_ptr(p.k, t, p.k_rs, EB);
  prefetch_l2(src + ((int64_t)h * D + lane * VE) * EB);
  if (lane == 0) prefetch_l2(p.pos + t);
}

// The (hi, lo) frequencies of lane `lane` of a head-row, for its VE elements
// i = (lane % (LPH/2)) * VE + e. The frequency table belongs to the version: it is written
// once, when the version is registered (and the registration waits for that copy), and is
// never written again, so kernels read it before griddepcontrol.wait, while the previous
// kernel of the stream still runs. Every RoPE lane of a grid reads the same few lines of
// the table; read after the wait, those reads queue behind each other at the L2 slices
// that hold the lines, on the critical path of every RoPE block. The same lane position
// has the same frequencies in every head-row, so a lane loads them once.
template <int DT, int D>
__device__ __forceinline__ void rope_lane_freqs(const float2* inv_freq, int lane, float* fq) {
  constexpr int VE = Act<DT>::VE;
  constexpr int HALF = D / VE / 2;
  const float* fr = reinterpret_cast<const float*>(inv_freq) + 2 * (lane % HALF) * VE;
#pragma unroll
  for (int q = 0; q < VE / 2; ++q) {
    const float4 f4 = ldg_f4(fr + 4 * q);
    fq[4 * q] = f4.x; fq[4 * q + 1] = f4.y; fq[4 * q + 2] = f4.z; fq[4 * q + 3] = f4.w;
  }
}

// One head-row (token t, head hh) handled by LPH = D / VE consecutive lanes, each lane
// owning VE consecutive elements. Rotate-half pairs element i with i + D/2, i.e. lane
// l with lane l ^ (LPH/2). hh < Hq: q head (rotated in place); hh < Hq + Hkv: k head
// (rotated into k_cache); else v head (copied into v_cache). fq holds the lane's
// frequencies (rope_lane_freqs). A head-row is processed in two steps: rope_row_load issues
// every load it needs -- the row slice, the position and the norm weights -- and
// rope_row_finish uses them, so a lane group that owns several head-rows issues all of
// their loads before it waits for any (one memory round trip in all).
template <int DT, int D>
__device__ __forceinline__ void rope_row_where(const RopeParams& p, int64_t unit, int64_t* t, int* h,
                                               bool* is_q, bool* is_v) {
  int hh;
  rope_unit_split(p, unit, t, &hh);
  rope_head_of(p, hh, h, is_q, is_v);
}

template <int DT, int D, bool QKNORM>
__device__ __forceinline__ void rope_row_load(const RopeParams& p, int64_t unit, int lane, uint4* raw,
                                              int32_t* pos, float* gg) {
  constexpr int VE = Act<DT>::VE;
  constexpr int EB = Act<DT>::BYTES;
  int64_t t;
  int h;
  bool is_q, is_v;
  rope_row_where<DT, D>(p, unit, &t, &h, &is_q, &is_v);
  const char* src = is_q ? row_ptr(p.q, t, p.q_rs, EB) : is_v ? row_ptr(p.v, t, p.v_rs, EB)
                                                             : row_ptr(p.k, t, p.k_rs, EB);
  src += ((int64_t)h * D + lane * VE) * EB;
  *raw = is_q ? ld16(src) : ldg16(src);
  *pos = __ldg(p.pos + t);
  if (QKNORM && !is_v) {
    const float* gam = (is_q ? p.gamma_q : p.gamma_k) + lane * VE;
#pragma unroll
    for (int q = 0; q < VE / 4; ++q) {
      const float4 g4 = ldg_f4(gam + 4 * q);
      gg[4 * q] = g4.x; gg[4 * q + 1] = g4.y; gg[4 * q + 2] = g4.z; gg[4 * q + 3] = g4.w;
    }
  }
}

template <int DT, int D, bool QKNORM>
__device__ __forceinline__ void rope_row_finish(const RopeParams& p, int64_t unit, int lane, const uint4 raw,
                                                const int32_t pos, const float* gg, const float* fq) {
  constexpr int VE = Act<DT>::VE;
  constexpr int LPH = D / VE;
  constexpr int HALF = LPH / 2;
  constexpr int EB = Act<DT>::BYTES;
  static_assert(LPH >= 2 && LPH <= 32 && (LPH & (LPH - 1)) == 0, "head size");
  const unsigned group_mask =
      (LPH == 32) ? 0xffffffffu : (((1u << LPH) - 1u) << ((threadIdx.x & 31) & ~(LPH - 1)));
  int64_t t;
  int h;
  bool is_q, is_v;
  rope_row_where<DT, D>(p, unit, &t, &h, &is_q, &is_v);
  if (pos < 0 || (int64_t)pos >= p.S) {
    if (lane == 0) atomicOr(p.err, kErrPos);
    return;
  }
  if (is_v) {  // bit copy into the cache
    st16(reinterpret_cast<char*>(p.v_cache) + (((int64_t)h * p.S + pos) * D + lane * VE) * EB, raw);
    return;
  }
  float x[VE];
  unpack<DT>(raw, x);
  if (QKNORM) {
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
  const bool low = lane < HALF;
  const float fpos = (float)pos;
  float y[VE];
#pragma unroll
  for (int e = 0; e < VE; ++e) {
    float sn, cs;
    rope_sincos(fpos, fq[2 * e], fq[2 * e + 1], &sn, &cs);
    // low half: x_i c - x_{i+D/2} s;  high half: x_{i+D/2} c + x_i s
    y[e] = low ? fmaf(x[e], cs, -other[e] * sn) : fmaf(x[e], cs, other[e] * sn);
  }
  if (is_q) {
    st16(row_ptr(p.q, t, p.q_rs, EB) + ((int64_t)h * D + lane * VE) * EB, pack<DT>(y));
  } else {
    char* dst = reinterpret_cast<char*>(p.k_cache) + (((int64_t)h * p.S + pos) * D + lane * VE) * EB;
    st16(dst, pack<DT>(y));
  }
}

template <int DT, int D, bool QKNORM>
__device__ __forceinline__ void rope_head_row(const RopeParams& p, int64_t unit, int lane, const float* fq) {
  uint4 raw;
  int32_t pos;
  float gg[Act<DT>::VE];
  rope_row_load<DT, D, QKNORM>(p, unit, lane, &raw, &pos, gg);
  rope_row_finish<DT, D, QKNORM>(p, unit, lane, raw, pos, gg, fq);
}

// K head-rows per lane group, for grids several waves long: lane group g (of G = 256 / LPH)
// of RoPE block rb owns the units rb * G * K + g + G * j, j < K -- with NH = 48 and K = 3 one
// token's q, k and v rows. A block then moves K times the bytes for the same fixed costs,
// which pays where blocks queue for slots (a 1024-token layer 39.7 -> 34.8 us) and not where
// a block's own latency is the step (one wave: slower per block). Rows of one token share
// the position and so every angle: the lane computes its sines and cosines once, for the
// token of the first row, and again only for a row of another token (NH not a multiple of
// G), reloading its frequencies then. All K rows' loads are issued before any is used.
template <int DT, int D, bool QKNORM, int K>
__device__ __forceinline__ void rope_rows(const RopeParams& p, const int64_t rb, const int lane, const int g,
                                          const float* fq) {
  constexpr int VE = Act<DT>::VE;
  constexpr int LPH = D / VE;
  constexpr int HALF = LPH / 2;
  constexpr int EB = Act<DT>::BYTES;
  constexpr int G = kThreads / LPH;
  const unsigned group_mask =
      (LPH == 32) ? 0xffffffffu : (((1u << LPH) - 1u) << ((threadIdx.x & 31) & ~(LPH - 1)));
  const int64_t nunits = p.T * p.NH;
  const int64_t u0 = rb * (int64_t)(G * K) + g;
  if (u0 >= nunits) return;
  // rows u0 + G * j: token and head-row of the first by one division, the rest by stepping
  int64_t t0;
  int hh0;
  rope_unit_split(p, u0, &t0, &hh0);
  uint4 raw[K];
  {
    int64_t t = t0;
    int hh = hh0;
#pragma unroll
    for (int j = 0; j < K; ++j) {
      if (j > 0) {
        hh += G;
        while (hh >= p.NH) { hh -= p.NH; ++t; }
      }
      if (u0 + (int64_t)G * j < nunits) {
        int h;
        bool is_q, is_v;
        rope_head_of(p, hh, &h, &is_q, &is_v);
        const char* src = is_q ? row_ptr(p.q, t, p.q_rs, EB) : is_v ? row_ptr(p.v, t, p.v_rs, EB)
                                                                   : row_ptr(p.k, t, p.k_rs, EB);
        src += ((int64_t)h * D + lane * VE) * EB;
        raw[j] = is_q ? ld16(src) : ldg16(src);
      }
    }
  }
  const int32_t pos0 = __ldg(p.pos + t0);
  float sn[VE], cs[VE];
#pragma unroll
  for (int e = 0; e < VE; ++e) rope_sincos((float)pos0, fq[2 * e], fq[2 * e + 1], &sn[e], &cs[e]);
  const bool low = lane < HALF;
  int64_t t = t0;
  int hh = hh0;
#pragma unroll
  for (int j = 0; j < K; ++j) {
    if (j > 0) {
      hh += G;
      while (hh >= p.NH) { hh -= p.NH; ++t; }
    }
    if (u0 + (int64_t)G * j >= nunits) break;
    int h;
    bool is_q, is_v;
    rope_head_of(p, hh, &h, &is_q, &is_v);
    // units ascend, so once a row belongs to a later token every following row does too
    const bool same = t == t0;
    const int32_t pos = same ? pos0 : __ldg(p.pos + t);
    if (pos < 0 || (int64_t)pos >= p.S) {
      if (lane == 0) atomicOr(p.err, kErrPos);
      continue;
    }
    if (is_v) {  // bit copy into the cache
      st16(reinterpret_cast<char*>(p.v_cache) + (((int64_t)h * p.S + pos) * D + lane * VE) * EB, raw[j]);
      continue;
    }
    float x[VE];
    unpack<DT>(raw[j], x);
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
    if (!same) {
      float f2[2 * VE];
      rope_lane_freqs<DT, D>(p.inv_freq, lane, f2);
#pragma unroll
      for (int e = 0; e < VE; ++e) rope_sincos((float)pos, f2[2 * e], f2[2 * e + 1], &sn[e], &cs[e]);
    }
    float y[VE];
#pragma unroll
    for (int e = 0; e < VE; ++e)
      y[e] = low ? fmaf(x[e], cs[e], -other[e] * sn[e]) : fmaf(x[e], cs[e], other[e] * sn[e]);
    if (is_q) {
      st16(row_ptr(p.q, t, p.q_rs, EB) + ((int64_t)h * D + lane * VE) * EB, pack<DT>(y));
    } else {
      st16(reinterpret_cast<char*>(p.k_cache) + (((int64_t)h * p.S + pos) * D + lane * VE) * EB, pack<DT>(y));
    }
  }
}

// ---------------------------------------------------------------- SwiGLU tile
template <int DT> __device__ __forceinline__ float silu_mul(float g, float u);
// bf16/fp16 outputs: fast exp and divide (relative error ~1e-6, far below the output ulp;
// for g below about -87 the result is -0, the limit of g * sigmoid(g)).
template <> __device__ __forceinline__ float silu_mul<DT_BF16>(float g, float u) {
  return __fdividef(g, 1.0f + __expf(-g)) * u;
}
template <> __device__ __forceinline__ float silu_mul<DT_FP16>(float g, float u) {
  return __fdividef(g, 1.0f + __expf(-g)) * u;
}
// fp32 outputs: full-precision exp and IEEE division.
template <> __device__ __forceinline__ float silu_mul<DT_FP32>(float g, float u) {
  return g / (1.0f + expf(-g)) * u;
}

// L2 prefetch of the gate and up lines of one SwiGLU tile (threads on a line boundary).
template <int DT, int UNROLL>
__device__ __forceinline__ void swiglu_prefetch(const SwigluParams& p, int64_t row, int64_t v0,
                                                int tid) {
  constexpr int VE = Act<DT>::VE;
  constexpr int EB = Act<DT>::BYTES;
  if ((tid & 7) != 0 || row >= p.T) return;
  const int64_t nvec = p.I / VE;
  const uint4* g = reinterpret_cast<const uint4*>(row_ptr(p.g, row, p.g_rs, EB));
  const uint4* u = reinterpret_cast<const uint4*>(row_ptr(p.u, row, p.u_rs, EB));
#pragma unroll
  for (int k = 0; k < UNROLL; ++k) {
    const int64_t vi = v0 + (int64_t)k * kThreads + tid;
    if (vi < nvec) {
      prefetch_l2(g + vi);
      prefetch_l2(u + vi);
    }
  }
}

// One tile of UNROLL * kThreads vectors of one row, starting at vector index v0.
template <int DT, int UNROLL>
__device__ __forceinline__ void swiglu_tile(const SwigluParams& p, int64_t row, int64_t v0,
                                            int tid) {
  constexpr int VE = Act<DT>::VE;
  constexpr int EB = Act<DT>::BYTES;
  const int64_t nvec = p.I / VE;
  const uint4* g = reinterpret_cast<const uint4*>(row_ptr(p.g, row, p.g_rs, EB));
  const uint4* u = reinterpret_cast<const uint4*>(row_ptr(p.u, row, p.u_rs, EB));
  uint4* o = reinterpret_cast<uint4*>(row_ptr(p.out, row, p.o_rs, EB));
  uint4 gv[UNROLL], uv[UNROLL];
#pragma unroll
  for (int k = 0; k < UNROLL; ++k) {
    const int64_t vi = v0 + (int64_t)k * kThreads + tid;
    if (vi < nvec) {
      gv[k] = ldg16(g + vi);
      uv[k] = ldg16(u + vi);
    }
  }
#pragma unroll
  for (int k = 0; k < UNROLL; ++k) {
    const int64_t vi = v0 + (int64_t)k * kThreads + tid;
    if (vi < nvec) {
      float gf[VE], uf[VE], of[VE];
      unpack<DT>(gv[k], gf);
      unpack<DT>(uv[k], uf);
#pragma unroll
      for (int e = 0; e < VE; ++e) of[e] = silu_mul<DT>(gf[e], uf[e]);
      st16(o + vi, pack<DT>(of));
    }
  }
}

}  // namespace trident
