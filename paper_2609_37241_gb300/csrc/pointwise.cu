// pointwise.cu -- FlagGems-style pointwise operators: silu, add, neg, masked_fill.
//
// These are operators of the paper's kernel benchmark (§4.1), where silu and masked_fill
// show its largest per-call gains (§4.2): the device work is a few bytes per element and
// the host orchestration around the launch dominates. The vector kernel tiles each row into
// UNROLL * 256 16-byte vectors, all loads of a tile issued before the first use (grid.y
// walks the rows); the generic kernel is a flat grid-stride loop with scalar accesses.
#include "device_common.cuh"
#include "measure.h"

namespace trident {

constexpr int kPwUnroll = 2;

template <int DT, int OP>
__device__ __forceinline__ float pw_apply(float a, float b, uint8_t m, float scalar) {
  if (OP == PW_SILU) return silu_mul<DT>(a, 1.0f);
  if (OP == PW_ADD) return a + b;
  if (OP == PW_NEG) return -a;
  return m ? scalar : a;  // PW_MASKED_FILL
}

template <int DT, int OP, int UNROLL>
__global__ void __launch_bounds__(kThreads) pointwise_vec_kernel(const PointwiseParams p) {
  pdl_trigger();
  constexpr int VE = Act<DT>::VE;
  constexpr int EB = Act<DT>::BYTES;
  const int64_t nvec = p.W / VE;
  const int64_t v0 = (int64_t)blockIdx.x * UNROLL * kThreads;
  if (p.prefetch && (threadIdx.x & 7) == 0 && blockIdx.y < p.T) {  // the first row's tile (prefetch_l2)
#pragma unroll
    for (int k = 0; k < UNROLL; ++k) {
      const int64_t vi = v0 + (int64_t)k * kThreads + threadIdx.x;
      if (vi < nvec) {
        prefetch_l2(reinterpret_cast<const uint4*>(row_ptr(p.a, blockIdx.y, p.a_rs, EB)) + vi);
        if (OP == PW_ADD) prefetch_l2(reinterpret_cast<const uint4*>(row_ptr(p.b, blockIdx.y, p.b_rs, EB)) + vi);
      }
    }
  }
  pdl_wait();
  for (int64_t row = blockIdx.y; row < p.T; row += gridDim.y) {
    const uint4* a = reinterpret_cast<const uint4*>(row_ptr(p.a, row, p.a_rs, EB));
    const uint4* b = reinterpret_cast<const uint4*>(row_ptr(p.b, row, p.b_rs, EB));
    const uint8_t* m = p.mask + row * p.m_rs;
    uint4* y = reinterpret_cast<uint4*>(row_ptr(p.y, row, p.y_rs, EB));
    uint4 av[UNROLL], bv[UNROLL];
    uint8_t mv[UNROLL][VE];
#pragma unroll
    for (int k = 0; k < UNROLL; ++k) {
      const int64_t vi = v0 + (int64_t)k * kThreads + threadIdx.x;
      if (vi < nvec) {
        av[k] = ldg16(a + vi);
        if (OP == PW_ADD) bv[k] = ldg16(b + vi);
        if (OP == PW_MASKED_FILL) {
          if (VE == 8) {
            const uint2 w = __ldg(reinterpret_cast<const uint2*>(m + vi * VE));
            memcpy(mv[k], &w, 8);
          } else {
            const uint32_t w = __ldg(reinterpret_cast<const uint32_t*>(m + vi * VE));
            memcpy(mv[k], &w, 4);
          }
        }
      }
    }
#pragma unroll
    for (int k = 0; k < UNROLL; ++k) {
      const int64_t vi = v0 + (int64_t)k * kThreads + threadIdx.x;
      if (vi < nvec) {
        float af[VE], bf[VE], of[VE];
        unpack<DT>(av[k], af);
        if (OP == PW_ADD) unpack<DT>(bv[k], bf);
#pragma unroll
        for (int e = 0; e < VE; ++e)
          of[e] = pw_apply<DT, OP>(af[e], OP == PW_ADD ? bf[e] : 0.f,
                                   OP == PW_MASKED_FILL ? mv[k][e] : (uint8_t)0, p.scalar);
        if (OP == PW_MASKED_FILL) {  // keep unmasked elements bit for bit (NaN payloads too)
          uint4 out = pack<DT>(of);
          uint16_t* o16 = reinterpret_cast<uint16_t*>(&out);
          const uint16_t* a16 = reinterpret_cast<const uint16_t*>(&av[k]);
          uint32_t* o32 = reinterpret_cast<uint32_t*>(&out);
          const uint32_t* a32 = reinterpret_cast<const uint32_t*>(&av[k]);
#pragma unroll
          for (int e = 0; e < VE; ++e) {
            if (!mv[k][e]) {
              if (EB == 2) o16[e] = a16[e];
              else o32[e] = a32[e];
            }
          }
          st16(y + vi, out);
        } else {
          st16(y + vi, pack<DT>(of));
        }
      }
    }
  }
}

template <int DT, int OP>
__global__ void __launch_bounds__(kThreads) pointwise_generic_kernel(const PointwiseParams p) {
  pdl_prologue();
  const int64_t total = p.T * p.W;
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < total; i += stride) {
    const int64_t row = i / p.W;
    const int64_t col = i - row * p.W;
    if (OP == PW_MASKED_FILL && !p.mask[row * p.m_rs + col]) {  // bit copy of x
      if (Act<DT>::BYTES == 2)
        reinterpret_cast<uint16_t*>(p.y)[row * p.y_rs + col] =
            reinterpret_cast<const uint16_t*>(p.a)[row * p.a_rs + col];
      else
        reinterpret_cast<uint32_t*>(p.y)[row * p.y_rs + col] =
            reinterpret_cast<const uint32_t*>(p.a)[row * p.a_rs + col];
      continue;
    }
    const float a = load_elem<DT>(p.a, row * p.a_rs + col);
    const float b = OP == PW_ADD ? load_elem<DT>(p.b, row * p.b_rs + col) : 0.f;
    store_elem<DT>(p.y, row * p.y_rs + col, pw_apply<DT, OP>(a, b, (uint8_t)1, p.scalar));
  }
}

template <int DT>
static const void* pick(int32_t op, bool vec) {
#define TRIDENT_PW(OPV)                                                                      \
  if (op == OPV) return vec ? (const void*)pointwise_vec_kernel<DT, OPV, kPwUnroll>            \
                            : (const void*)pointwise_generic_kernel<DT, OPV>;
  TRIDENT_PW(PW_SILU)
  TRIDENT_PW(PW_ADD)
  TRIDENT_PW(PW_NEG)
  TRIDENT_PW(PW_MASKED_FILL)
#undef TRIDENT_PW
  return nullptr;
}

// Latency-floor probe (trident_launch_floor): a kernel that does nothing but take part in
// programmatic dependent launch like every kernel of the library.
__global__ void empty_kernel() {
  pdl_trigger();
  pdl_wait();
}

const void* empty_kernel_entry() { return (const void*)empty_kernel; }

// Copy-floor probe (trident_copy_floor), see CopyFloorParams. With prefetch, a block's read
// lines go to L2 between the launch trigger and the wait, as the layer chain's blocks do.
__global__ void __launch_bounds__(kThreads) copy_floor_kernel(const CopyFloorParams p) {
  pdl_trigger();
  const int64_t g = gridDim.x;
  const int64_t rpb = (p.nr + g - 1) / g, wpb = (p.nw + g - 1) / g;
  const int64_t r0 = (int64_t)blockIdx.x * rpb, w0 = (int64_t)blockIdx.x * wpb;
  const uint4* src = static_cast<const uint4*>(p.src);
  uint4* dst = static_cast<uint4*>(p.dst);
  if (p.prefetch) {
    for (int64_t i = (int64_t)threadIdx.x * 8; i < rpb; i += (int64_t)kThreads * 8)
      if (r0 + i < p.nr) prefetch_l2(src + r0 + i);
  }
  pdl_wait();
  uint4 acc = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll 4
  for (int64_t i = threadIdx.x; i < rpb; i += kThreads) {
    if (r0 + i < p.nr) {
      const uint4 v = ldg16(src + r0 + i);
      acc.x ^= v.x; acc.y ^= v.y; acc.z ^= v.z; acc.w ^= v.w;
    }
  }
  for (int64_t j = threadIdx.x; j < wpb; j += kThreads)
    if (w0 + j < p.nw) st16(dst + w0 + j, acc);
}

const void* copy_floor_entry() { return (const void*)copy_floor_kernel; }

bool pointwise_kernel(int32_t op, int32_t dtype, int32_t variant, int64_t W, KernelEntry* out,
                      const char** why) {
  if (dtype != DT_BF16 && dtype != DT_FP16 && dtype != DT_FP32) { *why = "dtype"; return false; }
  if (W < 1) { *why = "W must be >= 1"; return false; }
  const int eb = dtype == DT_FP32 ? 4 : 2;
  const bool vec = variant != 1;
  if (vec && (W * eb) % 16 != 0) { *why = "vector pointwise needs W * elem_size % 16 == 0"; return false; }
  out->kind = vec ? KK_SWIGLU_TILE : KK_SWIGLU_FLAT;  // same grid rules as SwiGLU
  out->vec = vec ? 16 / eb : 1;
  out->unroll = vec ? kPwUnroll : 1;
  out->fn = dtype == DT_BF16 ? pick<DT_BF16>(op, vec) : dtype == DT_FP16 ? pick<DT_FP16>(op, vec)
                                                                         : pick<DT_FP32>(op, vec);
  if (!out->fn) { *why = "unknown pointwise op"; return false; }
  return true;
}

}  // namespace trident
