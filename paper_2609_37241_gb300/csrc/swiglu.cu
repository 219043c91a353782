// swiglu.cu -- SwiGLU activation: out = silu(g) * u, silu(g) = g / (1 + exp(-g)).
//
// silu is one of the paper's kernel benchmarks (§4.1) and its largest per-operator gain
// (§4.2); the gated form is how an LLM's MLP uses it. A pure stream: 6 bytes moved per
// bf16 element, one exp. The vector kernel tiles each row into blocks of
// UNROLL * 256 vectors and issues every load of a tile before the first use; grid.y walks
// the rows. The generic kernel is a flat grid-stride loop with scalar accesses.
#include "device_common.cuh"

namespace trident {

constexpr int kSwigluUnroll = 2;

template <int DT, int UNROLL>
__global__ void __launch_bounds__(kThreads) swiglu_vec_kernel(const SwigluParams p) {
  pdl_trigger();
  const int64_t v0 = (int64_t)blockIdx.x * UNROLL * kThreads;
  if (p.prefetch) swiglu_prefetch<DT, UNROLL>(p, blockIdx.y, v0, threadIdx.x);
  pdl_wait();
  for (int64_t row = blockIdx.y; row < p.T; row += gridDim.y)
    swiglu_tile<DT, UNROLL>(p, row, v0, threadIdx.x);
}

template <int DT>
__global__ void __launch_bounds__(kThreads) swiglu_generic_kernel(const SwigluParams p) {
  pdl_prologue();
  const int64_t total = p.T * p.I;
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < total; i += stride) {
    const int64_t row = i / p.I;
    const int64_t col = i - row * p.I;
    const float g = load_elem<DT>(p.g, row * p.g_rs + col);
    const float u = load_elem<DT>(p.u, row * p.u_rs + col);
    store_elem<DT>(p.out, row * p.o_rs + col, silu_mul<DT>(g, u));
  }
}

bool swiglu_kernel(int32_t dtype, int32_t variant, int64_t I, KernelEntry* out, const char** why) {
  if (dtype != DT_BF16 && dtype != DT_FP16 && dtype != DT_FP32) { *why = "dtype"; return false; }
  if (I < 1) { *why = "I must be >= 1"; return false; }
  const int eb = dtype == DT_FP32 ? 4 : 2;
  if (variant == 1) {  // GENERIC
    out->kind = KK_SWIGLU_FLAT;
    out->vec = 1;
    out->unroll = 1;
    out->fn = dtype == DT_BF16 ? (const void*)swiglu_generic_kernel<DT_BF16>
            : dtype == DT_FP16 ? (const void*)swiglu_generic_kernel<DT_FP16>
                               : (const void*)swiglu_generic_kernel<DT_FP32>;
    return true;
  }
  if ((I * eb) % 16 != 0) { *why = "vector SwiGLU needs I * elem_size % 16 == 0"; return false; }
  out->kind = KK_SWIGLU_TILE;
  out->vec = 16 / eb;
  out->unroll = kSwigluUnroll;
  out->fn = dtype == DT_BF16 ? (const void*)swiglu_vec_kernel<DT_BF16, kSwigluUnroll>
          : dtype == DT_FP16 ? (const void*)swiglu_vec_kernel<DT_FP16, kSwigluUnroll>
                             : (const void*)swiglu_vec_kernel<DT_FP32, kSwigluUnroll>;
  return true;
}

}  // namespace trident
