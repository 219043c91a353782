// noalloc.cu -- RoPE + KV-cache append that allocates nothing.
//
// The SCM path keeps two pieces of scratch memory in device allocations it makes itself:
// the frequency table of a RoPE version (cudaMalloc at registration) and the device
// status word (cudaMalloc at creation). Some callers cannot allocate device memory at
// all: a serving engine that has handed every byte of HBM to its own pool, or code running
// where a cudaMalloc would synchronise the device and stall other streams. For them,
// trident_rope_kv_noalloc runs the same vector RoPE/KV kernel with its scratch in a
// file-scope static device array of fixed size, so no call allocates anything (no
// cudaMalloc, no cudaFree, no allocating library routine).
//
// Scratch layout (kScratchBytes = 256 + 1024 bytes, held by every GPU that loads the
// library until the process exits): bytes [0, 4) the status word, bytes [256, end) the
// frequency table, (hi, lo) fp32 pairs of theta^(-2i/D) for i < D/2, at most kMaxPairs =
// 128 pairs (D <= 256). Every call first launches one small kernel on the caller's stream
// that clears the status word and rewrites the table for its own (theta, D), then the
// RoPE kernel. The host keeps no record of what the array holds, so nothing on the host
// can disagree with the device: whatever ran on the stream before, and whether or not an
// earlier launch failed, the RoPE kernel reads the table its own call wrote. The RoPE
// kernel reads its frequencies before griddepcontrol.wait; it is launched here without
// programmatic serialisation, so it starts only after the preparing kernel has finished.
#include <cuda_runtime.h>

#include <cmath>
#include <mutex>

#include "device_common.cuh"
#include "trident_scm.h"

namespace trident {
namespace {

constexpr size_t kTableOffset = 256;
constexpr int64_t kMaxPairs = 128;
constexpr size_t kScratchBytes = kTableOffset + size_t(kMaxPairs) * sizeof(float2);
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

struct DeviceScratch {
  std::once_flag once;
  cudaError_t setup_error = cudaSuccess;
  unsigned char* addr = nullptr;  // device address of g_scratch on this device
};
DeviceScratch g_dev[kMaxDevices];

// Prepares the scratch for one call: clears the status word and writes the frequency
// table f_i = theta^(-2i/D) in fp64, stored as (fp32(f), fp32(f - hi)), for i < D/2.
__global__ void prepare_scratch(uint32_t* status, float2* tab, int32_t D, double theta) {
  const int i = threadIdx.x;
  if (i == 0) *status = 0u;
  if (i < D / 2) {
    const double f = pow(theta, -2.0 * (double)i / (double)D);
    const float hi = (float)f;
    tab[i] = make_float2(hi, (float)(f - (double)hi));
  }
}

}  // namespace
}  // namespace trident

using namespace trident;

extern "C" __attribute__((visibility("default"))) int32_t trident_rope_kv_noalloc(
    const trident_args* args, void* stream, uint32_t* out_status) {
  RopeParams p;
  int32_t dtype = 0;
  bool qknorm = false;
  int32_t st = prepare_rope_args(args, &p, &dtype, &qknorm);
  if (st != TRIDENT_OK) return st;
  const int dev = args->t[0].device;
  if (dev >= kMaxDevices) return internal_fail(TRIDENT_ERR_INVALID, "device ordinal too large");
  int cur = -1;
  if (cudaGetDevice(&cur) != cudaSuccess || cur != dev)
    return internal_fail(TRIDENT_ERR_INVALID, "the tensors' device must be the current device");
  if (p.D / 2 > kMaxPairs)
    return internal_fail(TRIDENT_ERR_INVALID,
                         "D/2 exceeds the static scratch maximum of 128 frequency pairs (D <= 256)");
  KernelEntry ke;
  const char* why = "";
  if (!rope_kernel(dtype, TRIDENT_VARIANT_VECTOR, p.D, qknorm, &ke, &why))
    return internal_fail(TRIDENT_ERR_INVALID, why);

  // one-time set-up on this device: the device address of the static array
  DeviceScratch& ds = g_dev[dev];
  std::call_once(ds.once, [&] {
    void* a = nullptr;
    ds.setup_error = cudaGetSymbolAddress(&a, g_scratch);
    ds.addr = static_cast<unsigned char*>(a);
  });
  if (ds.setup_error != cudaSuccess || !ds.addr)
    return internal_fail(TRIDENT_ERR_CUDA, "cudaGetSymbolAddress of the scratch array failed");

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint32_t* status = reinterpret_cast<uint32_t*>(ds.addr);
  float2* table = reinterpret_cast<float2*>(ds.addr + kTableOffset);
  prepare_scratch<<<1, (unsigned)kMaxPairs, 0, s>>>(status, table, p.D, args->rope_theta);
  if (cudaGetLastError() != cudaSuccess)
    return internal_fail(TRIDENT_ERR_CUDA, "scratch preparation launch failed");
  p.inv_freq = table;
  p.err = status;
  const int64_t upb = rope_units_per_block(p.D, 2);
  const int64_t blocks = (p.T * p.NH + upb - 1) / upb;
  void* kargs[1] = {&p};
  if (cudaLaunchKernel(ke.fn, dim3((unsigned)(blocks < 0x7fffffff ? blocks : 0x7fffffff)), dim3(kThreads),
                       kargs, 0, s) != cudaSuccess)
    return internal_fail(TRIDENT_ERR_CUDA, "RoPE launch failed");
  if (out_status &&
      cudaMemcpyAsync(out_status, status, sizeof(uint32_t), cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return internal_fail(TRIDENT_ERR_CUDA, "status copy failed");
  if (cudaGetLastError() != cudaSuccess) return internal_fail(TRIDENT_ERR_CUDA, "launch error");
  return TRIDENT_OK;
}
