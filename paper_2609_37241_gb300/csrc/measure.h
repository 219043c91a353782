// measure.h -- parameters of the measurement kernels behind trident_launch_floor and
// trident_copy_floor. Neither is on the dispatch path: they give the floors the hot path's
// kernels are read against.
#pragma once
#include <stdint.h>

namespace trident {

// A copy with the traffic of a layer-chain launch and none of its arithmetic: block b of the
// grid reads the 16-byte vectors [b * rpb, (b + 1) * rpb) of src and writes [b * wpb, ...) of
// dst (rpb, wpb: the vector counts split evenly over the grid), every written vector the XOR
// of the vectors its thread read.
struct CopyFloorParams {
  const void* src;
  void* dst;
  int64_t nr, nw;    // 16-byte vectors read / written by the whole grid
  int32_t prefetch;  // 1: each block prefetches its read lines into L2 before the PDL wait
};

const void* copy_floor_entry();

}  // namespace trident
