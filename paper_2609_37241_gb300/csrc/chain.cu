// chain.cu -- one decoder layer's non-GEMM chain in a single launch.
//
//   add+RMSNorm(h, r0) -> x1, r1;  [q/k RMSNorm +] RoPE(q, k) + KV append;
//   add+RMSNorm(attn_out, r1) -> x2, r2;  SwiGLU(g, u) -> o
//
// The only data dependency inside the chain is r1 feeding the second norm, and it is
// row-local: the block that produces row t of r1 keeps it in registers and runs the
// second norm of row t itself. So no grid-wide barrier is needed; the launch is a
// horizontal fusion where blocks take different roles:
//   norm     two add+RMSNorm steps, one or two blocks per token (the longest per-block
//            work)
//   RoPE     RoPE/KV head-rows, (256 / (D/8)) per block, or three times that (three rows
//            of one token per lane group) on grids several waves long
//   SwiGLU   tiles of one row each, twice as wide on grids of many waves
// Grids are role-major ([norms | RoPE | SwiGLU], so the longest blocks start first), the
// smallest ones token-major (chain_block_tok), so that consecutive blocks mix roles. Under
// programmatic dependent launch, role-major grids that fit the resident slots with their
// own norm blocks run the LATE entry, whose short blocks trigger the next launch only at
// their exit (the next grid is then placed one norm block per SM). One launch replaces
// four, which is what matters at decode sizes, where each step moves well under a
// microsecond of HBM traffic. chain_step_kernel runs several independent calls' grids in
// one launch.
#include "device_common.cuh"

namespace trident {


// Norm role: part `part` (< SPLIT) of token `row`'s two add+RMSNorm steps.
template <int DT, int VPT, int SPLIT>
__device__ __forceinline__ void chain_norm(const ChainParams& c, const int64_t row, const int part) {
  constexpr int EB = Act<DT>::BYTES;
  constexpr int VE = Act<DT>::VE;
  const int tid = threadIdx.x;
  {
    // Both norms of one token. The second residual sum s2 = attn_out + round(s1) is
    // elementwise, so both sums of squares are formed before any reduction and reduced
    // together: one barrier. With a_split = 2 two CTAs share a token: each reads the whole
    // row (the sums need it) but loads only its half of both gamma vectors and writes only
    // its half of the four outputs, so no SM carries the token's full 56 KB. s1 and s2 are
    // recomputed from the packed inputs after the reduction rather than kept in registers.
    __shared__ float2 red[kThreads / 32];
    constexpr int PP = VPT / SPLIT;  // vectors per thread this CTA writes
    static_assert(VPT % SPLIT == 0, "split");
    const AddNormParams& n1 = c.n1;
    const AddNormParams& n2 = c.n2;
    uint4 hv[VPT], rv[VPT], av[VPT];
    float ga[PP][VE], gm[PP][VE];
    const uint4* hp = reinterpret_cast<const uint4*>(row_ptr(n1.x, row, n1.x_rs, EB));
    const uint4* rp = reinterpret_cast<const uint4*>(row_ptr(n1.r, row, n1.r_rs, EB));
    const uint4* ap = reinterpret_cast<const uint4*>(row_ptr(n2.x, row, n2.x_rs, EB));
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      const int64_t vi = (int64_t)v * kThreads + tid;
      hv[v] = ldg16(hp + vi);
      rv[v] = ldg16(rp + vi);
      av[v] = ldg16(ap + vi);
      if (v / PP == part) {
#pragma unroll
        for (int q = 0; q < VE / 4; ++q) {
          const float4 g1 = ldg_f4(n1.gamma + vi * VE + 4 * q);
          const float4 g2 = ldg_f4(n2.gamma + vi * VE + 4 * q);
          float* a = ga[v % PP];
          float* m = gm[v % PP];
          a[4 * q] = g1.x; a[4 * q + 1] = g1.y; a[4 * q + 2] = g1.z; a[4 * q + 3] = g1.w;
          m[4 * q] = g2.x; m[4 * q + 1] = g2.y; m[4 * q + 2] = g2.z; m[4 * q + 3] = g2.w;
        }
      }
    }
    uint4* r1p = reinterpret_cast<uint4*>(row_ptr(n1.r_out, row, n1.ro_rs, EB));
    uint4* r2p = reinterpret_cast<uint4*>(row_ptr(n2.r_out, row, n2.ro_rs, EB));
    float ss1 = 0.f, ss2 = 0.f;
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      const int64_t vi = (int64_t)v * kThreads + tid;
      float hf[VE], rf[VE], af[VE], s1[VE], s2[VE];
      unpack<DT>(hv[v], hf);
      unpack<DT>(rv[v], rf);
      unpack<DT>(av[v], af);
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        s1[e] = hf[e] + rf[e];
        ss1 = fmaf(s1[e], s1[e], ss1);
      }
      const uint4 r1 = pack<DT>(s1);
      float r1f[VE];
      unpack<DT>(r1, r1f);
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        s2[e] = af[e] + r1f[e];
        ss2 = fmaf(s2[e], s2[e], ss2);
      }
      if (v / PP == part) {
        st16(r1p + vi, r1);              // r1, then r2: in place (r2 = r1) keeps r2
        st16(r2p + vi, pack<DT>(s2));
      }
    }
    float2 sums = make_float2(ss1, ss2);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      sums.x += __shfl_xor_sync(0xffffffffu, sums.x, o);
      sums.y += __shfl_xor_sync(0xffffffffu, sums.y, o);
    }
    if ((tid & 31) == 0) red[tid >> 5] = sums;
    __syncthreads();
    float2 tot = make_float2(0.f, 0.f);
#pragma unroll
    for (int i = 0; i < kThreads / 32; ++i) {
      tot.x += red[i].x;
      tot.y += red[i].y;
    }
    const float inv1 = rsqrtf(tot.x * n1.inv_H + n1.eps);
    const float inv2 = rsqrtf(tot.y * n2.inv_H + n2.eps);
    uint4* x1p = reinterpret_cast<uint4*>(row_ptr(n1.y, row, n1.y_rs, EB));
    uint4* x2p = reinterpret_cast<uint4*>(row_ptr(n2.y, row, n2.y_rs, EB));
#pragma unroll
    for (int v = 0; v < VPT; ++v) {
      if (v / PP != part) continue;
      const int64_t vi = (int64_t)v * kThreads + tid;
      float hf[VE], rf[VE], af[VE], s1[VE], y1[VE], y2[VE];
      unpack<DT>(hv[v], hf);
      unpack<DT>(rv[v], rf);
      unpack<DT>(av[v], af);
#pragma unroll
      for (int e = 0; e < VE; ++e) s1[e] = hf[e] + rf[e];
      float r1f[VE];
      unpack<DT>(pack<DT>(s1), r1f);
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        y1[e] = s1[e] * inv1 * ga[v % PP][e];
        y2[e] = (af[e] + r1f[e]) * inv2 * gm[v % PP][e];
      }
      st16(x1p + vi, pack<DT>(y1));
      st16(x2p + vi, pack<DT>(y2));
    }
  }
}

// RoPE role: RoPE block rb (< nB), i.e. head-rows [rb * UPB, (rb + 1) * UPB) with UPB =
// rope_k * 256 / LPH (rope_rows with rope_k = 3 on grids several waves long); fq holds the
// lane's frequencies (rope_lane_freqs).
// Only the one-CTA-per-token entries (SPLIT 1: in-place calls, and grids too large for one
// wave) carry the rope_rows path, so the others keep their registers.
template <int DT, int D, bool QKNORM, bool ROWS3>
__device__ __forceinline__ void chain_rope(const ChainParams& c, const int64_t rb, const float* fq) {
  constexpr int LPH = D / Act<DT>::VE;
  if (ROWS3 && c.rope_k == 3) {
    rope_rows<DT, D, QKNORM, 3>(c.rope, rb, threadIdx.x % LPH, threadIdx.x / LPH, fq);
    return;
  }
  const int64_t unit = rb * (kThreads / LPH) + threadIdx.x / LPH;
  if (unit < c.rope.T * c.rope.NH) rope_head_row<DT, D, QKNORM>(c.rope, unit, threadIdx.x % LPH, fq);
}

// Before the PDL wait: the RoPE lane frequencies of a RoPE block (other roles load none).
template <int DT, int D>
__device__ __forceinline__ void chain_rope_freqs(const ChainParams& c, const bool is_rope, float* fq) {
  if (is_rope) rope_lane_freqs<DT, D>(c.rope.inv_freq, threadIdx.x % (D / Act<DT>::VE), fq);
}

// SwiGLU role: column tile `col_tile` of row `row`, SWU x 256 16-byte vectors of g and of u
// (kChainSwigluUnroll for one call's grid, kChainStepSwigluUnroll for a whole step's).
template <int DT, int SWU>
__device__ __forceinline__ void chain_swiglu(const ChainParams& c, const int64_t row, const int64_t col_tile) {
  swiglu_tile<DT, SWU>(c.sw, row, col_tile * SWU * kThreads, threadIdx.x);
}

// Row of SwiGLU tile `tile`. A single call's kernel divides by the host's multiplier
// (fast_div: the 64-token layer step 3.32 -> 3.29 us); the whole-step kernel (STEP), which
// reads its call's parameters at a block-varying index, keeps the division (the multiplier
// measured 3-5 % slower there).
template <bool STEP>
__device__ __forceinline__ int64_t swiglu_tile_row(const ChainParams& c, const int64_t tile) {
  if (STEP) return tile / c.sw_tiles_per_row;
  return fast_div((uint32_t)tile, c.sw_magic, c.sw_shift);
}

// Block b of one call's role-major grid (b < nA + nB + nC): [norms | RoPE | SwiGLU].
template <int DT, int VPT, int SPLIT, int D, bool QKNORM, int SWU, bool STEP>
__device__ __forceinline__ void chain_block(const ChainParams& c, const int b, const float* fq) {
  if (b < c.nA) {
    const int64_t row = b / SPLIT;
    chain_norm<DT, VPT, SPLIT>(c, row, b - (int)row * SPLIT);
  } else if (b < c.nA + c.nB) {
    chain_rope<DT, D, QKNORM, SPLIT == 1>(c, b - c.nA, fq);
  } else {
    const int64_t tile = b - c.nA - c.nB;
    if (tile >= c.sw_tiles) return;
    const int64_t row = swiglu_tile_row<STEP>(c, tile);
    chain_swiglu<DT, SWU>(c, row, tile - row * c.sw_tiles_per_row);
  }
}

// Token-major grid (SPLIT + rope_per_tok + sw_tiles_per_row, T): block (q, t) is token t's
// q-th block -- its norm parts, then its RoPE blocks, then its SwiGLU tiles. Blocks are
// dispatched x first, so consecutive blocks belong to one token and any few of them carry a
// mix of roles: under programmatic launch the blocks of a grid land on SMs as the previous
// kernel's blocks retire, several consecutive blocks on one SM, and a role-major order can
// give one SM four norm blocks (160 KB) while another gets 24 KB. Both indices come from
// special registers, so no remapped index stays live in a register through the body.
template <int DT, int VPT, int SPLIT, int D, bool QKNORM>
__device__ __forceinline__ void chain_block_tok(const ChainParams& c, const float* fq) {
  const int q = blockIdx.x;
  if (q < SPLIT) {
    chain_norm<DT, VPT, SPLIT>(c, blockIdx.y, q);
  } else if (q < SPLIT + c.rope_per_tok) {
    chain_rope<DT, D, QKNORM, false>(c, (int64_t)blockIdx.y * c.rope_per_tok + (q - SPLIT), fq);
  } else {
    chain_swiglu<DT, kChainSwigluUnroll>(c, blockIdx.y, q - SPLIT - c.rope_per_tok);
  }
}

// L2 prefetch of the lines a block reads first -- the norm rows, the RoPE head-rows and
// positions, the SwiGLU tile -- one prefetch per 128-byte line, between the launch trigger
// and the PDL wait (see prefetch_l2).
// A token's SPLIT norm blocks share its rows' lines: part p prefetches vectors v = p mod SPLIT.
template <int DT, int VPT, int SPLIT>
__device__ __forceinline__ void norm_prefetch(const ChainParams& c, const int64_t row, const int part) {
  constexpr int EB = Act<DT>::BYTES;
  constexpr int VE = Act<DT>::VE;
  const int tid = threadIdx.x;
  if ((tid & 3) != 0) return;  // a line is 8 threads' 16-byte row vectors, 4 threads' gamma floats
  const uint4* hp = reinterpret_cast<const uint4*>(row_ptr(c.n1.x, row, c.n1.x_rs, EB));
  const uint4* rp = reinterpret_cast<const uint4*>(row_ptr(c.n1.r, row, c.n1.r_rs, EB));
  const uint4* ap = reinterpret_cast<const uint4*>(row_ptr(c.n2.x, row, c.n2.x_rs, EB));
#pragma unroll
  for (int v = 0; v < VPT; ++v) {
    if (v % SPLIT != part) continue;
    const int64_t vi = (int64_t)v * kThreads + tid;
    if ((tid & 7) == 0) {
      prefetch_l2(hp + vi);
      prefetch_l2(rp + vi);
      prefetch_l2(ap + vi);
    }
    prefetch_l2(c.n1.gamma + vi * VE);  // this part's half of both norms' weights
    prefetch_l2(c.n2.gamma + vi * VE);
  }
}

// The token's RoPE head-rows (its q, k and v rows), prefetched by its norm blocks: part p of
// SPLIT takes head-rows [p * ceil(NH / SPLIT), ...), one thread per 128-byte line.
template <int DT, int SPLIT, int D>
__device__ __forceinline__ void norm_rope_prefetch(const ChainParams& c, const int64_t row, const int part) {
  constexpr int VE = Act<DT>::VE;
  constexpr int EB = Act<DT>::BYTES;
  constexpr int LINES = (D * EB + 127) / 128;      // 128-byte lines per head-row
  constexpr int LANES_PER_LINE = 128 / (VE * EB);  // lanes of a head-row per line
  const int per = (c.rope.NH + SPLIT - 1) / SPLIT;
  const int k = threadIdx.x / LINES;
  if (k >= per || part * per + k >= c.rope.NH) return;
  rope_prefetch<DT, D>(c.rope, row * c.rope.NH + part * per + k, (threadIdx.x % LINES) * LANES_PER_LINE);
}

// prefetch == 1: every block its own first lines; prefetch == 2: only the norm blocks, which
// take their token's rows and its RoPE head-rows (the other roles' own prefetches, issued by
// hundreds of blocks while the previous kernel finishes, measured slower).
template <int DT, int VPT, int SPLIT, int D, int SWU, bool STEP>
__device__ __forceinline__ void chain_prefetch(const ChainParams& c, const int b) {
  constexpr int LPH = D / Act<DT>::VE;
  const int tid = threadIdx.x;
  if (b < c.nA) {
    norm_prefetch<DT, VPT, SPLIT>(c, b / SPLIT, b % SPLIT);
    if (c.prefetch == 2) norm_rope_prefetch<DT, SPLIT, D>(c, b / SPLIT, b % SPLIT);
  } else if (c.prefetch == 2) {
    return;
  } else if (b < c.nA + c.nB) {
    if (c.rope_k != 1) return;  // several head-rows per lane group: grids too long to prefetch
    rope_prefetch<DT, D>(c.rope, (int64_t)(b - c.nA) * (kThreads / LPH) + tid / LPH, tid % LPH);
  } else {
    const int64_t tile = b - c.nA - c.nB;
    if (tile >= c.sw_tiles) return;
    const int64_t row = swiglu_tile_row<STEP>(c, tile);
    swiglu_prefetch<DT, SWU>(c.sw, row, (tile - row * c.sw_tiles_per_row) * SWU * kThreads, tid);
  }
}

template <int DT, int VPT, int SPLIT, int D>
__device__ __forceinline__ void chain_prefetch_tok(const ChainParams& c) {
  constexpr int LPH = D / Act<DT>::VE;
  const int tid = threadIdx.x, q = blockIdx.x;
  if (q < SPLIT) {
    norm_prefetch<DT, VPT, SPLIT>(c, blockIdx.y, q);
  } else if (q < SPLIT + c.rope_per_tok) {
    const int64_t rb = (int64_t)blockIdx.y * c.rope_per_tok + (q - SPLIT);
    rope_prefetch<DT, D>(c.rope, rb * (kThreads / LPH) + tid / LPH, tid % LPH);
  } else {
    swiglu_prefetch<DT, kChainSwigluUnroll>(
        c.sw, blockIdx.y, (int64_t)(q - SPLIT - c.rope_per_tok) * kChainSwigluUnroll * kThreads, tid);
  }
}

// Four resident blocks per SM for H 4096 (64 registers): the 64-token grid (576 blocks)
// then fits one wave on 152 SMs; a fifth register would drop it to three blocks per SM.
// LATE (role-major grids only): only the norm blocks trigger the next launch at their start,
// the RoPE and SwiGLU blocks at their exit. The next launch then starts once this grid's
// short blocks are gone, and its blocks are placed while several slots per SM are free, one
// norm block per SM, instead of filling each slot the moment it frees (up to four norm
// blocks on one SM). The trigger is otherwise the kernel's first instruction: even one
// parameter read ahead of it measured 0.05 us slower per launch.
template <int DT, int VPT, int SPLIT, int D, bool QKNORM, bool LATE, int SWU>
__global__ void __launch_bounds__(kThreads, VPT == 2 ? 4 : 2)
    chain_kernel(const __grid_constant__ ChainParams c) {
  if (!LATE || (int)blockIdx.x < c.nA) pdl_trigger();
  float fq[2 * Act<DT>::VE];
  if (!LATE && SWU == kChainSwigluUnroll && c.tok_grid) {
    if (c.prefetch) chain_prefetch_tok<DT, VPT, SPLIT, D>(c);
    chain_rope_freqs<DT, D>(c, (int)blockIdx.x >= SPLIT && (int)blockIdx.x < SPLIT + c.rope_per_tok, fq);
    pdl_wait();
    chain_block_tok<DT, VPT, SPLIT, D, QKNORM>(c, fq);
  } else {
    // A role-major grid fills the GPU: its RoPE blocks become resident only as the previous
    // kernel's blocks retire, and their frequency loads measured faster after the wait.
    const int b = blockIdx.x;
    if (c.prefetch) chain_prefetch<DT, VPT, SPLIT, D, SWU, false>(c, b);
    pdl_wait();
    chain_rope_freqs<DT, D>(c, b >= c.nA && b < c.nA + c.nB, fq);
    chain_block<DT, VPT, SPLIT, D, QKNORM, SWU, false>(c, b, fq);
  }
}

// Several independent calls in one launch: a block finds its call by binary search over
// the first-block table (uniform across the block, so the parameter reads broadcast).
// ROLE (one-CTA-per-token steps of one to two waves): role-major block order over the whole
// step -- every call's norm blocks, then every call's RoPE blocks, then every call's SwiGLU
// tiles -- so that the longer blocks fill the first wave (a separate entry: the call-major
// kernel measured about 1 % slower with this branch in it).
template <int DT, int VPT, int SPLIT, int D, bool QKNORM, bool ROLE>
__global__ void __launch_bounds__(kThreads, VPT == 2 ? 4 : 2)
    chain_step_kernel(const __grid_constant__ ChainStepParams p) {
  pdl_trigger();
  const int b = blockIdx.x;
  int lo = 0, hi = p.n - 1;
  if constexpr (ROLE) {
    const int r = b < p.role_first[1][0] ? 0 : (b < p.role_first[2][0] ? 1 : 2);
    const int32_t* f = p.role_first[r];
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (b >= f[mid]) lo = mid;
      else hi = mid - 1;
    }
    const ChainParams& c = p.c[lo];
    const int bl = b - f[lo] + (r == 0 ? 0 : (r == 1 ? c.nA : c.nA + c.nB));
    float fq[2 * Act<DT>::VE];
    chain_rope_freqs<DT, D>(c, r == 1, fq);
    pdl_wait();
    chain_block<DT, VPT, SPLIT, D, QKNORM, kChainStepSwigluUnroll, true>(c, bl, fq);
  } else {
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (b >= p.first[mid]) lo = mid;
      else hi = mid - 1;
    }
    const ChainParams& c = p.c[lo];
    const int bl = b - p.first[lo];
    if (c.prefetch) chain_prefetch<DT, VPT, SPLIT, D, kChainStepSwigluUnroll, true>(c, bl);
    float fq[2 * Act<DT>::VE];
    chain_rope_freqs<DT, D>(c, bl >= c.nA && bl < c.nA + c.nB, fq);
    pdl_wait();
    chain_block<DT, VPT, SPLIT, D, QKNORM, kChainStepSwigluUnroll, true>(c, bl, fq);
  }
}

template <int DT, int SPLIT, bool QK>
static void pick(int64_t H, const void** one, const void** step, const void** extra, const void** role) {
  // extra: for SPLIT 2 the LATE entry, for SPLIT 1 the wide-tile entry; role: for SPLIT 1
  // the role-major whole-step entry
  constexpr int per = kThreads * Act<DT>::VE;
  if (H == per * 2) {
    *one = (const void*)chain_kernel<DT, 2, SPLIT, 128, QK, false, kChainSwigluUnroll>;
    *step = (const void*)chain_step_kernel<DT, 2, SPLIT, 128, QK, false>;
    if constexpr (SPLIT == 2) *extra = (const void*)chain_kernel<DT, 2, SPLIT, 128, QK, true, kChainSwigluUnroll>;
    else *extra = (const void*)chain_kernel<DT, 2, SPLIT, 128, QK, false, kChainWideSwigluUnroll>;
    if constexpr (SPLIT == 1) *role = (const void*)chain_step_kernel<DT, 2, SPLIT, 128, QK, true>;
  } else if (H == per * 4) {
    *one = (const void*)chain_kernel<DT, 4, SPLIT, 128, QK, false, kChainSwigluUnroll>;
    *step = (const void*)chain_step_kernel<DT, 4, SPLIT, 128, QK, false>;
    if constexpr (SPLIT == 2) *extra = (const void*)chain_kernel<DT, 4, SPLIT, 128, QK, true, kChainSwigluUnroll>;
    else *extra = (const void*)chain_kernel<DT, 4, SPLIT, 128, QK, false, kChainWideSwigluUnroll>;
    if constexpr (SPLIT == 1) *role = (const void*)chain_step_kernel<DT, 4, SPLIT, 128, QK, true>;
  }
}

bool chain_kernel(int32_t dtype, int64_t H, int32_t D, bool qknorm, KernelEntry* out,
                  const char** why) {
  if (dtype != DT_BF16 && dtype != DT_FP16) { *why = "layer chain supports bf16 and fp16"; return false; }
  if (D != 128) { *why = "layer chain supports D = 128"; return false; }
  out->kind = KK_CHAIN;
  out->vec = 8;
  out->unroll = kChainSwigluUnroll;
  // fn: two blocks per token for the norms; fn_late: the same with the late launch trigger;
  // fn_inplace: one block per token (calls whose outputs overwrite inputs, and grids too
  // large for one wave); fn_wide: fn_inplace with wider SwiGLU tiles (grids of many waves);
  // fn_step*: the same for several calls per launch (fn_step_role: role-major order)
  out->fn = out->fn_inplace = out->fn_step = out->fn_step_inplace = out->fn_late = out->fn_wide =
      out->fn_step_role = nullptr;
  if (dtype == DT_BF16) {
    if (qknorm) {
      pick<DT_BF16, 2, true>(H, &out->fn, &out->fn_step, &out->fn_late, nullptr);
      pick<DT_BF16, 1, true>(H, &out->fn_inplace, &out->fn_step_inplace, &out->fn_wide, &out->fn_step_role);
    } else {
      pick<DT_BF16, 2, false>(H, &out->fn, &out->fn_step, &out->fn_late, nullptr);
      pick<DT_BF16, 1, false>(H, &out->fn_inplace, &out->fn_step_inplace, &out->fn_wide, &out->fn_step_role);
    }
  } else {
    if (qknorm) {
      pick<DT_FP16, 2, true>(H, &out->fn, &out->fn_step, &out->fn_late, nullptr);
      pick<DT_FP16, 1, true>(H, &out->fn_inplace, &out->fn_step_inplace, &out->fn_wide, &out->fn_step_role);
    } else {
      pick<DT_FP16, 2, false>(H, &out->fn, &out->fn_step, &out->fn_late, nullptr);
      pick<DT_FP16, 1, false>(H, &out->fn_inplace, &out->fn_step_inplace, &out->fn_wide, &out->fn_step_role);
    }
  }
  if (!out->fn) { *why = "layer chain supports H in {4096, 8192}"; return false; }
  return true;
}

}  // namespace trident
