// The literal row normaliser of Sec. 3.2.  A is sliced out of the causal
// prefill map over the context followed by the guide, so guide row r = (g, j)
// is normalised over every context key and over the guide keys 0..j:
//   lse[r] <- log( exp(lse_ctx[r]) + sum_{j' <= j} exp(sigma * q_r . kg_j') ).
// This kernel folds the guide-prefix term into the context normalisers that
// scoring pass 1 (or the caller) left in `lse`.  The work is tiny next to the
// context passes (G * L_t * (L_t + 1) / 2 dot products per document and head).
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "tp_device.cuh"
#include "tp_internal.h"

namespace tp {

namespace {

constexpr int kPrefixWarps = 8;
constexpr int kRowsPerWarp = 4;
constexpr int kRowsPerCta = kPrefixWarps * kRowsPerWarp;
constexpr int kKeyChunk = 32;  // guide keys per shared-memory chunk (one per lane)
constexpr int kMaxD = 128;

__device__ __forceinline__ float bf16_bits_to_f32(uint16_t b) {
  return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

// Merge of two (max, sum) pairs of exp terms; an empty pair is (-inf, 0).
__device__ __forceinline__ void merge_ms(float& m, float& s, float m2, float s2) {
  const float mm = fmaxf(m, m2);
  if (mm == -INFINITY) return;
  s = s * expf(m - mm) + s2 * expf(m2 - mm);
  m = mm;
}

// grid (ceil(rows / 32), batch * H_kv), 256 threads.  Warp w takes rows
// r0 + w + 8 i (i < 4) of unit (b, h) = blockIdx.y; in each chunk of 32 guide
// keys, lane l takes key j0 + l for all four rows at once.  The guide keys of
// the chunk sit transposed in shared memory ([d][33]: conflict-free for both
// the staging writes and the per-lane reads); the query rows are broadcast.
__global__ void __launch_bounds__(kPrefixWarps * 32) tp_prefix_kernel(const __grid_constant__ PrefixParams p) {
  __shared__ float qs[kRowsPerCta][kMaxD];
  __shared__ float kt[kMaxD][kKeyChunk + 1];
  grid_dep_launch();
  const int unit = blockIdx.y;
  const int b = unit / p.n_heads_kv;
  const int r0 = blockIdx.x * kRowsPerCta;
  const int d = p.head_dim, lt = p.guide_len;
  const size_t unit_row0 = static_cast<size_t>(unit) * p.rows;
  const uint16_t* qb = p.q + unit_row0 * d;
  const uint16_t* kg = p.k_guide + static_cast<size_t>(unit) * lt * d;

  for (int i = threadIdx.x; i < kRowsPerCta * d; i += blockDim.x) {
    const int rr = i / d, c = i - rr * d;
    const int r = r0 + rr;
    qs[rr][c] = r < p.rows ? bf16_bits_to_f32(qb[static_cast<size_t>(r) * d + c]) : 0.f;
  }
  int jmax = 0;  // the largest guide position among this CTA's rows
  for (int rr = 0; rr < kRowsPerCta && r0 + rr < p.rows; ++rr) jmax = max(jmax, (r0 + rr) % lt);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float m[kRowsPerWarp], s[kRowsPerWarp];
  int jrow[kRowsPerWarp];
#pragma unroll
  for (int i = 0; i < kRowsPerWarp; ++i) {
    m[i] = -INFINITY;
    s[i] = 0.f;
    const int r = r0 + warp + kPrefixWarps * i;
    jrow[i] = r < p.rows ? r % lt : -1;
  }
  for (int j0 = 0; j0 <= jmax; j0 += kKeyChunk) {
    __syncthreads();  // the previous chunk is consumed (and qs is complete)
    for (int i = threadIdx.x; i < kKeyChunk * d; i += blockDim.x) {
      const int l = i / d, c = i - l * d;
      kt[c][l] = j0 + l < lt ? bf16_bits_to_f32(kg[static_cast<size_t>(j0 + l) * d + c]) : 0.f;
    }
    __syncthreads();
    float acc[kRowsPerWarp] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
    for (int c = 0; c < d; ++c) {
      const float kv = kt[c][lane];
#pragma unroll
      for (int i = 0; i < kRowsPerWarp; ++i) acc[i] = fmaf(qs[warp + kPrefixWarps * i][c], kv, acc[i]);
    }
    const int jj = j0 + lane;
#pragma unroll
    for (int i = 0; i < kRowsPerWarp; ++i) {
      if (jj <= jrow[i]) merge_ms(m[i], s[i], acc[i] * p.sigma, 1.f);
    }
  }
#pragma unroll
  for (int i = 0; i < kRowsPerWarp; ++i) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m[i], o);
      const float s2 = __shfl_xor_sync(0xffffffffu, s[i], o);
      merge_ms(m[i], s[i], m2, s2);
    }
  }
  grid_dep_wait();  // the context normalisers come from scoring pass 1
  if (lane == 0) {
    const bool empty = p.off[b + 1] == p.off[b];
#pragma unroll
    for (int i = 0; i < kRowsPerWarp; ++i) {
      if (jrow[i] < 0) continue;
      const size_t at = unit_row0 + r0 + warp + kPrefixWarps * i;
      const float pre = m[i] + logf(s[i]);  // every row sees at least its own key
      // an empty document has no context terms (pass 1 writes no normaliser for it)
      const float ctx = empty ? -INFINITY : p.lse[at];
      float out = pre;
      if (ctx != -INFINITY) {
        const float mm = fmaxf(ctx, pre);
        out = mm + logf(expf(ctx - mm) + expf(pre - mm));
      }
      p.lse[at] = out;
    }
  }
}

}  // namespace

cudaError_t launch_prefix(const PrefixParams& p, bool dependent, cudaStream_t s) {
  const int units = p.batch * p.n_heads_kv;
  if (units <= 0 || p.rows <= 0) return cudaSuccess;
  if (p.head_dim > kMaxD) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((p.rows + kRowsPerCta - 1) / kRowsPerCta, units);
  cfg.blockDim = dim3(kPrefixWarps * 32);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = dependent ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, tp_prefix_kernel, p);
}

}  // namespace tp
