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

constexpr int kPrefixThreads = 256;
constexpr int kRowsPerCta = 32;   // 8 warps x 4 rows
constexpr int kKeyBlock = 128;    // 32 lanes x 4 keys
constexpr int kMaxD = 128;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.69314718055994531f;

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// Merge of two (max, sum) pairs of base-2 exp terms; an empty pair is (-inf, 0).
__device__ __forceinline__ void merge_ms2(float& m, float& s, float m2, float s2) {
  const float mm = fmaxf(m, m2);
  if (mm == -INFINITY) return;
  s = s * ex2(m - mm) + s2 * ex2(m2 - mm);
  m = mm;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Stages `count` bf16 rows of d elements (row stride d) into a transposed fp32
// tile t[c * ld + i] (i < count; rows past `count` are zero).  Each thread
// moves 16-byte pieces; consecutive threads take consecutive rows, so the
// transposed stores hit distinct banks.  All of a thread's loads are issued
// before the first store.
template <int PER>
__device__ __forceinline__ void stage_transposed(float* t, int ld, const uint16_t* src, int count,
                                                 int d) {
  const int pieces = d / 8;  // 16-byte pieces per row
  uint4 v[PER];
#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const int idx = threadIdx.x + u * kPrefixThreads;
    const int i = idx % ld, c8 = idx / ld;
    v[u] = make_uint4(0u, 0u, 0u, 0u);
    if (c8 < pieces && i < count)
      v[u] = *reinterpret_cast<const uint4*>(src + static_cast<size_t>(i) * d + c8 * 8);
  }
#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const int idx = threadIdx.x + u * kPrefixThreads;
    const int i = idx % ld, c8 = idx / ld;
    if (c8 >= pieces) continue;
    float* col = t + (c8 * 8) * ld + i;
    col[0 * ld] = bf16_lo(v[u].x);
    col[1 * ld] = bf16_hi(v[u].x);
    col[2 * ld] = bf16_lo(v[u].y);
    col[3 * ld] = bf16_hi(v[u].y);
    col[4 * ld] = bf16_lo(v[u].z);
    col[5 * ld] = bf16_hi(v[u].z);
    col[6 * ld] = bf16_lo(v[u].w);
    col[7 * ld] = bf16_hi(v[u].w);
  }
}

// grid (ceil(rows / 32), batch * H_kv), 256 threads, 80 KB of dynamic shared
// memory: the CTA's 32 query rows ([d][32]) and one block of 128 guide keys
// ([d][128]), both fp32 and transposed.  Warp w owns rows r0 + 4w .. 4w+3 and
// lane l keys kb + 4l .. 4l+3 of each key block: per feature c it reads one
// broadcast float4 of queries and one float4 of keys and does 16 FMAs.  Each
// lane keeps a running (max, sum) per row over its keys; the lanes merge at
// the end, and lane 0 folds the result into the row's normaliser.  All sums
// are kept in base-2 units (logits times sigma * log2(e)).
__global__ void __launch_bounds__(kPrefixThreads) tp_prefix_kernel(const __grid_constant__ PrefixParams p) {
  extern __shared__ float4 prefix_smem[];
  float* qs = reinterpret_cast<float*>(prefix_smem);     // [kMaxD][kRowsPerCta]
  float* kt = qs + kMaxD * kRowsPerCta;                  // [kMaxD][kKeyBlock]
  grid_dep_launch();
  const int unit = blockIdx.y;
  const int b = unit / p.n_heads_kv;
  const int r0 = blockIdx.x * kRowsPerCta;
  const int d = p.head_dim, lt = p.guide_len;
  const size_t unit_row0 = static_cast<size_t>(unit) * p.rows;
  const uint16_t* kg = p.k_guide + static_cast<size_t>(unit) * lt * d;
  const int nrows = min(kRowsPerCta, p.rows - r0);

  stage_transposed<kRowsPerCta * kMaxD / 8 / kPrefixThreads>(qs, kRowsPerCta, p.q + (unit_row0 + r0) * d,
                                                             nrows, d);
  int jmax = 0;  // the largest guide position among this CTA's rows
  for (int rr = 0; rr < nrows; ++rr) jmax = max(jmax, (r0 + rr) % lt);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float c2 = p.sigma * kLog2e;
  float m[4], s[4];
  int jrow[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    m[i] = -INFINITY;
    s[i] = 0.f;
    const int r = r0 + 4 * warp + i;
    jrow[i] = r < p.rows ? r % lt : -1;
  }
  for (int kb = 0; kb <= jmax; kb += kKeyBlock) {
    __syncthreads();  // the previous key block is consumed
    stage_transposed<kKeyBlock * kMaxD / 8 / kPrefixThreads>(kt, kKeyBlock, kg + static_cast<size_t>(kb) * d,
                                                             min(kKeyBlock, lt - kb), d);
    __syncthreads();
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[i][e] = 0.f;
#pragma unroll 4
    for (int c = 0; c < d; ++c) {
      const float4 qv = *reinterpret_cast<const float4*>(qs + c * kRowsPerCta + 4 * warp);
      const float4 kv = *reinterpret_cast<const float4*>(kt + c * kKeyBlock + 4 * lane);
      const float qa[4] = {qv.x, qv.y, qv.z, qv.w};
      const float ka[4] = {kv.x, kv.y, kv.z, kv.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[i][e] = fmaf(qa[i], ka[e], acc[i][e]);
    }
    // This block's terms per row, branch-free: the row's maximum over the
    // warp, then the sum of 2^(x - max); merged into the running pair.
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float x[4], lm = -INFINITY;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kb + 4 * lane + e;
        x[e] = key <= jrow[i] ? acc[i][e] * c2 : -INFINITY;  // causal: keys 0..j
        lm = fmaxf(lm, x[e]);
      }
      const float bm = warp_max(lm);
      float ls = 0.f;
      if (bm != -INFINITY) {
#pragma unroll
        for (int e = 0; e < 4; ++e) ls += ex2(x[e] - bm);
      }
      merge_ms2(m[i], s[i], bm, warp_sum(ls));
    }
  }
  grid_dep_wait();  // the context normalisers come from scoring pass 1
  if (lane < 4) {
    // every lane holds the warp's totals; lane i writes row i
    float mi = m[0], si = s[0];
    int ji = jrow[0];
#pragma unroll
    for (int i = 1; i < 4; ++i)
      if (lane == i) {
        mi = m[i];
        si = s[i];
        ji = jrow[i];
      }
    if (ji >= 0) {
      const size_t at = unit_row0 + r0 + 4 * warp + lane;
      const float pre = mi + lg2(si);  // every row sees at least its own key
      // an empty document has no context terms (pass 1 writes no normaliser for it)
      const float ctx = p.off[b + 1] == p.off[b] ? -INFINITY : p.lse[at] * kLog2e;
      float out = pre;
      if (ctx != -INFINITY) {
        const float mm = fmaxf(ctx, pre);
        out = mm + lg2(ex2(ctx - mm) + ex2(pre - mm));
      }
      p.lse[at] = out * kLn2;
    }
  }
}

}  // namespace

cudaError_t launch_prefix(const PrefixParams& p, bool dependent, cudaStream_t s) {
  const int units = p.batch * p.n_heads_kv;
  if (units <= 0 || p.rows <= 0) return cudaSuccess;
  if (p.head_dim > kMaxD || p.head_dim % 8 != 0) return cudaErrorInvalidValue;
  const size_t smem = sizeof(float) * kMaxD * (kRowsPerCta + kKeyBlock);
  cudaError_t e = set_smem_once(reinterpret_cast<const void*>(tp_prefix_kernel), 18);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((p.rows + kRowsPerCta - 1) / kRowsPerCta, units);
  cfg.blockDim = dim3(kPrefixThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = dependent ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, tp_prefix_kernel, p);
}

}  // namespace tp
