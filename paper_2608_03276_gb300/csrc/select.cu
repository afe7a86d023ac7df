// Top-budget selection per (document, KV head) (Sec. 3.4; Sec. 4 "Eviction":
// a uniform budget per head, heads selected independently), and the fused
// compaction of the kept rows.
//
// Scores are non-negative fp32, so their bit patterns order like their values
// once -0 and NaN are mapped to +0.  A three-digit radix select (11, 11 and
// 10 bits) finds the k-th largest key T and how many keys lie above it; the
// kept set is every key > T plus the first (k - above) keys equal to T in
// token order (the lowest-index tie-break), written in ascending order.
//
// Every kernel covers one 4096-token chunk of one (document, head) per CTA, so
// the whole GPU works on each stage:
//   score_hist  form keys (Eq. 1 pooling x gamma in the fused path) + digit-1 histogram
//   radix<2,3>  digit-2 / digit-3 histograms of the keys under the chosen prefix
//   count       threshold T per unit (chunk 0 records it) and (>T, ==T) counts per chunk
//   compact     ordered compaction into idx, then (fused path) the row gather:
//               K, V, Eq. 2 int8 codes of V, gamma
// Histograms are global (atomics on the few non-empty bins) and zeroed by the
// caller before score_hist.
#include "tp_device.cuh"

namespace tp {

namespace {

constexpr int kThreads = 512;
constexpr int kPer = kChunk / kThreads;  // tokens per thread
constexpr int kBins1 = 2048;             // bits 31..21
constexpr int kBins2 = 2048;             // bits 20..10
constexpr int kBins3 = 1024;             // bits 9..0
constexpr int kMaxHalf = 16;             // pooling half-window supported by the staging strip

__device__ __forceinline__ uint32_t score_key(float s) {
  return (s > 0.f) ? __float_as_uint(s) : 0u;  // -0, +0, NaN and negatives -> 0
}

struct Unit {
  int b, h, n, k;
  int64_t lo;
  size_t row;  // offset of the unit's first token in [H_kv, N] arrays
};

__device__ __forceinline__ Unit unit_of(const SelectParams& p) {
  Unit u;
  const int unit = blockIdx.y;
  u.b = unit / p.n_heads_kv;
  u.h = unit % p.n_heads_kv;
  u.lo = p.off[u.b];
  u.n = static_cast<int>(p.off[u.b + 1] - u.lo);
  u.k = p.kept[u.b];
  u.row = static_cast<size_t>(u.h) * p.n_total + u.lo;
  return u;
}

// Bin holding the `need`-th largest key (1-based) of a global histogram;
// *above = keys in higher bins.  Called by the whole block.
__device__ int find_digit(const int* ghist, int nbins, int need, int* above, int* scratch,
                          int* result) {
  const int per = nbins / kThreads;  // 2 or 4 bins per thread, highest bins first
  int cnt[4];
  int local = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    cnt[i] = i < per ? __ldcg(ghist + (nbins - 1 - (threadIdx.x * per + i))) : 0;
    local += cnt[i];
  }
  int total;
  int before = block_excl_scan(local, scratch, &total);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if (i < per && before < need && before + cnt[i] >= need) {
      result[0] = nbins - 1 - (threadIdx.x * per + i);
      result[1] = before;
    }
    before += cnt[i];
  }
  __syncthreads();
  *above = result[1];
  const int d = result[0];
  __syncthreads();
  return d;
}

// Adds the non-zero bins of a shared histogram into a global one.
__device__ __forceinline__ void flush_hist(const int* sh, int* gh, int nbins) {
  __syncthreads();
  for (int i = threadIdx.x; i < nbins; i += kThreads) {
    const int v = sh[i];
    if (v) atomicAdd(gh + i, v);
  }
}

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) score_hist_kernel(const __grid_constant__ SelectParams p) {
  __shared__ int hist[kBins1];
  __shared__ float strip[kChunk + 2 * kMaxHalf];
  const Unit u = unit_of(p);
  const int i0 = blockIdx.x * kChunk;
  if (i0 >= u.n) return;
  const int len = min(kChunk, u.n - i0);
  for (int i = threadIdx.x; i < kBins1; i += kThreads) hist[i] = 0;
  const int half = p.pool_kernel / 2;
  if (!p.scores_in) {
    const float* sk = p.skey + u.row;
    for (int j = threadIdx.x; j < len + 2 * half; j += kThreads) {
      const int i = i0 - half + j;
      strip[j] = (i >= 0 && i < u.n) ? sk[i] : 0.f;
    }
  }
  __syncthreads();
  const float inv_k = 1.0f / static_cast<float>(p.pool_kernel);
  for (int j = threadIdx.x; j < len; j += kThreads) {
    const size_t t = u.row + i0 + j;
    float s;
    if (p.scores_in) {
      s = p.scores_in[t];
    } else {
      float acc = 0.f;
      for (int o = 0; o <= 2 * half; ++o) acc += strip[j + o];
      s = acc * inv_k;
      if (!p.key_only) s *= p.gamma[t];
      if (p.scores_out) p.scores_out[t] = s;
    }
    const uint32_t key = score_key(s);
    p.keys[t] = key;
    atomicAdd(&hist[key >> 21], 1);
  }
  if (p.hist) flush_hist(hist, p.hist + static_cast<size_t>(blockIdx.y) * kHistInts, kBins1);
}

template <int PASS>
__global__ void __launch_bounds__(kThreads) radix_kernel(const __grid_constant__ SelectParams p) {
  __shared__ int hist[kBins2];
  __shared__ int scratch[33];
  __shared__ int result[2];
  const Unit u = unit_of(p);
  const int i0 = blockIdx.x * kChunk;
  if (i0 >= u.n || u.k <= 0 || u.k >= u.n) return;
  const int len = min(kChunk, u.n - i0);
  const int* gh = p.hist + static_cast<size_t>(blockIdx.y) * kHistInts;
  int above;
  const int d1 = find_digit(gh, kBins1, u.k, &above, scratch, result);
  uint32_t pre = static_cast<uint32_t>(d1);
  if (PASS == 3) {
    const int d2 = find_digit(gh + kBins1, kBins2, u.k - above, &above, scratch, result);
    pre = (pre << 11) | static_cast<uint32_t>(d2);
  }
  const int nb = PASS == 2 ? kBins2 : kBins3;
  for (int i = threadIdx.x; i < nb; i += kThreads) hist[i] = 0;
  __syncthreads();
  const uint32_t* keys = p.keys + u.row + i0;
  for (int j = threadIdx.x; j < len; j += kThreads) {
    const uint32_t key = keys[j];
    if (PASS == 2) {
      if ((key >> 21) == pre) atomicAdd(&hist[(key >> 10) & 0x7FF], 1);
    } else {
      if ((key >> 10) == pre) atomicAdd(&hist[key & 0x3FF], 1);
    }
  }
  flush_hist(hist, const_cast<int*>(gh) + (PASS == 2 ? kBins1 : kBins1 + kBins2), nb);
}

__global__ void __launch_bounds__(kThreads) count_kernel(const __grid_constant__ SelectParams p) {
  __shared__ int scratch[33];
  __shared__ int result[2];
  const Unit u = unit_of(p);
  const int i0 = blockIdx.x * kChunk;
  if (i0 >= u.n || u.k <= 0) return;
  const int len = min(kChunk, u.n - i0);
  int2* counts = p.counts + static_cast<size_t>(blockIdx.y) * p.max_chunks;
  if (u.k >= u.n) {  // everything kept
    if (threadIdx.x == 0) {
      counts[blockIdx.x] = make_int2(len, 0);
      if (blockIdx.x == 0) p.thresh[blockIdx.y] = make_int2(0, -1);
    }
    return;
  }
  const int* gh = p.hist + static_cast<size_t>(blockIdx.y) * kHistInts;
  int a1, a2, a3;
  const int d1 = find_digit(gh, kBins1, u.k, &a1, scratch, result);
  const int d2 = find_digit(gh + kBins1, kBins2, u.k - a1, &a2, scratch, result);
  const int d3 = find_digit(gh + kBins1 + kBins2, kBins3, u.k - a1 - a2, &a3, scratch, result);
  const uint32_t thr = (static_cast<uint32_t>(d1) << 21) | (static_cast<uint32_t>(d2) << 10) |
                       static_cast<uint32_t>(d3);
  const int need_eq = u.k - a1 - a2 - a3;
  const uint32_t* keys = p.keys + u.row + i0;
  int gt = 0, eq = 0;
  for (int j = threadIdx.x; j < len; j += kThreads) {
    const uint32_t key = keys[j];
    gt += key > thr;
    eq += key == thr;
  }
  int tg, te;
  block_excl_scan(gt, scratch, &tg);
  block_excl_scan(eq, scratch, &te);
  if (threadIdx.x == 0) {
    counts[blockIdx.x] = make_int2(tg, te);
    if (blockIdx.x == 0) p.thresh[blockIdx.y] = make_int2(static_cast<int>(thr), need_eq);
  }
}

// Copies one kept row: K lanes then V lanes (LPR lanes each), int8 codes of V.
template <int LPR>
__device__ __forceinline__ void copy_row(const SelectParams& p, const Unit& u, int64_t slot_index,
                                         int token, int lane_in_pair) {
  const bool is_v = lane_in_pair >= LPR;
  const int part = lane_in_pair % LPR;
  const int64_t tok = static_cast<int64_t>(u.h) * p.n_total + u.lo + token;
  const int64_t dst = slot_index * LPR + part;
  if (!is_v) {
    if (p.kc) reinterpret_cast<uint4*>(p.kc)[dst] =
        __ldcs(reinterpret_cast<const uint4*>(p.k) + tok * LPR + part);
  } else {
    const uint4 v = __ldcs(reinterpret_cast<const uint4*>(p.v) + tok * LPR + part);
    if (p.vc) reinterpret_cast<uint4*>(p.vc)[dst] = v;
    const float g = p.gamma[tok];
    if (p.vqc) reinterpret_cast<uint2*>(p.vqc)[dst] = quant8_bf16(v, g, p.qmax);
    if (p.gammac && part == 0) p.gammac[slot_index] = g;
  }
}

template <int LPR>
__global__ void __launch_bounds__(kThreads) compact_kernel(const __grid_constant__ SelectParams p) {
  __shared__ int scratch[33];
  __shared__ int2 list[kChunk];  // (slot, token) of the rows this CTA keeps
  __shared__ int nlist;
  const Unit u = unit_of(p);
  const int i0 = blockIdx.x * kChunk;
  const int64_t unit_slot0 = static_cast<int64_t>(blockIdx.y) * p.cap;
  // padding slots [k, cap): chunk 0 of the unit (also for empty documents)
  if (blockIdx.x == 0) {
    const int k0 = max(0, min(u.k, u.n));
    for (int64_t t = k0 + threadIdx.x; t < p.cap; t += kThreads) p.idx[unit_slot0 + t] = -1;
    if (p.gather) {
      constexpr int SPW = 32 / (2 * LPR);
      const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
      for (int64_t t = k0 + warp * SPW + lane / (2 * LPR); t < p.cap; t += (kThreads / 32) * SPW) {
        const int lp = lane % (2 * LPR);
        const int part = lp % LPR;
        const int64_t dst = (unit_slot0 + t) * LPR + part;
        if (lp < LPR) {
          if (p.kc) reinterpret_cast<uint4*>(p.kc)[dst] = make_uint4(0, 0, 0, 0);
        } else {
          if (p.vc) reinterpret_cast<uint4*>(p.vc)[dst] = make_uint4(0, 0, 0, 0);
          if (p.vqc) reinterpret_cast<uint2*>(p.vqc)[dst] = make_uint2(0, 0);
          if (p.gammac && part == 0) p.gammac[unit_slot0 + t] = 0.f;
        }
      }
    }
  }
  if (i0 >= u.n || u.k <= 0) return;
  const int len = min(kChunk, u.n - i0);
  const int2 th = p.thresh[blockIdx.y];
  const uint32_t thr = static_cast<uint32_t>(th.x);
  const int need_eq = th.y;  // -1: keep everything
  // tokens > T and == T in the chunks before this one
  const int2* counts = p.counts + static_cast<size_t>(blockIdx.y) * p.max_chunks;
  int gt_before = 0, eq_before = 0;
  for (int c = threadIdx.x; c < blockIdx.x; c += kThreads) {
    const int2 v = __ldcg(counts + c);
    gt_before += v.x;
    eq_before += v.y;
  }
  gt_before = block_sum(gt_before, scratch);
  eq_before = block_sum(eq_before, scratch);
  // ordered compaction: kPer consecutive tokens per thread.  A token's slot is
  // (tokens > T before it) + min(tokens == T before it, need_eq).
  const uint32_t* keys = p.keys + u.row + i0;
  const int j0 = threadIdx.x * kPer;
  int ngt = 0, neq = 0;
  uint32_t kk[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    const int j = j0 + e;
    kk[e] = j < len ? keys[j] : 0u;
    if (j < len) {
      if (need_eq < 0 || kk[e] > thr) ++ngt;
      else if (kk[e] == thr) ++neq;
    }
  }
  int tot;
  int gt_rank = gt_before + block_excl_scan(ngt, scratch, &tot);
  int eq_rank = eq_before + block_excl_scan(neq, scratch, &tot);
  if (threadIdx.x == 0) nlist = 0;
  __syncthreads();
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    const int j = j0 + e;
    if (j >= len) break;
    const bool is_gt = need_eq < 0 || kk[e] > thr;
    const bool is_eq = !is_gt && kk[e] == thr;
    if (is_gt || (is_eq && eq_rank < need_eq)) {
      const int slot = gt_rank + (need_eq < 0 ? 0 : min(eq_rank, need_eq));
      p.idx[unit_slot0 + slot] = i0 + j;
      if (p.gather) {
        const int at = atomicAdd(&nlist, 1);
        list[at] = make_int2(slot, i0 + j);
      }
    }
    gt_rank += is_gt;
    eq_rank += is_eq;
  }
  if (!p.gather) return;
  __syncthreads();
  constexpr int SPW = 32 / (2 * LPR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m = nlist;
  for (int e = warp * SPW + lane / (2 * LPR); e < m; e += (kThreads / 32) * SPW) {
    const int2 st = list[e];
    copy_row<LPR>(p, u, unit_slot0 + st.x, st.y, lane % (2 * LPR));
  }
}

}  // namespace

cudaError_t launch_select(const SelectParams& p, bool form_scores_only, cudaStream_t s) {
  const int units = p.batch * p.n_heads_kv;
  if (units <= 0 || p.max_chunks <= 0) return cudaSuccess;
  if (p.pool_kernel / 2 > kMaxHalf) return cudaErrorInvalidValue;
  const dim3 grid(p.max_chunks, units);
  score_hist_kernel<<<grid, kThreads, 0, s>>>(p);
  if (form_scores_only) return cudaGetLastError();
  radix_kernel<2><<<grid, kThreads, 0, s>>>(p);
  radix_kernel<3><<<grid, kThreads, 0, s>>>(p);
  count_kernel<<<grid, kThreads, 0, s>>>(p);
  if (p.head_dim == 64)
    compact_kernel<8><<<grid, kThreads, 0, s>>>(p);
  else
    compact_kernel<16><<<grid, kThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace tp
