// Top-budget selection per (document, KV head) (Sec. 3.4; Sec. 4 "Eviction":
// a uniform budget per head, heads selected independently).
//
// Scores are non-negative fp32, so their bit patterns order like their values
// once -0 and NaN are mapped to +0.  A three-digit radix select (11, 11 and
// 10 bits) finds the k-th largest key T and how many keys lie above it; an
// ordered block scan then keeps every key > T plus the first (k - above)
// keys equal to T in token order, which is the lowest-index tie-break.  The
// kept indices come out ascending.
//
// In the fused path the first pass also forms the scores themselves: Eq. 1's
// average pooling of the unpooled key scores (window K, zero outside the
// document, divisor K) times gamma (Eq. 3).
#include "tp_device.cuh"

namespace tp {

namespace {

constexpr int kThreads = 1024;
constexpr int kBins1 = 2048;  // bits 31..21
constexpr int kBins2 = 2048;  // bits 20..10
constexpr int kBins3 = 1024;  // bits 9..0
constexpr int kItems = 4;     // consecutive tokens per thread in the ordered scan

__device__ __forceinline__ uint32_t score_key(float s) {
  return (s > 0.f) ? __float_as_uint(s) : 0u;  // -0, +0, NaN and negatives -> 0
}

// Finds the bin holding the `need`-th largest element (1-based) of a histogram
// of `nbins` bins (bin index = digit value).  Returns the digit; *above gets
// the count of elements in higher bins.  All threads call it.
__device__ int find_digit(const int* hist, int nbins, int need, int* above, int* scratch,
                          int* result) {
  // Reverse order: position q holds bin nbins-1-q; per thread a run of bins.
  const int per = nbins / kThreads;  // 1 or 2
  int local = 0;
  for (int i = 0; i < per; ++i) local += hist[nbins - 1 - (threadIdx.x * per + i)];
  int total;
  int before = block_excl_scan(local, scratch, &total);
  for (int i = 0; i < per; ++i) {
    const int binv = nbins - 1 - (threadIdx.x * per + i);
    const int cnt = hist[binv];
    if (before < need && before + cnt >= need) {
      result[0] = binv;
      result[1] = before;
    }
    before += cnt;
  }
  __syncthreads();
  *above = result[1];
  const int d = result[0];
  __syncthreads();
  return d;
}

__global__ void __launch_bounds__(kThreads, 1) select_kernel(const __grid_constant__ SelectParams p) {
  __shared__ int hist[kBins1];
  __shared__ int scratch[33];
  __shared__ int result[2];
  const int unit = blockIdx.x;
  const int b = unit / p.n_heads_kv, h = unit % p.n_heads_kv;
  const int64_t lo = p.off[b];
  const int n = static_cast<int>(p.off[b + 1] - lo);
  const int k = p.kept[b];
  const size_t row = static_cast<size_t>(h) * p.n_total + lo;
  uint32_t* keys = p.keys + row;
  int32_t* out = p.idx + static_cast<size_t>(unit) * p.cap;

  // Pass 0: form the keys (pool x gamma in the fused path) and the top-digit histogram.
  for (int i = threadIdx.x; i < kBins1; i += kThreads) hist[i] = 0;
  __syncthreads();
  const int half = p.pool_kernel / 2;
  const float inv_k = 1.0f / static_cast<float>(p.pool_kernel);
  for (int i = threadIdx.x; i < n; i += kThreads) {
    float s;
    if (p.scores_in) {
      s = p.scores_in[row + i];
    } else {
      const float* sk = p.skey + row;
      float acc = 0.f;
      for (int o = -half; o <= half; ++o) {
        const int jj = i + o;
        if (jj >= 0 && jj < n) acc += sk[jj];
      }
      s = acc * inv_k;
      if (!p.key_only) s *= p.gamma[row + i];
      if (p.scores_out) p.scores_out[row + i] = s;
    }
    const uint32_t key = score_key(s);
    keys[i] = key;
    atomicAdd(&hist[key >> 21], 1);
  }
  __syncthreads();

  if (k <= 0) {
    for (int64_t t = threadIdx.x; t < p.cap; t += kThreads) out[t] = -1;
    return;
  }
  uint32_t thr = 0;
  int need_eq = 0;
  const bool all = k >= n;
  if (k > 0 && !all) {
    int above1, above2, above3;
    const int d1 = find_digit(hist, kBins1, k, &above1, scratch, result);
    int need = k - above1;
    for (int i = threadIdx.x; i < kBins2; i += kThreads) hist[i] = 0;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += kThreads) {
      const uint32_t key = keys[i];
      if ((key >> 21) == static_cast<uint32_t>(d1)) atomicAdd(&hist[(key >> 10) & 0x7FF], 1);
    }
    __syncthreads();
    const int d2 = find_digit(hist, kBins2, need, &above2, scratch, result);
    need -= above2;
    const uint32_t pre = (static_cast<uint32_t>(d1) << 11) | static_cast<uint32_t>(d2);
    for (int i = threadIdx.x; i < kBins3; i += kThreads) hist[i] = 0;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += kThreads) {
      const uint32_t key = keys[i];
      if ((key >> 10) == pre) atomicAdd(&hist[key & 0x3FF], 1);
    }
    __syncthreads();
    const int d3 = find_digit(hist, kBins3, need, &above3, scratch, result);
    need -= above3;
    thr = (pre << 10) | static_cast<uint32_t>(d3);
    need_eq = need;
  }

  // Ordered compaction: tokens in chunks of kThreads*kItems, kItems per thread.
  int kept_base = 0, eq_base = 0;
  for (int base = 0; base < n; base += kThreads * kItems) {
    const int i0 = base + threadIdx.x * kItems;
    bool gt[kItems], eq[kItems];
    int n_eq = 0;
#pragma unroll
    for (int e = 0; e < kItems; ++e) {
      const int i = i0 + e;
      bool g = false, q = false;
      if (i < n && k > 0) {
        if (all) {
          g = true;
        } else {
          const uint32_t key = keys[i];
          g = key > thr;
          q = key == thr;
        }
      }
      gt[e] = g;
      eq[e] = q;
      n_eq += q;
    }
    int eq_total;
    int eq_rank = eq_base + block_excl_scan(n_eq, scratch, &eq_total);
    bool keep[kItems];
    int n_keep = 0;
#pragma unroll
    for (int e = 0; e < kItems; ++e) {
      keep[e] = gt[e] || (eq[e] && eq_rank < need_eq);
      eq_rank += eq[e];
      n_keep += keep[e];
    }
    int keep_total;
    int pos = kept_base + block_excl_scan(n_keep, scratch, &keep_total);
#pragma unroll
    for (int e = 0; e < kItems; ++e)
      if (keep[e]) out[pos++] = i0 + e;
    kept_base += keep_total;
    eq_base += eq_total;
  }
  for (int64_t t = kept_base + threadIdx.x; t < p.cap; t += kThreads) out[t] = -1;
}

}  // namespace

cudaError_t launch_select(const SelectParams& p, cudaStream_t s) {
  const int units = p.batch * p.n_heads_kv;
  if (units <= 0) return cudaSuccess;
  select_kernel<<<units, kThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace tp
