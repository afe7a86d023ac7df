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
// One thread-block cluster of kClusterCtas CTAs handles one (document, head):
// CTA r owns a contiguous slice of the tokens.  Histograms and per-slice
// counts live in each CTA's shared memory and are summed across the cluster
// through distributed shared memory, separated by hardware cluster barriers,
// so the whole selection is one launch:
//   A  form keys (Eq. 1 pooling x gamma in the fused path), digit-1 histogram
//   B  digit-2 histogram under the chosen prefix        C  digit-3 histogram
//   D  (> T, == T) counts per slice, then the ordered compaction into idx.
// The kept rows are then copied by the grid-wide gather kernel.
#include <cooperative_groups.h>

#include "tp_device.cuh"

namespace cg = cooperative_groups;

namespace tp {

namespace {

constexpr int kThreads = 512;
constexpr int kPer = kChunk / kThreads;  // tokens per thread in one compaction round
constexpr int kBins1 = 2048;             // bits 31..21
constexpr int kBins2 = 2048;             // bits 20..10
constexpr int kBins3 = 1024;             // bits 9..0

__device__ __forceinline__ uint32_t score_key(float s) {
  return (s > 0.f) ? __float_as_uint(s) : 0u;  // -0, +0, NaN and negatives -> 0
}

// Adds one to hist[bin] for every active lane, one shared atomic per distinct
// bin in the warp (keys concentrate in few bins).  All 32 lanes must call it.
__device__ __forceinline__ void hist_add(int* hist, uint32_t bin, bool active) {
  const unsigned mask = __ballot_sync(0xffffffffu, active);
  if (!active) return;
  const unsigned peers = __match_any_sync(mask, bin);
  if ((threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
}

constexpr int kSliceKeys = 16384;  // keys of a CTA's slice kept in shared memory
constexpr int kMaxHalf = 16;       // largest pooling half-window of the staging strip

struct SelectSmem {
  uint32_t keys[kSliceKeys];
  float strip[kSliceKeys + 2 * kMaxHalf];  // unpooled key scores of a sub-slice + halo
  int hist1[kBins1];
  int hist2[kBins2];
  int hist3[kBins3];
  int counts[2];  // (> T, == T) in this CTA's slice
  int scratch[33];
  int result[2];
};

// Bin holding the `need`-th largest key (1-based) of the cluster-wide
// histogram (the sum of every CTA's shared histogram at byte offset `off`);
// *above = keys in higher bins.  Called by the whole block.
__device__ int cluster_digit(cg::cluster_group& cluster, SelectSmem& sm, const int* local_hist,
                             int nbins, int need, int* above) {
  const int per = nbins / kThreads;  // 2 or 4 bins per thread, highest bins first
  int cnt[4] = {0, 0, 0, 0};
  for (int r = 0; r < kClusterCtas; ++r) {
    const int* h = cluster.map_shared_rank(local_hist, r);
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (i < per) cnt[i] += h[nbins - 1 - (threadIdx.x * per + i)];
  }
  int local = 0;
#pragma unroll
  for (int i = 0; i < 4; ++i) local += cnt[i];
  int total;
  int before = block_excl_scan(local, sm.scratch, &total);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if (i < per && before < need && before + cnt[i] >= need) {
      sm.result[0] = nbins - 1 - (threadIdx.x * per + i);
      sm.result[1] = before;
    }
    before += cnt[i];
  }
  __syncthreads();
  *above = sm.result[1];
  const int d = sm.result[0];
  __syncthreads();
  return d;
}

__global__ void __cluster_dims__(kClusterCtas, 1, 1) __launch_bounds__(kThreads, 1)
    tp_select_kernel(const __grid_constant__ SelectParams p) {
  extern __shared__ uint8_t smem_raw[];
  SelectSmem& sm = *reinterpret_cast<SelectSmem*>(smem_raw);
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int unit = blockIdx.y;
  const int b = unit / p.n_heads_kv, h = unit % p.n_heads_kv;
  const int64_t lo = p.off[b];
  const int n = static_cast<int>(p.off[b + 1] - lo);
  const int k = p.kept[b];
  const size_t row = static_cast<size_t>(h) * p.n_total + lo;
  // this CTA's slice [s0, s1) of the document's tokens
  const int per_cta = (((n + kClusterCtas - 1) / kClusterCtas) + 3) & ~3;
  const int s0 = min(rank * per_cta, n), s1 = min(s0 + per_cta, n);
  // the slice's keys: in shared memory when they fit, else in the global scratch
  const bool in_smem = (s1 - s0 <= kSliceKeys);
  uint32_t* const keys_base = in_smem ? sm.keys : p.keys + row;
  const int kofs = in_smem ? s0 : 0;  // keys of token i live at keys_base[i - kofs]

  for (int i = threadIdx.x; i < kBins1; i += kThreads) {
    sm.hist1[i] = 0;
    sm.hist2[i] = 0;
  }
  for (int i = threadIdx.x; i < kBins3; i += kThreads) sm.hist3[i] = 0;
  __syncthreads();

  // A: keys of the slice (scores formed here in the fused path) + digit-1 histogram,
  // in sub-slices of kSliceKeys tokens whose key scores are staged with their halo
  const int half = p.pool_kernel / 2;
  const float inv_k = 1.0f / static_cast<float>(p.pool_kernel);
  for (int c0 = s0; c0 < s1; c0 += kSliceKeys) {
    const int c1 = min(c0 + kSliceKeys, s1);
    if (!p.scores_in) {
      const float* sk = p.skey + row;
      const int len = c1 - c0 + 2 * half;
      for (int j0 = threadIdx.x; j0 < len; j0 += 8 * kThreads) {
        float v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {  // eight independent loads in flight
          const int j = j0 + u * kThreads, i = c0 - half + j;
          v[u] = (j < len && i >= 0 && i < n) ? __ldg(sk + i) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (j0 + u * kThreads < len) sm.strip[j0 + u * kThreads] = v[u];
      }
      __syncthreads();
    }
    for (int base = c0; base < c1; base += 8 * kThreads) {
      float sv[8];
      bool live[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int i = base + u * kThreads + threadIdx.x;
        live[u] = i < c1;
        sv[u] = 0.f;
        if (live[u]) sv[u] = p.scores_in ? __ldg(p.scores_in + row + i)
                                         : (p.key_only ? 1.f : __ldg(p.gamma + row + i));
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int i = base + u * kThreads + threadIdx.x;
        uint32_t key = 0;
        if (live[u]) {
          float s = sv[u];
          if (!p.scores_in) {
            float acc = 0.f;
            const float* w = sm.strip + (i - c0);
            for (int o = 0; o <= 2 * half; ++o) acc += w[o];
            s = p.key_only ? acc * inv_k : (acc * inv_k) * sv[u];
            if (p.scores_out) p.scores_out[row + i] = s;
          }
          key = score_key(s);
          keys_base[i - kofs] = key;
        }
        if (!p.scores_only) hist_add(sm.hist1, key >> 21, live[u]);
      }
    }
    __syncthreads();
  }
  if (p.scores_only) return;  // no cluster-wide exchange follows

  const int64_t unit_slot0 = static_cast<int64_t>(unit) * p.cap;
  const int kk = max(0, min(k, n));
  if (rank == 0)
    for (int64_t t = kk + threadIdx.x; t < p.cap; t += kThreads) p.idx[unit_slot0 + t] = -1;
  cluster.sync();  // histograms of phase A complete everywhere

  uint32_t thr = 0;
  int need_eq = -1;  // -1: keep every token of the document
  if (kk > 0 && kk < n) {
    int above;
    const int d1 = cluster_digit(cluster, sm, sm.hist1, kBins1, kk, &above);
    int need = kk - above;
    for (int base = s0; base < s1; base += kThreads) {
      const int i = base + threadIdx.x;
      const uint32_t key = i < s1 ? keys_base[i - kofs] : 0u;
      hist_add(sm.hist2, (key >> 10) & 0x7FF, i < s1 && (key >> 21) == static_cast<uint32_t>(d1));
    }
    cluster.sync();
    const int d2 = cluster_digit(cluster, sm, sm.hist2, kBins2, need, &above);
    need -= above;
    const uint32_t pre = (static_cast<uint32_t>(d1) << 11) | static_cast<uint32_t>(d2);
    for (int base = s0; base < s1; base += kThreads) {
      const int i = base + threadIdx.x;
      const uint32_t key = i < s1 ? keys_base[i - kofs] : 0u;
      hist_add(sm.hist3, key & 0x3FF, i < s1 && (key >> 10) == pre);
    }
    cluster.sync();
    const int d3 = cluster_digit(cluster, sm, sm.hist3, kBins3, need, &above);
    need_eq = need - above;
    thr = (pre << 10) | static_cast<uint32_t>(d3);
  } else {
    // the cluster-wide barriers must match on every CTA
    cluster.sync();
    cluster.sync();
  }

  // D: counts of this slice, then prefix over the slices before it
  {
    int gt = 0, eq = 0;
    if (kk > 0) {
      for (int i = s0 + threadIdx.x; i < s1; i += kThreads) {
        const uint32_t key = keys_base[i - kofs];
        if (need_eq < 0 || key > thr) ++gt;
        else if (key == thr) ++eq;
      }
    }
    gt = block_sum(gt, sm.scratch);
    eq = block_sum(eq, sm.scratch);
    if (threadIdx.x == 0) {
      sm.counts[0] = gt;
      sm.counts[1] = eq;
    }
  }
  cluster.sync();
  int gt_before = 0, eq_before = 0;
  for (int r = 0; r < rank; ++r) {
    const int* c = cluster.map_shared_rank(sm.counts, r);
    gt_before += c[0];
    eq_before += c[1];
  }
  cluster.sync();  // no CTA leaves while another may still read its counts

  if (kk <= 0) return;
  // ordered compaction in rounds of kChunk tokens: a token's slot is
  // (tokens > T before it) + min(tokens == T before it, need_eq)
  for (int base = s0; base < s1; base += kChunk) {
    const int j0 = base + threadIdx.x * kPer;
    int ngt = 0, neq = 0;
    uint32_t kv[kPer];
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      const int j = j0 + e;
      kv[e] = j < s1 ? keys_base[j - kofs] : 0u;
      if (j < s1) {
        if (need_eq < 0 || kv[e] > thr) ++ngt;
        else if (kv[e] == thr) ++neq;
      }
    }
    int tot_gt, tot_eq;
    int gt_rank = gt_before + block_excl_scan(ngt, sm.scratch, &tot_gt);
    int eq_rank = eq_before + block_excl_scan(neq, sm.scratch, &tot_eq);
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      const int j = j0 + e;
      if (j >= s1) break;
      const bool is_gt = need_eq < 0 || kv[e] > thr;
      const bool is_eq = !is_gt && kv[e] == thr;
      if (is_gt || (is_eq && eq_rank < need_eq)) {
        const int slot = gt_rank + (need_eq < 0 ? 0 : min(eq_rank, need_eq));
        p.idx[unit_slot0 + slot] = j;
      }
      gt_rank += is_gt;
      eq_rank += is_eq;
    }
    gt_before += tot_gt;
    eq_before += tot_eq;
  }
}

}  // namespace

size_t select_smem_bytes() { return sizeof(SelectSmem); }

cudaError_t launch_select(const SelectParams& p, cudaStream_t s) {
  const int units = p.batch * p.n_heads_kv;
  if (units <= 0) return cudaSuccess;
  if (p.pool_kernel / 2 > kMaxHalf) return cudaErrorInvalidValue;
  const size_t smem = sizeof(SelectSmem);
  cudaError_t e = cudaFuncSetAttribute(tp_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  tp_select_kernel<<<dim3(kClusterCtas, units), kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

}  // namespace tp
