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
// One thread-block cluster of CL CTAs (8; 12 for documents of 64K tokens or
// more when every unit's cluster is resident at once; 4 when 8 per unit would
// not fit in one wave and every slice still fits in shared memory) handles one
// (document, head) -- or one (layer, document, head) when a stack of short
// layers is selected in one launch (four-CTA clusters, all resident):
// CTA r owns a contiguous slice of the tokens.  Histograms and per-slice
// counts live in each CTA's shared memory and are summed across the cluster
// through distributed shared memory, separated by hardware cluster barriers,
// so the whole selection is one launch:
//   A  form keys (Eq. 1 pooling x gamma in the fused path), digit-1 histogram
//   B  digit-2 histogram under the chosen prefix        C  digit-3 histogram
//   D  (> T, == T) counts per slice (read off its histograms), then the
//      ordered compaction into idx.
// The kept rows are then copied by the grid-wide gather kernel.
#include <cooperative_groups.h>


#include <cstddef>
#include <mutex>

#include "tp_device.cuh"

namespace cg = cooperative_groups;

namespace tp {

namespace {

constexpr int kThreads = 512;
// Digits of a key (bit 31 is always 0: keys are the bits of non-negative
// floats), so the first digit spends its 2048 bins on bits that vary
constexpr int kBins1 = 2048;             // bits 30..20
constexpr int kBins2 = 1024;             // bits 19..10
constexpr int kBins3 = 1024;             // bits 9..0

constexpr int kSliceKeys = 16384;  // keys of a CTA's slice kept in shared memory
constexpr int kMaxHalf = 16;       // largest pooling half-window of the staging strip

struct SelectSmem {
  uint32_t keys[kSliceKeys + kSliceKeys / 16];  // one padding word after every 16 keys
  // unpooled key scores of a sub-slice with its halo, and its scales (or given
  // scores); element g of the global array sits at [g - g_ref] with g_ref a
  // multiple of 4, so 16-byte groups of the two line up (4 floats of slack)
  float strip[kSliceKeys + 2 * kMaxHalf + 4];
  float vals[kSliceKeys + 4];
  int hist1[kBins1];
  int hist2[kBins2];
  int hist3[kBins3];
  // this CTA's slice of the cluster-summed histogram and its total, one
  // buffer per digit so that no search overwrites what another CTA may still
  // be reading from the previous one
  int red[3][kBins1 / 4];
  int red_total[3];
  int counts[2];  // (> T, == T) in this CTA's slice
  int scratch[33];
  int result[2];
  float norm2[2];  // this CTA's sums of squares of pooled key scores and scales
  float inv_norm[2];
};
static_assert(offsetof(SelectSmem, strip) % 16 == 0 && offsetof(SelectSmem, vals) % 16 == 0,
              "16-byte cp.async destinations must be 16-byte aligned");

// Sum of v over the block in a fixed order (warp trees, then warp totals).
__device__ __forceinline__ float block_sum_f(float v, float* warp_part) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) warp_part[warp] = v;
  __syncthreads();
  float t = 0.f;
  if (warp == 0) {
    t = lane < static_cast<int>(blockDim.x >> 5) ? warp_part[lane] : 0.f;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (lane == 0) warp_part[32] = t;
  }
  __syncthreads();
  t = warp_part[32];
  __syncthreads();
  return t;
}

// Address of `local` (a shared-memory object of this CTA) in cluster CTA `rank`.
__device__ __forceinline__ uint32_t dsmem(const void* local, int rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(local)), "r"(rank));
  return r;
}

__device__ __forceinline__ int ld_dsmem(uint32_t addr) {
  int v;
  asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
  return v;
}

// Bin holding the `need`-th largest key (1-based) of the cluster-wide
// histogram, i.e. the sum over the cluster of every CTA's `local_hist`;
// *above = keys in higher bins.  Called by every thread of every CTA of the
// cluster (it contains cluster barriers).
//   1. CTA r sums its slice of nbins/CL bins over the CL CTAs (remote loads).
//   2. Every CTA reads the CL slice totals, finds the slice holding the target
//      (highest bins first), and scans that slice's bins from its owner.
template <int CL>
__device__ int cluster_digit(cg::cluster_group& cluster, SelectSmem& sm, const int* local_hist,
                             int nbins, int need, int* above, int level) {
  int* const red = sm.red[level];
  int* const red_total = &sm.red_total[level];
  const int rank = static_cast<int>(cluster.block_rank());
  // CTA r owns bins [r slice, r slice + slice) (the last slice may be short
  // or empty when CL does not divide nbins); at most 512 bins: one per thread
  const int slice = (nbins + CL - 1) / CL;
  const int own = max(0, min(slice, nbins - rank * slice));
  if (static_cast<int>(threadIdx.x) < own) {
    const int bin = rank * slice + threadIdx.x;
    int v[CL];
#pragma unroll
    for (int r = 0; r < CL; ++r) v[r] = ld_dsmem(dsmem(local_hist + bin, r));
    int t = 0;
#pragma unroll
    for (int r = 0; r < CL; ++r) t += v[r];
    red[threadIdx.x] = t;
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    int t = 0;
    for (int i = threadIdx.x; i < own; i += 32) t += red[i];
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (threadIdx.x == 0) *red_total = t;
  }
  cluster.sync();  // every slice reduced
  // slice totals, highest slice first, and the slice that holds the target
  if (threadIdx.x == 0) {
    int before = 0, s_hit = 0, s_before = 0;
    for (int r = CL - 1; r >= 0; --r) {
      const int t = ld_dsmem(dsmem(red_total, r));
      if (before < need && before + t >= need) {
        s_hit = r;
        s_before = before;
      }
      before += t;
    }
    sm.result[0] = s_hit;
    sm.result[1] = s_before;
  }
  __syncthreads();
  const int s_hit = sm.result[0], s_before = sm.result[1];
  __syncthreads();
  // scan the hit slice's bins, highest first (one bin per thread)
  const int hit_own = max(0, min(slice, nbins - s_hit * slice));
  int cnt = 0;
  if (static_cast<int>(threadIdx.x) < hit_own) cnt = ld_dsmem(dsmem(&red[hit_own - 1 - threadIdx.x], s_hit));
  int total;
  const int before = s_before + block_excl_scan(cnt, sm.scratch, &total);
  if (static_cast<int>(threadIdx.x) < hit_own && before < need && before + cnt >= need) {
    sm.result[0] = s_hit * slice + (hit_own - 1 - threadIdx.x);
    sm.result[1] = before;
  }
  __syncthreads();
  *above = sm.result[1];
  const int d = sm.result[0];
  __syncthreads();  // sm.result is reused by the next search
  return d;
}

// CL: CTAs per (document, head) cluster.  BLEND: how the fused path combines
// the pooled key score with the scale (a compile-time choice, so the product
// kernel's per-token loop carries nothing for the other blends).
template <int CL, int BLEND, int KP>
__global__ void __launch_bounds__(kThreads, 1) tp_select_kernel(const __grid_constant__ SelectParams p) {
  extern __shared__ __align__(128) uint8_t smem_raw[];
  SelectSmem& sm = *reinterpret_cast<SelectSmem*>(smem_raw);
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  // clusters launch in blockIdx.y order: the longest documents' units first,
  // so that a second wave holds the shortest ones
  // with several layers in one launch, units are layer-major
  const int per_layer = p.batch * p.n_heads_kv;
  const int layer = static_cast<int>(blockIdx.y) / per_layer;
  const int yl = static_cast<int>(blockIdx.y) - layer * per_layer;
  const int b = p.order[yl / p.n_heads_kv], h = yl % p.n_heads_kv;
  const int unit = b * p.n_heads_kv + h;
  const bool merged = p.layers > 1;
  const float* const skey_in = merged ? p.skey_l[layer] : p.skey;
  const float* const gamma_in = merged ? p.gamma_l[layer] : p.gamma;
  uint32_t* const keys_g = merged ? p.keys_l[layer] : p.keys;
  int32_t* const idx_out = merged ? p.idx_l[layer] : p.idx;
  const int64_t lo = p.off[b];
  const int n = static_cast<int>(p.off[b + 1] - lo);
  const int k = p.kept[b];
  const size_t row = static_cast<size_t>(h) * p.n_total + lo;
  // this CTA's slice [s0, s1) of the document's tokens
  const int per_cta = (((n + CL - 1) / CL) + 3) & ~3;
  const int s0 = min(rank * per_cta, n), s1 = min(s0 + per_cta, n);
  // the slice's keys: in shared memory when they fit, else in the global scratch
  const bool in_smem = (s1 - s0 <= kSliceKeys);
  uint32_t* const keys_base = in_smem ? sm.keys : keys_g + row;
  // key of token i: keys_base[kpos(i)].  In shared memory every 16 keys are
  // followed by a padding word, so the compaction's runs of 16 consecutive
  // keys per thread start 17 words apart and its reads hit distinct banks.
  auto kpos = [&](int i) {
    const int r = in_smem ? i - s0 : i;
    return in_smem ? r + (r >> 4) : r;
  };

  grid_dep_launch();
  for (int i = threadIdx.x; i < kBins1; i += kThreads) sm.hist1[i] = 0;
  for (int i = threadIdx.x; i < kBins2; i += kThreads) sm.hist2[i] = 0;
  for (int i = threadIdx.x; i < kBins3; i += kThreads) sm.hist3[i] = 0;
  grid_dep_wait();  // key scores and scales come from the scoring kernels
  __syncthreads();

  // A: keys of the slice (scores formed here in the fused path) + digit-1 histogram,
  // in sub-slices of kSliceKeys tokens whose key scores are staged with their halo.
  // The normalised-add blend first sweeps the slice for the sums of squares of
  // the pooled key scores and of the scales, reduced over the cluster.
  const int half = p.pool_kernel / 2;
  const float inv_k = 1.0f / static_cast<float>(p.pool_kernel);
  const bool fused = !p.scores_in;
  float inv_na = 0.f, inv_nb = 0.f;
  auto sweep = [&](bool norms_only) {
    float sa = 0.f, sb = 0.f;
    for (int c0 = s0; c0 < s1; c0 += kSliceKeys) {
      const int c1 = min(c0 + kSliceKeys, s1);
      // Every load of the sub-slice goes out at once, straight into shared
      // memory (cp.async, 16-byte groups where aligned): the key scores with
      // their halo and the scales (or given scores).  Halo positions outside
      // the document are zero.  One global round trip per sub-slice.
      const float* vsrc = p.scores_in ? p.scores_in : (p.key_only ? nullptr : gamma_in);
      const int64_t g0 = static_cast<int64_t>(row);  // global index of token 0
      const int64_t sref = (g0 + c0 - half) & ~int64_t(3), vref = (g0 + c0) & ~int64_t(3);
      if (fused) {
        const int ia = max(c0 - half, 0), ib = min(c1 + half, n);  // halo inside the document
        stage_floats(sm.strip, skey_in, g0 + ia, g0 + ib, sref);
        for (int i = c0 - half + static_cast<int>(threadIdx.x); i < c1 + half; i += kThreads)
          if (i < ia || i >= ib) sm.strip[g0 + i - sref] = 0.f;
      }
      if (vsrc) stage_floats(sm.vals, vsrc, g0 + c0, g0 + c1, vref);
      cp_async_wait_all();
      __syncthreads();
      // four independent keys per trip, so their shared-memory loads overlap
      const float* vrow = sm.vals + (g0 + c0 - vref);             // token c0 at vrow[0]
      const float* srow = sm.strip + (g0 + c0 - half - sref);      // token c0's window at srow[0]
#pragma unroll 4
      for (int i = c0 + threadIdx.x; i < c1; i += kThreads) {
        const int r = i - c0;
        float sc = vsrc ? vrow[r] : 1.f;
        if (fused) {
          const float* w = srow + r;
          float acc;
          if (half == 2) {  // the default window of five, summed in the same order
            acc = (((w[0] + w[1]) + w[2]) + w[3]) + w[4];
          } else {
            acc = 0.f;
            for (int o = 0; o <= 2 * half; ++o) acc += w[o];
          }
          const float a = acc * inv_k, g = sc;
          if (norms_only) {
            sa += a * a;
            sb += g * g;
            continue;
          }
          if (p.key_only) {
            sc = a;
          } else if constexpr (BLEND == kBlendNormAdd) {
            sc = a * inv_na + g * inv_nb;
          } else if constexpr (BLEND == kBlendHarmonic) {
            const float den = a + g;
            sc = den > 0.f ? __fdiv_rn(2.f * a * g, den) : 0.f;
          } else {
            sc = a * g;
          }
          if (p.scores_out) p.scores_out[row + i] = sc;
        }
        const uint32_t key = score_key(sc);
        keys_base[kpos(i)] = key;
        if (!p.scores_only) atomicAdd(&sm.hist1[key >> 20], 1);
      }
      __syncthreads();
    }
    if (norms_only) {
      sa = block_sum_f(sa, reinterpret_cast<float*>(sm.scratch));
      sb = block_sum_f(sb, reinterpret_cast<float*>(sm.scratch));
      if (threadIdx.x == 0) {
        sm.norm2[0] = sa;
        sm.norm2[1] = sb;
      }
    }
  };
  if (BLEND == kBlendNormAdd && fused && !p.key_only) {
    sweep(true);
    cluster.sync();  // every CTA's sums are in place
    if (threadIdx.x == 0) {
      float ta = 0.f, tb = 0.f;  // summed in rank order: the same on every CTA
      for (int r = 0; r < CL; ++r) {
        ta += __int_as_float(ld_dsmem(dsmem(&sm.norm2[0], r)));
        tb += __int_as_float(ld_dsmem(dsmem(&sm.norm2[1], r)));
      }
      sm.inv_norm[0] = ta > 0.f ? __fdiv_rn(1.f, sqrtf(ta)) : 0.f;
      sm.inv_norm[1] = tb > 0.f ? __fdiv_rn(1.f, sqrtf(tb)) : 0.f;
    }
    cluster.sync();  // no CTA moves on (or leaves) while another still reads its sums
    inv_na = sm.inv_norm[0];
    inv_nb = sm.inv_norm[1];
  }
  sweep(false);
  if (p.scores_only) return;  // no cluster-wide exchange follows

  const int64_t unit_slot0 = static_cast<int64_t>(unit) * p.cap;
  const int kk = max(0, min(k, n));
  if (rank == 0)
    for (int64_t t = kk + threadIdx.x; t < p.cap; t += kThreads) idx_out[unit_slot0 + t] = -1;
  cluster.sync();  // histograms of phase A complete everywhere

  uint32_t thr = 0;
  int need_eq = -1;  // -1: keep every token of the document
  // this thread's share of the slice's counts of keys above T and equal to T
  int gt_part = 0, eq_part = 0;
  if (kk > 0 && kk < n) {
    int above;
    const int d1 = cluster_digit<CL>(cluster, sm, sm.hist1, kBins1, kk, &above, 0);
    int need = kk - above;
#pragma unroll 4
    for (int i = s0 + threadIdx.x; i < s1; i += kThreads) {
      const uint32_t key = keys_base[kpos(i)];
      if ((key >> 20) == static_cast<uint32_t>(d1)) atomicAdd(&sm.hist2[(key >> 10) & 0x3FF], 1);
    }
    cluster.sync();
    const int d2 = cluster_digit<CL>(cluster, sm, sm.hist2, kBins2, need, &above, 1);
    need -= above;
    const uint32_t pre = (static_cast<uint32_t>(d1) << 10) | static_cast<uint32_t>(d2);
#pragma unroll 4
    for (int i = s0 + threadIdx.x; i < s1; i += kThreads) {
      const uint32_t key = keys_base[kpos(i)];
      if ((key >> 10) == pre) atomicAdd(&sm.hist3[key & 0x3FF], 1);
    }
    cluster.sync();
    const int d3 = cluster_digit<CL>(cluster, sm, sm.hist3, kBins3, need, &above, 2);
    need_eq = need - above;
    thr = (pre << 10) | static_cast<uint32_t>(d3);
    // The slice's own histograms give its counts: a key above T lies in a
    // higher digit-1 bin, or shares digit 1 and lies in a higher digit-2 bin,
    // or shares both and lies in a higher digit-3 bin; keys equal to T fill
    // digit-3 bin d3.  (cluster_digit ends with a block barrier, so every
    // local histogram update is visible.)
    for (int i = d1 + 1 + static_cast<int>(threadIdx.x); i < kBins1; i += kThreads) gt_part += sm.hist1[i];
    for (int i = d2 + 1 + static_cast<int>(threadIdx.x); i < kBins2; i += kThreads) gt_part += sm.hist2[i];
    for (int i = d3 + 1 + static_cast<int>(threadIdx.x); i < kBins3; i += kThreads) gt_part += sm.hist3[i];
    if (threadIdx.x == 0) eq_part = sm.hist3[d3];
  } else {
    // the same cluster-wide barriers as the other branch: one per digit
    // search (three searches) and one after each of the two later histograms
#pragma unroll 1
    for (int i = 0; i < 5; ++i) cluster.sync();
  }

  // D: counts of this slice, then prefix over the slices before it
  {
    // with every token kept (need_eq < 0) the slice counts entirely above T
    int gt = need_eq < 0 ? (kk > 0 && threadIdx.x == 0 ? s1 - s0 : 0) : gt_part;
    int eq = need_eq < 0 ? 0 : eq_part;
    if (s1 - s0 < 32768) {  // one block sum of (> T) << 16 | (== T), no overflow
      const int both = block_sum((gt << 16) | eq, sm.scratch);
      gt = both >> 16;
      eq = both & 0xFFFF;
    } else {
      gt = block_sum(gt, sm.scratch);
      eq = block_sum(eq, sm.scratch);
    }
    if (threadIdx.x == 0) {
      sm.counts[0] = gt;
      sm.counts[1] = eq;
    }
  }
  cluster.sync();
  // counts of the slices before this one: lane r < rank reads CTA r's (one
  // round trip), a warp sum, shared with the block
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    int g = 0, e = 0;
    if (lane < rank) {
      g = ld_dsmem(dsmem(&sm.counts[0], lane));
      e = ld_dsmem(dsmem(&sm.counts[1], lane));
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      g += __shfl_xor_sync(0xffffffffu, g, o);
      e += __shfl_xor_sync(0xffffffffu, e, o);
    }
    if (lane == 0) {
      sm.result[0] = g;
      sm.result[1] = e;
    }
  }
  __syncthreads();
  int gt_before = sm.result[0], eq_before = sm.result[1];
  cluster.sync();  // no CTA leaves while another may still read its counts

  if (kk <= 0) return;
  // ordered compaction in rounds of KP tokens per thread: a token's slot is
  // (tokens > T before it) + min(tokens == T before it, need_eq)
  for (int base = s0; base < s1; base += KP * kThreads) {
    const int j0 = base + threadIdx.x * KP;
    int ngt = 0, neq = 0;
    uint32_t kv[KP];
#pragma unroll
    for (int e = 0; e < KP; ++e) {
      const int j = j0 + e;
      kv[e] = j < s1 ? keys_base[kpos(j)] : 0u;
      if (j < s1) {
        if (need_eq < 0 || kv[e] > thr) ++ngt;
        else if (kv[e] == thr) ++neq;
      }
    }
    // one scan of packed counts: (> T) in the high 16 bits, (== T) in the low
    int tot;
    const int pre = block_excl_scan((ngt << 16) | neq, sm.scratch, &tot);
    const int tot_gt = tot >> 16, tot_eq = tot & 0xFFFF;
    int gt_rank = gt_before + (pre >> 16);
    int eq_rank = eq_before + (pre & 0xFFFF);
#pragma unroll
    for (int e = 0; e < KP; ++e) {
      const int j = j0 + e;
      if (j >= s1) break;
      const bool is_gt = need_eq < 0 || kv[e] > thr;
      const bool is_eq = !is_gt && kv[e] == thr;
      if (is_gt || (is_eq && eq_rank < need_eq)) {
        const int slot = gt_rank + (need_eq < 0 ? 0 : min(eq_rank, need_eq));
        idx_out[unit_slot0 + slot] = j;
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

template <int CL, int BLEND, int KP>
cudaError_t launch_select_t(const SelectParams& p, int units, size_t smem, bool dependent,
                            cudaStream_t s, int slot) {
  cudaError_t e = set_smem_once(reinterpret_cast<const void*>(tp_select_kernel<CL, BLEND, KP>), slot);
  if (e != cudaSuccess) return e;
  if (CL > 8) {  // clusters above the portable size of 8
    e = cudaFuncSetAttribute(reinterpret_cast<const void*>(tp_select_kernel<CL, BLEND, KP>),
                             cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(CL, units);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = CL;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = dependent ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, tp_select_kernel<CL, BLEND, KP>, p);
}

template <int CL, int KP = 16>
cudaError_t launch_select_blend(const SelectParams& p, int units, size_t smem, bool dependent,
                                cudaStream_t s, int slot0) {
  switch (p.blend) {
    case kBlendNormAdd:
      return launch_select_t<CL, kBlendNormAdd, KP>(p, units, smem, dependent, s, slot0 + 1);
    case kBlendHarmonic:
      return launch_select_t<CL, kBlendHarmonic, KP>(p, units, smem, dependent, s, slot0 + 2);
    default: return launch_select_t<CL, kBlendProduct, KP>(p, units, smem, dependent, s, slot0);
  }
}

// How many clusters of CL selection CTAs can be resident at once (0 if the
// query is refused), cached per CUDA context.
template <int CL>
int select_max_clusters(size_t smem, int slot) {
  constexpr int kEntries = 16;
  static std::mutex mu;
  static unsigned long long ctxs[kEntries];
  static int answers[kEntries];
  static int used;
  const unsigned long long ctx = context_key();
  {
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < used; ++i)
      if (ctxs[i] == ctx) return answers[i];
  }
  const void* fn = reinterpret_cast<const void*>(tp_select_kernel<CL, kBlendProduct, 16>);
  int n = 0;
  if (set_smem_once(fn, slot) == cudaSuccess &&
      (CL <= 8 || cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess)) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(CL, 1);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CL;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) n = 0;
  }
  cudaGetLastError();  // a refused query leaves no error behind
  std::lock_guard<std::mutex> lock(mu);
  if (ctx != 0 && used < kEntries) {
    ctxs[used] = ctx;
    answers[used++] = n;
  }
  return n;
}

cudaError_t launch_select(const SelectParams& p, bool dependent, cudaStream_t s) {
  const int units = p.batch * p.n_heads_kv * (p.layers > 1 ? p.layers : 1);
  if (units <= 0) return cudaSuccess;
  if (p.layers > kMaxSelectLayers) return cudaErrorInvalidValue;
  if (p.pool_kernel / 2 > kMaxHalf) return cudaErrorInvalidValue;
  const size_t smem = sizeof(SelectSmem);
  int dev = 0, sms = 148;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t n_max = 0;
  for (int b = 0; b < p.batch; ++b) n_max = p.off[b + 1] - p.off[b] > n_max ? p.off[b + 1] - p.off[b] : n_max;
  // shared-memory attribute slots: 12..14 for four-CTA clusters, 15..17 for
  // eight, 21..23 and 56..58 for twelve
  // Long documents (64K tokens and more): twelve CTAs per unit when every
  // unit's cluster is resident at once (8 such clusters fit on a 152-SM GB300:
  // 128K, 8 heads: 163.5 against 166.4 us per caller-normaliser layer).
  // Slices above 16 tokens per thread (128K: 10.9K tokens) compact in one
  // round of 22 per thread rather than two of 16 (1.8 us per 128K layer; 22
  // per thread everywhere was slower on shorter slices).
  if (n_max >= 65536 && select_max_clusters<12>(smem, 21) >= units) {
    const int64_t per_cta = (((n_max + 11) / 12) + 3) & ~int64_t(3);
    if (per_cta > 16 * kThreads) return launch_select_blend<12, 22>(p, units, smem, dependent, s, 56);
    return launch_select_blend<12>(p, units, smem, dependent, s, 21);
  }
  // Several layers in one launch: four-CTA clusters, which the caller checked
  // are all resident at once (select_merge_layers).
  if (p.layers > 1 && (n_max + 3) / 4 <= kSliceKeys)
    return launch_select_blend<4>(p, units, smem, dependent, s, 12);
  // Fewer, larger slices when eight CTAs per unit would need more than one wave.
  if (units * 8 > sms && (n_max + 3) / 4 <= kSliceKeys)
    return launch_select_blend<4>(p, units, smem, dependent, s, 12);
  return launch_select_blend<8>(p, units, smem, dependent, s, 15);
}

int select_merge_layers(int units_per_layer, int64_t n_max) {
  if (units_per_layer <= 0 || (n_max + 3) / 4 > kSliceKeys) return 1;
  const int clusters = select_max_clusters<4>(sizeof(SelectSmem), 12);
  const int layers = clusters / units_per_layer;
  return layers < 1 ? 1 : (layers > kMaxSelectLayers ? kMaxSelectLayers : layers);
}

}  // namespace tp
