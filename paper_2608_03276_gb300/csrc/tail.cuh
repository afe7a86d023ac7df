// The fused tail of scoring pass 2: a layer's top-budget selection (Sec. 3.4;
// Sec. 4 "Eviction": a uniform budget per KV head, heads selected
// independently) and the compaction of the kept rows, run by the same CTAs
// that scored the keys, right after their scoring loop.
//
// The CTAs of one (document, KV head) unit each own a contiguous key range.
// The selection is the three-digit radix select of the standalone selection
// kernel (11, 11 and 10 bits of the fp32 score's bit pattern, lowest token
// index first among equal scores), with the unit's histograms summed in global
// memory instead of a cluster's shared memory:
//   B1  every range's unpooled key scores are in global memory (Eq. 1's
//       pooling reads up to 16 scores of each neighbouring range);
//       radix keys of the range (pooled score x gamma, Eq. 3) into shared
//       memory, digit-1 histogram added into the unit's global histogram
//   B2  digit 1 (every CTA reads the same histogram and takes the same
//       decision); digit-2 histogram         B3  digit 2; digit-3 histogram
//   B4  threshold T: each range's (> T, == T) counts
//   B5  ordered compaction: a range's kept tokens take consecutive slots after
//       those of the ranges before it
//   B6  the unit's kept rows copied into the compressed cache, split evenly
//       over the unit's CTAs
// A barrier is an arrival counter per unit in the workspace (release add,
// acquire poll), bounded by the same 2 s limit as every other wait.  The host
// enables the tail only when the whole grid is resident at once (at most one
// CTA per SM and no more CTAs than SMs), so no CTA waits on one that cannot
// start.
#pragma once

#include "tp_device.cuh"

namespace tp {

constexpr int kTailChunk = 4096;   // tokens whose inputs are staged at once
constexpr int kTailHalfMax = 16;   // largest pooling half-window (pool kernel <= 33)
constexpr int kTailBins1 = 2048;   // key bits 31..21
constexpr int kTailBins2 = 2048;   // key bits 20..10
constexpr int kTailBins3 = 1024;   // key bits 9..0
constexpr int kTailPer = 16;       // tokens per thread in one compaction round
static_assert(kTailBins1 + kTailBins2 + kTailBins3 == kTailHistInts, "histogram layout");

struct TailSmem {
  uint32_t keys[kTailMaxKeys + kTailMaxKeys / 16];  // one padding word after every 16 keys
  // unpooled key scores of a chunk with its halo, and its scales: element g of
  // the global array sits at [g - g_ref], g_ref a multiple of 4
  float strip[kTailChunk + 2 * kTailHalfMax + 4];
  float vals[kTailChunk + 4];
  int hist[kTailBins1];  // this range's histogram of the current digit
  int scratch[33];
  int result[2];
};
static_assert(sizeof(uint32_t) * (kTailMaxKeys + kTailMaxKeys / 16) % 16 == 0 &&
                  sizeof(float) * (kTailChunk + 2 * kTailHalfMax + 4) % 16 == 0,
              "16-byte cp.async destinations must be 16-byte aligned");

__device__ __forceinline__ void red_release_add(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Stages global floats src[ga, gb) into dst[g - g_ref] (g_ref a multiple of 4,
// dst 16-byte aligned), reading through L2 only: the values were written by
// other CTAs of this grid.  16-byte cp.async.cg over the aligned middle, plain
// L2 loads at the two ragged ends.  Called by every thread of the block;
// complete after cp_async_wait_all() and a barrier.
__device__ __forceinline__ void stage_floats_l2(float* dst, const float* src, int64_t ga,
                                                int64_t gb, int64_t g_ref) {
  if (gb <= ga) return;
  const int64_t a4 = (ga + 3) & ~int64_t(3), b4 = gb & ~int64_t(3);
  // a caller's array need only be 4-byte aligned: then every load is 4 bytes
  if (a4 >= b4 || (reinterpret_cast<uintptr_t>(src) & 15) != 0) {
    for (int64_t g = ga + threadIdx.x; g < gb; g += blockDim.x) dst[g - g_ref] = __ldcg(src + g);
    return;
  }
  const int64_t groups = (b4 - a4) >> 2;
  for (int64_t q = threadIdx.x; q < groups; q += blockDim.x) {
    const int64_t g = a4 + 4 * q;
    cp_async16(dst + (g - g_ref), src + g);
  }
  const int head = static_cast<int>(a4 - ga), tail = static_cast<int>(gb - b4);
  if (static_cast<int>(threadIdx.x) < head) {
    const int64_t g = ga + threadIdx.x;
    dst[g - g_ref] = __ldcg(src + g);
  } else if (static_cast<int>(threadIdx.x) >= 32 && static_cast<int>(threadIdx.x) < 32 + tail) {
    const int64_t g = b4 + (threadIdx.x - 32);
    dst[g - g_ref] = __ldcg(src + g);
  }
}

// Adds this range's histogram into the unit's global one (non-zero bins only)
// and clears it for the next digit.
__device__ __forceinline__ void tail_flush_hist(int* gh, int* lh, int nbins) {
  __syncthreads();
  for (int i = threadIdx.x; i < nbins; i += blockDim.x) {
    const int c = lh[i];
    if (c) {
      atomicAdd(gh + i, c);
      lh[i] = 0;
    }
  }
}

// Bin of the unit histogram gh[nbins] holding the need-th largest key
// (1-based); *above = keys in higher bins.  Threads 0..511 read nbins/512
// consecutive bins each, highest first; every CTA of the unit reads the same
// counts and takes the same decision.  Called by every thread of the block.
__device__ __forceinline__ int tail_digit(const int* gh, int nbins, int need, int* above,
                                          TailSmem& sm) {
  const int per = nbins / 512;  // 4 (2048 bins) or 2 (1024 bins)
  int cnt[4] = {0, 0, 0, 0};
  int sum = 0;
  if (threadIdx.x < 512) {
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (j < per) {
        cnt[j] = __ldcg(gh + (nbins - 1 - (static_cast<int>(threadIdx.x) * per + j)));
        sum += cnt[j];
      }
  }
  int total;
  int before = block_excl_scan(sum, sm.scratch, &total);
  if (threadIdx.x < 512 && before < need && before + sum >= need) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (j < per && before + cnt[j] >= need) {
        sm.result[0] = nbins - 1 - (static_cast<int>(threadIdx.x) * per + j);
        sm.result[1] = before;
        break;
      }
      before += cnt[j];
    }
  }
  __syncthreads();
  *above = sm.result[1];
  const int d = sm.result[0];
  __syncthreads();  // sm.result is reused by the next search
  return d;
}

// Copies kept slots [sa, sb) of a unit (indices already in p.idx) into the
// compressed cache: K and V rows, their Eq. 2 codes from gamma, and gamma.
// A group of D/8 lanes moves one slot, four slots per lane in flight.
template <int D>
__device__ __forceinline__ void tail_gather(const KeyScoreParams& p, int64_t g0, int64_t slot0,
                                            int64_t sa, int64_t sb, int n) {
  constexpr int LPR = D / 8;
  constexpr int UNR = 4;
  const int part = threadIdx.x % LPR;
  const int ngroups = blockDim.x / LPR;
  const uint4* kin = reinterpret_cast<const uint4*>(p.k);
  const uint4* vin = reinterpret_cast<const uint4*>(p.v);
  for (int64_t s = sa + threadIdx.x / LPR; s < sb; s += static_cast<int64_t>(ngroups) * UNR) {
    int32_t j[UNR];
    uint4 kv[UNR], vv[UNR];
    float g[UNR];
#pragma unroll
    for (int u = 0; u < UNR; ++u) {
      const int64_t t = s + static_cast<int64_t>(u) * ngroups;
      j[u] = t < sb ? __ldcg(p.idx + slot0 + t) : -1;
      if (j[u] >= n) j[u] = -1;  // never read outside the document
    }
#pragma unroll
    for (int u = 0; u < UNR; ++u) {
      kv[u] = vv[u] = make_uint4(0, 0, 0, 0);
      g[u] = 0.f;
      if (j[u] >= 0) {
        const int64_t tok = g0 + j[u];
        kv[u] = __ldcs(kin + tok * LPR + part);
        vv[u] = __ldcs(vin + tok * LPR + part);
        g[u] = __ldcg(p.gamma + tok);
      }
    }
#pragma unroll
    for (int u = 0; u < UNR; ++u) {
      const int64_t t = s + static_cast<int64_t>(u) * ngroups;
      if (t >= sb) continue;
      const int64_t slot = slot0 + t;
      const int64_t dst = slot * LPR + part;
      if (p.kc) reinterpret_cast<uint4*>(p.kc)[dst] = kv[u];
      if (p.vc) reinterpret_cast<uint4*>(p.vc)[dst] = vv[u];
      if (p.vqc) {
        if (p.bits == 8)
          reinterpret_cast<uint2*>(p.vqc)[dst] = quant8_packed(vv[u], g[u], p.qmax);
        else
          reinterpret_cast<uint32_t*>(p.vqc)[dst] = quant4_packed(vv[u], g[u], p.qmax);
      }
      if (p.gammac && part == 0) p.gammac[slot] = g[u];
    }
  }
}

// Fills slots [sa, sb) of a unit as unused: idx -1, zero rows and scale.
template <int D>
__device__ __forceinline__ void tail_clear(const KeyScoreParams& p, int64_t slot0, int64_t sa,
                                           int64_t sb) {
  constexpr int LPR = D / 8;
  const int part = threadIdx.x % LPR;
  const int ngroups = blockDim.x / LPR;
  for (int64_t t = sa + threadIdx.x / LPR; t < sb; t += ngroups) {
    const int64_t slot = slot0 + t;
    const int64_t dst = slot * LPR + part;
    if (part == 0) {
      p.idx[slot] = -1;
      if (p.gammac) p.gammac[slot] = 0.f;
    }
    if (p.kc) reinterpret_cast<uint4*>(p.kc)[dst] = make_uint4(0, 0, 0, 0);
    if (p.vc) reinterpret_cast<uint4*>(p.vc)[dst] = make_uint4(0, 0, 0, 0);
    if (p.vqc) {
      if (p.bits == 8) reinterpret_cast<uint2*>(p.vqc)[dst] = make_uint2(0, 0);
      else reinterpret_cast<uint32_t*>(p.vqc)[dst] = 0u;
    }
  }
}

// The tail of one CTA: document b, head h, this CTA the c-th of the ncta CTAs
// of the unit, owning key tiles t0 .. t0+nt-1 of the n-token document.  Every
// thread of the block calls it after the scoring loop (the shared memory of
// the scoring pipeline is free again).
template <int D>
__device__ void keyscore_tail(const KeyScoreParams& p, uint8_t* smem, int b, int h, int c,
                              int ncta, int t0, int nt, int n, int64_t doc_lo,
                              volatile int* abort_flag) {
  TailSmem& sm = *reinterpret_cast<TailSmem*>(smem);
  const int unit = b * p.n_heads_kv + h;
  int* const ctr = p.tsync + 2 * unit;  // arrivals, departures
  int* const gh1 = p.thist + static_cast<size_t>(unit) * kTailHistInts;
  int* const gh2 = gh1 + kTailBins1;
  int* const gh3 = gh2 + kTailBins2;
  const int kk = max(0, min(p.kept[b], n));
  const bool radix = kk > 0 && kk < n;
  const int phases = 1 + (radix ? 3 : 0) + (kk > 0 ? 2 : 0);
  const int s0 = t0 * kKeyTile, s1 = min((t0 + nt) * kKeyTile, n);
  const int64_t g0 = static_cast<int64_t>(h) * p.n_total + doc_lo;  // token 0 of the document
  const int64_t slot0 = static_cast<int64_t>(unit) * p.cap;
  const int cta_lin = blockIdx.y * gridDim.x + blockIdx.x;
  int arrived = 0;  // thread 0's arrivals on ctr
  int phase = 0;

  // barrier over the unit's CTAs: every CTA's global writes before it are
  // visible to every CTA after it
  auto unit_sync = [&]() -> bool {
    ++phase;
    __syncthreads();
    if (threadIdx.x == 0 && !*abort_flag) {
      __threadfence();
      red_release_add(ctr, 1);
      ++arrived;
      const int target = phase * ncta;
      if (ld_acquire(ctr) < target) {
        const uint64_t tw = global_timer_ns();
        while (ld_acquire(ctr) < target) {
          if (global_timer_ns() - tw > kWaitLimitNs) {
            *abort_flag = 1;
            break;
          }
          __nanosleep(64);
        }
      }
      __threadfence();
    }
    __syncthreads();
    return *abort_flag == 0;
  };
  // leaves the unit's barriers: the last CTA to leave resets the counters for
  // the next layer (no CTA of the unit polls them any more)
  auto leave = [&]() {
    if (threadIdx.x == 0) {
      if (phases > arrived) red_release_add(ctr, phases - arrived);
      const int old = atomicAdd(ctr + 1, 1);
      if (old == ncta - 1) {
        atomicExch(ctr, 0);
        atomicExch(ctr + 1, 0);
      }
    }
  };
  auto bail = [&]() {
    if (threadIdx.x == 0) set_status(p.status, TP_ERR_TIMEOUT);
    leave();
  };

  if (*abort_flag) {
    bail();
    return;
  }
  // this CTA's share of the unit's histograms starts at zero (before B1, so
  // every CTA adds into zeroed bins after it)
  if (radix) {
    const int za = kTailHistInts * c / ncta, zb = kTailHistInts * (c + 1) / ncta;
    for (int i = za + threadIdx.x; i < zb; i += blockDim.x) gh1[i] = 0;
  }
  for (int i = threadIdx.x; i < kTailBins1; i += blockDim.x) sm.hist[i] = 0;
  if (!unit_sync()) {  // B1
    bail();
    return;
  }

  // radix keys of the range: Eq. 1 pooling of the key scores (zero outside the
  // document, divisor K), times gamma (Eq. 3) or a blend
  const int half = p.pool_kernel / 2;
  const float inv_k = 1.0f / static_cast<float>(p.pool_kernel);
  auto kpos = [&](int i) {
    const int r = i - s0;
    return r + (r >> 4);
  };
  for (int c0 = s0; c0 < s1; c0 += kTailChunk) {
    const int c1 = min(c0 + kTailChunk, s1);
    const int64_t sref = (g0 + c0 - half) & ~int64_t(3), vref = (g0 + c0) & ~int64_t(3);
    const int ia = max(c0 - half, 0), ib = min(c1 + half, n);  // halo inside the document
    stage_floats_l2(sm.strip, p.skey, g0 + ia, g0 + ib, sref);
    for (int i = c0 - half + static_cast<int>(threadIdx.x); i < c1 + half; i += blockDim.x)
      if (i < ia || i >= ib) sm.strip[g0 + i - sref] = 0.f;
    if (!p.key_only) stage_floats_l2(sm.vals, p.gamma, g0 + c0, g0 + c1, vref);
    cp_async_wait_all();
    __syncthreads();
    const float* vrow = sm.vals + (g0 + c0 - vref);         // token c0 at vrow[0]
    const float* srow = sm.strip + (g0 + c0 - half - sref);  // token c0's window at srow[0]
#pragma unroll 4
    for (int i = c0 + threadIdx.x; i < c1; i += blockDim.x) {
      const int r = i - c0;
      const float* w = srow + r;
      float acc;
      if (half == 2) {  // the default window of five, summed in the same order
        acc = (((w[0] + w[1]) + w[2]) + w[3]) + w[4];
      } else {
        acc = 0.f;
        for (int o = 0; o <= 2 * half; ++o) acc += w[o];
      }
      const float a = acc * inv_k;
      float sc;
      if (p.key_only) {
        sc = a;
      } else if (p.blend == kBlendHarmonic) {
        const float g = vrow[r];
        const float den = a + g;
        sc = den > 0.f ? __fdiv_rn(2.f * a * g, den) : 0.f;
      } else {
        sc = a * vrow[r];
      }
      if (p.scores_out) p.scores_out[g0 + i] = sc;
      const uint32_t key = score_key(sc);
      sm.keys[kpos(i)] = key;
      if (radix) atomicAdd(&sm.hist[key >> 21], 1);
    }
    __syncthreads();
  }

  uint32_t thr = 0;
  int need_eq = -1;  // -1: every token of the document is kept
  if (radix) {
    tail_flush_hist(gh1, sm.hist, kTailBins1);
    if (!unit_sync()) {  // B2
      bail();
      return;
    }
    int above;
    const int d1 = tail_digit(gh1, kTailBins1, kk, &above, sm);
    int need = kk - above;
#pragma unroll 4
    for (int i = s0 + threadIdx.x; i < s1; i += blockDim.x) {
      const uint32_t key = sm.keys[kpos(i)];
      if ((key >> 21) == static_cast<uint32_t>(d1)) atomicAdd(&sm.hist[(key >> 10) & 0x7FF], 1);
    }
    tail_flush_hist(gh2, sm.hist, kTailBins2);
    if (!unit_sync()) {  // B3
      bail();
      return;
    }
    const int d2 = tail_digit(gh2, kTailBins2, need, &above, sm);
    need -= above;
    const uint32_t pre = (static_cast<uint32_t>(d1) << 11) | static_cast<uint32_t>(d2);
#pragma unroll 4
    for (int i = s0 + threadIdx.x; i < s1; i += blockDim.x) {
      const uint32_t key = sm.keys[kpos(i)];
      if ((key >> 10) == pre) atomicAdd(&sm.hist[key & 0x3FF], 1);
    }
    tail_flush_hist(gh3, sm.hist, kTailBins3);
    if (!unit_sync()) {  // B4
      bail();
      return;
    }
    const int d3 = tail_digit(gh3, kTailBins3, need, &above, sm);
    need_eq = need - above;
    thr = (pre << 10) | static_cast<uint32_t>(d3);
  }

  if (kk > 0) {
    // (> T, == T) counts of this range
    int gt = 0, eq = 0;
#pragma unroll 4
    for (int i = s0 + threadIdx.x; i < s1; i += blockDim.x) {
      const uint32_t key = sm.keys[kpos(i)];
      if (need_eq < 0 || key > thr) ++gt;
      else if (key == thr) ++eq;
    }
    gt = block_sum(gt, sm.scratch);
    eq = block_sum(eq, sm.scratch);
    if (threadIdx.x == 0) {
      p.tcount[2 * cta_lin] = gt;
      p.tcount[2 * cta_lin + 1] = eq;
    }
    if (!unit_sync()) {  // B5
      bail();
      return;
    }
    // counts of the unit's ranges before this one (CTAs c' < c of this head row)
    if (threadIdx.x < 32) {
      int a = 0, e = 0;
      const int lin0 = cta_lin - c;
      for (int j = threadIdx.x; j < c; j += 32) {
        a += __ldcg(p.tcount + 2 * (lin0 + j));
        e += __ldcg(p.tcount + 2 * (lin0 + j) + 1);
      }
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) {
        a += __shfl_xor_sync(0xffffffffu, a, o);
        e += __shfl_xor_sync(0xffffffffu, e, o);
      }
      if (threadIdx.x == 0) {
        sm.result[0] = a;
        sm.result[1] = e;
      }
    }
    __syncthreads();
    int gt_before = sm.result[0], eq_before = sm.result[1];
    __syncthreads();
    // ordered compaction: a kept token's slot is (tokens > T before it) +
    // min(tokens == T before it, need_eq)
    const int round = static_cast<int>(blockDim.x) * kTailPer;
    for (int base = s0; base < s1; base += round) {
      const int j0 = base + static_cast<int>(threadIdx.x) * kTailPer;
      int ngt = 0, neq = 0;
      uint32_t kv[kTailPer];
#pragma unroll
      for (int e = 0; e < kTailPer; ++e) {
        const int j = j0 + e;
        kv[e] = j < s1 ? sm.keys[kpos(j)] : 0u;
        if (j < s1) {
          if (need_eq < 0 || kv[e] > thr) ++ngt;
          else if (kv[e] == thr) ++neq;
        }
      }
      // one scan of packed counts: (> T) in the high 16 bits, (== T) in the low
      int tot;
      const int pre = block_excl_scan((ngt << 16) | neq, sm.scratch, &tot);
      int gt_rank = gt_before + (pre >> 16);
      int eq_rank = eq_before + (pre & 0xFFFF);
#pragma unroll
      for (int e = 0; e < kTailPer; ++e) {
        const int j = j0 + e;
        if (j >= s1) break;
        const bool is_gt = need_eq < 0 || kv[e] > thr;
        const bool is_eq = !is_gt && kv[e] == thr;
        if (is_gt || (is_eq && eq_rank < need_eq)) {
          const int slot = gt_rank + (need_eq < 0 ? 0 : min(eq_rank, need_eq));
          if (slot < kk) p.idx[slot0 + slot] = j;  // always true when the counts agree
        }
        gt_rank += is_gt;
        eq_rank += is_eq;
      }
      gt_before += tot >> 16;
      eq_before += tot & 0xFFFF;
    }
    if (!unit_sync()) {  // B6: every kept index of the unit is written
      bail();
      return;
    }
    tail_gather<D>(p, g0, slot0, static_cast<int64_t>(kk) * c / ncta,
                   static_cast<int64_t>(kk) * (c + 1) / ncta, n);
  }
  // unused slots kk .. cap-1 of the unit, split over its CTAs
  const int64_t spare = p.cap - kk;
  if (spare > 0)
    tail_clear<D>(p, slot0, kk + spare * c / ncta, kk + spare * (c + 1) / ncta);
  // documents without tokens have no CTAs: every CTA of the grid clears a
  // share of their rows
  const int ctas = gridDim.x * gridDim.y;
  for (int bb = 0; bb < p.docs.batch; ++bb) {
    if (p.docs.off[bb + 1] != p.docs.off[bb]) continue;
    for (int hh = 0; hh < p.n_heads_kv; ++hh) {
      const int64_t s_lo = static_cast<int64_t>(bb * p.n_heads_kv + hh) * p.cap;
      tail_clear<D>(p, s_lo, p.cap * cta_lin / ctas, p.cap * (cta_lin + 1) / ctas);
    }
  }
  leave();
}

}  // namespace tp
