// The fused tail of scoring pass 2: a layer's top-budget selection (Sec. 3.4;
// Sec. 4 "Eviction": a uniform budget per KV head, heads selected
// independently) and the compaction of the kept rows, run by the same CTAs
// that scored the keys.
//
// The CTAs of one (document, KV head) unit each own a contiguous key range.
// The selection is the three-digit radix select of the standalone selection
// kernel (11, 11 and 10 bits of the fp32 score's bit pattern, lowest token
// index first among equal scores), with the unit's histograms summed in global
// memory instead of a cluster's shared memory.
//
// During the scoring loop two otherwise idle warps of each CTA turn every
// scored tile into radix keys (Eq. 1 pooling x gamma, Eq. 3) and count their
// top digit (tail_keys_in_loop).  A key needs the scores up to K/2 tokens to
// its right, so the keys of the last K/2 tokens of a range wait for the next
// CTA's first tile, which that CTA announces with a flag as soon as it is
// scored.  After the loop (keyscore_tail):
//   B1  the unit's digit-1 histogram is complete and every key is written;
//       digit 1 (every CTA reads the same histogram and takes the same
//       decision); digit-2 histogram       B2  digit 2; digit-3 histogram
//   B3  threshold T: each range's (> T, == T) counts
//   B4  ordered compaction: a range's kept tokens take consecutive slots after
//       those of the ranges before it (warp ballots)
//   B5  the unit's kept rows copied into the compressed cache, split evenly
//       over the unit's CTAs
// A barrier is an arrival counter per unit in the workspace (release add,
// acquire poll), bounded by the same 2 s limit as every other wait.  The host
// enables the tail only when the whole grid is resident at once (at most one
// CTA per SM and no more CTAs than SMs), so no CTA waits on one that cannot
// start.
#pragma once

#include "tp_device.cuh"

namespace tp {

constexpr int kTailBins1 = 2048;   // key bits 31..21
constexpr int kTailBins2 = 2048;   // key bits 20..10
constexpr int kTailBins3 = 1024;   // key bits 9..0
constexpr int kKeyWarp0 = 18;      // first of the two key warps of pass 2
constexpr int kKeyThreads = 64;
static_assert(kTailBins1 + kTailBins2 + kTailBins3 == kTailHistInts, "histogram layout");

struct TailSmem {
  // the range's keys: token i at keys[g0 + i - kref], kref = (g0 + first) & ~3
  uint32_t keys[kTailMaxKeys + 4];
  int hist[kTailBins2];   // this range's histogram of digit 2 or 3
  int scratch[33];
  int result[2];
  int wsum[2][32];        // per-warp (> T, == T) counts, then their exclusive prefix
};
static_assert(sizeof(uint32_t) * (kTailMaxKeys + 4) % 16 == 0, "16-byte cp.async destinations");

__device__ __forceinline__ void red_release_add(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release(int* p, int v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Stages 32-bit words src[ga, gb) into dst[g - g_ref] (g_ref a multiple of 4,
// dst 16-byte aligned), reading through L2 only: 16-byte cp.async.cg over the
// aligned middle, plain L2 loads at the two ragged ends (or everywhere when
// src is not 16-byte aligned).  Called by every thread of the block; complete
// after cp_async_wait_all() and a barrier.
__device__ __forceinline__ void stage_words_l2(uint32_t* dst, const uint32_t* src, int64_t ga,
                                               int64_t gb, int64_t g_ref) {
  if (gb <= ga) return;
  const int64_t a4 = (ga + 3) & ~int64_t(3), b4 = gb & ~int64_t(3);
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

// Radix key of token i of the document whose token 0 is global index g0
// (Eq. 1 pooling of the unpooled key scores, zero outside [0, n), divisor K;
// then Eq. 3's product with gamma, or the harmonic blend, or the key score
// alone); the combined score goes to scores_out when asked.  Reads through L2.
__device__ __forceinline__ uint32_t tail_key(const KeyScoreParams& p, int64_t g0, int i, int n,
                                             int half, float inv_k) {
  const float* w = p.skey + g0 + i - half;
  float acc;
  if (half == 2 && i >= 2 && i + 2 < n) {  // the default window of five, summed in the same order
    acc = (((__ldcg(w) + __ldcg(w + 1)) + __ldcg(w + 2)) + __ldcg(w + 3)) + __ldcg(w + 4);
  } else {
    acc = 0.f;
    for (int o = 0; o <= 2 * half; ++o) {
      const int t = i - half + o;
      acc += (t >= 0 && t < n) ? __ldcg(w + o) : 0.f;
    }
  }
  const float a = acc * inv_k;
  float sc;
  if (p.key_only) {
    sc = a;
  } else if (p.blend == kBlendHarmonic) {
    const float g = __ldcg(p.gamma + g0 + i);
    const float den = a + g;
    sc = den > 0.f ? __fdiv_rn(2.f * a * g, den) : 0.f;
  } else {
    sc = a * __ldcg(p.gamma + g0 + i);
  }
  if (p.scores_out) p.scores_out[g0 + i] = sc;
  return score_key(sc);
}

// Digit-1 count of a key in the packed 16-bit histogram (bins 2w and 2w + 1
// share word w; a range holds at most kTailMaxKeys keys, so no count overflows).
__device__ __forceinline__ void hist16_add(uint32_t* hist16, uint32_t key) {
  const uint32_t bin = key >> 21;
  atomicAdd(hist16 + (bin >> 1), 1u << ((bin & 1u) << 4));
}

// Waits until *count reaches `target` (bounded like every wait).
__device__ __forceinline__ bool wait_count(volatile int* count, int target, volatile int* abort_flag) {
  if (*count >= target) return true;
  const uint64_t t0 = global_timer_ns();
  while (*count < target) {
    if (*abort_flag) return false;
    if (global_timer_ns() - t0 > kWaitLimitNs) {
      *abort_flag = 1;
      return false;
    }
    __nanosleep(64);
  }
  return true;
}

// The two key warps during the scoring loop: keys of tokens [o0, ilim) of the
// CTA's range, tile by tile, as the epilogue announces scored tiles on
// `tiles_done` (four arrivals per tile).  ilim stops K/2 tokens short of the
// range's end unless the range ends the document.  After tile 0 is scored its
// keys... and the CTA's flag tells the previous CTA of the unit that the
// scores it needs for its last K/2 keys are in memory.
__device__ void tail_keys_in_loop(const KeyScoreParams& p, uint32_t* hist16, volatile int* tiles_done,
                                  int c, int t0, int nt, int n, int64_t doc_lo, int h,
                                  volatile int* abort_flag) {
  const int tid = static_cast<int>(threadIdx.x) - kKeyWarp0 * 32;
  for (int i = tid; i < kTailBins1 / 2; i += kKeyThreads) hist16[i] = 0;
  asm volatile("bar.sync 1, %0;" ::"n"(kKeyThreads) : "memory");  // the two key warps only
  const int half = p.pool_kernel / 2;
  const float inv_k = 1.0f / static_cast<float>(p.pool_kernel);
  const int s0 = t0 * kKeyTile, s1 = min((t0 + nt) * kKeyTile, n);
  const int o0 = c == 0 ? 0 : min(s0 + half, n);
  const int ilim = s1 >= n ? n : s1 - half;
  const int64_t g0 = static_cast<int64_t>(h) * p.n_total + doc_lo;
  const int cta_lin = blockIdx.y * gridDim.x + blockIdx.x;
  for (int lt = 0; lt < nt; ++lt) {
    if (!wait_count(tiles_done, 4 * min(lt + 2, nt), abort_flag)) return;
    if (lt == 0 && tid == 0) {
      __threadfence();
      st_release(p.tflag + cta_lin, p.epoch);
    }
    const int a = max(o0, s0 + lt * kKeyTile), e = min(s0 + (lt + 1) * kKeyTile, ilim);
    for (int i = a + tid; i < e; i += kKeyThreads) {
      const uint32_t key = tail_key(p, g0, i, n, half, inv_k);
      p.keys[g0 + i] = key;
      hist16_add(hist16, key);
    }
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
// of the unit, owning key tiles t0 .. t0+nt-1 of the n-token document; its
// key range is [o0, o1) (the tiles' tokens shifted right by K/2, see above).
// `hist16` holds the digit-1 counts of the keys the key warps formed.  Every
// thread of the block calls it after the scoring loop (the shared memory of
// the scoring pipeline is free again).
template <int D>
__device__ void keyscore_tail(const KeyScoreParams& p, uint8_t* smem, uint32_t* hist16, int b,
                              int h, int c, int ncta, int t0, int nt, int n, int64_t doc_lo,
                              volatile int* abort_flag) {
  TailSmem& sm = *reinterpret_cast<TailSmem*>(smem);
  const int unit = b * p.n_heads_kv + h;
  int* const ctr = p.tsync + 2 * unit;  // arrivals, departures
  int* const gh1 = p.thist + static_cast<size_t>(unit) * kTailHistInts;
  int* const gh2 = gh1 + kTailBins1;
  int* const gh3 = gh2 + kTailBins2;
  const int kk = max(0, min(p.kept[b], n));
  const bool radix = kk > 0 && kk < n;
  const int phases = 1 + (radix ? 2 : 0) + (kk > 0 ? 2 : 0);
  const int half = p.pool_kernel / 2;
  const int s1 = min((t0 + nt) * kKeyTile, n);
  const int o0 = c == 0 ? 0 : min(t0 * kKeyTile + half, n);
  const int o1 = c == ncta - 1 ? n : min(s1 + half, n);
  const int64_t g0 = static_cast<int64_t>(h) * p.n_total + doc_lo;  // token 0 of the document
  const int64_t kref = (g0 + o0) & ~int64_t(3);
  const int64_t slot0 = static_cast<int64_t>(unit) * p.cap;
  const int cta_lin = blockIdx.y * gridDim.x + blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
  int arrived = 0;  // thread 0's arrivals on ctr
  int phase = 0;
  auto key_at = [&](int i) { return sm.keys[g0 + i - kref]; };

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
          __nanosleep(32);
        }
      }
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
  // keys of the last K/2 tokens of the range: their windows reach into the
  // next CTA's first tile, announced by that CTA's flag
  if (c < ncta - 1) {
    if (threadIdx.x == 0) {
      const int* flag = p.tflag + cta_lin + 1;
      const uint64_t tw = global_timer_ns();
      while (ld_acquire(flag) < p.epoch) {
        if (global_timer_ns() - tw > kWaitLimitNs) {
          *abort_flag = 1;
          break;
        }
        __nanosleep(32);
      }
    }
    __syncthreads();
    if (*abort_flag) {
      bail();
      return;
    }
    const float inv_k = 1.0f / static_cast<float>(p.pool_kernel);
    for (int i = max(o0, s1 - half) + static_cast<int>(threadIdx.x); i < o1; i += blockDim.x) {
      const uint32_t key = tail_key(p, g0, i, n, half, inv_k);
      p.keys[g0 + i] = key;
      hist16_add(hist16, key);
    }
  }
  __syncthreads();
  // the range's digit-1 counts into the unit's histogram, and its keys into
  // shared memory (in flight across the barrier)
  if (radix) {
    for (int w = threadIdx.x; w < kTailBins1 / 2; w += blockDim.x) {
      const uint32_t v = hist16[w];
      if (v & 0xFFFFu) atomicAdd(gh1 + 2 * w, static_cast<int>(v & 0xFFFFu));
      if (v >> 16) atomicAdd(gh1 + 2 * w + 1, static_cast<int>(v >> 16));
    }
  }
  if (kk > 0) stage_words_l2(sm.keys, p.keys, g0 + o0, g0 + o1, kref);
  for (int i = threadIdx.x; i < kTailBins2; i += blockDim.x) sm.hist[i] = 0;
  cp_async_wait_all();
  if (!unit_sync()) {  // B1: digit-1 histogram complete, every key written
    bail();
    return;
  }

  uint32_t thr = 0;
  int need_eq = -1;  // -1: every token of the document is kept
  if (radix) {
    int above;
    const int d1 = tail_digit(gh1, kTailBins1, kk, &above, sm);
    int need = kk - above;
#pragma unroll 4
    for (int i = o0 + threadIdx.x; i < o1; i += blockDim.x) {
      const uint32_t key = key_at(i);
      if ((key >> 21) == static_cast<uint32_t>(d1)) atomicAdd(&sm.hist[(key >> 10) & 0x7FF], 1);
    }
    tail_flush_hist(gh2, sm.hist, kTailBins2);
    if (!unit_sync()) {  // B2
      bail();
      return;
    }
    const int d2 = tail_digit(gh2, kTailBins2, need, &above, sm);
    need -= above;
    const uint32_t pre = (static_cast<uint32_t>(d1) << 11) | static_cast<uint32_t>(d2);
#pragma unroll 4
    for (int i = o0 + threadIdx.x; i < o1; i += blockDim.x) {
      const uint32_t key = key_at(i);
      if ((key >> 10) == pre) atomicAdd(&sm.hist[key & 0x3FF], 1);
    }
    tail_flush_hist(gh3, sm.hist, kTailBins3);
    if (!unit_sync()) {  // B3
      bail();
      return;
    }
    const int d3 = tail_digit(gh3, kTailBins3, need, &above, sm);
    need_eq = need - above;
    thr = (pre << 10) | static_cast<uint32_t>(d3);
  }

  if (kk > 0) {
    // warp w owns the chunk [w0, w1) of the range, a multiple of 32 tokens long
    const int m = o1 - o0;
    const int chunk = ((m + nwarps - 1) / nwarps + 31) & ~31;
    const int w0 = min(o0 + warp * chunk, o1), w1 = min(w0 + chunk, o1);
    int gt = 0, eq = 0;
    for (int j = w0 + lane; j < w1; j += 32) {
      const uint32_t key = key_at(j);
      if (need_eq < 0 || key > thr) ++gt;
      else if (key == thr) ++eq;
    }
    gt = __reduce_add_sync(0xffffffffu, gt);
    eq = __reduce_add_sync(0xffffffffu, eq);
    if (lane == 0) {
      sm.wsum[0][warp] = gt;
      sm.wsum[1][warp] = eq;
    }
    __syncthreads();
    if (threadIdx.x == 0) {  // the range's counts, and each warp's prefix within it
      int a = 0, e = 0;
      for (int w = 0; w < nwarps; ++w) {
        const int tg = sm.wsum[0][w], te = sm.wsum[1][w];
        sm.wsum[0][w] = a;
        sm.wsum[1][w] = e;
        a += tg;
        e += te;
      }
      p.tcount[2 * cta_lin] = a;
      p.tcount[2 * cta_lin + 1] = e;
    }
    if (!unit_sync()) {  // B3 / B4: every range's counts are in memory
      bail();
      return;
    }
    // zero this CTA's share of the unit's histograms for the next layer:
    // every CTA read them before arriving here
    if (radix) {
      const int za = kTailHistInts * c / ncta, zb = kTailHistInts * (c + 1) / ncta;
      for (int i = za + threadIdx.x; i < zb; i += blockDim.x) gh1[i] = 0;
    }
    // counts of the unit's ranges before this one (CTAs c' < c of this head row)
    if (warp == 0) {
      int a = 0, e = 0;
      const int lin0 = cta_lin - c;
      for (int j = lane; j < c; j += 32) {
        a += __ldcg(p.tcount + 2 * (lin0 + j));
        e += __ldcg(p.tcount + 2 * (lin0 + j) + 1);
      }
      a = __reduce_add_sync(0xffffffffu, a);
      e = __reduce_add_sync(0xffffffffu, e);
      if (lane == 0) {
        sm.result[0] = a;
        sm.result[1] = e;
      }
    }
    __syncthreads();
    // ordered compaction by warp ballots: a kept token's slot is (tokens > T
    // before it) + min(tokens == T before it, need_eq)
    int gbase = sm.result[0] + sm.wsum[0][warp], ebase = sm.result[1] + sm.wsum[1][warp];
    const uint32_t below = (1u << lane) - 1u;
    for (int j0 = w0; j0 < w1; j0 += 32) {
      const int j = j0 + lane;
      const uint32_t key = j < w1 ? key_at(j) : 0u;
      const bool is_gt = j < w1 && (need_eq < 0 || key > thr);
      const bool is_eq = j < w1 && !is_gt && key == thr;
      const uint32_t mg = __ballot_sync(0xffffffffu, is_gt), me = __ballot_sync(0xffffffffu, is_eq);
      const int gr = gbase + __popc(mg & below), er = ebase + __popc(me & below);
      if (is_gt || (is_eq && er < need_eq)) {
        const int slot = gr + (need_eq < 0 ? 0 : min(er, need_eq));
        if (slot < kk) p.idx[slot0 + slot] = j;  // always true when the counts agree
      }
      gbase += __popc(mg);
      ebase += __popc(me);
    }
    if (!unit_sync()) {  // B4 / B5: every kept index of the unit is written
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
