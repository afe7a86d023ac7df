// Guide-to-context scoring on tcgen05 tensor cores (Sec. 3.2, Eq. 1).
//
// The guide block of one KV head (M = G*L_t stacked query rows, at most 512)
// against the document's keys is a dense M x n x d contraction.  Exact
// per-row softmax normalisation needs every row's log-sum-exp before any
// column (per-key) sum can be formed, so the scores take two passes:
//
//   pass 1 (tp_lse_kernel)      D[row, key] = Q K^T in TMEM, one thread per guide
//                            row keeps a running (max, sum of 2^x) over the
//                            CTA's key tiles; the last CTA of a (document,
//                            head) merges the partials into lse[row].
//   pass 2 (tp_keyscore_kernel) D[key, row] = K Q^T in TMEM (keys on lanes), one
//                            thread per key sums exp(x*sigma - lse[row]) over all
//                            rows of the group: s_key[key] (mean over G).
//
// Both passes stream 128-key tiles of K with TMA (128-byte swizzle, an
// evict-first L2 policy: read once) through a ring of shared-memory stages;
// one thread issues the MMAs; four epilogue warpgroups drain TMEM.  Warp roles
// per CTA (18 warps, 20 with the V-scale warps):
//   warp 0  TMEM owner + TMA producer      warp 1  MMA issuer
//   warps 2-17  epilogue warpgroups 0-3 (warp w reads TMEM lanes 32*(w%4)..)
//   warps 18-19 Eq. 2 scales from a V ring (pass 1; pass 2 with the caller's
//               normalisers)
//
// With row normalisers given by the caller there is no pass 1: pass 2 forms
// the scales too (tp_keyscore_kernel<D, true, NH>, where the guide block fits beside
// two K and two V stages: up to 256 guide rows at d = 128), or, for
// more rows, tp_keyscore_pair_kernel runs it on two-CTA clusters sharing each
// MMA (tcgen05 cta_group::2), each CTA holding half of the guide block so that
// the V ring fits beside it.
#include <math.h>

#include <mutex>

#include "tp_device.cuh"

namespace tp {

namespace {

constexpr int kThreads = 576;      // pass 2: TMA, MMA, 16 epilogue warps
constexpr int kLseThreads = 640;   // pass 1: the same plus 2 V-scale warps
constexpr int kVWarp0 = 18;        // first V-scale warp of pass 1
constexpr int kVStages = 3;        // V-tile ring depth of pass 1
constexpr int kVStages2 = 2;       // V-tile ring depth of pass 2 when it forms the scales
constexpr int kEpiWarp0 = 2;  // first epilogue warp
constexpr int kEpiWarps = 16;  // four warpgroups
constexpr uint32_t kHalfTileBytes = 128 * 128;  // 128 keys x 64 bf16

struct ScoreSmem {
  uint32_t q, k, bars, misc, extra, total;
};

// Byte offsets inside the (1024-aligned) dynamic shared memory.
__host__ __device__ inline ScoreSmem score_layout(int head_dim, int rows_pad, int stages,
                                                  uint32_t extra_bytes) {
  ScoreSmem L;
  const int nkh = head_dim / 64;
  L.q = 0;
  L.k = static_cast<uint32_t>(nkh * rows_pad * 128);
  L.bars = L.k + static_cast<uint32_t>(stages) * nkh * kHalfTileBytes;
  L.misc = L.bars + static_cast<uint32_t>(2 * stages + 16) * 8;
  L.extra = (L.misc + 16 + 15) & ~15u;
  L.total = L.extra + extra_bytes;
  return L;
}

// Pass 2 extras after its barriers: up to 1 KB of alignment, the row-offset
// operands of the extra K step (key side 128 x 32 B, guide side rows x 32 B),
// the epilogue partials [4 tiles][4][128 keys].
__host__ __device__ inline uint32_t keyscore_extra_bytes(int rows_pad) {
  return 1024u + 128u * 32u + static_cast<uint32_t>(rows_pad) * 32u + 4u * 4u * 128u * 4u;
}

__device__ __forceinline__ uint8_t* aligned_smem(uint8_t* raw) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
}

// Bounded wait that ignores the abort flag (used only while unwinding).
__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > kWaitLimitNs) return;
  }
}

__device__ __forceinline__ float2 lse_merge(float2 a, float2 b) {
  const float m = fmaxf(a.x, b.x);
  if (m == -INFINITY) return make_float2(-INFINITY, 0.f);
  return make_float2(m, a.y * ex2(a.x - m) + b.y * ex2(b.x - m));
}

// Value i of a 64-column span held as two 32-register chunks.
#define TP_X64(i) __uint_as_float((i) < 32 ? ra[(i) & 31] : rb[(i) & 31])

__device__ __forceinline__ float max64(const uint32_t (&ra)[32], const uint32_t (&rb)[32]) {
  float t[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    t[k] = fmax3(TP_X64(8 * k), TP_X64(8 * k + 1), TP_X64(8 * k + 2));
    t[k] = fmax3(t[k], TP_X64(8 * k + 3), TP_X64(8 * k + 4));
    t[k] = fmax3(t[k], TP_X64(8 * k + 5), TP_X64(8 * k + 6));
    t[k] = fmaxf(t[k], TP_X64(8 * k + 7));
  }
  return fmaxf(fmax3(fmax3(t[0], t[1], t[2]), fmax3(t[3], t[4], t[5]), t[6]), t[7]);
}

// sum_i 2^(x_i * c2 + off) over a 64-column span, four packed partial sums.
__device__ __forceinline__ float sum_exp2_64(const uint32_t (&ra)[32], const uint32_t (&rb)[32],
                                             float c2, float off) {
  float2 a[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                 make_float2(0.f, 0.f)};
  const float2 cc = make_float2(c2, c2), oo = make_float2(off, off);
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const float2 y = ffma2(make_float2(TP_X64(2 * i), TP_X64(2 * i + 1)), cc, oo);
    a[i & 3] = fadd2(a[i & 3], make_float2(ex2(y.x), ex2(y.y)));
  }
  const float2 t = fadd2(fadd2(a[0], a[1]), fadd2(a[2], a[3]));
  return t.x + t.y;
}
#undef TP_X64

// A 64-column span of a guide row's logits (two 32-column chunks) into the
// running (offset m, sum z) of pass 1, both in log2 units:
// z = sum 2^(x*c2 - m).  The offset is refreshed from the exact maximum of the
// span only when it is unset or the span's sum would leave the safe range
// (2^64); otherwise no max is computed.  Columns >= `valid` are masked in place.
__device__ __forceinline__ void lse_chunk64(uint32_t (&ra)[32], uint32_t (&rb)[32], int col0,
                                            int valid, float c2, float& m, float& z) {
  if (valid < col0 + 64) {
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      if (col0 + i >= valid) ra[i] = 0xFF800000u;  // -inf
      if (col0 + 32 + i >= valid) rb[i] = 0xFF800000u;
    }
  }
  float s = 0.f;
  bool exact = (m == -INFINITY);
  if (!exact) {
    s = sum_exp2_64(ra, rb, c2, -m);
    exact = !(s <= 0x1p64f);
  }
  if (exact) {
    const float mn = fmaxf(m, max64(ra, rb) * c2);
    if (mn == -INFINITY) return;
    s = sum_exp2_64(ra, rb, c2, -mn);
    z *= ex2(m - mn);
    m = mn;
  }
  z += s;
  if (z > 0x1p64f) {
    z *= 0x1p-64f;
    m += 64.f;
  }
}


// Eq. 2 scales of the 128 V rows of one staged, 128-byte-swizzled tile: V
// warp vw (of two) reduces rows 64 vw .. 64 vw + 63, two per lane.  The
// swizzle only permutes 16-byte chunks within a row, so a row's absmax may read
// its chunks in any order: lane l reads chunk position cc ^ (row & 7), so that
// eight consecutive rows cover all banks at every step.  Row r's scale goes to
// gamma_rows[r] for r < valid (absmax as bf16 bits, then one IEEE division).
template <int NKH>
__device__ __forceinline__ void vscale_tile(const uint8_t* tile, int vw, int lane, float* gamma_rows,
                                            int valid, float qmax) {
#pragma unroll
  for (int rr = 0; rr < 2; ++rr) {
    const int r = vw * 64 + rr * 32 + lane;
    uint32_t mx = 0;
#pragma unroll
    for (int kh = 0; kh < NKH; ++kh)
#pragma unroll
      for (int cc = 0; cc < 8; ++cc) {
        const uint4 u =
            *reinterpret_cast<const uint4*>(tile + kh * kHalfTileBytes + r * 128 + ((cc ^ (r & 7)) << 4));
        mx = __vmaxu2(mx, u.x & 0x7FFF7FFFu);
        mx = __vmaxu2(mx, u.y & 0x7FFF7FFFu);
        mx = __vmaxu2(mx, u.z & 0x7FFF7FFFu);
        mx = __vmaxu2(mx, u.w & 0x7FFF7FFFu);
      }
    const uint32_t a16 = max(mx & 0xFFFFu, mx >> 16);
    if (r < valid) gamma_rows[r] = __fdiv_rn(__uint_as_float(a16 << 16), qmax);
  }
}

// One 32-column chunk of a key's logits in pass 2: sum_r 2^(D_r * c2), where
// the accumulator D already holds logit_r - lse_r / sigma (the row offset
// enters the contraction as an extra K step).
__device__ __forceinline__ float key_chunk(const uint32_t (&r)[32], float c2) {
  float2 a[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                 make_float2(0.f, 0.f)};
  const float2 cc = make_float2(c2, c2);
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const float2 y = fmul2(make_float2(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1])), cc);
    a[i & 3] = fadd2(a[i & 3], make_float2(ex2(y.x), ex2(y.y)));
  }
  const float2 t = fadd2(fadd2(a[0], a[1]), fadd2(a[2], a[3]));
  return t.x + t.y;
}

// Issues the TMA loads of the guide block (all rows_pad rows, both K halves).
template <int D>
__device__ __forceinline__ void load_guide(uint8_t* sQ, const CUtensorMap* tmq, int rows_pad,
                                           int group_index, uint64_t* bar) {
  constexpr int NKH = D / 64;
  const int qbox = rows_pad < 256 ? rows_pad : 256;
  mbar_arrive_expect_tx(bar, static_cast<uint32_t>(NKH * rows_pad * 128));
#pragma unroll
  for (int kh = 0; kh < NKH; ++kh)
    for (int r0 = 0; r0 < rows_pad; r0 += qbox)
      tma_load_3d(sQ + (kh * rows_pad + r0) * 128, tmq, kh * 64, r0, group_index, bar);
}

// ---------------------------------------------------------------------------
// Pass 1: per-row log-sum-exp of the scaled logits.
//
// The group's guide rows stay in tensor memory for the whole CTA (the MMA's A
// operand, NRB row blocks of 128 rows), so each MMA reads only the K tile from
// shared memory.  Job (tile, row block) accumulates D[row, key] for 128 keys
// into one of NB rotating TMEM buffers; all four epilogue warpgroups share
// every job (warpgroup g owns columns 32g..32g+31), each thread keeping a
// running (offset, sum) per row block for its row.
//
// With p.gamma set, the same CTA also produces the Eq. 2 scale of every token
// of its key range: the producer streams the V tiles into a second ring and
// two warps reduce each row's absmax (the V stream hides under the scoring).
// ---------------------------------------------------------------------------
template <int D, int NRB>
__global__ void __launch_bounds__(kLseThreads, 1)
    tp_lse_kernel(const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv,
               const __grid_constant__ CUtensorMap tmq, const __grid_constant__ LseParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = aligned_smem(smem_raw);
  constexpr int NKH = D / 64;
  constexpr uint32_t KT = NKH * kHalfTileBytes;
  constexpr int ACOLS = NRB * D / 2;                       // TMEM columns of the guide rows
  constexpr int NB = (512 - ACOLS) / 128 < 3 ? (512 - ACOLS) / 128 : 3;  // accumulator buffers
  const int stages = p.stages, rows_pad = NRB * 128;
  const bool with_v = p.gamma != nullptr;
  const ScoreSmem L = score_layout(D, 0, stages + kVStages, 0);
  uint8_t* sK = smem + L.k;
  uint8_t* sV = sK + stages * KT;
  uint64_t* full_k = reinterpret_cast<uint64_t*>(smem + L.bars);
  uint64_t* empty_k = full_k + stages;
  uint64_t* tfull = empty_k + stages;  // [NB]
  uint64_t* tempty = tfull + 3;        // [NB], one arrival per epilogue warp
  uint64_t* drain = tempty + 3;
  uint64_t* full_v = drain + 1;        // [kVStages]
  uint64_t* empty_v = full_v + kVStages;  // [kVStages], one arrival per V warp
  uint64_t* q_full = empty_v + kVStages;   // the guide block has landed in the K ring
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L.misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L.misc + 4);
  int* last_flag = reinterpret_cast<int*>(smem + L.misc + 8);
  // [4 warpgroups][rows_pad] row statistics, written once the K ring is idle
  float2* stats = reinterpret_cast<float2*>(sK);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint64_t kv_policy = l2_evict_first_policy();  // K and V are read once
  const int h = blockIdx.y;
  const int b = find_doc(p.docs, blockIdx.x);
  const int c = blockIdx.x - p.docs.cta[b];
  const int ncta_doc = p.docs.cta[b + 1] - p.docs.cta[b];
  const int64_t doc_lo = p.docs.off[b];
  const int n = static_cast<int>(p.docs.off[b + 1] - doc_lo);
  const int ntiles = (n + kKeyTile - 1) / kKeyTile;
  const int t0 = c * p.tiles_per_cta;
  const int nt = min(p.tiles_per_cta, ntiles - t0);
  grid_dep_launch();

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(&full_k[s], 1);
      mbar_init(&empty_k[s], 1);
    }
    for (int i = 0; i < NB; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], kEpiWarps / 2);  // one group of eight warps drains a buffer
    }
    mbar_init(drain, 1);
    for (int i = 0; i < kVStages; ++i) {
      mbar_init(&full_v[i], 1);
      mbar_init(&empty_v[i], 2);
    }
    mbar_init(q_full, 1);
    *abort_flag = 0;
    *last_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // Guide rows -> TMEM columns [0, ACOLS).  The block arrives by TMA in the
  // (still idle) K ring, 128-byte swizzled; warpgroup g then writes row block
  // g, warp quadrant q its 32 rows, one row per thread (rows >= M arrive as
  // zeros).  The swizzle puts 16-byte chunk c of row r at chunk c ^ (r & 7),
  // so a warp's 32 rows read conflict-free.
  // The V ring is idle meanwhile: its first tiles are requested right away.
  const int v_pre = with_v ? min(kVStages, nt) : 0;
  auto issue_v = [&](int lt) {
    const int vs = lt % kVStages;
    mbar_arrive_expect_tx(&full_v[vs], KT);
    const int y = static_cast<int>(doc_lo + static_cast<int64_t>(t0 + lt) * kKeyTile);
#pragma unroll
    for (int kh = 0; kh < NKH; ++kh)
      tma_load_3d_hint(sV + vs * KT + kh * kHalfTileBytes, &tmv, kh * 64, y, h, &full_v[vs], kv_policy);
  };
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&tmq);
    if (with_v) prefetch_tensormap(&tmv);
    for (int lt = 0; lt < v_pre; ++lt) issue_v(lt);
    const int qbox = rows_pad < 256 ? rows_pad : 256;
    mbar_arrive_expect_tx(q_full, static_cast<uint32_t>(NKH * rows_pad * 128));
#pragma unroll
    for (int kh = 0; kh < NKH; ++kh)
      for (int r0 = 0; r0 < rows_pad; r0 += qbox)
        tma_load_3d(sK + (kh * rows_pad + r0) * 128, &tmq, kh * 64, r0, b * p.n_heads_kv + h, q_full);
  }
  if (warp >= kEpiWarp0 && warp < kVWarp0) {
    const int g = (warp - kEpiWarp0) >> 2, quad = warp & 3;
    if (g < NRB && mbar_wait(q_full, 0, abort_flag)) {
      const int row = g * 128 + quad * 32 + lane;
#pragma unroll
      for (int part = 0; part < D / 64; ++part) {
        const uint8_t* src = sK + (part * rows_pad + row) * 128;
        uint32_t r[32];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const uint4 v = *reinterpret_cast<const uint4*>(src + ((i ^ (row & 7)) << 4));
          r[4 * i] = v.x;
          r[4 * i + 1] = v.y;
          r[4 * i + 2] = v.z;
          r[4 * i + 3] = v.w;
        }
        tmem_st32(tmem + (static_cast<uint32_t>(quad * 32) << 16) + g * (D / 2) + part * 32, r);
      }
    }
    fence_proxy_async_smem();  // the K stream overwrites the block next
  }
  if (warp == 0 && lane == 0 && *abort_flag) mbar_drain(q_full, 0);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  // epilogue: running (offset, sum) per row block this warp sees (two with NRB = 4)
  float m[2] = {-INFINITY, -INFINITY}, z[2] = {0.f, 0.f};

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tensormap(&tmk);
      int issued = 0, issued_v = v_pre;
      for (int lt = 0; lt < nt; ++lt) {
        const int s = lt % stages, use = lt / stages;
        if (use > 0 && !mbar_wait(&empty_k[s], (use - 1) & 1, abort_flag)) break;
        mbar_arrive_expect_tx(&full_k[s], KT);
        const int y = static_cast<int>(doc_lo + static_cast<int64_t>(t0 + lt) * kKeyTile);
#pragma unroll
        for (int kh = 0; kh < NKH; ++kh)
          tma_load_3d_hint(sK + s * KT + kh * kHalfTileBytes, &tmk, kh * 64, y, h, &full_k[s], kv_policy);
        issued = lt + 1;
        if (lt >= v_pre && with_v) {
          if (!mbar_wait(&empty_v[lt % kVStages], (lt / kVStages - 1) & 1, abort_flag)) break;
          issue_v(lt);
          issued_v = lt + 1;
        }
      }
      if (*abort_flag) {  // let in-flight copies land before the CTA exits
        for (int lt = max(0, issued - stages); lt < issued; ++lt)
          mbar_drain(&full_k[lt % stages], (lt / stages) & 1);
        for (int lt = max(0, issued_v - kVStages); lt < issued_v; ++lt)
          mbar_drain(&full_v[lt % kVStages], (lt / kVStages) & 1);
      }
    }
    __syncwarp();
  } else if (warp >= kVWarp0) {
    // Eq. 2 scales, two warps per tile
    if (with_v) {
      const int vw = warp - kVWarp0;
      // launched as a dependent of the previous layer's compaction, which may
      // still read the scale buffer: no store before it has finished
      grid_dep_wait();
      for (int lt = 0; lt < nt; ++lt) {
        const int vs = lt % kVStages;
        if (!mbar_wait(&full_v[vs], (lt / kVStages) & 1, abort_flag)) break;
        const int tok0 = (t0 + lt) * kKeyTile;
        vscale_tile<NKH>(sV + vs * KT, vw, lane, p.gamma + static_cast<size_t>(h) * p.n_total + doc_lo + tok0,
                         n - tok0, p.qmax);
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty_v[vs]);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, kKeyTile);
      bool ok = true;
      for (int lt = 0; ok && lt < nt; ++lt) {
        const int s = lt % stages;
        if (!mbar_wait(&full_k[s], (lt / stages) & 1, abort_flag)) break;
        tc_fence_after();
#pragma unroll
        for (int rb = 0; rb < NRB; ++rb) {
          const int j = lt * NRB + rb, buf = j % NB, use = j / NB;
          if (use > 0 && !mbar_wait(&tempty[buf], (use - 1) & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t dt = tmem + static_cast<uint32_t>(ACOLS + buf * 128);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const int kh = kk >> 2, k16 = kk & 3;
            const uint64_t bd = sdesc_k128(smem_u32(sK + s * KT + kh * kHalfTileBytes + k16 * 32));
            mma_bf16_ts(dt, tmem + rb * (D / 2) + kk * 8, bd, idesc, kk > 0 ? 1u : 0u);
          }
          mma_commit(&tfull[buf]);
        }
        mma_commit(&empty_k[s]);
      }
      mma_commit(drain);  // completes once every MMA issued above has finished
      mbar_drain(drain, 0);
    }
    __syncwarp();
  } else {
    // Two groups of eight warps take alternate jobs (group G = jobs j with
    // j % 2 == G), so one group's TMEM loads overlap the other's arithmetic.
    // In a group, warpgroup half h owns columns 64h..64h+63 of the job.
    const int wg = (warp - kEpiWarp0) >> 2, grp = wg >> 1, hcol = wg & 1, quad = warp & 3;
    const float c2 = p.c2;
    const uint32_t tcol = tmem + (static_cast<uint32_t>(quad * 32) << 16) + ACOLS + hcol * 64;
    const int njobs = nt * NRB;
    bool ok = true;
    for (int j = grp; ok && j < njobs; j += 2) {
      const int buf = j % NB, lt = j / NRB;
      if (!mbar_wait(&tfull[buf], (j / NB) & 1, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t ra[32], rb[32];
      tmem_ld32_async(tcol + buf * 128, ra);
      tmem_ld32_async(tcol + buf * 128 + 32, rb);
      tmem_wait(ra);
      tmem_wait(rb);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[buf]);
      const int valid = min(kKeyTile, n - (t0 + lt) * kKeyTile);
      // row block j % NRB: this group sees rb = grp, grp + 2 (NRB = 4), grp (NRB = 2), 0 (NRB = 1)
      const int slot = NRB == 4 ? (j % NRB) >> 1 : 0;
      if (slot == 0) lse_chunk64(ra, rb, hcol * 64, valid, c2, m[0], z[0]);
      else lse_chunk64(ra, rb, hcol * 64, valid, c2, m[NRB == 4 ? 1 : 0], z[NRB == 4 ? 1 : 0]);
    }
  }
  // Every stream has landed and every MMA has finished: the K ring is free.
  __syncthreads();
  // The workspace partials, normalisers and counters may still be in use by
  // the previous layer's kernels when this one runs as their dependent.
  grid_dep_wait();

  const bool aborted = *abort_flag != 0;
  if (aborted) {
    if (threadIdx.x == 0) set_status(p.status, TP_ERR_TIMEOUT);
  } else {
    if (warp >= kEpiWarp0 && warp < kVWarp0) {
      const int g = (warp - kEpiWarp0) >> 2, grp = g >> 1, quad = warp & 3;
#pragma unroll
      for (int rb = 0; rb < NRB; ++rb) {
        // this warp's (offset, sum) for row block rb, or the empty pair
        float2 st = make_float2(-INFINITY, 0.f);
        if (NRB == 1) st = make_float2(m[0], z[0]);
        else if (NRB == 2 && rb == grp) st = make_float2(m[0], z[0]);
        else if (NRB == 4 && (rb & 1) == grp) st = make_float2(m[rb >> 1], z[rb >> 1]);
        stats[g * rows_pad + rb * 128 + quad * 32 + lane] = st;
      }
    }
    __syncthreads();
    for (int r = threadIdx.x; r < rows_pad; r += blockDim.x) {
      float2 acc = make_float2(-INFINITY, 0.f);
#pragma unroll
      for (int g = 0; g < 4; ++g) acc = lse_merge(acc, stats[g * rows_pad + r]);
      p.partials[(static_cast<size_t>(h) * gridDim.x + blockIdx.x) * rows_pad + r] = acc;
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
      const int prev = atomicAdd(&p.counters[h * p.docs.batch + b], 1);
      *last_flag = (prev == ncta_doc - 1) ? 1 : 0;
      // every CTA of this (document, head) has counted: the last one leaves the
      // counter zero again, so the next layer of a stack needs no reset
      if (prev == ncta_doc - 1) p.counters[h * p.docs.batch + b] = 0;
    }
    __syncthreads();
    if (*last_flag) {
      __threadfence();
      const float2* part =
          p.partials + (static_cast<size_t>(h) * gridDim.x + p.docs.cta[b]) * rows_pad;
      for (int r = threadIdx.x; r < p.rows; r += blockDim.x) {
        // merged in CTA order, eight partials in flight at a time
        float2 acc = make_float2(-INFINITY, 0.f);
        for (int c0 = 0; c0 < ncta_doc; c0 += 8) {
          float2 v[8];
#pragma unroll
          for (int u = 0; u < 8; ++u)
            if (c0 + u < ncta_doc) v[u] = __ldcg(part + static_cast<size_t>(c0 + u) * rows_pad + r);
#pragma unroll
          for (int u = 0; u < 8; ++u)
            if (c0 + u < ncta_doc) acc = lse_merge(acc, v[u]);
        }
        p.lse[(static_cast<size_t>(b) * p.n_heads_kv + h) * p.rows + r] =
            (acc.x + lg2(acc.y)) * 0.69314718055994531f;
      }
    }
  }
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ---------------------------------------------------------------------------
// Pass 2: s_key[key] = (1/G) sum over rows of 2^(x*c2 - lse[row]*log2(e)).
//
// Keys sit on TMEM lanes (D[key, row] = K Q^T); each MMA job covers one
// 128-key tile and one 256-row part of the guide block (N).  Two groups of
// eight epilogue warps take alternate jobs, each draining one of two TMEM
// buffers; a warp's partial sum for its key over its chunks of a job goes to
// one of four rotating shared-memory slots, and a tile's partials are added in
// a fixed order once all have arrived (bounded mbarrier waits).  NH (one or two
// parts) and FULL (every part eight 32-row chunks) are template parameters,
// so the epilogue is unrolled for the shape with no per-chunk guards.
//
// VS (the caller's normalisers, at most 256 guide rows): the same CTA also
// forms the Eq. 2 scale of every token of its key range from a V ring, as in
// pass 1, so the layer reads K and V once.  The normalisers are then inputs of
// the call: as a programmatic dependent (the next layer of a stack) the kernel
// waits for its predecessor only before its first store.
// ---------------------------------------------------------------------------
template <int D, bool VS, int NH, bool FULL>
__global__ void __launch_bounds__(VS ? kLseThreads : kThreads, 1)
    tp_keyscore_kernel(const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv,
                       const __grid_constant__ CUtensorMap tmq, const __grid_constant__ KeyScoreParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = aligned_smem(smem_raw);
  constexpr int NKH = D / 64;
  constexpr uint32_t KT = NKH * kHalfTileBytes;
  constexpr int VST = VS ? kVStages2 : 0;
  const int stages = p.stages, rows_pad = p.rows_pad, rows_mma = p.rows_mma;
  constexpr int nh = NH;  // 256-row parts of the guide block per key tile
  const ScoreSmem L = score_layout(D, rows_pad, stages + VST, keyscore_extra_bytes(rows_pad));
  uint8_t* sQ = smem + L.q;
  uint8_t* sK = smem + L.k;
  uint8_t* sV = sK + stages * KT;  // VS: the V ring after the K ring
  uint64_t* full_k = reinterpret_cast<uint64_t*>(smem + L.bars);
  uint64_t* empty_k = full_k + stages;
  uint64_t* q_full = empty_k + stages;
  uint64_t* tfull = q_full + 1;   // [2 TMEM buffers]
  uint64_t* tempty = tfull + 2;   // [2 TMEM buffers], one arrival per epilogue warp
  uint64_t* drain = tempty + 2;
  uint64_t* pdone = drain + 1;    // [4] partial slots complete, one arrival per warp
  uint64_t* full_v = pdone + 4;   // VS: [VST]
  uint64_t* empty_v = full_v + VST;  // VS: [VST], one arrival per V warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L.misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L.misc + 4);
  // Row offsets as an extra K step of the contraction (32-byte swizzled,
  // K-major): key side [1, 1, 1, 0, ...], guide side (hi, mid, lo, 0, ...) with
  // hi + mid + lo = -lse[row] / sigma (three bf16 parts, exact to ~2^-24).
  uint8_t* a_aug = smem + ((L.extra + 1023u) & ~1023u);               // [128 keys][32 B]
  uint8_t* b_aug = a_aug + 128 * 32;                                  // [rows_pad][32 B]
  float* part = reinterpret_cast<float*>(b_aug + rows_pad * 32);      // [4][4][128]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint64_t kv_policy = l2_evict_first_policy();  // K and V are read once
  const int h = blockIdx.y;
  const int b = find_doc(p.docs, blockIdx.x);
  const int c = blockIdx.x - p.docs.cta[b];
  const int64_t doc_lo = p.docs.off[b];
  const int n = static_cast<int>(p.docs.off[b + 1] - doc_lo);
  const int ntiles = (n + kKeyTile - 1) / kKeyTile;
  const int t0 = c * p.tiles_per_cta;
  const int nt = min(p.tiles_per_cta, ntiles - t0);

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(&full_k[s], 1);
      mbar_init(&empty_k[s], 1);
    }
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], kEpiWarps / 2);  // one group of eight warps drains a buffer
    }
    mbar_init(drain, 1);
    for (int i = 0; i < 4; ++i) mbar_init(&pdone[i], 8 * nh);
    for (int i = 0; i < VST; ++i) {
      mbar_init(&full_v[i], 1);
      mbar_init(&empty_v[i], 2);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  // The guide block and the first K (and V) tiles are inputs of the whole
  // layer: they may load while the predecessor finishes, requested by the
  // thread that initialised their barriers, before the allocation.
  const int k_pre = min(stages, nt), v_pre = min(VST, nt);
  auto issue_v = [&](int lt) {
    const int vs = lt % kVStages2;
    mbar_arrive_expect_tx(&full_v[vs], KT);
    const int y = static_cast<int>(doc_lo + static_cast<int64_t>(t0 + lt) * kKeyTile);
#pragma unroll
    for (int kh = 0; kh < NKH; ++kh)
      tma_load_3d_hint(sV + vs * KT + kh * kHalfTileBytes, &tmv, kh * 64, y, h, &full_v[vs], kv_policy);
  };
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&tmk);
    prefetch_tensormap(&tmq);
    if (VS) prefetch_tensormap(&tmv);
    load_guide<D>(sQ, &tmq, rows_pad, b * p.n_heads_kv + h, q_full);
    for (int lt = 0; lt < k_pre; ++lt) {
      mbar_arrive_expect_tx(&full_k[lt], KT);
      const int y = static_cast<int>(doc_lo + static_cast<int64_t>(t0 + lt) * kKeyTile);
#pragma unroll
      for (int kh = 0; kh < NKH; ++kh)
        tma_load_3d_hint(sK + lt * KT + kh * kHalfTileBytes, &tmk, kh * 64, y, h, &full_k[lt], kv_policy);
    }
    for (int lt = 0; lt < v_pre; ++lt) issue_v(lt);
  }
  __syncwarp();  // warp 0 reconverges before its collective allocation
  grid_dep_launch();
  if (warp == 0) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (!VS) grid_dep_wait();  // the row normalisers come from pass 1
  {
    const float* lse = p.lse + (static_cast<size_t>(b) * p.n_heads_kv + h) * p.rows;
    for (int r = threadIdx.x; r < 128 + rows_pad; r += blockDim.x) {
      uint4 c0;
      uint8_t* row;
      if (r < 128) {  // key side: three ones
        row = a_aug + r * 32;
        c0 = make_uint4(0x3F803F80u, 0x00003F80u, 0u, 0u);
      } else {        // guide side: the row's offset in three parts
        const int g = r - 128;
        row = b_aug + g * 32;
        const float v = g < p.rows ? -(lse[g] * 1.4426950408889634f) / p.c2 : -1.0e30f;
        const uint32_t hi = bf16_bits_rn(v);
        const float r1 = v - __uint_as_float(hi << 16);
        const uint32_t mid = bf16_bits_rn(r1);
        const uint32_t lo = bf16_bits_rn(r1 - __uint_as_float(mid << 16));
        c0 = make_uint4(hi | (mid << 16), lo, 0u, 0u);
      }
      const int rr = r < 128 ? r : r - 128;
      const int pos = (rr >> 2) & 1;  // 32-byte swizzle: chunk c at c ^ ((row >> 2) & 1)
      *reinterpret_cast<uint4*>(row + pos * 16) = c0;
      *reinterpret_cast<uint4*>(row + (pos ^ 1) * 16) = make_uint4(0u, 0u, 0u, 0u);
    }
    fence_proxy_async_smem();  // read by the tensor core
  }
  __syncthreads();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // K tiles as their stages free up; with VS each V tile once the V warps
      // have released its stage (the V stream runs beside the scoring)
      int issued = k_pre, issued_v = v_pre;
      bool ok = true;
      for (int lt = k_pre; ok && lt < nt; ++lt) {
        const int s = lt % stages, use = lt / stages;
        if (use > 0 && !mbar_wait(&empty_k[s], (use - 1) & 1, abort_flag)) break;
        mbar_arrive_expect_tx(&full_k[s], KT);
        const int y = static_cast<int>(doc_lo + static_cast<int64_t>(t0 + lt) * kKeyTile);
#pragma unroll
        for (int kh = 0; kh < NKH; ++kh)
          tma_load_3d_hint(sK + s * KT + kh * kHalfTileBytes, &tmk, kh * 64, y, h, &full_k[s], kv_policy);
        issued = lt + 1;
        if (VS) {
          for (; issued_v <= lt && issued_v < nt; ++issued_v) {
            const int vs = issued_v % kVStages2;
            if (!mbar_wait(&empty_v[vs], (issued_v / kVStages2 - 1) & 1, abort_flag)) {
              ok = false;
              break;
            }
            issue_v(issued_v);
          }
        }
      }
      if (VS) {
        for (; ok && issued_v < nt; ++issued_v) {
          const int vs = issued_v % kVStages2;
          if (!mbar_wait(&empty_v[vs], (issued_v / kVStages2 - 1) & 1, abort_flag)) break;
          issue_v(issued_v);
        }
      }
      if (*abort_flag) {  // let in-flight copies land before the CTA exits
        mbar_drain(q_full, 0);
        for (int lt = max(0, issued - stages); lt < issued; ++lt)
          mbar_drain(&full_k[lt % stages], (lt / stages) & 1);
        if (VS)
          for (int lt = max(0, issued_v - kVStages2); lt < issued_v; ++lt)
            mbar_drain(&full_v[lt % kVStages2], (lt / kVStages2) & 1);
      }
    }
    __syncwarp();
  } else if (VS && warp >= kVWarp0) {
    // Eq. 2 scales of the CTA's key range, two warps per tile
    const int vw = warp - kVWarp0;
    grid_dep_wait();  // the previous layer's kernels may still read the scales
    for (int lt = 0; lt < nt; ++lt) {
      const int vs = lt % kVStages2;
      if (!mbar_wait(&full_v[vs], (lt / kVStages2) & 1, abort_flag)) break;
      const int tok0 = (t0 + lt) * kKeyTile;
      vscale_tile<NKH>(sV + vs * KT, vw, lane, p.gamma + static_cast<size_t>(h) * p.n_total + doc_lo + tok0,
                       n - tok0, p.qmax);
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_v[vs]);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = mbar_wait(q_full, 0, abort_flag);
      for (int lt = 0; ok && lt < nt; ++lt) {
        const int s = lt % stages;
        if (!mbar_wait(&full_k[s], (lt / stages) & 1, abort_flag)) break;
        tc_fence_after();
        for (int hh = 0; hh < nh; ++hh) {
          const int j = lt * nh + hh, buf = j & 1, use = j >> 1;
          if (use > 0 && !mbar_wait(&tempty[buf], (use - 1) & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int nrows = min(256, rows_mma - 256 * hh);
          const uint32_t idesc = idesc_bf16_f32(128, nrows);
          const uint32_t dt = tmem + static_cast<uint32_t>(buf * 256);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const int kh = kk >> 2, k16 = kk & 3;
            const uint64_t a = sdesc_k128(smem_u32(sK + s * KT + kh * kHalfTileBytes + k16 * 32));
            const uint64_t bd =
                sdesc_k128(smem_u32(sQ + (kh * rows_pad + hh * 256) * 128 + k16 * 32));
            mma_bf16_ss(dt, a, bd, idesc, kk > 0 ? 1u : 0u);
          }
          mma_bf16_ss(dt, sdesc_k32(smem_u32(a_aug)), sdesc_k32(smem_u32(b_aug + hh * 256 * 32)),
                      idesc, 1u);
          mma_commit(&tfull[buf]);
        }
        mma_commit(&empty_k[s]);
      }
      mma_commit(drain);
      mbar_drain(drain, 0);
    }
    __syncwarp();
  } else {
    // Two groups of eight warps take alternate jobs: job j = lt * nh + hh goes
    // to group j & 1, which drains TMEM buffer j & 1, so one group's TMEM loads
    // overlap the other group's arithmetic.  In a group, warp (cg, quad)
    // reduces TMEM lanes 32 quad .. 32 quad + 31 (keys) over the column chunks
    // 4 cg .. 4 cg + 3; the second pair of chunks loads while the first pair is
    // reduced, and the buffer is released once all four are in registers.
    const int e = warp - kEpiWarp0, grp = e >> 3, cg = (e >> 2) & 1, quad = warp & 3;
    const float c2 = p.c2;
    const uint32_t tlane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    bool ok = true, stored = false;
    for (int lt = 0; lt < nt; ++lt) {
      float* slot = part + (lt & 3) * 4 * 128;  // partials (hh, cg) of this tile's keys
      uint64_t* done = &pdone[lt & 3];
      for (int hh = 0; hh < nh; ++hh) {
        const int j = lt * nh + hh, buf = j & 1;
        if (buf != grp) continue;
        if (ok && !mbar_wait(&tfull[buf], (j >> 1) & 1, abort_flag)) ok = false;
        if (!ok) continue;
        tc_fence_after();
        const int nch = FULL ? 8 : min(256, rows_mma - 256 * hh) / 32;
        const uint32_t tb = tlane + buf * 256;
        const int ch = 4 * cg;
        float acc = 0.f;
        uint32_t ra[32], rb[32];
        if (ch < nch) tmem_ld32_async(tb + ch * 32, ra);
        if (ch + 1 < nch) tmem_ld32_async(tb + (ch + 1) * 32, rb);
        if (ch < nch) tmem_wait(ra);
        if (ch + 1 < nch) tmem_wait(rb);
        if (ch < nch) acc += key_chunk(ra, c2);
        if (ch + 2 < nch) tmem_ld32_async(tb + (ch + 2) * 32, ra);
        if (ch + 1 < nch) acc += key_chunk(rb, c2);
        if (ch + 3 < nch) tmem_ld32_async(tb + (ch + 3) * 32, rb);
        if (ch + 2 < nch) tmem_wait(ra);
        if (ch + 3 < nch) tmem_wait(rb);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[buf]);
        if (ch + 2 < nch) acc += key_chunk(ra, c2);
        if (ch + 3 < nch) acc += key_chunk(rb, c2);
        slot[(hh * 2 + cg) * 128 + quad * 32 + lane] = acc;
        __syncwarp();
        if (lane == 0) mbar_arrive(done);
      }
      // The cg = 0 warps of the group that ran the tile's last job sum the
      // partials in a fixed order once every warp of the tile's jobs has
      // arrived on the slot's barrier (phase lt / 4).  No warp reaches the same
      // slot four tiles on before this read: that job needs a TMEM buffer that
      // this group releases only after it.
      const int fin = (lt * nh + nh - 1) & 1;
      if (grp == fin && cg == 0) {
        if (ok && !mbar_wait(done, (lt >> 2) & 1, abort_flag)) ok = false;
        if (ok) {
          if (VS && !stored) {
            grid_dep_wait();  // the previous layer's selection may still read the key scores
            stored = true;
          }
          const int kl = quad * 32 + lane;
          float s4 = slot[kl] + slot[128 + kl];
          if (nh == 2) s4 = (s4 + slot[256 + kl]) + slot[384 + kl];
          const int key = (t0 + lt) * kKeyTile + kl;
          if (key < n) p.skey[static_cast<size_t>(h) * p.n_total + doc_lo + key] = s4 * p.inv_group;
        }
      }
    }
  }
  __syncthreads();
  if (*abort_flag != 0 && threadIdx.x == 0) set_status(p.status, TP_ERR_TIMEOUT);
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ---------------------------------------------------------------------------
// Pass 2 and the Eq. 2 scales on a CTA pair (tcgen05 cta_group::2), for row
// normalisers given by the caller: one kernel reads K and V once.
//
// The two CTAs of a cluster share each MMA: a pair tile is 256 keys, the even
// CTA streaming keys 0..127 of it and the odd CTA keys 128..255 (A split along
// M), and every job's guide rows are split in halves (B split along N).  Each
// CTA therefore keeps only half of the guide block in shared memory, which
// leaves room for a V ring: as in pass 1, two warps reduce each of the CTA's
// V rows to its absmax while the scoring runs.  Each CTA's tensor memory
// receives D[key, row] for its own 128 keys and all rows of the job, so the
// epilogue is that of the one-CTA kernel.
//
// The even CTA's warp 1 issues the MMAs and multicasts every completion to
// both CTAs (TMEM buffer full, K stage free, drain).  The odd CTA's warp 1
// relays the arrival of each of its K stages to the even CTA, and its
// epilogue warps release a TMEM buffer on the even CTA's barrier, so the MMA
// thread waits for both halves of every operand and of every drained buffer.
//
// Launched as a programmatic dependent (the next layer of a stack after the
// previous layer's compaction), the kernel loads and scores at once (its
// inputs are the layer's) and waits for its predecessor only before its first
// store of a scale or a key score.
// ---------------------------------------------------------------------------

struct PairSmem {
  uint32_t q, k, v, bars, misc, a_aug, b_aug, part, total;
};

// Byte offsets inside the (1024-aligned) dynamic shared memory of one CTA:
// guide half [nh jobs][D/64 halves][128 rows][128 B], the K ring, the V ring,
// barriers, the row-offset operands (key side 128 x 32 B; guide side
// [nh][128 rows][32 B]) and the epilogue partials [4 tiles][4][128 keys].
__host__ __device__ inline PairSmem pair_layout(int head_dim, int nh, int stages) {
  PairSmem L;
  const int nkh = head_dim / 64;
  L.q = 0;
  L.k = static_cast<uint32_t>(nh * nkh) * kHalfTileBytes;
  L.v = L.k + static_cast<uint32_t>(stages * nkh) * kHalfTileBytes;
  L.bars = L.v + static_cast<uint32_t>(kVStages2 * nkh) * kHalfTileBytes;
  L.misc = L.bars + static_cast<uint32_t>(3 * stages + 2 * kVStages2 + 16) * 8;
  L.a_aug = (L.misc + 16 + 1023) & ~1023u;
  L.b_aug = L.a_aug + 128u * 32u;
  L.part = L.b_aug + static_cast<uint32_t>(nh) * 128u * 32u;
  L.total = L.part + 4u * 4u * 128u * 4u;
  return L;
}

template <int D, int NH, bool FULL>
__global__ void __launch_bounds__(kLseThreads, 1)
    tp_keyscore_pair_kernel(const __grid_constant__ CUtensorMap tmk,
                            const __grid_constant__ CUtensorMap tmv,
                            const __grid_constant__ CUtensorMap tmq,
                            const __grid_constant__ KeyScoreParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = aligned_smem(smem_raw);
  constexpr int NKH = D / 64;
  constexpr uint32_t KT = NKH * kHalfTileBytes;
  constexpr int kPairTile = 2 * kKeyTile;
  const int stages = p.stages, rows_mma = p.rows_mma;
  constexpr int nh = NH;  // 256-row parts of the guide block per pair tile
  const PairSmem L = pair_layout(D, nh, stages);
  uint8_t* sQ = smem + L.q;
  uint8_t* sK = smem + L.k;
  uint8_t* sV = smem + L.v;
  uint64_t* full_k = reinterpret_cast<uint64_t*>(smem + L.bars);
  uint64_t* empty_k = full_k + stages;  // multicast by the MMA thread's commits
  uint64_t* pfull = empty_k + stages;   // even CTA: the odd CTA's stage has landed
  uint64_t* full_v = pfull + stages;    // [kVStages2]
  uint64_t* empty_v = full_v + kVStages2;  // [kVStages2], one arrival per V warp
  uint64_t* q_full = empty_v + kVStages2;
  uint64_t* tfull = q_full + 1;         // [2 TMEM buffers], multicast
  uint64_t* tempty = tfull + 2;         // [2] even CTA: one arrival per epilogue warp of the pair
  uint64_t* drain = tempty + 2;         // multicast
  uint64_t* pdone = drain + 1;          // [4] partial slots complete, one arrival per warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L.misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L.misc + 4);
  uint8_t* a_aug = smem + L.a_aug;
  uint8_t* b_aug = smem + L.b_aug;
  float* part = reinterpret_cast<float*>(smem + L.part);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint64_t kv_policy = l2_evict_first_policy();  // K and V are read once
  const uint32_t rank = cluster_ctarank();  // 0 issues the MMAs
  const int h = blockIdx.y;
  const int pair = static_cast<int>(blockIdx.x >> 1);
  const int b = find_doc(p.docs, pair);
  const int c = pair - p.docs.cta[b];
  const int64_t doc_lo = p.docs.off[b];
  const int n = static_cast<int>(p.docs.off[b + 1] - doc_lo);
  const int ntiles = (n + kPairTile - 1) / kPairTile;
  const int t0 = c * p.tiles_per_cta;
  const int nt = min(p.tiles_per_cta, ntiles - t0);
  const int key0 = static_cast<int>(rank) * kKeyTile;  // this CTA's half of a pair tile
  auto tile_row = [&](int lt) {
    return static_cast<int>(doc_lo + static_cast<int64_t>(t0 + lt) * kPairTile + key0);
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(&full_k[s], 1);
      mbar_init(&empty_k[s], 1);
      mbar_init(&pfull[s], 1);
    }
    for (int i = 0; i < kVStages2; ++i) {
      mbar_init(&full_v[i], 1);
      mbar_init(&empty_v[i], 2);
    }
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], kEpiWarps);  // eight warps of each CTA drain a buffer
    }
    mbar_init(drain, 1);
    for (int i = 0; i < 4; ++i) mbar_init(&pdone[i], 8 * nh);
    *abort_flag = 0;
    fence_barrier_init();
  }
  // This CTA's half of every job's guide rows, its first K and V tiles,
  // requested by the thread that initialised their barriers, before the
  // cluster barrier and the allocation.
  const int k_pre = min(stages, nt), v_pre = min(kVStages2, nt);
  auto issue_v = [&](int lt) {
    const int vs = lt % kVStages2;
    mbar_arrive_expect_tx(&full_v[vs], KT);
#pragma unroll
    for (int kh = 0; kh < NKH; ++kh)
      tma_load_3d_hint(sV + vs * KT + kh * kHalfTileBytes, &tmv, kh * 64, tile_row(lt), h, &full_v[vs], kv_policy);
  };
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&tmk);
    prefetch_tensormap(&tmv);
    prefetch_tensormap(&tmq);
    mbar_arrive_expect_tx(q_full, static_cast<uint32_t>(nh * NKH) * kHalfTileBytes);
    for (int hh = 0; hh < nh; ++hh) {
      const int half = min(256, rows_mma - 256 * hh) / 2;
      const int r0 = 256 * hh + static_cast<int>(rank) * half;
#pragma unroll
      for (int kh = 0; kh < NKH; ++kh)
        tma_load_3d(sQ + (hh * NKH + kh) * kHalfTileBytes, &tmq, kh * 64, r0, b * p.n_heads_kv + h,
                    q_full);
    }
    for (int lt = 0; lt < k_pre; ++lt) {
      mbar_arrive_expect_tx(&full_k[lt], KT);
#pragma unroll
      for (int kh = 0; kh < NKH; ++kh)
        tma_load_3d_hint(sK + lt * KT + kh * kHalfTileBytes, &tmk, kh * 64, tile_row(lt), h, &full_k[lt], kv_policy);
    }
    for (int lt = 0; lt < v_pre; ++lt) issue_v(lt);
  }
  __syncwarp();  // warp 0 reconverges before the cluster barrier and the allocation
  grid_dep_launch();
  // both CTAs are running and their barriers are initialised before the
  // collective allocation and any remote arrival
  cluster_sync_all();
  if (warp == 0) {
    tmem_alloc_pair(tmem_slot, 512);
    tmem_relinquish_pair();
  }
  {
    // the caller's row normalisers: an input of the layer
    const float* lse = p.lse + (static_cast<size_t>(b) * p.n_heads_kv + h) * p.rows;
    for (int r = threadIdx.x; r < 128 + nh * 128; r += blockDim.x) {
      uint4 c0;
      uint8_t* row;
      int rr;
      if (r < 128) {  // key side: three ones
        rr = r;
        row = a_aug + r * 32;
        c0 = make_uint4(0x3F803F80u, 0x00003F80u, 0u, 0u);
      } else {        // guide side: the offset of row i of this CTA's half of job hh
        const int hh = (r - 128) >> 7, i = (r - 128) & 127;
        const int half = min(256, rows_mma - 256 * hh) / 2;
        const int g = 256 * hh + static_cast<int>(rank) * half + i;
        rr = i;
        row = b_aug + (hh * 128 + i) * 32;
        const float v = (i < half && g < p.rows) ? -(lse[g] * 1.4426950408889634f) / p.c2 : -1.0e30f;
        const uint32_t hi = bf16_bits_rn(v);
        const float r1 = v - __uint_as_float(hi << 16);
        const uint32_t mid = bf16_bits_rn(r1);
        const uint32_t lo = bf16_bits_rn(r1 - __uint_as_float(mid << 16));
        c0 = make_uint4(hi | (mid << 16), lo, 0u, 0u);
      }
      const int pos = (rr >> 2) & 1;  // 32-byte swizzle: chunk c at c ^ ((row >> 2) & 1)
      *reinterpret_cast<uint4*>(row + pos * 16) = c0;
      *reinterpret_cast<uint4*>(row + (pos ^ 1) * 16) = make_uint4(0u, 0u, 0u, 0u);
    }
    fence_proxy_async_smem();  // read by the tensor core
  }
  // Before the first MMA: the odd CTA's guide half has landed and both CTAs'
  // offset operands and tensor memory are in place.
  if (warp == 1 && lane == 0 && rank == 1) mbar_wait(q_full, 0, abort_flag);
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // K tiles as their stages free up; each V tile once the V warps have
      // released its stage (the V stream runs beside the scoring)
      int issued = k_pre, issued_v = v_pre;
      bool ok = true;
      for (int lt = k_pre; ok && lt < nt; ++lt) {
        const int s = lt % stages, use = lt / stages;
        if (use > 0 && !mbar_wait(&empty_k[s], (use - 1) & 1, abort_flag)) break;
        mbar_arrive_expect_tx(&full_k[s], KT);
#pragma unroll
        for (int kh = 0; kh < NKH; ++kh)
          tma_load_3d_hint(sK + s * KT + kh * kHalfTileBytes, &tmk, kh * 64, tile_row(lt), h, &full_k[s], kv_policy);
        issued = lt + 1;
        for (; issued_v <= lt && issued_v < nt; ++issued_v) {
          const int vs = issued_v % kVStages2;
          if (!mbar_wait(&empty_v[vs], (issued_v / kVStages2 - 1) & 1, abort_flag)) {
            ok = false;
            break;
          }
          issue_v(issued_v);
        }
      }
      for (; ok && issued_v < nt; ++issued_v) {
        const int vs = issued_v % kVStages2;
        if (!mbar_wait(&empty_v[vs], (issued_v / kVStages2 - 1) & 1, abort_flag)) break;
        issue_v(issued_v);
      }
      if (*abort_flag) {  // let in-flight copies land before the CTA exits
        mbar_drain(q_full, 0);
        for (int lt = max(0, issued - stages); lt < issued; ++lt)
          mbar_drain(&full_k[lt % stages], (lt / stages) & 1);
        for (int lt = max(0, issued_v - kVStages2); lt < issued_v; ++lt)
          mbar_drain(&full_v[lt % kVStages2], (lt / kVStages2) & 1);
      }
    }
    __syncwarp();
  } else if (warp >= kVWarp0) {
    // Eq. 2 scales of this CTA's 128 keys of each pair tile
    const int vw = warp - kVWarp0;
    grid_dep_wait();  // the previous layer's kernels may still read the scales
    for (int lt = 0; lt < nt; ++lt) {
      const int vs = lt % kVStages2;
      if (!mbar_wait(&full_v[vs], (lt / kVStages2) & 1, abort_flag)) break;
      const int tok0 = (t0 + lt) * kPairTile + key0;
      vscale_tile<NKH>(sV + vs * KT, vw, lane, p.gamma + static_cast<size_t>(h) * p.n_total + doc_lo + tok0,
                       n - tok0, p.qmax);
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_v[vs]);
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 1) {
      // relay: each of this CTA's K stages has landed
      const uint32_t pfull0 = cluster_addr(pfull, 0);
      for (int lt = 0; lt < nt; ++lt) {
        const int s = lt % stages;
        if (!mbar_wait(&full_k[s], (lt / stages) & 1, abort_flag)) break;
        mbar_arrive_cluster(pfull0 + static_cast<uint32_t>(s) * 8u);
      }
      mbar_drain(drain, 0);  // the pair's last MMA has completed
    } else if (lane == 0) {
      bool ok = mbar_wait(q_full, 0, abort_flag);
      for (int lt = 0; ok && lt < nt; ++lt) {
        const int s = lt % stages;
        if (!mbar_wait(&full_k[s], (lt / stages) & 1, abort_flag)) break;
        if (!mbar_wait_cluster(&pfull[s], (lt / stages) & 1, abort_flag)) break;
        tc_fence_after();
        for (int hh = 0; hh < nh; ++hh) {
          const int j = lt * nh + hh, buf = j & 1, use = j >> 1;
          if (use > 0 && !mbar_wait(&tempty[buf], (use - 1) & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int nrows = min(256, rows_mma - 256 * hh);
          const uint32_t idesc = idesc_bf16_f32(256, nrows);
          const uint32_t dt = tmem + static_cast<uint32_t>(buf * 256);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const int kh = kk >> 2, k16 = kk & 3;
            const uint64_t a = sdesc_k128(smem_u32(sK + s * KT + kh * kHalfTileBytes + k16 * 32));
            const uint64_t bd = sdesc_k128(smem_u32(sQ + (hh * NKH + kh) * kHalfTileBytes + k16 * 32));
            mma_bf16_ss_pair(dt, a, bd, idesc, kk > 0 ? 1u : 0u);
          }
          mma_bf16_ss_pair(dt, sdesc_k32(smem_u32(a_aug)), sdesc_k32(smem_u32(b_aug + hh * 128 * 32)),
                           idesc, 1u);
          mma_commit_pair(&tfull[buf]);
        }
        mma_commit_pair(&empty_k[s]);
      }
      mma_commit_pair(drain);
      mbar_drain(drain, 0);
    }
    __syncwarp();
  } else {
    // The epilogue of the one-CTA kernel on this CTA's 128 keys; a drained
    // buffer is released on the even CTA's barrier (a CTA-scope arrival: it
    // reports completed tensor-memory loads, not data).
    const int e = warp - kEpiWarp0, grp = e >> 3, cg = (e >> 2) & 1, quad = warp & 3;
    const float c2 = p.c2;
    const uint32_t tlane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    const uint32_t tempty0 = cluster_addr(tempty, 0);
    bool ok = true, stored = false;
    for (int lt = 0; lt < nt; ++lt) {
      float* slot = part + (lt & 3) * 4 * 128;
      uint64_t* done = &pdone[lt & 3];
      for (int hh = 0; hh < nh; ++hh) {
        const int j = lt * nh + hh, buf = j & 1;
        if (buf != grp) continue;
        if (ok && !mbar_wait(&tfull[buf], (j >> 1) & 1, abort_flag)) ok = false;
        if (!ok) continue;
        tc_fence_after();
        const int nch = FULL ? 8 : min(256, rows_mma - 256 * hh) / 32;
        const uint32_t tb = tlane + buf * 256;
        const int ch = 4 * cg;
        float acc = 0.f;
        uint32_t ra[32], rb[32];
        if (ch < nch) tmem_ld32_async(tb + ch * 32, ra);
        if (ch + 1 < nch) tmem_ld32_async(tb + (ch + 1) * 32, rb);
        if (ch < nch) tmem_wait(ra);
        if (ch + 1 < nch) tmem_wait(rb);
        if (ch < nch) acc += key_chunk(ra, c2);
        if (ch + 2 < nch) tmem_ld32_async(tb + (ch + 2) * 32, ra);
        if (ch + 1 < nch) acc += key_chunk(rb, c2);
        if (ch + 3 < nch) tmem_ld32_async(tb + (ch + 3) * 32, rb);
        if (ch + 2 < nch) tmem_wait(ra);
        if (ch + 3 < nch) tmem_wait(rb);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (rank == 0) mbar_arrive(&tempty[buf]);
          else mbar_arrive_remote(tempty0 + static_cast<uint32_t>(buf) * 8u);
        }
        if (ch + 2 < nch) acc += key_chunk(ra, c2);
        if (ch + 3 < nch) acc += key_chunk(rb, c2);
        slot[(hh * 2 + cg) * 128 + quad * 32 + lane] = acc;
        __syncwarp();
        if (lane == 0) mbar_arrive(done);
      }
      const int fin = (lt * nh + nh - 1) & 1;
      if (grp == fin && cg == 0) {
        if (ok && !mbar_wait(done, (lt >> 2) & 1, abort_flag)) ok = false;
        if (ok) {
          if (!stored) {
            grid_dep_wait();  // the previous layer's selection may still read the key scores
            stored = true;
          }
          const int kl = quad * 32 + lane;
          float s4 = slot[kl] + slot[128 + kl];
          if (nh == 2) s4 = (s4 + slot[256 + kl]) + slot[384 + kl];
          const int key = (t0 + lt) * kPairTile + key0 + kl;
          if (key < n) p.skey[static_cast<size_t>(h) * p.n_total + doc_lo + key] = s4 * p.inv_group;
        }
      }
    }
  }
  __syncthreads();
  if (*abort_flag != 0 && threadIdx.x == 0) set_status(p.status, TP_ERR_TIMEOUT);
  // neither CTA releases its tensor memory or leaves while the pair's MMAs or
  // the other CTA's remote arrivals may still touch it
  tc_fence_before();
  cluster_sync_all();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, 512);
  }
}

}  // namespace

size_t lse_smem_bytes(int head_dim, int rows_pad, int stages) {
  (void)rows_pad;  // the guide rows live in tensor memory; V has its own ring
  return score_layout(head_dim, 0, stages + kVStages, 0).total + 1024;
}

size_t keyscore_smem_bytes(int head_dim, int rows_pad, int stages, bool scales) {
  return score_layout(head_dim, rows_pad, stages + (scales ? kVStages2 : 0),
                      keyscore_extra_bytes(rows_pad)).total + 1024;
}

size_t keyscore_pair_smem_bytes(int head_dim, int rows_mma, int stages) {
  return pair_layout(head_dim, (rows_mma + 255) / 256, stages).total + 1024;
}

template <int D, int NRB>
cudaError_t launch_lse_t(const CUtensorMap& tmk, const CUtensorMap& tmv, const CUtensorMap& tmq,
                         const LseParams& p, dim3 grid, size_t smem, bool dependent, cudaStream_t s) {
  cudaError_t e = set_smem_once(reinterpret_cast<const void*>(tp_lse_kernel<D, NRB>),
                                1 + (D == 128 ? 3 : 0) + (NRB == 1 ? 0 : NRB == 2 ? 1 : 2));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kLseThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = dependent ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, tp_lse_kernel<D, NRB>, tmk, tmv, tmq, p);
}

cudaError_t launch_lse(const CUtensorMap& tmk, const CUtensorMap& tmv, const CUtensorMap& tmq,
                       const LseParams& p, int head_dim, dim3 grid, size_t smem, bool dependent,
                       cudaStream_t s) {
  if (head_dim == 128) {
    if (p.nrb == 1) return launch_lse_t<128, 1>(tmk, tmv, tmq, p, grid, smem, dependent, s);
    if (p.nrb == 2) return launch_lse_t<128, 2>(tmk, tmv, tmq, p, grid, smem, dependent, s);
    return launch_lse_t<128, 4>(tmk, tmv, tmq, p, grid, smem, dependent, s);
  }
  if (p.nrb == 1) return launch_lse_t<64, 1>(tmk, tmv, tmq, p, grid, smem, dependent, s);
  if (p.nrb == 2) return launch_lse_t<64, 2>(tmk, tmv, tmq, p, grid, smem, dependent, s);
  return launch_lse_t<64, 4>(tmk, tmv, tmq, p, grid, smem, dependent, s);
}

template <int D, bool VS, int NH, bool FULL>
cudaError_t launch_keyscore_t(const CUtensorMap& tmk, const CUtensorMap& tmv, const CUtensorMap& tmq,
                              const KeyScoreParams& p, dim3 grid, size_t smem, bool dependent,
                              cudaStream_t s) {
  // shared-memory attribute slots 32..47, one per instantiation
  const int slot = 32 + ((D == 64) << 3 | VS << 2 | (NH == 2) << 1 | !FULL);
  cudaError_t e = set_smem_once(reinterpret_cast<const void*>(tp_keyscore_kernel<D, VS, NH, FULL>), slot);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(VS ? kLseThreads : kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = dependent ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, tp_keyscore_kernel<D, VS, NH, FULL>, tmk, tmv, tmq, p);
}

template <int D, bool VS>
cudaError_t launch_keyscore_d(const CUtensorMap& tmk, const CUtensorMap& tmv, const CUtensorMap& tmq,
                              const KeyScoreParams& p, dim3 grid, size_t smem, bool dependent,
                              cudaStream_t s) {
  const bool full = p.rows_mma % 256 == 0;
  if (p.rows_mma > 256)
    return full ? launch_keyscore_t<D, VS, 2, true>(tmk, tmv, tmq, p, grid, smem, dependent, s)
                : launch_keyscore_t<D, VS, 2, false>(tmk, tmv, tmq, p, grid, smem, dependent, s);
  return full ? launch_keyscore_t<D, VS, 1, true>(tmk, tmv, tmq, p, grid, smem, dependent, s)
              : launch_keyscore_t<D, VS, 1, false>(tmk, tmv, tmq, p, grid, smem, dependent, s);
}

// The guide block is taken in 256-row parts per key tile, one or two, each of
// eight 32-row chunks except perhaps the last: both are compile-time, so each
// shape gets its own unrolled epilogue with no per-chunk guards where every
// part is whole.  Against run-time counts, per 128K layer at 512 rows, pass 2
// takes 88.6 against 107.8 us.
cudaError_t launch_keyscore(const CUtensorMap& tmk, const CUtensorMap& tmv, const CUtensorMap& tmq,
                            const KeyScoreParams& p, int head_dim, dim3 grid, size_t smem,
                            bool dependent, cudaStream_t s) {
  if (p.gamma)
    return head_dim == 128 ? launch_keyscore_d<128, true>(tmk, tmv, tmq, p, grid, smem, dependent, s)
                           : launch_keyscore_d<64, true>(tmk, tmv, tmq, p, grid, smem, dependent, s);
  return head_dim == 128 ? launch_keyscore_d<128, false>(tmk, tmv, tmq, p, grid, smem, dependent, s)
                         : launch_keyscore_d<64, false>(tmk, tmv, tmq, p, grid, smem, dependent, s);
}

namespace {

// The pair kernel for a head dim and guide block: one or two 256-row parts per
// pair tile, whole or not (compile-time, as in tp_keyscore_kernel).
template <int D>
const void* keyscore_pair_fn_d(int rows_mma) {
  const bool full = rows_mma % 256 == 0;
  if (rows_mma > 256)
    return full ? reinterpret_cast<const void*>(tp_keyscore_pair_kernel<D, 2, true>)
                : reinterpret_cast<const void*>(tp_keyscore_pair_kernel<D, 2, false>);
  return full ? reinterpret_cast<const void*>(tp_keyscore_pair_kernel<D, 1, true>)
              : reinterpret_cast<const void*>(tp_keyscore_pair_kernel<D, 1, false>);
}

const void* keyscore_pair_fn(int head_dim, int rows_mma) {
  return head_dim == 128 ? keyscore_pair_fn_d<128>(rows_mma) : keyscore_pair_fn_d<64>(rows_mma);
}

// The instantiation keyscore_pair_fn names, launched.
template <int D>
cudaError_t launch_pair_d(const cudaLaunchConfig_t& cfg, const CUtensorMap& tmk, const CUtensorMap& tmv,
                          const CUtensorMap& tmq, const KeyScoreParams& p) {
  const bool full = p.rows_mma % 256 == 0;
  if (p.rows_mma > 256)
    return full ? cudaLaunchKernelEx(&cfg, tp_keyscore_pair_kernel<D, 2, true>, tmk, tmv, tmq, p)
                : cudaLaunchKernelEx(&cfg, tp_keyscore_pair_kernel<D, 2, false>, tmk, tmv, tmq, p);
  return full ? cudaLaunchKernelEx(&cfg, tp_keyscore_pair_kernel<D, 1, true>, tmk, tmv, tmq, p)
              : cudaLaunchKernelEx(&cfg, tp_keyscore_pair_kernel<D, 1, false>, tmk, tmv, tmq, p);
}

// shared-memory attribute slots 48..55, one per instantiation
int keyscore_pair_slot(int head_dim, int rows_mma) {
  return 48 + ((head_dim == 64) << 2 | (rows_mma > 256) << 1 | (rows_mma % 256 != 0));
}

cudaLaunchConfig_t pair_config(dim3 grid, size_t smem, cudaStream_t s, cudaLaunchAttribute (&attr)[2],
                               bool dependent) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kLseThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = dependent ? 2 : 1;
  return cfg;
}

}  // namespace

int keyscore_pair_max_clusters(int head_dim, int rows_mma, size_t smem) {
  // answers cached per (CUDA context, kernel, shared memory)
  constexpr int kEntries = 32;
  const void* fn = keyscore_pair_fn(head_dim, rows_mma);
  struct Entry {
    unsigned long long ctx;
    const void* fn;
    size_t smem;
    int clusters;
  };
  static std::mutex mu;
  static Entry cache[kEntries];
  static int used;
  const unsigned long long ctx = context_key();
  {
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < used; ++i)
      if (cache[i].ctx == ctx && cache[i].fn == fn && cache[i].smem == smem) return cache[i].clusters;
  }
  if (set_smem_once(fn, keyscore_pair_slot(head_dim, rows_mma)) != cudaSuccess) return 0;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = pair_config(dim3(2, 1), smem, 0, attr, false);
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, fn, &cfg) != cudaSuccess)
    clusters = 0;
  cudaGetLastError();  // a refused query leaves no error behind
  std::lock_guard<std::mutex> lock(mu);
  if (ctx != 0 && used < kEntries) cache[used++] = Entry{ctx, fn, smem, clusters};
  return clusters;
}

cudaError_t launch_keyscore_pair(const CUtensorMap& tmk, const CUtensorMap& tmv,
                                 const CUtensorMap& tmq, const KeyScoreParams& p, int head_dim,
                                 dim3 grid, size_t smem, bool dependent, cudaStream_t s) {
  cudaError_t e =
      set_smem_once(keyscore_pair_fn(head_dim, p.rows_mma), keyscore_pair_slot(head_dim, p.rows_mma));
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = pair_config(grid, smem, s, attr, dependent);
  return head_dim == 128 ? launch_pair_d<128>(cfg, tmk, tmv, tmq, p)
                         : launch_pair_d<64>(cfg, tmk, tmv, tmq, p);
}

}  // namespace tp
