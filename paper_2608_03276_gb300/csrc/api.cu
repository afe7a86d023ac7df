// C ABI of the TaskPress compression path (include/taskpress.h): argument
// checks, launch planning, workspace carving, TMA descriptors and the kernel
// sequence of each entry point.  Nothing here allocates device memory.
#include <math.h>
#include <string.h>

#include <algorithm>
#include <mutex>

#include "tp_internal.h"

namespace tp {
namespace {

constexpr size_t kAlign = 256;
constexpr int kMaxSmem = 232448;  // opt-in dynamic shared memory per block on sm_100-class GPUs

size_t align_up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

struct Plan {
  int hq, hkv, d, lt, g, batch;
  int64_t n_total;
  int64_t off[kMaxBatch + 1];
  // The scoring kernels see one block of at most TP_MAX_ROWS stacked guide
  // rows, [row0, row0 + rows) of the rows_full = G * L_t rows; a plan made by
  // make_plan holds the first block, block_plan the others.
  int rows_full, blocks, row0;
  int rows, nrb, rows_pad, rows_mma;
  int tiles_per_cta, grid_x;
  int32_t cta[kMaxBatch + 1];
  int stages1, stages2;
  size_t smem1, smem2;
  // pass 2 forming the Eq. 2 scales too (caller's normalisers): K stages and
  // shared memory, stages2s = 0 where two K stages and the V ring do not fit
  // next to the guide block (more than 256 guide rows: CTA pairs then)
  int stages2s;
  size_t smem2s;
  float c2, inv_group, sigma;
  int bits;     // Eq. 2 code width: 8 or 4
  float qmax;   // 2^(bits-1) - 1
  int32_t kept[kMaxBatch];
  int64_t cap;
  // workspace offsets (ws_lse holds one block's normalisers; with more than
  // one block, ws_lse_full all of them and ws_skey_part a block's key scores)
  size_t ws_status, ws_partials, ws_lse, ws_skey, ws_gamma, ws_keys, ws_lse_full, ws_skey_part,
      ws_total;
};

int num_sms() {
  int dev = 0, sms = 148;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms > 0 ? sms : 148;
}

// The row-block fields of a plan for a block of `rows` stacked guide rows:
// 128-row blocks of pass 1, the MMA extent of pass 2, and the deepest K-tile
// rings that fit next to the guide block.
int set_rows(Plan* P, int rows) {
  P->rows = rows;
  const int rb = (rows + 127) / 128;
  P->nrb = rb <= 1 ? 1 : (rb <= 2 ? 2 : 4);
  P->rows_pad = 128 * P->nrb;
  P->rows_mma = (rows + 31) / 32 * 32;
  P->stages1 = 6;  // K ring of pass 1 (next to its V ring)
  while (P->stages1 > 1 && lse_smem_bytes(P->d, P->rows_pad, P->stages1) > kMaxSmem) --P->stages1;
  P->stages2 = 4;
  while (P->stages2 > 1 && keyscore_smem_bytes(P->d, P->rows_pad, P->stages2, false) > kMaxSmem)
    --P->stages2;
  P->smem1 = lse_smem_bytes(P->d, P->rows_pad, P->stages1);
  // pass 1 stages the guide block, and at the end its row statistics, through
  // its K ring
  if (size_t(P->stages1) * (P->d / 64) * 16384 <
      std::max(size_t(P->d / 64) * P->rows_pad * 128, size_t(4) * P->rows_pad * sizeof(float2)))
    return TP_ERR_UNSUPPORTED_SHAPE;
  P->smem2 = keyscore_smem_bytes(P->d, P->rows_pad, P->stages2, false);
  if (P->smem1 > size_t(kMaxSmem) || P->smem2 > size_t(kMaxSmem)) return TP_ERR_UNSUPPORTED_SHAPE;
  P->stages2s = 4;
  while (P->stages2s >= 2 && keyscore_smem_bytes(P->d, P->rows_pad, P->stages2s, true) > kMaxSmem)
    --P->stages2s;
  if (P->stages2s < 2) P->stages2s = 0;
  P->smem2s = P->stages2s ? keyscore_smem_bytes(P->d, P->rows_pad, P->stages2s, true) : 0;
  return TP_OK;
}

int64_t kept_for(int64_t n, double ratio, int64_t budget) {
  if (budget >= 0) return budget < n ? budget : n;
  return tp_budget(n, ratio);
}

// Validates the problem and fills the plan.  `need_select` adds the kept
// counts (ratio/budget must then be valid).
int make_plan(const tp_problem* p, double ratio, int64_t budget, bool need_select, Plan* P) {
  if (!p || !P) return TP_ERR_INVALID_ARG;
  if (p->n_heads_kv <= 0 || p->n_heads_q <= 0 || p->n_heads_q % p->n_heads_kv != 0)
    return TP_ERR_INVALID_ARG;
  if (p->guide_len <= 0 || p->batch <= 0 || p->batch > kMaxBatch || !p->doc_offsets)
    return TP_ERR_INVALID_ARG;
  if (p->head_dim != 64 && p->head_dim != 128) return TP_ERR_UNSUPPORTED_SHAPE;
  if (p->pool_kernel < 1 || p->pool_kernel % 2 == 0 || p->pool_kernel > 33)
    return TP_ERR_UNSUPPORTED_SHAPE;
  if (p->quant_bits != 8 && p->quant_bits != 4) return TP_ERR_UNSUPPORTED_SHAPE;
  const uint32_t score_flags = TP_SCORE_KEY_ONLY | TP_SCORE_NORM_ADD | TP_SCORE_HARMONIC;
  if (p->flags & ~score_flags) return TP_ERR_INVALID_ARG;
  const uint32_t f = p->flags;
  if ((f & (f - 1)) != 0) return TP_ERR_INVALID_ARG;  // at most one score flag
  memset(P, 0, sizeof(*P));
  P->hq = p->n_heads_q;
  P->hkv = p->n_heads_kv;
  P->d = p->head_dim;
  P->lt = p->guide_len;
  P->g = p->n_heads_q / p->n_heads_kv;
  P->batch = p->batch;
  if (p->doc_offsets[0] != 0) return TP_ERR_INVALID_ARG;
  for (int b = 0; b <= p->batch; ++b) {
    P->off[b] = p->doc_offsets[b];
    if (b > 0 && (P->off[b] < P->off[b - 1] || P->off[b] - P->off[b - 1] > INT32_MAX / 2))
      return TP_ERR_INVALID_ARG;
  }
  P->n_total = P->off[p->batch];
  if (P->n_total > (int64_t(1) << 31) - 256) return TP_ERR_UNSUPPORTED_SHAPE;
  const int64_t rows = int64_t(P->g) * P->lt;
  if (rows > TP_MAX_GUIDE_ROWS) return TP_ERR_UNSUPPORTED_SHAPE;
  P->rows_full = static_cast<int>(rows);
  P->blocks = static_cast<int>((rows + TP_MAX_ROWS - 1) / TP_MAX_ROWS);
  P->row0 = 0;
  const double sigma = p->softmax_scale > 0 ? double(p->softmax_scale) : 1.0 / sqrt(double(P->d));
  P->c2 = static_cast<float>(sigma * 1.4426950408889634);
  P->sigma = static_cast<float>(sigma);
  P->bits = p->quant_bits;
  P->qmax = static_cast<float>((1 << (p->quant_bits - 1)) - 1);
  P->inv_group = 1.0f / static_cast<float>(P->g);

  // Key tiles per CTA: the smallest T whose CTA count fits one wave.
  const int sms = num_sms();
  int64_t tiles_total = 0;
  for (int b = 0; b < P->batch; ++b) tiles_total += (P->off[b + 1] - P->off[b] + 127) / 128;
  tiles_total *= P->hkv;
  int64_t T = tiles_total > 0 ? (tiles_total + sms - 1) / sms : 1;
  if (T < 1) T = 1;
  for (int iter = 0; iter < 64; ++iter) {
    int64_t ctas = 0;
    for (int b = 0; b < P->batch; ++b) ctas += ((P->off[b + 1] - P->off[b] + 127) / 128 + T - 1) / T;
    if (ctas * P->hkv <= sms) break;
    ++T;
  }
  P->tiles_per_cta = static_cast<int>(T);
  P->cta[0] = 0;
  for (int b = 0; b < P->batch; ++b) {
    const int64_t tiles = (P->off[b + 1] - P->off[b] + 127) / 128;
    P->cta[b + 1] = P->cta[b] + static_cast<int32_t>((tiles + T - 1) / T);
  }
  P->grid_x = P->cta[P->batch];

  // The first block of guide rows (all of them up to TP_MAX_ROWS).
  const int st_rows = set_rows(P, static_cast<int>(std::min<int64_t>(rows, TP_MAX_ROWS)));
  if (st_rows != TP_OK) return st_rows;

  P->cap = 0;
  if (need_select) {
    for (int b = 0; b < P->batch; ++b) {
      const int64_t k = kept_for(P->off[b + 1] - P->off[b], ratio, budget);
      if (k < 0) return TP_ERR_INVALID_ARG;
      P->kept[b] = static_cast<int32_t>(k);
      if (k > P->cap) P->cap = k;
    }
  }

  const size_t units = size_t(P->hkv) * P->batch;

  // [status | counters] are zeroed at the start of a call.
  size_t o = 0;
  P->ws_status = o;
  o = align_up(o + sizeof(int) * (1 + units));
  P->ws_partials = o;
  o = align_up(o + sizeof(float2) * size_t(P->hkv) * P->grid_x * P->rows_pad);
  P->ws_lse = o;
  o = align_up(o + sizeof(float) * size_t(P->batch) * P->hkv * P->rows);
  P->ws_skey = o;
  o = align_up(o + sizeof(float) * size_t(P->hkv) * P->n_total);
  P->ws_gamma = o;
  o = align_up(o + sizeof(float) * size_t(P->hkv) * P->n_total);
  P->ws_keys = o;
  o = align_up(o + sizeof(uint32_t) * size_t(P->hkv) * P->n_total);
  P->ws_lse_full = P->ws_skey_part = o;
  if (P->blocks > 1) {
    P->ws_lse_full = o;
    o = align_up(o + sizeof(float) * size_t(P->batch) * P->hkv * P->rows_full);
    P->ws_skey_part = o;
    o = align_up(o + sizeof(float) * size_t(P->hkv) * P->n_total);
  }
  P->ws_total = o;
  return TP_OK;
}

// --- TMA descriptors ---------------------------------------------------------
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static std::once_flag once;
  static EncodeTiledFn fn = nullptr;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(f);
  });
  return fn;
}

// 3-D bf16 view {d, rows, planes} with a {64, box_rows, 1} box, 128-byte
// swizzle; consecutive planes lie plane_rows rows apart (rows by default).
bool encode_3d(CUtensorMap* map, const void* base, int d, int64_t rows, int64_t planes,
               int box_rows, int64_t plane_rows = -1) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  if (plane_rows < 0) plane_rows = rows;
  cuuint64_t dims[3] = {cuuint64_t(d), cuuint64_t(rows), cuuint64_t(planes)};
  cuuint64_t strides[2] = {cuuint64_t(d) * 2, cuuint64_t(d) * 2 * cuuint64_t(plane_rows)};
  cuuint32_t box[3] = {64, cuuint32_t(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15) == 0; }

int cuda_status(cudaError_t e) { return e == cudaSuccess ? TP_OK : TP_ERR_CUDA; }

// The guide rows of a plan's block: rows [row0, row0 + rows) of every
// (document, head) group of G * L_t rows (a row offset of a multiple of
// TP_MAX_ROWS keeps the base 16-byte aligned).
bool encode_q(CUtensorMap* map, const Plan& P, const void* q, int box_rows) {
  const char* base = static_cast<const char*>(q) + size_t(P.row0) * P.d * 2;
  return encode_3d(map, base, P.d, P.rows, int64_t(P.batch) * P.hkv, box_rows, P.rows_full);
}

bool encode_maps(const Plan& P, const void* q, const void* k, CUtensorMap* tmk, CUtensorMap* tmq) {
  return encode_3d(tmk, k, P.d, P.n_total, P.hkv, 128) &&
         encode_q(tmq, P, q, P.rows_pad < 256 ? P.rows_pad : 256);
}

// Alignment mask of a code buffer: a thread stores 8 codes at once (8 bytes,
// or 4 at b = 4).
uintptr_t code_align(const Plan& P) { return P.bits == 8 ? 7 : 3; }

DocTable doc_table(const Plan& P) {
  DocTable docs;
  memset(&docs, 0, sizeof(docs));
  docs.batch = P.batch;
  for (int b = 0; b <= P.batch; ++b) {
    docs.off[b] = P.off[b];
    docs.cta[b] = P.cta[b];
  }
  return docs;
}

// Pass 1: row normalisers into `lse` ([batch, H_kv, rows]), and the Eq. 2
// scales of every token into `gamma` when v/gamma are given.  The counters and
// the status word at the head of the workspace must be zero.
int run_lse(const Plan& P, const CUtensorMap& tmk, const CUtensorMap& tmq, const void* q,
            const void* v, float* gamma, float* lse, char* ws, cudaStream_t s, bool dependent = false) {
  CUtensorMap tmv = tmk;
  if (gamma && !encode_3d(&tmv, v, P.d, P.n_total, P.hkv, 128)) return TP_ERR_CUDA;
  int* status = reinterpret_cast<int*>(ws + P.ws_status);
  LseParams lp;
  memset(&lp, 0, sizeof(lp));
  lp.docs = doc_table(P);
  lp.q = static_cast<const uint16_t*>(q);
  lp.gamma = gamma;
  lp.qmax = P.qmax;
  lp.n_total = P.n_total;
  lp.n_heads_kv = P.hkv;
  lp.rows = P.rows;
  lp.rows_pad = P.rows_pad;
  lp.nrb = P.nrb;
  lp.tiles_per_cta = P.tiles_per_cta;
  lp.stages = P.stages1;
  lp.c2 = P.c2;
  lp.partials = reinterpret_cast<float2*>(ws + P.ws_partials);
  lp.lse = lse;
  lp.counters = status + 1;
  lp.status = status;
  return cuda_status(
      launch_lse(tmk, tmv, tmq, lp, P.d, dim3(P.grid_x, P.hkv), P.smem1, dependent, s));
}

// Pass 2 with the Eq. 2 scales on CTA pairs: tiles of 256 keys, the smallest
// count per pair whose pairs (over all heads) are resident at once, and the
// deepest K ring that fits next to half of the guide block and the V ring.
struct PairGeometry {
  int tiles;                   // pair tiles per pair
  int pairs;                   // pairs per head
  int32_t cta[kMaxBatch + 1];  // pair prefix per document
  int stages;
  size_t smem;
};

bool pair_geometry(const Plan& P, PairGeometry* G) {
  G->stages = 4;
  while (G->stages > 1 && keyscore_pair_smem_bytes(P.d, P.rows_mma, G->stages) > size_t(kMaxSmem))
    --G->stages;
  G->smem = keyscore_pair_smem_bytes(P.d, P.rows_mma, G->stages);
  if (G->smem > size_t(kMaxSmem)) return false;
  const int clusters = keyscore_pair_max_clusters(P.d, P.rows_mma, G->smem);
  if (clusters <= 0) return false;
  int64_t tiles_total = 0;
  for (int b = 0; b < P.batch; ++b) tiles_total += (P.off[b + 1] - P.off[b] + 255) / 256;
  tiles_total *= P.hkv;
  int64_t T = tiles_total > 0 ? (tiles_total + clusters - 1) / clusters : 1;
  if (T < 1) T = 1;
  int64_t pairs = 0;
  for (int iter = 0; iter < 64; ++iter) {
    pairs = 0;
    for (int b = 0; b < P.batch; ++b) pairs += ((P.off[b + 1] - P.off[b] + 255) / 256 + T - 1) / T;
    if (pairs * P.hkv <= clusters) break;
    ++T;
  }
  if (pairs * P.hkv > clusters || pairs == 0) return false;
  G->tiles = static_cast<int>(T);
  G->cta[0] = 0;
  for (int b = 0; b < P.batch; ++b)
    G->cta[b + 1] = G->cta[b] + static_cast<int32_t>(((P.off[b + 1] - P.off[b] + 255) / 256 + T - 1) / T);
  G->pairs = G->cta[P.batch];
  return true;
}

// Pass 2: unpooled key scores [H_kv, N] from the row normalisers.
int run_keyscore(const Plan& P, const CUtensorMap& tmk, const void* q, const float* lse,
                 float* skey, int* status, bool dependent, cudaStream_t s) {
  KeyScoreParams kp;
  memset(&kp, 0, sizeof(kp));
  kp.docs = doc_table(P);
  kp.n_heads_kv = P.hkv;
  kp.rows = P.rows;
  kp.rows_pad = P.rows_pad;
  kp.rows_mma = P.rows_mma;
  kp.tiles_per_cta = P.tiles_per_cta;
  kp.stages = P.stages2;
  kp.c2 = P.c2;
  kp.inv_group = P.inv_group;
  kp.n_total = P.n_total;
  kp.lse = lse;
  kp.skey = skey;
  kp.status = status;
  CUtensorMap tmq;
  if (!encode_q(&tmq, P, q, P.rows_pad < 256 ? P.rows_pad : 256)) return TP_ERR_CUDA;
  return cuda_status(
      launch_keyscore(tmk, tmk, tmq, kp, P.d, dim3(P.grid_x, P.hkv), P.smem2, dependent, s));
}

// With the caller's row normalisers: the key scores and the Eq. 2 scales of
// every token in one kernel (K and V each read once): one CTA per key range
// with up to 256 guide rows, CTA pairs above (each CTA then holds half of the
// guide block).  Returns kNoFusedScales, launching nothing, where neither fits
// (pairs that would not all be resident at once); the caller then runs the
// quantiser and pass 2.
constexpr int kNoFusedScales = 1;  // positive: every TP_ERR_* code is negative

bool fused_scales_fit(const Plan& P) {
  PairGeometry G;
  return P.stages2s > 0 || pair_geometry(P, &G);
}

int run_keyscore_scales(const Plan& P, const void* q, const void* k, const void* v,
                        const float* lse, float* skey, float* gamma, int* status, bool dependent,
                        cudaStream_t s) {
  PairGeometry G;
  const bool single = P.stages2s > 0;
  if (!single && !pair_geometry(P, &G)) return kNoFusedScales;
  CUtensorMap tmk, tmv, tmq;
  const int qbox = single ? (P.rows_pad < 256 ? P.rows_pad : 256) : 128;
  if (!encode_3d(&tmk, k, P.d, P.n_total, P.hkv, 128) ||
      !encode_3d(&tmv, v, P.d, P.n_total, P.hkv, 128) ||
      !encode_q(&tmq, P, q, qbox))
    return TP_ERR_CUDA;
  KeyScoreParams kp;
  memset(&kp, 0, sizeof(kp));
  kp.docs = doc_table(P);
  kp.n_heads_kv = P.hkv;
  kp.rows = P.rows;
  kp.rows_pad = P.rows_pad;
  kp.rows_mma = P.rows_mma;
  kp.c2 = P.c2;
  kp.inv_group = P.inv_group;
  kp.n_total = P.n_total;
  kp.lse = lse;
  kp.skey = skey;
  kp.gamma = gamma;
  kp.qmax = P.qmax;
  kp.status = status;
  if (single) {
    kp.tiles_per_cta = P.tiles_per_cta;
    kp.stages = P.stages2s;
    return cuda_status(
        launch_keyscore(tmk, tmv, tmq, kp, P.d, dim3(P.grid_x, P.hkv), P.smem2s, dependent, s));
  }
  for (int b = 0; b <= P.batch; ++b) kp.docs.cta[b] = G.cta[b];
  kp.tiles_per_cta = G.tiles;
  kp.stages = G.stages;
  return cuda_status(launch_keyscore_pair(tmk, tmv, tmq, kp, P.d, dim3(2 * G.pairs, P.hkv), G.smem,
                                          dependent, s));
}

// The guide-prefix fold of the literal normaliser (`lse` in place).
int run_prefix(const Plan& P, const void* q, const void* k_guide, float* lse, bool dependent,
               cudaStream_t s) {
  PrefixParams pp;
  memset(&pp, 0, sizeof(pp));
  for (int b = 0; b <= P.batch; ++b) pp.off[b] = P.off[b];
  pp.q = static_cast<const uint16_t*>(q);
  pp.k_guide = static_cast<const uint16_t*>(k_guide);
  pp.lse = lse;
  pp.batch = P.batch;
  pp.n_heads_kv = P.hkv;
  pp.rows = P.rows_full;  // the fold reads and rewrites whole rows of every block
  pp.guide_len = P.lt;
  pp.head_dim = P.d;
  pp.sigma = P.sigma;
  return cuda_status(launch_prefix(pp, dependent, s));
}

// The plan of block `blk` of the guide rows (rows blk * TP_MAX_ROWS onwards).
int block_plan(const Plan& P, int blk, Plan* B) {
  *B = P;
  B->row0 = blk * TP_MAX_ROWS;
  return set_rows(B, std::min(TP_MAX_ROWS, P.rows_full - B->row0));
}

// Columns [col0, col0 + cols) of `units` rows of floats, from rows src_pitch
// floats apart to rows dst_pitch floats apart (device to device, in stream
// order).
int copy_cols(float* dst, int dst_pitch, const float* src, int src_pitch, int cols, size_t units,
              cudaStream_t s) {
  if (units == 0 || cols == 0) return TP_OK;
  return cuda_status(cudaMemcpy2DAsync(dst, sizeof(float) * dst_pitch, src, sizeof(float) * src_pitch,
                                       sizeof(float) * cols, units, cudaMemcpyDeviceToDevice, s));
}

// Scoring of a guide longer than one block of TP_MAX_ROWS stacked rows
// (P.blocks > 1), leaving the unpooled key scores in the workspace like
// run_scoring.  A row's normaliser involves that row alone, so every block
// runs the passes on its own rows; the key scores (Eq. 1: a sum over all rows
// of the group) are the blocks' sums added in block order, and the Eq. 2
// scales come with block 0's pass over V.  Without the caller's normalisers
// or a guide-prefix fold, block b's pass 2 follows its own pass 1.  Otherwise
// the normalisers are first gathered into their full [batch, H_kv, M] layout
// (the caller's, or pass 1's followed by the fold, which reads whole rows),
// and each block's columns are copied out before its pass 2.  Launches go in
// plain stream order.
int run_scoring_blocks(const Plan& P, const void* q, const void* k, const void* v, float* gamma,
                       const float* lse_in, const void* k_guide, char* ws, cudaStream_t s,
                       float* skey_out = nullptr) {
  float* const lse_b = reinterpret_cast<float*>(ws + P.ws_lse);
  float* const lse_f = reinterpret_cast<float*>(ws + P.ws_lse_full);
  float* const skey = skey_out ? skey_out : reinterpret_cast<float*>(ws + P.ws_skey);
  float* const part = reinterpret_cast<float*>(ws + P.ws_skey_part);
  int* const status = reinterpret_cast<int*>(ws + P.ws_status);
  const size_t units = size_t(P.batch) * P.hkv;
  const int64_t nkey = int64_t(P.hkv) * P.n_total;
  const bool gathered = lse_in || k_guide;
  CUtensorMap tmk;
  if (!encode_3d(&tmk, k, P.d, P.n_total, P.hkv, 128)) return TP_ERR_CUDA;
  int st;
  if (!lse_in) {
    for (int blk = 0; blk < P.blocks; ++blk) {
      Plan B;
      if ((st = block_plan(P, blk, &B)) != TP_OK) return st;
      CUtensorMap tmq;
      if (!encode_q(&tmq, B, q, B.rows_pad < 256 ? B.rows_pad : 256)) return TP_ERR_CUDA;
      if ((st = run_lse(B, tmk, tmq, q, blk == 0 ? v : nullptr, blk == 0 ? gamma : nullptr, lse_b,
                        ws, s)) != TP_OK)
        return st;
      if (gathered) {
        if ((st = copy_cols(lse_f + B.row0, P.rows_full, lse_b, B.rows, B.rows, units, s)) != TP_OK)
          return st;
        continue;
      }
      if ((st = run_keyscore(B, tmk, q, lse_b, blk == 0 ? skey : part, status, false, s)) != TP_OK)
        return st;
      if (blk > 0 && launch_add(skey, part, nkey, num_sms(), s) != cudaSuccess) return TP_ERR_CUDA;
    }
    if (!gathered) return TP_OK;
    if (k_guide && (st = run_prefix(P, q, k_guide, lse_f, false, s)) != TP_OK) return st;
  }
  const float* const src = lse_in ? lse_in : lse_f;
  for (int blk = 0; blk < P.blocks; ++blk) {
    Plan B;
    if ((st = block_plan(P, blk, &B)) != TP_OK) return st;
    if ((st = copy_cols(lse_b, B.rows, src + B.row0, P.rows_full, B.rows, units, s)) != TP_OK)
      return st;
    float* const out = blk == 0 ? skey : part;
    if (lse_in && blk == 0 && gamma) {
      // the caller's normalisers: block 0's kernel also forms the scales
      st = run_keyscore_scales(B, q, k, v, lse_b, out, gamma, status, false, s);
      if (st == kNoFusedScales) {
        if (launch_vquant(static_cast<const uint16_t*>(v), nullptr, gamma, nkey, P.d, P.qmax, P.bits,
                          num_sms(), s) != cudaSuccess)
          return TP_ERR_CUDA;
        st = run_keyscore(B, tmk, q, lse_b, out, status, false, s);
      }
    } else {
      st = run_keyscore(B, tmk, q, lse_b, out, status, false, s);
    }
    if (st != TP_OK) return st;
    if (blk > 0 && launch_add(skey, part, nkey, num_sms(), s) != cudaSuccess) return TP_ERR_CUDA;
  }
  return TP_OK;
}

// Both scoring passes (with the Eq. 2 scales fused into the first when gamma
// is given, and the guide prefix folded into the normalisers between them when
// k_guide is given); leaves the unpooled key scores in the workspace (or in
// skey_out).
int run_scoring(const Plan& P, const void* q, const void* k, const void* v, float* gamma, char* ws,
                cudaStream_t s, const void* k_guide = nullptr, bool dependent = false,
                float* skey_out = nullptr) {
  if (P.n_total == 0 || P.grid_x == 0) return TP_OK;
  if (P.blocks > 1) return run_scoring_blocks(P, q, k, v, gamma, nullptr, k_guide, ws, s, skey_out);
  CUtensorMap tmk, tmq;
  if (!encode_maps(P, q, k, &tmk, &tmq)) return TP_ERR_CUDA;
  float* lse = reinterpret_cast<float*>(ws + P.ws_lse);
  int st = run_lse(P, tmk, tmq, q, v, gamma, lse, ws, s, dependent);
  if (st != TP_OK) return st;
  if (k_guide && (st = run_prefix(P, q, k_guide, lse, true, s)) != TP_OK) return st;
  return run_keyscore(P, tmk, q, lse, skey_out ? skey_out : reinterpret_cast<float*>(ws + P.ws_skey),
                      reinterpret_cast<int*>(ws + P.ws_status), true, s);
}

// Stacks of layers of short documents select several layers in one launch
// when the caller's workspace holds their key scores, scales and key scratch
// side by side (tp_workspace_bytes_stack): slot 0 is the plan's own regions,
// slots 1.. follow the plan's workspace.
constexpr int64_t kMergeMaxTokens = 65536;  // four-CTA slices stay in shared memory

int64_t max_doc_len(const Plan& P) {
  int64_t m = 0;
  for (int b = 0; b < P.batch; ++b) m = std::max(m, P.off[b + 1] - P.off[b]);
  return m;
}

int stack_slots(const Plan& P, int n_layers) {
  if (n_layers < 2 || max_doc_len(P) > kMergeMaxTokens) return 1;
  return std::min(n_layers, kMaxSelectLayers);
}

size_t slot_bytes(const Plan& P) { return 3 * align_up(sizeof(float) * size_t(P.hkv) * P.n_total); }

struct Slot {
  float* skey;
  float* gamma;
  uint32_t* keys;
};

Slot stack_slot(const Plan& P, char* ws, int i) {
  if (i == 0)
    return {reinterpret_cast<float*>(ws + P.ws_skey), reinterpret_cast<float*>(ws + P.ws_gamma),
            reinterpret_cast<uint32_t*>(ws + P.ws_keys)};
  const size_t a = align_up(sizeof(float) * size_t(P.hkv) * P.n_total);
  char* base = ws + P.ws_total + size_t(i - 1) * slot_bytes(P);
  return {reinterpret_cast<float*>(base), reinterpret_cast<float*>(base + a),
          reinterpret_cast<uint32_t*>(base + 2 * a)};
}

// Layers per selection launch for a stack: as many as the workspace holds
// slots for and as fit in one wave of four-CTA selection clusters; 1 for the
// normalised-add score (its per-document norms are summed over a cluster, so
// the cluster size must not change with the grouping).
int stack_group(const Plan& P, uint32_t flags, int n_layers, size_t ws_bytes) {
  int g = stack_slots(P, n_layers);
  if (g < 2 || (flags & TP_SCORE_NORM_ADD)) return 1;
  while (g > 1 && P.ws_total + size_t(g - 1) * slot_bytes(P) > ws_bytes) --g;
  if (g < 2) return 1;
  return std::min(g, select_merge_layers(P.batch * P.hkv, max_doc_len(P)));
}

int blend_of(uint32_t flags) {
  if (flags & TP_SCORE_NORM_ADD) return kBlendNormAdd;
  if (flags & TP_SCORE_HARMONIC) return kBlendHarmonic;
  return kBlendProduct;
}

void fill_select(const Plan& P, char* ws, SelectParams* sp) {
  memset(sp, 0, sizeof(*sp));
  for (int b = 0; b <= P.batch; ++b) sp->off[b] = P.off[b];
  for (int b = 0; b < P.batch; ++b) sp->kept[b] = P.kept[b];
  // the selection launches the longest documents' clusters first (ties in
  // document order): with more clusters than fit at once, the last wave then
  // holds the shortest documents
  for (int b = 0; b < P.batch; ++b) sp->order[b] = static_cast<int16_t>(b);
  std::stable_sort(sp->order, sp->order + P.batch, [&](int16_t x, int16_t y) {
    return P.off[x + 1] - P.off[x] > P.off[y + 1] - P.off[y];
  });
  sp->batch = P.batch;
  sp->n_heads_kv = P.hkv;
  sp->head_dim = P.d;
  sp->n_total = P.n_total;
  sp->cap = P.cap;
  sp->pool_kernel = 1;
  sp->keys = reinterpret_cast<uint32_t*>(ws + P.ws_keys);
}

int zero_head(const Plan& P, char* ws, cudaStream_t s) {
  return cudaMemsetAsync(ws + P.ws_status, 0, P.ws_partials - P.ws_status, s) == cudaSuccess
             ? TP_OK
             : TP_ERR_CUDA;
}

void fill_gather(const Plan& P, GatherParams* gp) {
  memset(gp, 0, sizeof(*gp));
  for (int b = 0; b <= P.batch; ++b) gp->off[b] = P.off[b];
  gp->batch = P.batch;
  gp->n_heads_kv = P.hkv;
  gp->head_dim = P.d;
  gp->n_total = P.n_total;
  gp->cap = P.cap;
  gp->qmax = P.qmax;
  gp->bits = P.bits;
}

// The fused layer.  Without `lse`: two scoring passes (the first also forms
// the Eq. 2 scales), with the guide prefix folded into the normalisers between
// them when `k_guide` is given.  With the caller's row normalisers `lse`: one
// pass over V for the scales, then the key-score pass with those normalisers.
int compress_layer(const tp_problem* p, const void* q, const void* k, const void* v,
                   const float* lse_in, const void* k_guide, double keep_ratio, int64_t budget,
                   int32_t* idx, void* kc, void* vc, int8_t* vqc, float* gammac, float* scores,
                   float* gamma, void* ws, size_t ws_bytes, void* stream) {
  Plan P;
  int st = make_plan(p, keep_ratio, budget, true, &P);
  if (st != TP_OK) return st;
  if (!q || !k || !v || (!idx && P.cap > 0) || !aligned16(q) || !aligned16(k) || !aligned16(v))
    return TP_ERR_INVALID_ARG;
  if ((kc && !aligned16(kc)) || (vc && !aligned16(vc)) ||
      (vqc && (reinterpret_cast<uintptr_t>(vqc) & code_align(P))))
    return TP_ERR_INVALID_ARG;
  if (!ws || ws_bytes < P.ws_total || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)))
    return TP_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  float* g = gamma ? gamma : reinterpret_cast<float*>(w + P.ws_gamma);
  if ((st = zero_head(P, w, s)) != TP_OK) return st;
  if (!lse_in) {
    if ((st = run_scoring(P, q, k, v, g, w, s, k_guide)) != TP_OK) return st;
  } else if (P.n_total > 0 && P.grid_x > 0 && P.blocks > 1) {
    if ((st = run_scoring_blocks(P, q, k, v, g, lse_in, nullptr, w, s)) != TP_OK) return st;
  } else if (P.n_total > 0 && P.grid_x > 0) {
    float* const skey = reinterpret_cast<float*>(w + P.ws_skey);
    int* const status = reinterpret_cast<int*>(w + P.ws_status);
    st = run_keyscore_scales(P, q, k, v, lse_in, skey, g, status, false, s);
    if (st == kNoFusedScales) {
      if (launch_vquant(static_cast<const uint16_t*>(v), nullptr, g, int64_t(P.hkv) * P.n_total, P.d,
                        P.qmax, P.bits, num_sms(), s) != cudaSuccess)
        return TP_ERR_CUDA;
      CUtensorMap tmk, tmq;
      if (!encode_maps(P, q, k, &tmk, &tmq)) return TP_ERR_CUDA;
      st = run_keyscore(P, tmk, q, lse_in, skey, status, true, s);
    }
    if (st != TP_OK) return st;
  }
  SelectParams sp;
  fill_select(P, w, &sp);
  sp.pool_kernel = p->pool_kernel;
  sp.key_only = (p->flags & TP_SCORE_KEY_ONLY) ? 1 : 0;
  sp.blend = blend_of(p->flags);
  sp.skey = reinterpret_cast<const float*>(w + P.ws_skey);
  sp.gamma = g;
  sp.scores_out = scores;
  sp.idx = idx;
  cudaError_t e2 = launch_select(sp, true, s);
  if (e2 != cudaSuccess) return TP_ERR_CUDA;
  if (P.cap == 0) return TP_OK;
  GatherParams gp;
  fill_gather(P, &gp);
  gp.k = static_cast<const uint16_t*>(k);
  gp.v = static_cast<const uint16_t*>(v);
  gp.gamma = g;
  gp.idx = idx;
  gp.kc = static_cast<uint16_t*>(kc);
  gp.vc = static_cast<uint16_t*>(vc);
  gp.vqc = vqc;
  gp.gammac = gammac;
  return cuda_status(launch_gather(gp, true, s));
}

// The selection of layers l0 .. l0 + gl - 1 of a stack (one launch; their key
// scores and scales in slots 0 .. gl - 1) and their compactions, each a
// programmatic dependent of the kernel before it.
int stack_tail(const Plan& P, const tp_problem* p, int l0, int gl, const void* const* k,
               const void* const* v, int32_t* const* idx, void* const* kc, void* const* vc,
               int8_t* const* vqc, float* const* gammac, char* w, cudaStream_t s) {
  SelectParams sp;
  fill_select(P, w, &sp);
  sp.pool_kernel = p->pool_kernel;
  sp.key_only = (p->flags & TP_SCORE_KEY_ONLY) ? 1 : 0;
  sp.blend = blend_of(p->flags);
  const Slot s0 = stack_slot(P, w, 0);
  sp.skey = s0.skey;
  sp.gamma = s0.gamma;
  sp.idx = idx ? idx[l0] : nullptr;
  if (gl > 1) {
    sp.layers = gl;
    for (int i = 0; i < gl; ++i) {
      const Slot sl = stack_slot(P, w, i);
      sp.skey_l[i] = sl.skey;
      sp.gamma_l[i] = sl.gamma;
      sp.keys_l[i] = sl.keys;
      sp.idx_l[i] = idx ? idx[l0 + i] : nullptr;
    }
  }
  if (launch_select(sp, true, s) != cudaSuccess) return TP_ERR_CUDA;
  if (P.cap == 0) return TP_OK;
  for (int i = 0; i < gl; ++i) {
    const int l = l0 + i;
    GatherParams gp;
    fill_gather(P, &gp);
    gp.k = static_cast<const uint16_t*>(k[l]);
    gp.v = static_cast<const uint16_t*>(v[l]);
    gp.gamma = stack_slot(P, w, i).gamma;
    gp.idx = idx[l];
    gp.kc = kc ? static_cast<uint16_t*>(kc[l]) : nullptr;
    gp.vc = vc ? static_cast<uint16_t*>(vc[l]) : nullptr;
    gp.vqc = vqc ? vqc[l] : nullptr;
    gp.gammac = gammac ? gammac[l] : nullptr;
    const int st = cuda_status(launch_gather(gp, true, s));
    if (st != TP_OK) return st;
  }
  return TP_OK;
}

}  // namespace


// ---------------------------------------------------------------------------
// Fixed device scratch for tp_guide_lse_static: the status word, the per-
// (document, head) counters and the per-CTA partial sums of pass 1.  Every
// GPU that loads the library holds it until the process exits.
// ---------------------------------------------------------------------------
constexpr size_t kStaticScratchBytes = size_t(2) << 20;  // 2 MiB
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

namespace {

// The array's device address belongs to one CUDA context: a context created
// after cudaDeviceReset, or a second context on the same device, holds its
// own copy at another address.  Addresses are therefore cached by the
// context's process-unique ID (cuCtxGetId), never by device number.
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

struct CtxFns {
  CtxGetCurrentFn get_current = nullptr;
  CtxGetIdFn get_id = nullptr;
};

const CtxFns& ctx_fns() {
  static std::once_flag once;
  static CtxFns fns;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      fns.get_current = reinterpret_cast<CtxGetCurrentFn>(f);
    f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      fns.get_id = reinterpret_cast<CtxGetIdFn>(f);
  });
  return fns;
}

constexpr int kStaticCacheSlots = 64;
std::mutex g_static_mu;
struct StaticSlot {
  unsigned long long ctx_id;
  void* ptr;
};
StaticSlot g_static_cache[kStaticCacheSlots];
int g_static_used = 0;

// ID of the calling thread's current context; when the thread has none yet,
// the runtime's primary context of the current device is made current first.
int current_ctx_id(unsigned long long* id) {
  const CtxFns& fns = ctx_fns();
  if (!fns.get_current || !fns.get_id) return TP_ERR_CUDA;
  CUcontext ctx = nullptr;
  if (fns.get_current(&ctx) != CUDA_SUCCESS) return TP_ERR_CUDA;
  if (!ctx) {
    void* ptr = nullptr;  // any runtime call that needs a context binds the primary one
    if (cudaGetSymbolAddress(&ptr, g_static_scratch) != cudaSuccess) return TP_ERR_CUDA;
    if (fns.get_current(&ctx) != CUDA_SUCCESS || !ctx) return TP_ERR_CUDA;
  }
  return fns.get_id(ctx, id) == CUDA_SUCCESS ? TP_OK : TP_ERR_CUDA;
}

// Device address of g_static_scratch in the current context (host code cannot
// use the symbol itself as an address): looked up on the first call in each
// context and cached by context ID.  The ID check runs on every call; it is a
// query of the driver's context state and needs no device work.
int static_scratch(char** out) {
  unsigned long long id = 0;
  int st = current_ctx_id(&id);
  if (st != TP_OK) return st;
  std::lock_guard<std::mutex> lock(g_static_mu);
  for (int i = 0; i < g_static_used; ++i)
    if (g_static_cache[i].ctx_id == id) {
      *out = static_cast<char*>(g_static_cache[i].ptr);
      return TP_OK;
    }
  void* ptr = nullptr;
  if (cudaGetSymbolAddress(&ptr, g_static_scratch) != cudaSuccess || !ptr) return TP_ERR_CUDA;
  if (g_static_used < kStaticCacheSlots) g_static_cache[g_static_used++] = {id, ptr};
  *out = static_cast<char*>(ptr);
  return TP_OK;
}

}  // namespace

unsigned long long context_key() {
  unsigned long long id = 0;
  return current_ctx_id(&id) == TP_OK ? id : 0ull;
}

// Kernel attributes belong to a CUDA context as well: the cache is keyed by
// the context's ID, so a context created after cudaDeviceReset, or a second
// context on the device, sets them again.
cudaError_t set_smem_once(const void* kernel, int slot) {
  constexpr int kSlots = 64, kCtxPerSlot = 8;
  static std::mutex mu;
  static unsigned long long done[kSlots][kCtxPerSlot];
  static int used[kSlots];
  const unsigned long long key = context_key();
  if (slot < 0 || slot >= kSlots || key == 0)
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem);
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < used[slot]; ++i)
    if (done[slot][i] == key) return cudaSuccess;
  const cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem);
  if (e == cudaSuccess && used[slot] < kCtxPerSlot) done[slot][used[slot]++] = key;
  return e;
}

}  // namespace tp

using namespace tp;

extern "C" {

int64_t tp_budget(int64_t n, double keep_ratio) {
  if (n < 0 || !(keep_ratio >= 0.0 && keep_ratio <= 1.0)) return -1;
  const double dn = static_cast<double>(n);
  const double prod = keep_ratio * dn;
  const double slack = 1e-9 * dn;
  double k = ceil(prod - slack);
  if (k < 0) k = 0;
  if (k > dn) k = dn;
  return static_cast<int64_t>(k);
}

int64_t tp_kept_capacity(const tp_problem* p, double keep_ratio, int64_t budget) {
  Plan P;
  if (make_plan(p, keep_ratio, budget, true, &P) != TP_OK) return -1;
  return P.cap;
}

size_t tp_workspace_bytes(const tp_problem* p, double keep_ratio, int64_t budget) {
  Plan P;
  const bool sel = budget >= 0 || (keep_ratio >= 0.0 && keep_ratio <= 1.0);
  if (make_plan(p, keep_ratio, budget, sel, &P) != TP_OK) return 0;
  return P.ws_total;
}

size_t tp_workspace_bytes_stack(const tp_problem* p, double keep_ratio, int64_t budget, int n_layers) {
  Plan P;
  const bool sel = budget >= 0 || (keep_ratio >= 0.0 && keep_ratio <= 1.0);
  if (n_layers < 0 || make_plan(p, keep_ratio, budget, sel, &P) != TP_OK) return 0;
  return P.ws_total + size_t(stack_slots(P, n_layers) - 1) * slot_bytes(P);
}

int tp_stack_layers_per_selection(const tp_problem* p, double keep_ratio, int64_t budget,
                                  int n_layers, size_t ws_bytes) {
  Plan P;
  if (n_layers < 1 || make_plan(p, keep_ratio, budget, true, &P) != TP_OK) return -1;
  return stack_group(P, p->flags, n_layers, ws_bytes);
}

int tp_quantize_v(const tp_problem* p, const void* v, int8_t* vq, float* gamma, void* stream) {
  Plan P;
  int st = make_plan(p, 0.0, 0, false, &P);
  if (st != TP_OK) return st;
  if (!v || !gamma || !aligned16(v) || (vq && (reinterpret_cast<uintptr_t>(vq) & code_align(P))))
    return TP_ERR_INVALID_ARG;
  return cuda_status(launch_vquant(static_cast<const uint16_t*>(v), vq, gamma,
                                   int64_t(P.hkv) * P.n_total, P.d, P.qmax, P.bits, num_sms(),
                                   static_cast<cudaStream_t>(stream)));
}

int tp_quantize_rows(const void* x, int64_t rows, int head_dim, int quant_bits, void* xq,
                     float* scale, void* stream) {
  if (rows < 0 || (head_dim != 64 && head_dim != 128) || (quant_bits != 8 && quant_bits != 4))
    return rows < 0 ? TP_ERR_INVALID_ARG : TP_ERR_UNSUPPORTED_SHAPE;
  if (rows == 0) return TP_OK;
  if (!x || !scale || !aligned16(x) ||
      (xq && (reinterpret_cast<uintptr_t>(xq) & (quant_bits == 8 ? 7u : 3u))))
    return TP_ERR_INVALID_ARG;
  const float qmax = static_cast<float>((1 << (quant_bits - 1)) - 1);
  return cuda_status(launch_vquant(static_cast<const uint16_t*>(x), xq, scale, rows, head_dim, qmax,
                                   quant_bits, num_sms(), static_cast<cudaStream_t>(stream)));
}

int tp_guide_scores(const tp_problem* p, const void* q, const void* k, const float* gamma,
                    float* scores, void* ws, size_t ws_bytes, void* stream) {
  Plan P;
  int st = make_plan(p, 0.0, 0, false, &P);
  if (st != TP_OK) return st;
  const bool key_only = (p->flags & TP_SCORE_KEY_ONLY) != 0;
  if (!q || !k || !scores || (!gamma && !key_only) || !aligned16(q) || !aligned16(k))
    return TP_ERR_INVALID_ARG;
  if (!ws || ws_bytes < P.ws_total || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)))
    return TP_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  if ((st = zero_head(P, w, s)) != TP_OK) return st;
  if ((st = run_scoring(P, q, k, nullptr, nullptr, w, s)) != TP_OK) return st;
  SelectParams sp;
  fill_select(P, w, &sp);
  sp.pool_kernel = p->pool_kernel;
  sp.key_only = key_only ? 1 : 0;
  sp.blend = blend_of(p->flags);
  sp.skey = reinterpret_cast<const float*>(w + P.ws_skey);
  sp.gamma = gamma;
  sp.scores_out = scores;
  sp.scores_only = 1;
  return cuda_status(launch_select(sp, true, s));
}

int tp_guide_lse(const tp_problem* p, const void* q, const void* k, const void* v, float* lse,
                 float* gamma, void* ws, size_t ws_bytes, void* stream) {
  Plan P;
  int st = make_plan(p, 0.0, 0, false, &P);
  if (st != TP_OK) return st;
  if (!q || !k || !lse || !aligned16(q) || !aligned16(k)) return TP_ERR_INVALID_ARG;
  if ((v == nullptr) != (gamma == nullptr) || (v && !aligned16(v))) return TP_ERR_INVALID_ARG;
  if (!ws || ws_bytes < P.ws_total || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)))
    return TP_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  if ((st = zero_head(P, w, s)) != TP_OK) return st;
  if (P.n_total == 0 || P.grid_x == 0) return TP_OK;
  CUtensorMap tmk, tmq;
  if (!encode_maps(P, q, k, &tmk, &tmq)) return TP_ERR_CUDA;
  if (P.blocks == 1) return run_lse(P, tmk, tmq, q, v, gamma, lse, w, s);
  // a long guide: block by block through the workspace into lse's columns
  float* const lse_b = reinterpret_cast<float*>(w + P.ws_lse);
  for (int blk = 0; blk < P.blocks; ++blk) {
    Plan B;
    if ((st = block_plan(P, blk, &B)) != TP_OK) return st;
    if (!encode_q(&tmq, B, q, B.rows_pad < 256 ? B.rows_pad : 256)) return TP_ERR_CUDA;
    if ((st = run_lse(B, tmk, tmq, q, blk == 0 ? v : nullptr, blk == 0 ? gamma : nullptr, lse_b, w,
                      s)) != TP_OK)
      return st;
    if ((st = copy_cols(lse + B.row0, P.rows_full, lse_b, B.rows, B.rows, size_t(P.batch) * P.hkv,
                        s)) != TP_OK)
      return st;
  }
  return TP_OK;
}

int tp_guide_lse_static(const tp_problem* p, const void* q, const void* k, const void* v,
                        float* lse, float* gamma, void* stream) {
  Plan P;
  int st = make_plan(p, 0.0, 0, false, &P);
  if (st != TP_OK) return st;
  if (!q || !k || !lse || !aligned16(q) || !aligned16(k)) return TP_ERR_INVALID_ARG;
  if ((v == nullptr) != (gamma == nullptr) || (v && !aligned16(v))) return TP_ERR_INVALID_ARG;
  if (P.blocks > 1) return TP_ERR_UNSUPPORTED_SHAPE;  // the blocks need a workspace
  // pass 1 touches the workspace only up to the end of its partial sums
  if (P.ws_lse > kStaticScratchBytes) return TP_ERR_WORKSPACE;
  char* w = nullptr;
  if ((st = static_scratch(&w)) != TP_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((st = zero_head(P, w, s)) != TP_OK) return st;  // counters must start at zero
  if (P.n_total == 0 || P.grid_x == 0) return TP_OK;
  CUtensorMap tmk, tmq;
  if (!encode_maps(P, q, k, &tmk, &tmq)) return TP_ERR_CUDA;
  return run_lse(P, tmk, tmq, q, v, gamma, lse, w, s);
}

int tp_guide_key_scores(const tp_problem* p, const void* q, const void* k, const void* v,
                        const float* lse, float* key_scores, float* gamma, void* stream) {
  Plan P;
  int st = make_plan(p, 0.0, 0, false, &P);
  if (st != TP_OK) return st;
  if (!q || !k || !lse || !key_scores || !aligned16(q) || !aligned16(k)) return TP_ERR_INVALID_ARG;
  if ((v == nullptr) != (gamma == nullptr) || (v && !aligned16(v))) return TP_ERR_INVALID_ARG;
  if (P.blocks > 1) return TP_ERR_UNSUPPORTED_SHAPE;  // the blocks' sums need a workspace
  if (P.n_total == 0 || P.grid_x == 0) return TP_OK;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (v) {
    st = run_keyscore_scales(P, q, k, v, lse, key_scores, gamma, nullptr, false, s);
    if (st != kNoFusedScales) return st;
    if (launch_vquant(static_cast<const uint16_t*>(v), nullptr, gamma, int64_t(P.hkv) * P.n_total,
                      P.d, P.qmax, P.bits, num_sms(), s) != cudaSuccess)
      return TP_ERR_CUDA;
  }
  CUtensorMap tmk, tmq;
  if (!encode_maps(P, q, k, &tmk, &tmq)) return TP_ERR_CUDA;
  return run_keyscore(P, tmk, q, lse, key_scores, nullptr, false, s);
}

int tp_select(const tp_problem* p, const float* scores, double keep_ratio, int64_t budget,
              int32_t* idx, void* ws, size_t ws_bytes, void* stream) {
  Plan P;
  int st = make_plan(p, keep_ratio, budget, true, &P);
  if (st != TP_OK) return st;
  if (!scores || (!idx && P.cap > 0)) return TP_ERR_INVALID_ARG;
  if (!ws || ws_bytes < P.ws_total || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)))
    return TP_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  if ((st = zero_head(P, w, s)) != TP_OK) return st;
  SelectParams sp;
  fill_select(P, w, &sp);
  sp.scores_in = scores;
  sp.idx = idx;
  return cuda_status(launch_select(sp, false, s));
}

int tp_compact(const tp_problem* p, const void* k, const void* v, const float* gamma,
               const int32_t* idx, double keep_ratio, int64_t budget, void* kc, void* vc,
               int8_t* vqc, float* gammac, void* stream) {
  Plan P;
  int st = make_plan(p, keep_ratio, budget, true, &P);
  if (st != TP_OK) return st;
  if (P.cap == 0) return TP_OK;
  if (!k || !v || !gamma || !idx || !aligned16(k) || !aligned16(v)) return TP_ERR_INVALID_ARG;
  if ((kc && !aligned16(kc)) || (vc && !aligned16(vc)) ||
      (vqc && (reinterpret_cast<uintptr_t>(vqc) & code_align(P))))
    return TP_ERR_INVALID_ARG;
  GatherParams gp;
  fill_gather(P, &gp);
  gp.k = static_cast<const uint16_t*>(k);
  gp.v = static_cast<const uint16_t*>(v);
  gp.gamma = gamma;
  gp.idx = idx;
  gp.kc = static_cast<uint16_t*>(kc);
  gp.vc = static_cast<uint16_t*>(vc);
  gp.vqc = vqc;
  gp.gammac = gammac;
  return cuda_status(launch_gather(gp, false, static_cast<cudaStream_t>(stream)));
}

int tp_compress_layer(const tp_problem* p, const void* q, const void* k, const void* v,
                      double keep_ratio, int64_t budget, int32_t* idx, void* kc, void* vc,
                      int8_t* vqc, float* gammac, float* scores, float* gamma, void* ws,
                      size_t ws_bytes, void* stream) {
  return compress_layer(p, q, k, v, nullptr, nullptr, keep_ratio, budget, idx, kc, vc, vqc, gammac,
                        scores, gamma, ws, ws_bytes, stream);
}

int tp_compress_layer_lse(const tp_problem* p, const void* q, const void* k, const void* v,
                          const float* lse, double keep_ratio, int64_t budget, int32_t* idx,
                          void* kc, void* vc, int8_t* vqc, float* gammac, float* scores,
                          float* gamma, void* ws, size_t ws_bytes, void* stream) {
  if (!lse) return TP_ERR_INVALID_ARG;
  return compress_layer(p, q, k, v, lse, nullptr, keep_ratio, budget, idx, kc, vc, vqc, gammac,
                        scores, gamma, ws, ws_bytes, stream);
}

int tp_compress_layer_guide(const tp_problem* p, const void* q, const void* k, const void* v,
                            const void* k_guide, double keep_ratio, int64_t budget, int32_t* idx,
                            void* kc, void* vc, int8_t* vqc, float* gammac, float* scores,
                            float* gamma, void* ws, size_t ws_bytes, void* stream) {
  if (!k_guide || !aligned16(k_guide)) return TP_ERR_INVALID_ARG;
  return compress_layer(p, q, k, v, nullptr, k_guide, keep_ratio, budget, idx, kc, vc, vqc, gammac,
                        scores, gamma, ws, ws_bytes, stream);
}

int tp_compress_layers(const tp_problem* p, int n_layers, const void* const* q,
                       const void* const* k, const void* const* v, double keep_ratio,
                       int64_t budget, int32_t* const* idx, void* const* kc, void* const* vc,
                       int8_t* const* vqc, float* const* gammac, void* ws, size_t ws_bytes,
                       void* stream) {
  Plan P;
  int st = make_plan(p, keep_ratio, budget, true, &P);
  if (st != TP_OK) return st;
  if (n_layers < 0 || (n_layers > 0 && (!q || !k || !v || (!idx && P.cap > 0))))
    return TP_ERR_INVALID_ARG;
  for (int l = 0; l < n_layers; ++l) {
    if (!q[l] || !k[l] || !v[l] || !aligned16(q[l]) || !aligned16(k[l]) || !aligned16(v[l]))
      return TP_ERR_INVALID_ARG;
    if (P.cap > 0 && !idx[l]) return TP_ERR_INVALID_ARG;
    if ((kc && kc[l] && !aligned16(kc[l])) || (vc && vc[l] && !aligned16(vc[l])) ||
        (vqc && vqc[l] && (reinterpret_cast<uintptr_t>(vqc[l]) & code_align(P))))
      return TP_ERR_INVALID_ARG;
  }
  if (!ws || ws_bytes < P.ws_total || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)))
    return TP_ERR_WORKSPACE;
  if (n_layers == 0) return TP_OK;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  // one reset for the whole stack: pass 1 leaves its counters zero again
  if ((st = zero_head(P, w, s)) != TP_OK) return st;
  const int group = stack_group(P, p->flags, n_layers, ws_bytes);
  for (int l0 = 0; l0 < n_layers; l0 += group) {
    const int gl = std::min(group, n_layers - l0);
    for (int i = 0; i < gl; ++i) {
      // each layer's pass 1 is a dependent of the kernel before it (the
      // previous layer's pass 2, compaction or selection): its prologue
      // overlaps that kernel's tail, and it waits for it before its first store
      const Slot sl = stack_slot(P, w, i);
      const int l = l0 + i;
      if ((st = run_scoring(P, q[l], k[l], v[l], sl.gamma, w, s, nullptr, l > 0, sl.skey)) != TP_OK)
        return st;
    }
    if ((st = stack_tail(P, p, l0, gl, k, v, idx, kc, vc, vqc, gammac, w, s)) != TP_OK) return st;
  }
  return TP_OK;
}

int tp_compress_layers_lse(const tp_problem* p, int n_layers, const void* const* q,
                           const void* const* k, const void* const* v, const float* const* lse,
                           double keep_ratio, int64_t budget, int32_t* const* idx, void* const* kc,
                           void* const* vc, int8_t* const* vqc, float* const* gammac, void* ws,
                           size_t ws_bytes, void* stream) {
  Plan P;
  int st = make_plan(p, keep_ratio, budget, true, &P);
  if (st != TP_OK) return st;
  if (n_layers < 0 || (n_layers > 0 && (!q || !k || !v || !lse || (!idx && P.cap > 0))))
    return TP_ERR_INVALID_ARG;
  for (int l = 0; l < n_layers; ++l) {
    if (!q[l] || !k[l] || !v[l] || !lse[l] || !aligned16(q[l]) || !aligned16(k[l]) ||
        !aligned16(v[l]))
      return TP_ERR_INVALID_ARG;
    if (P.cap > 0 && !idx[l]) return TP_ERR_INVALID_ARG;
    if ((kc && kc[l] && !aligned16(kc[l])) || (vc && vc[l] && !aligned16(vc[l])) ||
        (vqc && vqc[l] && (reinterpret_cast<uintptr_t>(vqc[l]) & code_align(P))))
      return TP_ERR_INVALID_ARG;
  }
  if (!ws || ws_bytes < P.ws_total || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)))
    return TP_ERR_WORKSPACE;
  if (n_layers == 0) return TP_OK;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  int* const status = reinterpret_cast<int*>(w + P.ws_status);
  const bool scored = P.n_total > 0 && P.grid_x > 0;
  if ((st = zero_head(P, w, s)) != TP_OK) return st;
  // Per layer: the key scores with the Eq. 2 scales (one kernel on CTA pairs),
  // then the selection and the compaction, each a programmatic dependent of
  // the kernel before it.  A layer's scoring kernel loads and scores while the
  // kernel before it finishes and waits for it only before its first store;
  // the compaction completes after its selection (it waited for it), which
  // was the last reader of the key scores, and is itself the last reader of
  // the scales, so one buffer of each serves every group of layers.  Without
  // resident pairs a layer runs the quantiser and pass 2 instead.
  const int group = stack_group(P, p->flags, n_layers, ws_bytes);
  for (int l0 = 0; l0 < n_layers; l0 += group) {
    const int gl = std::min(group, n_layers - l0);
    for (int i = 0; scored && i < gl; ++i) {
      const Slot sl = stack_slot(P, w, i);
      const int l = l0 + i;
      if (P.blocks > 1) {
        // a long guide: plain stream order
        if ((st = run_scoring_blocks(P, q[l], k[l], v[l], sl.gamma, lse[l], nullptr, w, s, sl.skey)) !=
            TP_OK)
          return st;
        continue;
      }
      st = run_keyscore_scales(P, q[l], k[l], v[l], lse[l], sl.skey, sl.gamma, status, l > 0, s);
      if (st == kNoFusedScales) {
        if (launch_vquant(static_cast<const uint16_t*>(v[l]), nullptr, sl.gamma,
                          int64_t(P.hkv) * P.n_total, P.d, P.qmax, P.bits, num_sms(), s) != cudaSuccess)
          return TP_ERR_CUDA;
        CUtensorMap tmk, tmq;
        if (!encode_maps(P, q[l], k[l], &tmk, &tmq)) return TP_ERR_CUDA;
        st = run_keyscore(P, tmk, q[l], lse[l], sl.skey, status, true, s);
      }
      if (st != TP_OK) return st;
    }
    if ((st = stack_tail(P, p, l0, gl, k, v, idx, kc, vc, vqc, gammac, w, s)) != TP_OK) return st;
  }
  return TP_OK;
}

int tp_guide_prefix_lse(const tp_problem* p, const void* q, const void* k_guide, float* lse,
                        void* stream) {
  Plan P;
  int st = make_plan(p, 0.0, 0, false, &P);
  if (st != TP_OK) return st;
  if (!q || !k_guide || !lse || !aligned16(q) || !aligned16(k_guide)) return TP_ERR_INVALID_ARG;
  return run_prefix(P, q, k_guide, lse, false, static_cast<cudaStream_t>(stream));
}

int tp_compress_kernel_count(const tp_problem* p, double keep_ratio, int64_t budget, int mode) {
  Plan P;
  if (mode < 0 || mode > 2 || make_plan(p, keep_ratio, budget, true, &P) != TP_OK) return -1;
  int kernels = P.cap > 0 ? 2 : 1;  // selection [+ compaction]
  if (P.n_total > 0 && P.grid_x > 0) {
    // per further block of guide rows: its passes and one addition of its key
    // scores (the copies of normalisers between blocks are not kernels)
    const int more = P.blocks - 1;
    if (mode == 1)  // the key scores with the scales in one kernel, else the quantiser and pass 2
      kernels += (fused_scales_fit(P) ? 1 : 2) + 2 * more;
    else
      kernels += (mode == 2 ? 3 : 2) + 3 * more;  // pass 1, [prefix fold,] pass 2
  }
  return kernels;
}

int tp_selftest_wait_timeout(void* ws, size_t ws_bytes, int64_t limit_ns, void* stream) {
  if (!ws || ws_bytes < sizeof(int) || (reinterpret_cast<uintptr_t>(ws) & 3)) return TP_ERR_WORKSPACE;
  if (limit_ns <= 0 || limit_ns > 1000000000) return TP_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(ws, 0, sizeof(int), s) != cudaSuccess) return TP_ERR_CUDA;
  return cuda_status(launch_wait_selftest(static_cast<int*>(ws), static_cast<uint64_t>(limit_ns), s));
}

int tp_check_status(const void* ws, size_t ws_bytes, void* stream) {
  if (!ws || ws_bytes < sizeof(int)) return TP_ERR_WORKSPACE;
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return TP_ERR_CUDA;
  int status = 0;
  if (cudaMemcpy(&status, ws, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return TP_ERR_CUDA;
  return status == 0 ? TP_OK : status;
}

const char* tp_status_string(int status) {
  switch (status) {
    case TP_OK: return "ok";
    case TP_ERR_INVALID_ARG: return "invalid argument";
    case TP_ERR_WORKSPACE: return "workspace missing or too small";
    case TP_ERR_UNSUPPORTED_SHAPE: return "unsupported shape";
    case TP_ERR_CUDA: return "CUDA error";
    case TP_ERR_TIMEOUT: return "device-side wait timed out";
    default: return "unknown status";
  }
}

}  // extern "C"
