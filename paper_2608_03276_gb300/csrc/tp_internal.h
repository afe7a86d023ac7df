// Internal interface between the C-ABI layer (api.cu) and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/taskpress.h"

namespace tp {

constexpr int kKeyTile = 128;      // context keys per MMA tile
constexpr int kMaxBatch = TP_MAX_BATCH;

// Where each document's CTAs start inside a head's row of the grid, and where
// each document's tokens start.  Passed by value (kernel parameter space).
struct DocTable {
  int64_t off[kMaxBatch + 1];      // token offsets, off[batch] = N
  int32_t cta[kMaxBatch + 1];      // CTA prefix per document (grid.x = cta[batch])
  int32_t batch;
};

__host__ __device__ inline int find_doc(const DocTable& t, int cta) {
  int lo = 0, hi = t.batch - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (t.cta[mid] <= cta) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Pass 1: per-row log-sum-exp partials over a CTA's key tiles, then the
// per-(document, head) merge by the last CTA to finish.
struct LseParams {
  DocTable docs;
  const uint16_t* q;  // guide rows [batch * H_kv, rows, d] bf16
  float* gamma;       // Eq. 2 scales [H_kv, N] written alongside, or null
  float qmax;
  int64_t n_total;
  int n_heads_kv;
  int rows;          // M = G * L_t
  int rows_pad;      // 128 * nrb
  int nrb;           // 128-row blocks of the guide (1, 2 or 4)
  int tiles_per_cta;
  int stages;        // K-tile ring depth
  float c2;          // softmax scale * log2(e)
  float2* partials;  // [H_kv, grid.x, rows_pad] (max2, sum)
  float* lse;        // [batch, H_kv, rows] natural-log sum-exp of scaled logits
  int* counters;     // [H_kv * batch], zero at launch
  int* status;
};

// Pass 2: per-key sum over all guide rows of exp(logit - lse).
struct KeyScoreParams {
  DocTable docs;     // CTA prefix per document (pair prefix for the pair kernel)
  int n_heads_kv;
  int rows;
  int rows_pad;
  int rows_mma;      // rows rounded up to 32 (the MMA N extent, split in 256s)
  int tiles_per_cta; // 128-key tiles per CTA (256-key pair tiles per pair)
  int stages;
  float c2;
  float inv_group;
  int64_t n_total;
  const float* lse;  // [batch, H_kv, rows] natural log
  float* skey;       // [H_kv, N]
  float* gamma;      // Eq. 2 scales [H_kv, N] written alongside, or null
  float qmax;
  int* status;
};


// Blends of the pooled key score a and the scale g (Eq. 3 and the Sec. 4.4
// aggregation ablation): a * g; a / ||a||_2 + g / ||g||_2 per (document,
// head); 2 a g / (a + g).
constexpr int kBlendProduct = 0;
constexpr int kBlendNormAdd = 1;
constexpr int kBlendHarmonic = 2;

// Layers one selection launch may take at once (a stack of short documents).
constexpr int kMaxSelectLayers = 8;

struct SelectParams {
  int64_t off[kMaxBatch + 1];
  int32_t kept[kMaxBatch];   // k_b per document
  int16_t order[kMaxBatch];  // documents in the order their clusters launch (longest first)
  int batch;
  int n_heads_kv;
  int head_dim;
  int64_t n_total;
  int64_t cap;
  int pool_kernel;           // >= 1, odd
  int key_only;
  int blend;                 // kBlendProduct (Eq. 3), kBlendNormAdd or kBlendHarmonic
  int scores_only;           // form the scores (and keys) and stop
  const float* scores_in;    // combined scores (tp_select) or null
  const float* skey;         // unpooled key scores (fused path) or null
  const float* gamma;        // per-token scale (fused path) or null
  float* scores_out;         // optional combined scores out (fused path)
  uint32_t* keys;            // [H_kv, N] scratch
  int32_t* idx;              // [batch, H_kv, cap]
  // layers > 1: the selections of that many layers of one problem in one
  // launch (units layer-major), each layer with its own key scores, scales,
  // key scratch and kept indices; skey, gamma, keys and idx above are then
  // unused.  Only the fused path with the product, harmonic or key-only score
  // merges layers, and never with scores_in / scores_out.
  int layers;
  const float* skey_l[kMaxSelectLayers];
  const float* gamma_l[kMaxSelectLayers];
  uint32_t* keys_l[kMaxSelectLayers];
  int32_t* idx_l[kMaxSelectLayers];
};

struct GatherParams {
  int64_t off[kMaxBatch + 1];
  int batch;
  int n_heads_kv;
  int head_dim;
  int64_t n_total;
  int64_t cap;
  float qmax;
  int bits;           // 8: int8 codes; 4: two codes per byte
  const uint16_t* k;
  const uint16_t* v;
  const float* gamma;
  const int32_t* idx;
  uint16_t* kc;
  uint16_t* vc;
  int8_t* vqc;
  float* gammac;
};

// The literal normaliser: the guide's causal prefix folded into each guide
// row's context normaliser, in place.
struct PrefixParams {
  int64_t off[kMaxBatch + 1];  // token offsets (an empty document has no context term)
  const uint16_t* q;           // guide rows [batch * H_kv, rows, d] bf16
  const uint16_t* k_guide;     // guide keys [batch * H_kv, L_t, d] bf16
  float* lse;                  // [batch, H_kv, rows], read and rewritten
  int batch;
  int n_heads_kv;
  int rows;                    // M = G * L_t, row r = (g, j) with j = r mod L_t
  int guide_len;
  int head_dim;
  float sigma;                 // logit scale
};

// Launchers (return cudaError_t of the launch).
cudaError_t launch_vquant(const uint16_t* v, void* vq, float* gamma, int64_t rows, int head_dim,
                          float qmax, int bits, int num_sms, cudaStream_t s);
// Pass 1.  `dependent`: launched as a programmatic dependent of the previous
// layer's last kernel (a stack of layers in one call); it then waits for that
// kernel before its first store.
cudaError_t launch_lse(const CUtensorMap& tmk, const CUtensorMap& tmv, const CUtensorMap& tmq,
                       const LseParams& p, int head_dim, dim3 grid, size_t smem, bool dependent,
                       cudaStream_t s);
// Pass 2, one CTA per key range.  `dependent`: launch as a programmatic
// dependent of the previous kernel in the stream (only where that kernel and
// this one belong to one layer's sequence, whose inputs were written before
// its first kernel started); it waits for it before reading the normalisers.
// With p.gamma set (the caller's normalisers, at most 256 guide rows) it also
// forms the Eq. 2 scales from V (map tmv) and waits only before its first
// store.
cudaError_t launch_keyscore(const CUtensorMap& tmk, const CUtensorMap& tmv, const CUtensorMap& tmq,
                            const KeyScoreParams& p, int head_dim, dim3 grid, size_t smem,
                            bool dependent, cudaStream_t s);
// Pass 2 with the caller's normalisers and the Eq. 2 scales (p.gamma) in one
// kernel on CTA pairs (two-CTA clusters sharing each MMA); grid.x is twice the
// number of pairs.  The guide map has 128-row boxes (each CTA loads half of
// every job's rows).  `dependent`: it waits for the previous kernel only
// before its first store.
cudaError_t launch_keyscore_pair(const CUtensorMap& tmk, const CUtensorMap& tmv,
                                 const CUtensorMap& tmq, const KeyScoreParams& p, int head_dim,
                                 dim3 grid, size_t smem, bool dependent, cudaStream_t s);
// How many CTA pairs of the pair kernel for this head dim and guide block can
// be resident at once (0 when the device or the query refuses a two-CTA
// cluster of that size).
int keyscore_pair_max_clusters(int head_dim, int rows_mma, size_t smem);
// acc[i] += x[i] for i < n (16-byte aligned buffers): the key scores of a
// later block of guide rows added to the earlier blocks' sum.
cudaError_t launch_add(float* acc, const float* x, int64_t n, int num_sms, cudaStream_t s);
cudaError_t launch_select(const SelectParams& p, bool dependent, cudaStream_t s);
// How many layers of a problem with `units_per_layer` (document, head) units
// and documents of at most n_max tokens one selection launch can take with
// every cluster resident at once and every slice in shared memory (four-CTA
// clusters); 1 when merging layers would not fit (or the device is not asked:
// no GPU, or the query is refused).
int select_merge_layers(int units_per_layer, int64_t n_max);
cudaError_t launch_gather(const GatherParams& p, bool dependent, cudaStream_t s);
cudaError_t launch_prefix(const PrefixParams& p, bool dependent, cudaStream_t s);
cudaError_t launch_wait_selftest(int* status, uint64_t limit_ns, cudaStream_t s);

// Raises a kernel's dynamic shared-memory limit to the device maximum, once per
// (kernel slot, CUDA context); `slot` names the kernel in a small registry.
cudaError_t set_smem_once(const void* kernel, int slot);
// The current CUDA context's process-unique ID (cuCtxGetId; the device's
// primary context is bound first when none is current), 0 if unavailable.
// Caches of per-context state (kernel attributes, co-residency answers) are
// keyed by it.
unsigned long long context_key();

// Shared-memory layout sizes of the scoring kernels (host side).
size_t lse_smem_bytes(int head_dim, int rows_pad, int stages);
size_t keyscore_smem_bytes(int head_dim, int rows_pad, int stages, bool scales);
size_t keyscore_pair_smem_bytes(int head_dim, int rows_mma, int stages);

}  // namespace tp
