/*
 * taskpress.h - C ABI of the TaskPress prefill-time KV-cache compression path
 * for GB300 (sm_103a).
 *
 * TaskPress (Sec. 3) keeps, for every KV head of a layer, the context tokens
 * that a short task guide attends to most (Eq. 1), weighted by each token's
 * per-token V quantisation scale (Eq. 2, Eq. 3), and evicts the rest with a
 * uniform per-head budget (Sec. 4, "Eviction").  This library runs that step
 * on one GPU: score, select, and compact the kept K/V into a reusable cache.
 *
 * Conventions shared by every call
 * --------------------------------
 *  - All tensor pointers are DEVICE pointers to contiguous row-major memory,
 *    owned by the caller.  The library allocates nothing (tp_guide_lse_static's
 *    fixed device array aside) and keeps no state between calls apart from
 *    small per-CUDA-context caches, each guarded by a mutex: kernel attributes
 *    already set, the device's answers to cluster co-residency queries, and
 *    that array's device address.  TMA descriptors are encoded on every call.
 *  - bf16 tensors are passed as `const void*` (IEEE bfloat16 bit patterns).
 *  - Shapes (d = head_dim, N = total tokens = doc_offsets[batch]):
 *        Q guide   [batch, H_q, L_t, d]   bf16, post-RoPE guide queries
 *        K, V      [H_kv, N, d]           bf16, documents packed along N
 *        gamma     [H_kv, N]              fp32 per-token V scale
 *        Vq        [H_kv, N, d*b/8]       Eq. 2 codes (see below)
 *        scores    [H_kv, N]              fp32 combined scores s_i
 *        idx       [batch, H_kv, cap]     int32, doc-local kept indices
 *        Kc, Vc    [batch, H_kv, cap, d]  bf16 compressed cache
 *        Vqc       [batch, H_kv, cap, d*b/8] Eq. 2 codes
 *        gammac    [batch, H_kv, cap]     fp32
 *    where cap = tp_kept_capacity(...).  Document b keeps k_b <= cap tokens;
 *    slots k_b..cap-1 of its rows are filled with idx = -1 and zero bytes.
 *  - Codes (b = quant_bits): b = 8, one int8 per value; b = 4 (the 4-bit KV
 *    of the paper's experiments, Sec. 4), two per byte, channel 2i in the
 *    low nibble and channel 2i+1 in the high nibble, each 4-bit two's
 *    complement.  Code buffers are 8-byte (b = 8) or 4-byte (b = 4) aligned.
 *  - Query head h belongs to KV head h / (H_q / H_kv) (contiguous groups).
 *  - Every call takes a cudaStream_t (passed as void*; NULL = legacy default
 *    stream), enqueues its kernels and returns without synchronising.
 *    Launch errors are reported through the return code; errors raised while
 *    the kernels run surface at the next synchronisation of the stream.
 *  - Return value: TP_OK (0) or a negative TP_ERR_* code; outputs are
 *    undefined after an error.
 *  - CUDA graphs: every call can be captured.  The first call of a problem
 *    shape on a device sets kernel attributes and asks the device how many
 *    thread-block clusters fit at once (the launch geometry depends on it);
 *    make one call of the shape outside the capture first.
 *  - Inputs must be finite.  NaN scores are ranked as 0 (never preferred).
 */
#ifndef TASKPRESS_H_
#define TASKPRESS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
#define TP_OK 0
#define TP_ERR_INVALID_ARG (-1)       /* null pointer, bad count, bad ratio     */
#define TP_ERR_WORKSPACE (-2)         /* workspace missing or too small          */
#define TP_ERR_UNSUPPORTED_SHAPE (-3) /* d not in {64,128}, even pool kernel, .. */
#define TP_ERR_CUDA (-4)              /* a CUDA runtime/driver call failed       */
#define TP_ERR_TIMEOUT (-5)           /* a device-side wait gave up (see below)  */

/* Flags (tp_problem.flags). */
#define TP_SCORE_KEY_ONLY 0x1u /* s_i = pooled key score only (Sec. 4.3.1 ablation) */
/* The other blends of the Sec. 4.4 aggregation ablation (at most one flag):
 *   TP_SCORE_NORM_ADD  s_i = s_key_i / ||s_key||_2 + gamma_i / ||gamma||_2, the
 *                      L2 norms taken over one document and KV head (a zero
 *                      norm drops its term);
 *   TP_SCORE_HARMONIC  s_i = 2 s_key_i gamma_i / (s_key_i + gamma_i), 0 where
 *                      the sum is 0 (the paper prints ',' for '+'). */
#define TP_SCORE_NORM_ADD 0x2u
#define TP_SCORE_HARMONIC 0x4u

/* Limits. */
#define TP_MAX_BATCH 256   /* documents per call                              */
#define TP_MAX_ROWS 512    /* stacked guide rows one scoring pass holds        */
#define TP_MAX_GUIDE_ROWS 8192 /* G * L_t stacked guide rows per KV head      */
/* A guide of more than TP_MAX_ROWS stacked rows (more than 512 / G tokens,
 * such as the 256- and 1024-token guides of the paper's TTFT study, Sec.
 * 4.2.3, at G = 4) is scored in blocks of TP_MAX_ROWS rows.  A row's
 * normaliser involves only that row, so each block runs both scoring passes on
 * its own rows (one more pass over K per block and pass; the Eq. 2 scales come
 * with the first block); the key scores, a sum over all rows (Eq. 1), are the
 * blocks' fp32 sums added in block order.  The fused entry points,
 * tp_guide_scores, tp_guide_lse and tp_guide_prefix_lse take such guides, and
 * their workspace grows by one fp32 normaliser per guide row, document and
 * head plus one fp32 key score per token and head.  tp_guide_key_scores and
 * tp_guide_lse_static, which take no workspace, return
 * TP_ERR_UNSUPPORTED_SHAPE for them, and every entry point does above
 * TP_MAX_GUIDE_ROWS rows. */

/*
 * One layer's compression problem.
 *   n_heads_q, n_heads_kv : H_q, H_kv (H_q a multiple of H_kv)
 *   head_dim              : d, 64 or 128
 *   guide_len             : L_t, the task guide's token count (Sec. 3.2)
 *   batch                 : number of documents packed along the token axis
 *   doc_offsets           : HOST pointer to batch+1 non-decreasing int64
 *                           offsets, doc_offsets[0] = 0; document b owns
 *                           tokens [doc_offsets[b], doc_offsets[b+1]).
 *   pool_kernel           : K of Eq. 1's average pooling; odd, 1..33 (default 5)
 *   quant_bits            : b of Eq. 2: 8 or 4
 *   softmax_scale         : logit scale; <= 0 means 1/sqrt(d)
 *   flags                 : 0 (Eq. 3 product), or one of TP_SCORE_KEY_ONLY,
 *                           TP_SCORE_NORM_ADD, TP_SCORE_HARMONIC
 */
typedef struct tp_problem {
  int32_t n_heads_q;
  int32_t n_heads_kv;
  int32_t head_dim;
  int32_t guide_len;
  int32_t batch;
  int32_t pool_kernel;
  int32_t quant_bits;
  float softmax_scale;
  uint32_t flags;
  const int64_t* doc_offsets;
} tp_problem;

/*
 * Tokens kept per head for a keep ratio (Sec. 4: the eviction ratio is the
 * pruned share, so keep = 1 - eviction).  Returns ceil(ratio*n - 1e-9*n)
 * clamped to [0, n] (the small offset keeps exact decimal products such as
 * 0.07*100 from rounding up), or -1 when n < 0 or the ratio is not in [0, 1].
 */
int64_t tp_budget(int64_t n, double keep_ratio);

/*
 * Capacity of the per-(document, head) output rows: max over documents of
 * k_b, where k_b = min(budget, n_b) when budget >= 0, else
 * tp_budget(n_b, keep_ratio).  Returns -1 on invalid arguments.
 */
int64_t tp_kept_capacity(const tp_problem* p, double keep_ratio, int64_t budget);

/*
 * Bytes of device workspace that tp_guide_scores, tp_select and
 * tp_compress_layer need for this problem (0 on invalid arguments).  The
 * workspace is caller-owned scratch, 256-byte aligned, with no required
 * contents; it must not be shared by calls that may overlap on the GPU.
 */
size_t tp_workspace_bytes(const tp_problem* p, double keep_ratio, int64_t budget);

/*
 * Workspace for tp_compress_layers / tp_compress_layers_lse over n_layers
 * layers (0 on invalid arguments).  For documents of at most 65536 tokens it
 * adds, for up to 7 further layers, room for one more layer's key scores,
 * scales and selection scratch (12 bytes per token and head each); otherwise,
 * and for one layer, it equals tp_workspace_bytes.  Given such a workspace the
 * stack calls select several consecutive layers in one launch, as many as the
 * workspace holds and as the device runs at once (one four-CTA cluster per
 * layer, document and head, all resident); the product, harmonic and
 * key-only scores only (the normalised-add score sums its norms over a
 * cluster, so it keeps one layer per launch).  The kept sets are the exact
 * top-k of the same scores either way, so results do not depend on the
 * grouping.  (A selection launch is bound by latency, not bandwidth: its
 * cluster barriers and distributed shared-memory round trips cost the same
 * for one layer as for several.)
 */
size_t tp_workspace_bytes_stack(const tp_problem* p, double keep_ratio, int64_t budget,
                                int n_layers);

/*
 * How many consecutive layers tp_compress_layers / tp_compress_layers_lse
 * select per launch for this problem, stack depth and workspace size (a
 * planning query: 1 when the workspace has no room for more, for documents
 * above 65536 tokens, for the normalised-add score, or where the device's
 * answer to the cluster co-residency query is not available); -1 on invalid
 * arguments.  Needs the device current, as the stack calls do.
 */
int tp_stack_layers_per_selection(const tp_problem* p, double keep_ratio, int64_t budget,
                                  int n_layers, size_t ws_bytes);

/*
 * Eq. 2 (Sec. 3.3) for every token of V: gamma_i = max_c |v_ic| / qmax with
 * qmax = 2^(b-1) - 1 (127 or 7; fp32, IEEE round-to-nearest division) and
 * codes q_ic = clamp(rint(v_ic / gamma_i), -qmax, qmax) (IEEE fp32 quotient,
 * round-half-even; gamma_i = 0 gives q_i = 0).  v: [H_kv, N, d] bf16 in;
 * vq: [H_kv, N, d*b/8] codes out, stored as described above (may be NULL to
 * compute gamma only); gamma: [H_kv, N] fp32 out.
 */
int tp_quantize_v(const tp_problem* p, const void* v, int8_t* vq, float* gamma, void* stream);

/*
 * The Eq. 2 rule for any rows of d bf16 values (for example the compacted K,
 * which makes the compressed cache fully quantised; the paper's experiments
 * store both K and V in 4 bits, Sec. 4): scale[r] = max_c |x_rc| / qmax and
 * codes clamp(rint(x_rc / scale[r]), -qmax, qmax) exactly as tp_quantize_v,
 * qmax = 2^(quant_bits-1) - 1.  x: [rows, d] bf16, 16-byte aligned;
 * xq: [rows, d*quant_bits/8] codes out (may be NULL); scale: [rows] fp32 out.
 * head_dim: 64 or 128; quant_bits: 8 or 4.  No problem description needed.
 */
int tp_quantize_rows(const void* x, int64_t rows, int head_dim, int quant_bits, void* xq,
                     float* scale, void* stream);

/*
 * Combined importance s_i of every context token (Sec. 3.2-3.4):
 *   A = softmax over the context of sigma * Q_guide K^T, per guide row
 *       (the guide-to-context block of the prefill attention map, Sec. 3.2),
 *   s_key_i = (1/K) sum_{k=-K/2..K/2} (1/G) sum_{rows r of the group} A[r, i+k]
 *       (Eq. 1; rows are the G*L_t guide rows of the KV head's query heads,
 *       terms outside the document are zero),
 *   s_i = s_key_i * gamma_i (Eq. 3), or s_key_i with TP_SCORE_KEY_ONLY, or
 *   the TP_SCORE_NORM_ADD / TP_SCORE_HARMONIC blend.
 * q: [batch, H_q, L_t, d] bf16; k: [H_kv, N, d] bf16; gamma: [H_kv, N] fp32
 * (may be NULL only with TP_SCORE_KEY_ONLY); scores: [H_kv, N] fp32 out.
 * ws / ws_bytes: workspace of at least tp_workspace_bytes(p, 0, 0).
 */
int tp_guide_scores(const tp_problem* p, const void* q, const void* k, const float* gamma,
                    float* scores, void* ws, size_t ws_bytes, void* stream);

/*
 * Stage 1 of the scores (Sec. 3.2): the softmax normaliser of every guide row,
 *   lse[b, h, r] = log sum_{i in document b} exp(sigma * q_r . k_i)
 * for the M = G*L_t stacked guide rows r of KV head h (rows ordered query
 * head-major within the group, then guide token).  q, k as in tp_guide_scores;
 * lse: [batch, H_kv, M] fp32 out (natural log).  Empty documents are skipped.
 * With v ([H_kv, N, d] bf16) and gamma ([H_kv, N] fp32 out) both non-NULL, the
 * same pass also writes the Eq. 2 scales of every token (as tp_quantize_v),
 * reading V alongside K; both NULL skips that.
 * ws / ws_bytes: workspace of at least tp_workspace_bytes(p, 0, 0).
 */
int tp_guide_lse(const tp_problem* p, const void* q, const void* k, const void* v, float* lse,
                 float* gamma, void* ws, size_t ws_bytes, void* stream);

/*
 * tp_guide_lse without a caller workspace.  The paper has no counterpart; this
 * entry point exists for callers that cannot allocate device memory: code
 * that runs inside a CUDA stream capture or a host framework's launch hook
 * where calling the allocator is not allowed, or plugins that are handed
 * only a stream and the tensors they must read and write.  Arguments and
 * results are those of tp_guide_lse; the scratch it needs (status word,
 * counters, partial sums) lives in a fixed 2 MiB device array inside the
 * library, which every GPU that loads the library keeps until exit.
 *  - Guides of more than TP_MAX_ROWS stacked rows return
 *    TP_ERR_UNSUPPORTED_SHAPE (their blocks need a workspace).
 *  - Problems whose pass-1 scratch exceeds 2 MiB are rejected with
 *    TP_ERR_WORKSPACE (typical shapes need well under 1 MiB: about
 *    8 bytes x number of SMs x guide rows, plus 4 bytes per document and head).
 *  - The first call in each CUDA context looks up that array's device address
 *    (cudaGetSymbolAddress) with the context current; make that first call
 *    before any stream capture.  The address is cached by the context's ID
 *    (cuCtxGetId), checked on every call: cudaDeviceReset or a second
 *    context on the same device gets its own copy of the array and its own
 *    lookup, and a reset context's address is never reused.
 *  - All calls share the one array: calls that may overlap on the GPU (other
 *    streams, other threads) race and must be serialised by the caller.
 *  - Nothing is allocated: no cudaMalloc, cudaFree or allocating library call.
 */
int tp_guide_lse_static(const tp_problem* p, const void* q, const void* k, const void* v,
                        float* lse, float* gamma, void* stream);

/*
 * Stage 2 of the scores (Sec. 3.2, Eq. 1's inner sums): given the row
 * normalisers `lse` ([batch, H_kv, M] fp32, natural log, e.g. from
 * tp_guide_lse or from the caller's own prefill attention), writes the
 * unpooled key score of every context token,
 *   key_scores[h, off_b + i] = (1/G) sum_r exp(sigma * q_r . k_i - lse[b, h, r]).
 * Needs no workspace.  key_scores: [H_kv, N] fp32 out.  Guides of more than
 * TP_MAX_ROWS stacked rows return TP_ERR_UNSUPPORTED_SHAPE (their blocks need
 * a workspace: use tp_guide_scores or a fused entry point).
 * With v ([H_kv, N, d] bf16) and gamma ([H_kv, N] fp32 out) both non-NULL, the
 * same kernel also writes the Eq. 2 scales of every token (as tp_quantize_v),
 * reading V alongside K (one CTA per key range up to 256 guide rows, two-CTA
 * clusters above; a separate V pass where those pairs would not all be
 * resident at once); both NULL skips that.
 */
int tp_guide_key_scores(const tp_problem* p, const void* q, const void* k, const void* v,
                        const float* lse, float* key_scores, float* gamma, void* stream);

/*
 * Top-budget selection per (document, KV head) (Sec. 3.4; Sec. 4 uniform
 * per-head budget): the k_b largest scores of each document's rows, equal
 * scores resolved towards the lower token index, -0 treated as +0, NaN as 0.
 * scores: [H_kv, N] fp32; idx: [batch, H_kv, cap] int32 out, doc-local,
 * strictly ascending in each row, then -1 padding.  keep_ratio / budget as in
 * tp_kept_capacity.  ws: tp_workspace_bytes(p, keep_ratio, budget) bytes.
 */
int tp_select(const tp_problem* p, const float* scores, double keep_ratio, int64_t budget,
              int32_t* idx, void* ws, size_t ws_bytes, void* stream);

/*
 * Order-preserving compaction of the kept tokens (Sec. 3.1: the compressed
 * cache of the selected index subset).  For every (document b, head h, slot t)
 * with j = idx[b,h,t] >= 0:  Kc = K[h, off_b + j], Vc = V[h, off_b + j],
 * Vqc = Eq. 2 codes of that V row with scale gamma[h, off_b + j],
 * gammac = gamma[h, off_b + j]; slots with idx = -1 are zero-filled.
 * Any of kc, vc, vqc, gammac may be NULL to skip that output.
 */
int tp_compact(const tp_problem* p, const void* k, const void* v, const float* gamma,
               const int32_t* idx, double keep_ratio, int64_t budget, void* kc, void* vc,
               int8_t* vqc, float* gammac, void* stream);

/*
 * The fused per-layer path: Eq. 2 scales, Eq. 1 / Eq. 3 scores, per-head
 * top-budget selection and compaction, all on `stream` with no host
 * synchronisation.  Outputs as in tp_select and tp_compact; `scores` and
 * `gamma` ([H_kv, N] fp32) are optional outputs (NULL to skip).
 * Kernels: the normalising pass (which also forms the Eq. 2 scales), the
 * key-score pass, the selection and the compaction (none when nothing is
 * kept), each a programmatic dependent of the one before;
 * tp_compress_kernel_count says how many kernels a call launches.
 */
int tp_compress_layer(const tp_problem* p, const void* q, const void* k, const void* v,
                      double keep_ratio, int64_t budget, int32_t* idx, void* kc, void* vc,
                      int8_t* vqc, float* gammac, float* scores, float* gamma, void* ws,
                      size_t ws_bytes, void* stream);

/*
 * tp_compress_layer with the caller's row normalisers: `lse` ([batch, H_kv, M]
 * fp32, natural log, rows ordered as in tp_guide_lse) replaces the normalising
 * pass, so the scores take one pass over K (Sec. 3.2).  The
 * method slices A out of the full prefill attention map; a caller that keeps
 * that attention's per-row log-sum-exp for the guide rows passes it here and
 * gets the paper's literal normaliser, which also counts the guide's own
 * causal prefix.  With lse from tp_guide_lse the result equals
 * tp_compress_layer's.  The same kernel forms the key scores and the Eq. 2
 * scales, so K and V are each read once: one CTA per key range for up to 256
 * guide rows, two-CTA clusters sharing each tensor-core MMA (each CTA holding
 * half of the guide block) above.  Where those pairs would not all be
 * resident at once (more than 76 (document, KV head) units of more than 256
 * rows on a 152-SM GPU) the scales come from a separate pass over V.
 * Other arguments, outputs and workspace as in tp_compress_layer.
 */
int tp_compress_layer_lse(const tp_problem* p, const void* q, const void* k, const void* v,
                          const float* lse, double keep_ratio, int64_t budget, int32_t* idx,
                          void* kc, void* vc, int8_t* vqc, float* gammac, float* scores,
                          float* gamma, void* ws, size_t ws_bytes, void* stream);

/*
 * The literal row normaliser (Sec. 3.2).  A is sliced out of the causal
 * prefill map over the context followed by the guide, so guide row
 * r = (g, j) (rows ordered as in tp_guide_lse, j = r mod L_t) is normalised
 * over every context key of its document and over the guide keys 0..j:
 *   lse[b, h, r] <- log( exp(lse[b, h, r]) + sum_{j' <= j} exp(sigma q_r . kg[b, h, j']) ).
 * Folds the guide-prefix term into `lse` in place ([batch, H_kv, M] fp32,
 * natural log, as tp_guide_lse writes it).  For an empty document the input
 * row is ignored and the output is the prefix term alone.
 * q: [batch, H_q, L_t, d] bf16; k_guide: [batch, H_kv, L_t, d] bf16, the
 * guide's post-RoPE keys from the same prefill (16-byte aligned, as q).
 * The arithmetic is fp32 (exact bf16 products, fp32 sums, expf / logf).
 */
int tp_guide_prefix_lse(const tp_problem* p, const void* q, const void* k_guide, float* lse,
                        void* stream);

/*
 * tp_compress_layer with the literal normaliser: between the two scoring
 * passes the guide prefix is folded into each row's normaliser as in
 * tp_guide_prefix_lse.  k_guide: [batch, H_kv, L_t, d] bf16 device pointer.
 * Other arguments, outputs and workspace as in tp_compress_layer.
 */
int tp_compress_layer_guide(const tp_problem* p, const void* q, const void* k, const void* v,
                            const void* k_guide, double keep_ratio, int64_t budget, int32_t* idx,
                            void* kc, void* vc, int8_t* vqc, float* gammac, float* scores,
                            float* gamma, void* ws, size_t ws_bytes, void* stream);

/*
 * A stack of n_layers layers of one problem in one call (the per-layer path of
 * tp_compress_layer, layer after layer, on `stream`).  q, k, v, idx, kc, vc,
 * vqc and gammac are HOST arrays of n_layers device pointers, each laid out as
 * in tp_compress_layer; kc, vc, vqc and gammac (the arrays, or entries of
 * them) may be NULL to skip that output.  The workspace is reset once for the
 * whole stack and layer l's first kernel is launched as a programmatic
 * dependent of layer l - 1's last one, so consecutive layers overlap at their
 * boundary.  Results equal n_layers calls of tp_compress_layer.  ws_bytes as
 * for tp_compress_layer (one layer's workspace serves the whole stack), or
 * tp_workspace_bytes_stack(p, keep_ratio, budget, n_layers) bytes, with which
 * short layers are selected several at a time (see there).
 */
int tp_compress_layers(const tp_problem* p, int n_layers, const void* const* q,
                       const void* const* k, const void* const* v, double keep_ratio,
                       int64_t budget, int32_t* const* idx, void* const* kc, void* const* vc,
                       int8_t* const* vqc, float* const* gammac, void* ws, size_t ws_bytes,
                       void* stream);

/*
 * A stack of n_layers layers with the caller's row normalisers (as
 * tp_compress_layer_lse, layer after layer, on `stream`); lse is a HOST array
 * of n_layers device pointers, each [batch, H_kv, M] fp32 (natural log).
 * Other arguments as in tp_compress_layers.  Each layer's scoring kernel is a
 * programmatic dependent of the kernel before it: it loads and scores at once
 * and waits for that kernel only before its first store.  Results equal
 * n_layers calls of tp_compress_layer_lse bit for bit.  ws_bytes as for
 * tp_compress_layers (tp_workspace_bytes or tp_workspace_bytes_stack).
 */
int tp_compress_layers_lse(const tp_problem* p, int n_layers, const void* const* q,
                           const void* const* k, const void* const* v, const float* const* lse,
                           double keep_ratio, int64_t budget, int32_t* const* idx, void* const* kc,
                           void* const* vc, int8_t* const* vqc, float* const* gammac, void* ws,
                           size_t ws_bytes, void* stream);

/*
 * How many kernels one fused call launches for this problem (mode 0:
 * tp_compress_layer, 1: tp_compress_layer_lse, 2: tp_compress_layer_guide;
 * tp_compress_layers launches mode 0's count per layer, tp_compress_layers_lse
 * mode 1's); -1 on invalid arguments.  A planning query: it launches nothing
 * (for mode 1 above 256 guide rows it asks the current device how many CTA
 * pairs can be resident; without a device it counts the separate V pass).
 */
int tp_compress_kernel_count(const tp_problem* p, double keep_ratio, int64_t budget, int mode);

/*
 * Synchronises `stream`, then reads the device status word that the kernels of
 * the last call on this workspace left.  Every device-side wait in the
 * kernels is bounded; one that gives up records TP_ERR_TIMEOUT there and the
 * kernel returns early (its outputs are then undefined).  Returns TP_OK,
 * TP_ERR_TIMEOUT, or TP_ERR_CUDA if the synchronisation itself failed.
 */
int tp_check_status(const void* ws, size_t ws_bytes, void* stream);

/*
 * Self-test of the failure path: one thread waits, through the same bounded
 * mbarrier wait every kernel uses, on a barrier that nothing arrives at.
 * After limit_ns (0 < limit_ns <= 1e9) it gives up, records TP_ERR_TIMEOUT in
 * the workspace status word (which this call first zeroes) and the kernel
 * returns normally; tp_check_status(ws, ...) then reports TP_ERR_TIMEOUT and
 * the context stays usable.  Nothing faults, traps or hangs.
 */
int tp_selftest_wait_timeout(void* ws, size_t ws_bytes, int64_t limit_ns, void* stream);

/* Human-readable name of a status code (static storage). */
const char* tp_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* TASKPRESS_H_ */
