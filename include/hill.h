/*
 * hill.h -- C ABI of libhill.so: GB300 (sm_103a) kernels for the per-decode-
 * step token-importance evaluation of HillInfer (arxiv 2602.18750).
 *
 * One decode step of one layer: score the current query against every cached
 * key (Eq. 1, Sec. 2.1), aggregate the scores per token over all query heads
 * (Sec. 4.1 column-sum of attention weights, or the raw inner product of
 * Sec. 4.4), optionally add them to a running per-token importance, select
 * the top-k tokens per sequence (Sec. 3.1, Sec. 4.2), and run the decode
 * attention over the selected tokens only (Sec. 4.1, workflow step 6).
 *
 * Conventions shared by every call
 * --------------------------------
 * - All tensor pointers are DEVICE pointers owned by the caller; the library
 *   never allocates, frees or retains them.  Scratch space comes from the
 *   caller's workspace `ws` (size from hill_workspace_bytes; 16-byte aligned;
 *   its contents need no initialisation and are not preserved between calls).
 * - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy default
 *   stream).  A returned HILL_OK means the work was enqueued.  Two calls that
 *   share a workspace must be ordered on the GPU (same stream).
 * - Kernels are launched as programmatic dependents of the previous kernel on
 *   the stream.  The first kernel of a call may read the call's inputs (q,
 *   the 16-bit K cache, lens, k) before its dependency wait, so those must be
 *   complete when the call is issued in stream order: work that writes them
 *   must not be a kernel that triggers its dependents early
 *   (griddepcontrol.launch_dependents) and writes them afterwards.  Ordinary
 *   kernels and copies satisfy this.  Outputs and workspace are written only
 *   after the wait.
 * - Host-side validation failures return immediately and launch nothing.
 *   Launch failures return HILL_ERR_CUDA.  Conditions only visible on the
 *   device (a budget larger than max_k, a selected index outside the cache, a
 *   copy that never completed) set a device error word; hill_sync_status()
 *   reports and clears it.  No kernel traps or spins without a bound.
 * - Layouts (element strides, the head dimension contiguous):
 *     q        [B][H][d]          strides q_sb, q_sh
 *     k_cache  [B][Hkv][cap][d]   strides k_sb, k_sh, k_sn
 *     v_cache  [B][Hkv][cap][d]   strides v_sb, v_sh, v_sn
 *     lens, k, count  [B] int32;  scores, accum  [B][cap] float32 (row = cap);
 *     idx      [B][max_k] int32;  out  [B][H][d] float32, contiguous.
 *   Every stride must be a multiple of 8 elements and q/k/v 16-byte aligned.
 *   Query head h reads KV head h / (H / Hkv) (contiguous grouping).
 * - lens[b] counts the cached tokens of sequence b including the token
 *   generated this step (the caller appends its K/V first); it is clamped to
 *   [0, cap] on the device.  Entries of scores/accum at j >= lens[b] are not
 *   touched.  k[b] is clamped to [0, lens[b]].
 * - Supported: head_dim 128; any H and Hkv with H a multiple of Hkv (MHA,
 *   GQA with any group size G = H / Hkv, MQA); B <= 512; fp16 or bf16 q/K/V.
 *   Groups of more than 8 query heads are scored in passes of at most 8 over
 *   the same keys, except with at most 4 KV heads (MQA-like), where one pass
 *   scores up to 32 query heads of each KV head from every key tile; the
 *   attention takes up to 16 query heads per pass over the gathered rows.
 *   More than 32 KV heads are scored in passes of at most 32 (e.g. 40 KV
 *   heads: two passes of 20), each pass streaming only its own heads' keys.
 */
#ifndef HILL_H_
#define HILL_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  HILL_OK = 0,
  HILL_ERR_INVALID_ARG = 1,  /* bad pointer, size, stride or alignment       */
  HILL_ERR_UNSUPPORTED = 2,  /* valid but not built (head_dim, group size)    */
  HILL_ERR_WORKSPACE = 3,    /* ws NULL or smaller than hill_workspace_bytes */
  HILL_ERR_CUDA = 4,         /* a CUDA runtime call or launch failed          */
  HILL_ERR_TIMEOUT = 5,      /* a bounded device wait expired (device word)   */
  HILL_ERR_DEVICE = 6        /* a device-side argument check fired (device word) */
} hill_status;

typedef enum { HILL_F16 = 0, HILL_BF16 = 1 } hill_dtype;

/* Importance rule.  ATTN (the paper's definition, Sec. 4.1): per (b, h) the
 * softmax of z = q.K/sqrt(d) over j < lens[b], summed over all H query heads.
 * RAW (Sec. 4.4 "Algorithmic Simplification"): the sum over heads of z itself
 * (no softmax); the 1/sqrt(d) scale is kept. */
typedef enum { HILL_SCORE_ATTN = 0, HILL_SCORE_RAW = 1 } hill_score_mode;

typedef struct {
  int32_t batch;         /* B  >= 0                                   */
  int32_t num_q_heads;   /* H  >= 1                                   */
  int32_t num_kv_heads;  /* Hkv >= 1, H % Hkv == 0                    */
  int32_t head_dim;      /* d (128)                                   */
  int32_t capacity;      /* cap: allocated tokens per (b, kv head)    */
  int32_t dtype;         /* hill_dtype of q, K and V                  */
  int64_t q_sb, q_sh;             /* element strides of q             */
  int64_t k_sb, k_sh, k_sn;       /* element strides of k_cache       */
  int64_t v_sb, v_sh, v_sn;       /* element strides of v_cache       */
} hill_desc;

/* Bytes of workspace that any call below needs for this descriptor, mode and
 * index width (the maximum over the four calls).  Returns 0 for an invalid
 * descriptor.  Queries the current device's SM count. */
size_t hill_workspace_bytes(const hill_desc* desc, hill_score_mode mode, int32_t max_k);

/* Per-token importance (Eq. 1 with Sec. 4.1 or Sec. 4.4):
 *   ATTN: scores[b][j] = sum_h softmax_{j'<lens[b]}(q_h . K_{g(h),j'} / sqrt(d))[j]
 *   RAW : scores[b][j] = sum_h q_h . K_{g(h),j} / sqrt(d)
 * for j < lens[b].  If accum != NULL it is also updated: accum[b][j] +=
 * scores[b][j] (running importance across decode steps; a newly appended
 * token must hold 0 in accum before its first step).  scores is required. */
hill_status hill_score(const hill_desc* desc, const void* q, const void* k_cache,
                       const int32_t* lens, hill_score_mode mode, float* scores,
                       float* accum, void* ws, size_t ws_bytes, void* stream);

/* Top-k selection (Sec. 3.1 top-alpha retention, Sec. 4.2 global top-alpha):
 * for each b, the first n_b = min(k[b], lens[b]) tokens j < lens[b] in the
 * order (scores[b][j] descending, j ascending) -- a lower index wins a tie --
 * written to idx[b][0..n_b) in ascending index order, idx[b][n_b..max_k) =
 * -1, count[b] = n_b.  If n_b > max_k, count[b] = max_k and the device error
 * word records HILL_ERR_DEVICE.  -0.0 ranks equal to +0.0; keys must be
 * finite. */
hill_status hill_topk_select(const hill_desc* desc, const float* scores, const int32_t* lens,
                             const int32_t* k, int32_t max_k, int32_t* idx, int32_t* count,
                             void* ws, size_t ws_bytes, void* stream);

/* Decode attention over the selected tokens only (Sec. 4.1, workflow step 6; Eq. 1
 * restricted to the selected set, softmax renormalised over it):
 *   out[b][h][:] = sum_{t<count[b]} p_t V[b][g(h)][idx[b][t]][:],
 *   p = softmax_t(q_h . K[b][g(h)][idx[b][t]] / sqrt(d)).
 * count[b] == 0 gives zeros.  count[b] is clamped to [0, max_k]; an index
 * outside [0, cap) is skipped and recorded as HILL_ERR_DEVICE. */
hill_status hill_gather_sparse_attn(const hill_desc* desc, const void* q, const void* k_cache,
                                    const void* v_cache, const int32_t* idx, const int32_t* count,
                                    int32_t max_k, float* out, void* ws, size_t ws_bytes,
                                    void* stream);

/* The whole step for one layer, in the order of the evaluation workflow of
 * Sec. 4.1 (steps 4-6: score the cached keys against the current query,
 * keep the top-alpha critical tokens, attend over those only): hill_score,
 * then hill_topk_select on accum (if given) else on this step's scores, then
 * (if out != NULL) hill_gather_sparse_attn over the selection.  scores may be
 * NULL (then the step's scores live in the workspace).  Results equal those
 * of the three separate calls. */
hill_status hill_evict_step(const hill_desc* desc, const void* q, const void* k_cache,
                            const void* v_cache, const int32_t* lens, const int32_t* k,
                            int32_t max_k, hill_score_mode mode, float* accum, float* scores,
                            int32_t* idx, int32_t* count, float* out, void* ws,
                            size_t ws_bytes, void* stream);

/* BKP bookkeeping (Sec. 4.2, Bidirectional KV Cache Pools), applied to the
 * kept set of one HBM tier.  Two metrics decide which tokens stay:
 *  - temporal-aware pinning: the W = min(recent, lens[b]) most recent tokens
 *    [lens[b] - W, lens[b]) are always kept;
 *  - the older tokens [0, lens[b] - W) are ranked as in hill_topk_select and
 *    the first min(k[b], lens[b] - W) of them are kept;
 *  - frequency-aware tracking: hits (nullable, [B][cap] uint16, caller-
 *    owned and persistent across steps; the paper's 2-byte-per-token hit-rate
 *    table) gains +1, saturating at 65535, at every kept token.
 * idx[b] lists the kept tokens in ascending order (the window last), count[b]
 * = kept tokens.  If the window plus the ranked tokens exceed max_k, the
 * window keeps its max_k most recent tokens, the ranked part gets what is
 * left, and HILL_ERR_DEVICE is recorded.  recent < 0 is HILL_ERR_INVALID_ARG;
 * recent = 0 with hits = NULL is exactly hill_topk_select. */
hill_status hill_topk_select_bkp(const hill_desc* desc, const float* scores, const int32_t* lens,
                                 const int32_t* k, int32_t recent, int32_t max_k, int32_t* idx,
                                 int32_t* count, uint16_t* hits, void* ws, size_t ws_bytes,
                                 void* stream);

/* hill_evict_step with the BKP selection of hill_topk_select_bkp in place of
 * the plain top-k (same other arguments; recent = 0 with hits = NULL is
 * exactly hill_evict_step). */
hill_status hill_evict_step_bkp(const hill_desc* desc, const void* q, const void* k_cache,
                                const void* v_cache, const int32_t* lens, const int32_t* k,
                                int32_t recent, int32_t max_k, hill_score_mode mode, float* accum,
                                float* scores, int32_t* idx, int32_t* count, uint16_t* hits, float* out,
                                void* ws, size_t ws_bytes, void* stream);

/* The same step in two calls, for the layer-pipelined evaluation of Sec. 4.3
 * (the evaluation of layer i + 1 overlaps the rest of layer i): while the
 * normalisation and selection of one layer run on a second stream, the K
 * stream of the next layer proceeds on the first.
 *
 * hill_evict_step_begin launches the scoring kernel: it streams the K cache
 * once and writes, in ATTN mode, the logits and per-CTA softmax partials into
 * the workspace, in RAW mode the per-token sums into scores (and accum +=).
 * It reads q, k_cache and lens.
 *
 * hill_evict_step_end completes the step from the workspace: in ATTN mode the
 * normalisation (scores, accum += as in hill_score), then the top-k selection
 * of hill_topk_select_bkp (recent = 0 and hits = NULL: exactly
 * hill_topk_select) on accum if given, else on this step's scores.  It reads
 * no keys.  Its kernels run beside a scoring kernel of another layer: the
 * normalisation's finalize fits next to a scoring CTA on one SM, and the
 * selection uses the SMs the scoring grid of begin leaves free.
 *
 * Both calls of one step take the same desc, lens, max_k, mode, accum,
 * scores and ws (sized by hill_workspace_bytes); end may be issued on another
 * stream than begin, after an event recorded behind begin.  The workspace
 * belongs to the step from begin until end has completed: a pipeline over
 * layers rotates n >= 2 workspaces and issues begin of layer l + n only after
 * end of layer l.  One workspace per layer leaves the K stream without any
 * wait inside a decode step (fastest); two or three bound the memory.  The
 * scoring kernel of begin takes 17/20 of the SMs, so that end's kernels have
 * room beside it.  Results equal those of
 * hill_evict_step_bkp without attention, the ATTN scores within rounding (the
 * smaller scoring grid and the two-kernel normalisation combine the softmax
 * partials in another order); the selection follows the same rule on the
 * step's own scores.  Attention: hill_gather_sparse_attn on idx and count
 * afterwards. */
hill_status hill_evict_step_begin(const hill_desc* desc, const void* q, const void* k_cache,
                                  const int32_t* lens, int32_t max_k, hill_score_mode mode, float* accum,
                                  float* scores, void* ws, size_t ws_bytes, void* stream);
/* hill_evict_step_begin with the keys scored from their E4M3 shadow (k8,
 * kscale as in hill_score_f8 below): the split form of hill_evict_step_f8's
 * evaluation, completed by hill_evict_step_end in the same way. */
hill_status hill_evict_step_begin_f8(const hill_desc* desc, const void* q, const uint8_t* k8, const float* kscale,
                                     const int32_t* lens, int32_t max_k, hill_score_mode mode, float* accum,
                                     float* scores, void* ws, size_t ws_bytes, void* stream);
hill_status hill_evict_step_end(const hill_desc* desc, const int32_t* lens, const int32_t* k, int32_t recent,
                                int32_t max_k, hill_score_mode mode, float* accum, float* scores,
                                int32_t* idx, int32_t* count, uint16_t* hits, void* ws, size_t ws_bytes,
                                void* stream);

/* Per-KV-head selection (a variant of the evaluation: the paper evaluates at
 * token level for every head topology, Sec. 5.3; here each KV head keeps its
 * own set).  The importance is aggregated over the G query heads of each KV
 * head only,
 *   ATTN: s[b][g][j] = sum_{h in group g} softmax_{j'<lens[b]}(z[b,h,j'])[j]
 *   RAW : s[b][g][j] = sum_{h in group g} z[b,h,j],
 * written to scores [B][Hkv][cap] (caller-owned, required unless accum
 * [B][Hkv][cap] is given; then accum += s and the ranking uses accum).  The
 * top min(k[b], lens[b]) tokens of every (b, g) go to idx [B][Hkv][max_k]
 * (ascending, -1 padded) and count [B][Hkv], and if out != NULL the query
 * heads of KV head g attend over idx[b][g] only.  B * Hkv <= 512. */
hill_status hill_evict_step_kvh(const hill_desc* desc, const void* q, const void* k_cache,
                                const void* v_cache, const int32_t* lens, const int32_t* k, int32_t max_k,
                                hill_score_mode mode, float* accum, float* scores, int32_t* idx,
                                int32_t* count, float* out, void* ws, size_t ws_bytes, void* stream);

/* Asymmetric-precision scoring (Sec. 4.4, CEC): the evaluation ranks tokens
 * with low-precision inner products, while the attention keeps the original
 * 16-bit keys and values.  On this GPU the low precision is OCP FP8 E4M3
 * (its tensor-core rate is ~14x that of INT8 here), one scale per key row:
 *   k8     [B][Hkv][cap][128] uint8 E4M3 codes, dense, 16-byte aligned;
 *   kscale [B][Hkv][cap32] float32, cap32 = cap rounded up to 32, dense.
 * A row's codes are e4m3(K_i * (448 / amax)) with amax = max_i |K_i| (float32
 * product, round to nearest even, saturating) and its scale is amax / 448.
 * The query is cast the same way per (b, h) inside the scoring kernel, and
 *   z8 = (sum_i e4m3(q)_i e4m3(K)_i) * s_q * s_k / sqrt(d)
 * replaces the logit of Eq. 1 in the importance (ATTN or RAW, as hill_score).
 *
 * hill_quantize_k writes the shadow of rows [row_begin[b], row_end[b]) of
 * every KV head (device arrays [B], clamped to [0, cap]); max_rows bounds
 * row_end - row_begin over b (e.g. 1 to add this step's token, cap to build
 * the whole shadow). */
hill_status hill_quantize_k(const hill_desc* desc, const void* k_cache, const int32_t* row_begin,
                            const int32_t* row_end, int32_t max_rows, uint8_t* k8, float* kscale,
                            void* stream);

/* hill_score on the E4M3 shadow (same outputs and workspace as hill_score). */
hill_status hill_score_f8(const hill_desc* desc, const void* q, const uint8_t* k8, const float* kscale,
                          const int32_t* lens, hill_score_mode mode, float* scores, float* accum,
                          void* ws, size_t ws_bytes, void* stream);

/* hill_evict_step with the scoring on the E4M3 shadow; the sparse attention
 * (out != NULL) reads the original k_cache and v_cache.  k_cache and v_cache
 * may be NULL when out is NULL. */
hill_status hill_evict_step_f8(const hill_desc* desc, const void* q, const uint8_t* k8, const float* kscale,
                               const void* k_cache, const void* v_cache, const int32_t* lens,
                               const int32_t* k, int32_t max_k, hill_score_mode mode, float* accum,
                               float* scores, int32_t* idx, int32_t* count, float* out, void* ws,
                               size_t ws_bytes, void* stream);

/* Synchronises `stream`, then returns and clears the device error word of the
 * current device: HILL_ERR_TIMEOUT if a bounded wait expired, HILL_ERR_DEVICE
 * if a device-side argument check fired, HILL_ERR_CUDA if the synchronisation
 * itself failed, else HILL_OK. */
hill_status hill_sync_status(void* stream);

/* Static, human-readable name of a status. */
const char* hill_status_string(hill_status status);

/* Largest scratch, in bytes, that hill_score_noalloc may use: 16 MiB. */
#define HILL_SCORE_NOALLOC_MAX_SCRATCH (16u << 20)

/* hill_score for callers that cannot allocate device memory.  (The paper
 * has no counterpart; this is a deployment convenience.)  Some callers have
 * no way to obtain a workspace: a plug-in running inside a host application
 * that owns the whole device-memory budget and forbids its own cudaMalloc, a
 * latency-critical decode loop where an allocation could block or fail at an
 * unpredictable moment, or a binding from a language without a CUDA
 * allocator.  This entry point takes the same arguments as hill_score minus
 * the workspace and computes exactly what hill_score computes; its scratch is
 * a fixed HILL_SCORE_NOALLOC_MAX_SCRATCH-byte array built into the library,
 * which every GPU that loads the library holds until the process exits.
 *  - It allocates nothing: no cudaMalloc, cudaFree or allocating library call.
 *  - The first call on each device looks up that array's device address
 *    (cudaGetSymbolAddress, no allocation); make that first call on a device
 *    before any stream capture.
 *  - A call needing more scratch than the array holds returns
 *    HILL_ERR_WORKSPACE without launching anything.  ATTN mode needs
 *    4*B*H*cap bytes of logits, 8*B*H*P bytes of softmax partials and
 *    8*B*H bytes of statistics, each rounded up to 256 bytes; P = min(SMs,
 *    B * ceil(cap / 32)) * W partial slots, W = 8 / Hkv rounded down when
 *    Hkv <= 4 and H / Hkv >= 5, else 1 (SMs = the device's multiprocessor
 *    count).  RAW mode needs none.
 *  - All calls share the array, and it keeps whatever the last call left;
 *    no entry of it needs to start at zero (a call reads only what it wrote).
 *    Calls that overlap on the GPU (two streams, or two host threads without
 *    ordering) race on it: order them on one stream. */
hill_status hill_score_noalloc(const hill_desc* desc, const void* q, const void* k_cache,
                               const int32_t* lens, hill_score_mode mode, float* scores,
                               float* accum, void* stream);

/* Number of kernels this library has launched (or recorded into a CUDA graph
 * under stream capture) in this process so far, over all devices.  Lets a
 * caller count the kernels one call or one captured graph contains. */
uint64_t hill_kernel_launches(void);

/* Self-test of the bounded waits every kernel uses (no counterpart in the
 * paper): launches one warp that waits on a barrier nothing will complete,
 * for limit_us microseconds (1 .. 1e6), then gives up.  The wait expiring is
 * recorded like any other: the next hill_sync_status() returns
 * HILL_ERR_TIMEOUT, and the stream and context stay usable. */
hill_status hill_selftest_wait(uint32_t limit_us, void* stream);

/* ABI version of this header (major * 100 + minor). */
int32_t hill_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* HILL_H_ */
