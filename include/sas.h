/*
 * sas.h -- C ABI of the GB300 (sm_103a) SAS attention forward library.
 *
 * SAS ("Simple Attention Sparsification", arXiv 2609.13141) is trainable
 * block-sparse attention for causal language models.  Keys and values are cut
 * into blocks of b = 64 tokens.  A selector scores the historical blocks of
 * every query, the scores become gates g = softmax(s) (Sec. 4.3), the Top-K
 * blocks are kept (Eq. selected_context) and attention runs over the query's
 * own block B_0 (causal, unit gate) plus the kept blocks, with log g added
 * to the logits of the kept blocks (Eq. ours_train; Alg. 1 step 4).  The
 * inference form (Alg. 2) drops the log g bias.
 *
 * Conventions shared by every entry point:
 *   - All tensor arguments are DEVICE pointers owned by the caller.  The
 *     library never frees them and keeps no reference after the call.
 *   - bf16 tensors are passed as void* and hold IEEE bfloat16 values.
 *   - Layouts are dense row-major with the shapes given; Q, K, V, O are
 *     [B, H, N, d] ("BHND").  Base pointers must be 16-byte aligned.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Calls are
 *     asynchronous on that stream; the library synchronises only inside
 *     sas_create / sas_destroy / sas_mlp_fwd's first use of a larger size /
 *     the sas_get_* readers.
 *   - A handle's device workspace (kept lists, tile union lists, the attention
 *     kernel's work counter, the MLP hidden activation) is reused by every
 *     call on it, so calls on one handle must not overlap on the GPU: issue
 *     them on one stream (or order the streams with events), and use one
 *     handle per concurrently running stream.
 *   - Arguments are checked before anything is launched; on an argument error
 *     nothing is written and the call returns SAS_ERR_INVALID_ARG or
 *     SAS_ERR_UNSUPPORTED.  sas_last_error(h) then describes the problem.
 *   - Every wait inside a kernel is bounded.  A wait that runs out sets a
 *     device status word (read with sas_get_device_status) and the kernel
 *     returns early; nothing traps.
 *   - There is no CPU fallback: without a usable sm_103a device, calls return
 *     SAS_ERR_CUDA.
 */
#ifndef SAS_H
#define SAS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    SAS_OK = 0,
    SAS_ERR_INVALID_ARG = 1,   /* null/misaligned pointer, bad size, bad enum   */
    SAS_ERR_UNSUPPORTED = 2,   /* valid but outside what the kernels implement  */
    SAS_ERR_CUDA = 3,          /* a CUDA runtime/driver call failed             */
    SAS_ERR_TIMEOUT = 4,       /* a bounded in-kernel wait ran out              */
    SAS_ERR_OOM = 5            /* workspace allocation failed                   */
} sas_status;

/* Gate form of the historical blocks.
 *   TRAIN_SOFT : Eq. ours_train, logits of a kept block get + log g_m.
 *   INFER_HARD : Alg. 2, kept blocks enter unbiased (the forward of the hard
 *                Top-K gate, Sec. 4.2 "ranking preservation"). */
/*   TRAIN_HARD_STE : the hard Top-K gate trained through the straight-through
 *                estimator (Sec. 4.2 "ranking preservation", App. D, Eq.
 *                rank_unbounded): the forward is that of INFER_HARD; the
 *                backward adds the gate gradient of every historical block,
 *                kept or dropped, with the soft gates g = softmax(s) standing in
 *                for the hard ones (see sas_attention_bwd).  Sparse scope,
 *                softmax gates in the inner position. */
typedef enum { SAS_MODE_TRAIN_SOFT = 0, SAS_MODE_INFER_HARD = 1, SAS_MODE_TRAIN_HARD_STE = 2 } sas_mode;

/* Where the selector scores s come from (Alg. 1 step 1).
 *   SCORES_GIVEN  : the caller passes s as a [B, H, N, C] fp32 table.
 *   MEANPOOL_PROJ : s_im = bf16(Wq q_i) . bf16(Wk mean(K_Bm)) / sqrt(d_sel),
 *                   a mean-pooled block-summary selector (the paper relies on
 *                   pooled block summaries, App. B, and a gate-query projection
 *                   dotted against them, Sec. 6.3; its exact AttnGate is not
 *                   described, this is the library's reading). */
typedef enum { SAS_SEL_SCORES_GIVEN = 0, SAS_SEL_MEANPOOL_PROJ = 1 } sas_selector;

/* Gate activation phi of Eq. general_gate, g = phi(s) over the row's
 * historical blocks (Sec. 4.2 "gate activation"; the current block keeps
 * g_0 = 1).  Selection is the same for all three (Top-K of s).
 *   SOFTMAX : g = softmax(s) over the C_i historical blocks (the SAS form).
 *   SIGMOID : g = sigmoid(s), independent gates.
 *   LOGIT   : s itself is added to the logits, i.e. log g = s. */
typedef enum { SAS_GATE_SOFTMAX = 0, SAS_GATE_SIGMOID = 1, SAS_GATE_LOGIT = 2 } sas_gate_act;

/* Gate position (Sec. 4.2 "gate position"), TRAIN_SOFT mode only:
 *   INNER : o = softmax(q K^T + log g) V (Eq. ours_train, the SAS form).
 *   OUTER : o = softmax(q K^T) (g . V): the softmax runs over the plain
 *           logits and each kept block's value rows are scaled by its g;
 *           LSE is then that of the plain logits. */
typedef enum { SAS_GATE_INNER = 0, SAS_GATE_OUTER = 1 } sas_gate_pos;

/* Training scope (Sec. 4.2 "training scope"; Table 1 settings 9-11):
 *   SPARSE : only the Top-K historical blocks enter the attention (the SAS
 *            form, Eq. spa with the gates of Eq. ours_train).
 *   FULL   : no Top-K: every historical block of a row enters with its
 *            log-gate, softmax(q K^T + log g) V over the row's whole history
 *            (Eq. fula with the gates, setting 9).  Needs the softmax gate in
 *            the inner position and [B, H, N, d] inputs (max_seqs = 0); topk
 *            is not used; sel_idx / sel_logg must be NULL.
 *            With the learned selector the handle keeps a [B, Hkv, N, C]
 *            fp32 score table (the dense gate table the paper's kernel
 *            reads, App. E); with given scores the caller's table is read.
 * The stochastic approximation of the full scope (full*, setting 11) is the
 * sparse scope with noise added to the scores: sas_attention_fwd_noisy. */
typedef enum { SAS_SCOPE_SPARSE = 0, SAS_SCOPE_FULL = 1 } sas_scope;

typedef struct {
    int32_t B, H, N, d;   /* batch, heads, tokens (N <= 2^30), head dim (d in {64, 128}) */
    int32_t block;        /* block size b; must be 64 (Sec. 4.2.1 setup)             */
    int32_t topk;         /* K historical blocks kept per query, 0 <= K <= 64         */
    float sm_scale;       /* softmax scale on q.k; 0 selects 1/sqrt(d) (Alg. 3)       */
    int32_t mode;         /* sas_mode                                                 */
    int32_t selector;     /* sas_selector                                             */
    int32_t d_sel;        /* selector dim d_sel in {64, 128}; 0 selects d             */
    int32_t gate_act;     /* sas_gate_act (0 = SOFTMAX, the SAS default)               */
    int32_t gate_pos;     /* sas_gate_pos (0 = INNER, the SAS default)                 */
    int32_t Hkv;          /* KV heads (GQA); 0 selects H.  H must be a multiple of it:
                             query head h uses KV head h / (H / Hkv), and the G = H / Hkv
                             query heads of a group share one selection (Sec. 5.3;
                             Sec. 5 inference implementation): one score table
                             per group, given or from the learned selector's group
                             gate query.                                               */
    int32_t max_seqs;     /* 0: [B, H, N, d] batches of N-token sequences.  > 0: packed
                             variable-length sequences, at most max_seqs of them, in
                             [H, N, d] tensors whose token axis (N = capacity) holds
                             them back to back (sas_attention_fwd_varlen); needs B = 1. */
    int32_t max_seqlen;   /* packed mode: longest sequence (1 .. N; 0 selects N); the
                             score table has C = ceil(max_seqlen / 64) columns         */
    int32_t scope;        /* sas_scope (0 = SPARSE, the SAS default)                   */
} sas_config;

typedef struct sas_handle sas_handle;

/* Validates cfg, allocates the handle's device workspace (projected block
 * summaries, per-tile block lists, internal selection buffers) on the
 * current device and returns the handle in *out.  Synchronous. */
sas_status sas_create(const sas_config* cfg, sas_handle** out);

/* Frees the workspace.  Waits for the device first.  NULL is a no-op. */
void sas_destroy(sas_handle* h);

/* SAS training-mode forward of one attention layer: Alg. 1 steps 1-4
 * (selector scores, gates g = softmax(s), Top-K, gated sparse attention),
 * with the fused-kernel structure of Alg. 3 (skip blocks no query in a tile
 * keeps, online softmax, O and LSE outputs).
 *
 *   Q         bf16 [B, H, N, d]                                       (in)
 *   K, V      bf16 [B, Hkv, N, d] (Hkv = H without GQA)               (in)
 *   scores    fp32 [B, Hkv, N, C], C = ceil(N / 64); row i reads entries
 *             0 .. floor(i/64)-1 and ignores the rest.  Required for
 *             SCORES_GIVEN, must be NULL for MEANPOOL_PROJ.  Scores must
 *             be finite.                                              (in)
 *   Wq        bf16 [Hkv, d_sel, G d], G = H / Hkv: the gate-query
 *             projection of each KV group, applied to its G query heads'
 *             rows concatenated head by head, q~ = bf16(Wq [q_0; ...;
 *             q_{G-1}]) ([H, d_sel, d] without GQA);
 *   Wk        bf16 [Hkv, d_sel, d] key projection of the block summaries.
 *             Linear-layer layout [out, in]; required for MEANPOOL_PROJ,
 *             NULL otherwise.                                         (in)
 *   O         bf16 [B, H, N, d]                                       (out)
 *   LSE       fp32 [B, H, N] natural-log log-sum-exp of each row's
 *             gated logits (Alg. 3 output); may be NULL.              (out)
 *   sel_idx   int32 [B, Hkv, N, topk]: each row's kept historical blocks
 *             (per group) in ascending order, padded with -1; may be
 *             NULL.                                                   (out)
 *   sel_logg  fp32 [B, Hkv, N, topk]: log g of the kept blocks under the
 *             handle's gate activation (same order, 0 where padded);
 *             may be NULL.                                            (out)
 *
 * Top-K is exact-K: ties go to the lower block index; rows with at most K
 * historical blocks keep all of them. */
sas_status sas_attention_fwd(sas_handle* h,
                             const void* Q, const void* K, const void* V,
                             const float* scores,
                             const void* Wq, const void* Wk,
                             void* O, float* LSE,
                             int32_t* sel_idx, float* sel_logg,
                             void* stream);

/* full* training scope (Table 1 setting 11, Sec. 4.2: the full scope
 * approximated stochastically, the scores perturbed by noise before the gate
 * activation and the Top-K): sas_attention_fwd with s~ = s + noise in place of the scores
 * s, for the gate activation and for the Top-K alike.  The sum is formed in
 * fp32: s~ = fp32(s + noise) with s the given score or, for the learned
 * selector, fp32(q~ . K~ / sqrt(d_sel)).
 *   noise  fp32 [B, Hkv, N, C], C = ceil(N / 64), the same layout as given
 *          scores (entries m >= floor(i/64) are not read); finite.  DEVICE.
 * Sparse-scope handles of [B, H, N, d] inputs only; other arguments as in
 * sas_attention_fwd.  sel_logg reports log g of the noisy scores. */
sas_status sas_attention_fwd_noisy(sas_handle* h,
                                   const void* Q, const void* K, const void* V,
                                   const float* scores,
                                   const void* Wq, const void* Wk,
                                   const float* noise,
                                   void* O, float* LSE,
                                   int32_t* sel_idx, float* sel_logg,
                                   void* stream);

/* Backward of sas_attention_fwd (Alg. 4 of App. E; gate and score gradients
 * of App. D), for d = 128, any gate activation and position, any mode.  In
 * the outer position (o = softmax(z) (g . V)) dV takes P g dO, dS = P (g dP -
 * Delta), and a block's dlogg is the row sum of P g dP.
 * The kept sets are those of the forward (the Top-K choice is a constant of
 * the backward), and the per-tile block lists are read from the handle: call
 * it after the sas_attention_fwd of the same inputs on this handle, with no
 * other forward in between.  With grouped-query attention (Hkv < H) a
 * group's K, V, kept sets and gates serve its H / Hkv query heads, so dK, dV
 * and the gate gradients are sums over those heads (Sec. 3.3).  After a
 * forward on head-packed tiles (see sas_get_attention_work) the backward runs
 * on the same tiles, batched or packed, when a sequence holds at most
 * 2047 - G of them (G (N + 127) / 128 with N the longest sequence); else on
 * tiles of one query head.  The gradients are the same either way, up to the
 * order of floating-point sums.
 *
 * Full training scope (a SAS_SCOPE_FULL handle; Sec. 4.2, Eq. scope_grad):
 * every historical block of a row is kept and gated, so dlogg holds one
 * entry per historical block ([B, Hkv, N, C], entry m for block m) and the
 * score gradient is ds = dlogg - g sum(dlogg) over the whole history.  With
 * given scores, `scores` is required (the log-gates s - LSE are rebuilt from
 * it); with the learned selector the handle's score table is used.
 *
 * Hard Top-K gate under the straight-through estimator (a
 * SAS_MODE_TRAIN_HARD_STE handle, given scores, [B, H, N, d] inputs): dQ, dK
 * and dV are those of the hard forward (kept blocks unbiased, the rest
 * dropped); the gate gradient covers every historical block, dropped ones
 * included, each weighted by exp(z - LSE) under the hard forward's LSE (Eq.
 * rank_unbounded).  dlogg [B, Hkv, N, C] holds x_m = g_m dL/dg^_m for block m
 * (g = softmax(s) over the row's history, g^ the estimator's gate), and
 * dscores = x - g sum(x) = g (dg^ - sum g dg^).  `scores` is required.
 * Both forms build per-row lists of every historical block ([B, Hkv, N, C]
 * int32 + fp32 of handle workspace, allocated by the first such call).
 *
 * Packed sequences (a handle created with max_seqs > 0): the backward of the
 * last sas_attention_fwd_varlen on the handle, whose tile table it reads;
 * the layouts drop B ([H, N, d], [Hkv, N, C], ...), every sequence is its
 * own problem (no gradient crosses sequences), and rows past cu[num_seqs]
 * of dQ, dK, dV, dlogg and dscores are not written.
 *
 *   Q, O       bf16 [B, H, N, d]; LSE fp32 [B, H, N]: the forward's      (in)
 *   K, V       bf16 [B, Hkv, N, d]                                       (in)
 *   dO         bf16 [B, H, N, d] gradient of the loss w.r.t. O          (in)
 *   sel_idx, sel_logg: the forward's outputs, or NULL if the forward
 *              was given NULL for them                                   (in)
 *   scores     fp32 [B, Hkv, N, C] given scores; needed for dscores and by
 *              the full scope and hard-STE forms                         (in)
 *   dQ         bf16 [B, H, N, d]; dK, dV bf16 [B, Hkv, N, d]             (out)
 *   dlogg      fp32 [B, Hkv, N, topk] dL/d(log g) of each kept block, in
 *              the order of sel_idx, summed over the group's query heads
 *              (0 where padded; all 0 in INFER_HARD mode); [B, Hkv, N, C]
 *              by block for the full scope and hard-STE; may be NULL     (out)
 *   dscores    fp32 [B, Hkv, N, C] dL/ds of the given scores, sparse scope:
 *              ds_m = dlogg_m [m kept] - g_m sum_kept dlogg, 0 past each
 *              row's history (sigmoid gates: dlogg_m (1 - g_m) [m kept];
 *              raw logits: dlogg_m [m kept]); SCORES_GIVEN handles only,
 *              else NULL.
 *              g_m = exp(s_m - LSE_i) takes the row's log-normaliser
 *              LSE_i = s_m - log g_m from its first kept entry, so the
 *              scores must be the ones the forward selected with     (out)
 * N (packed: max_seqlen) must not exceed 262016 (2047 tiles of 128 rows).  The first call
 * allocates the handle's backward workspace (synchronously); later calls are
 * asynchronous and can be captured in a CUDA graph when B * H * T * (T + 1)
 * * 512 bytes <= 8 GiB (T = ceil(N / 128)) and that much memory is free at the
 * first call.  Otherwise every call reads back how many blocks the forward's
 * tiles visit, to size a buffer, and so synchronises with its stream once. */
sas_status sas_attention_bwd(sas_handle* h,
                             const void* Q, const void* K, const void* V,
                             const float* scores,
                             const void* O, const float* LSE, const void* dO,
                             const int32_t* sel_idx, const float* sel_logg,
                             void* dQ, void* dK, void* dV,
                             float* dlogg, float* dscores,
                             void* stream);

/* Packed variable-length form of sas_attention_fwd, on a handle created
 * with max_seqs > 0.  Sequence s holds rows cu_seqlens[s] .. cu_seqlens[s+1]-1
 * of the token axis and is its own causal problem: its blocks of 64 tokens
 * start at its first row, and no row attends outside its sequence (with the
 * learned selector each sequence is scored against the summaries of its own
 * blocks).
 *
 *   cu_seqlens int32 [num_seqs + 1], DEVICE: cu[0] = 0, non-decreasing,
 *              every length <= max_seqlen, cu[num_seqs] <= N.  Checked on
 *              the device: offsets that break this set the device status
 *              word to SAS_ERR_INVALID_ARG and nothing is computed.     (in)
 *   num_seqs   1 .. max_seqs
 *   Q          bf16 [H, N, d]; K, V bf16 [Hkv, N, d]                     (in)
 *   scores     fp32 [Hkv, N, C], C = ceil(max_seqlen / 64); row cu[s] + t
 *              reads entries 0 .. floor(t/64)-1 (blocks of its sequence).
 *              SCORES_GIVEN; NULL for MEANPOOL_PROJ                        (in)
 *   Wq, Wk     the learned selector's projections as in sas_attention_fwd
 *              (MEANPOOL_PROJ); NULL with given scores                     (in)
 *   O          bf16 [H, N, d]; LSE fp32 [H, N] (may be NULL)            (out)
 *   sel_idx, sel_logg  [Hkv, N, topk] as in sas_attention_fwd, block
 *              indices counted within the row's sequence (may be NULL) (out)
 * Rows past cu[num_seqs] are not written.  Graph-capturable (no host
 * synchronisation). */
sas_status sas_attention_fwd_varlen(sas_handle* h, const int32_t* cu_seqlens, int32_t num_seqs,
                                    const void* Q, const void* K, const void* V, const float* scores,
                                    const void* Wq, const void* Wk,
                                    void* O, float* LSE, int32_t* sel_idx, float* sel_logg, void* stream);

/* Dense MLP sublayer Y = GELU(X W1^T + b1) W2^T + b2 with the exact (erf)
 * GELU.  SAS itself does not define or change the MLP; this is the plain
 * transformer MLP that completes a layer.
 *   X  bf16 [T, D]; W1 bf16 [F, D]; b1 bf16 [F] or NULL;
 *   W2 bf16 [D, F]; b2 bf16 [D] or NULL; Y bf16 [T, D].
 * D and F must be multiples of 64; T >= 1.  The hidden activation
 * GELU(X W1^T + b1) is kept as a bf16 [T, F] tensor in handle-owned
 * memory, allocated (synchronously) the first time a call needs more. */
sas_status sas_mlp_fwd(sas_handle* h,
                       const void* X, const void* W1, const void* b1,
                       const void* W2, const void* b2, void* Y,
                       int64_t T, int64_t D, int64_t F,
                       void* stream);

/* Handle-free variant of sas_mlp_fwd that allocates no device memory.
 * (The paper has no counterpart: this serves callers, not the method.)
 *
 * Who needs it: callers that cannot call cudaMalloc while they run the
 * layer -- code recording a CUDA graph on its stream, plug-ins whose host
 * framework owns all device memory, services that must keep a fixed device
 * footprint.  sas_mlp_fwd would allocate its hidden buffer through a handle;
 * this entry point instead keeps the bf16 hidden activation [T, F] in a fixed
 * array of SAS_MLP_NOALLOC_MAX_HIDDEN_BYTES (32 MiB) compiled into the
 * library, which every GPU that loads the library reserves until the process
 * exits.  It calls no allocator (neither CUDA's nor any library's).
 *
 * Arguments, layouts and result are those of sas_mlp_fwd (X, W1, b1, W2, b2,
 * Y are caller-owned device buffers).  T * F * 2 must not exceed
 * SAS_MLP_NOALLOC_MAX_HIDDEN_BYTES; larger sizes are rejected with
 * SAS_ERR_UNSUPPORTED before anything runs.
 *
 * The first call on each device looks the array's device address up with
 * cudaGetSymbolAddress (with that device current); make that first call
 * before any stream capture starts.  All calls on a device share the one
 * array, and it keeps whatever the last call left in it: two calls whose
 * work overlaps on the GPU (different streams without ordering between
 * them) race on it and may corrupt each other's results.  Calls ordered on
 * one stream are safe.
 *
 * The return value covers what the host can check before launching.  What
 * the kernels find while they run (a bounded wait that ran out, misaligned
 * shared memory: Y is then incomplete) is latched in a per-device status
 * word, read with sas_mlp_noalloc_get_device_status. */
#define SAS_MLP_NOALLOC_MAX_HIDDEN_BYTES (32u * 1024u * 1024u)
sas_status sas_mlp_fwd_noalloc(const void* X, const void* W1, const void* b1,
                               const void* W2, const void* b2, void* Y,
                               int64_t T, int64_t D, int64_t F,
                               void* stream);

/* Status word of sas_mlp_fwd_noalloc on the current device (there is no
 * handle to hold one).  Synchronises the device, then writes to *out_status
 * what the kernels of every earlier call recorded -- SAS_OK, SAS_ERR_TIMEOUT
 * (a bounded wait ran out) or SAS_ERR_CUDA (a kernel found its shared memory
 * not 1024-byte aligned) -- and clears it.  Allocates nothing.  Returns
 * SAS_ERR_CUDA if the synchronisation or the read fails. */
sas_status sas_mlp_noalloc_get_device_status(int32_t* out_status);

/* Static text for a status code. */
const char* sas_status_str(sas_status s);

/* Text of the last error recorded on this handle ("" if none). */
const char* sas_last_error(const sas_handle* h);

/* Reads and clears the device status word: SAS_OK, SAS_ERR_TIMEOUT (a
 * bounded wait ran out) or SAS_ERR_CUDA (a kernel found its shared memory
 * not 1024-byte aligned and returned without computing).  Synchronises the
 * device first. */
sas_status sas_get_device_status(sas_handle* h, int32_t* out_status);

/* Per-kernel timing with CUDA events recorded on the launch stream around
 * every kernel.  sas_set_timing(h, 1) starts recording (and clears earlier
 * records); sas_get_timings synchronises, then writes, for each kernel kind,
 * the number of launches and the summed milliseconds.  Kinds, in order:
 * 0 block summaries, 1 (unused: the selector's query projection runs inside
 * the selection kernel), 2 selection, 3 attention, 4 MLP up-projection +
 * GELU, 5 MLP down-projection, 6 attention backward (all its kernels).
 * n_kinds <= 7. */
#define SAS_NUM_KERNEL_KINDS 7
sas_status sas_set_timing(sas_handle* h, int32_t enable);
sas_status sas_get_timings(sas_handle* h, int64_t* launches, double* total_ms, int32_t n_kinds);

/* Total number of kernels this handle has launched since creation. */
int64_t sas_launch_count(const sas_handle* h);

/* Failure-path diagnostics: the budget, in SM clock cycles, of every bounded
 * wait in the main loops of the kernels this handle launches from now on
 * (0 restores the default of about 2 s).  A budget too short for the work
 * makes those waits give up: the kernels then record SAS_ERR_TIMEOUT in the
 * device status word and return early, leaving their outputs incomplete.
 * The waits that drain a kernel's own copies and tensor-core work before it
 * exits keep at least the default budget, so nothing is left in flight and
 * the context stays usable.  Not for production use. */
sas_status sas_set_wait_limit(sas_handle* h, int64_t cycles);

/* Copies the per-tile count of historical blocks the attention kernel
 * processes (the union of the kept blocks of the tile's 128 query rows,
 * excluding the tile's own two diagonal blocks) from the last forward:
 * out[B * Hkv * T], one per KV group and tile slot, T = ceil(N/128).  A
 * packed-sequence handle has T = ceil(N/128) + max_seqs slots per group, of
 * which the first sum_s ceil(n_s/128) hold the sequences' tiles (longest key
 * history first).  Synchronises. */
sas_status sas_get_tile_union_counts(sas_handle* h, int32_t* host_out, int64_t n);

/* The work of the last attention forward: *tiles 128-row tiles computed and
 * *tile_blocks (tile, 64-key block) products, each 4 * 128 * 64 * d FLOPs
 * over QK^T and PV whether or not every row of the tile keeps the block.
 * Tiles hold 128 rows of one query head, or with GQA (G >= 2, 128 a multiple
 * of 8 G, sparse scope) 128 / G tokens of each of the G query heads of a KV
 * group: those share one kept list per token, so a tile visits the union of
 * 128 / G tokens' kept blocks and its one diagonal block (head-packed tiles;
 * packed sequences: G such tiles per 128-row tile of a sequence, the last
 * ones possibly past its end and empty).  Synchronises. */
sas_status sas_get_attention_work(sas_handle* h, int64_t* tiles, int64_t* tile_blocks);

/* Failure-path self-test: launches one block that waits on an mbarrier that
 * nothing completes, with the library's bounded wait and a limit of
 * `limit_cycles` SM clock cycles, and returns in *host_status what the
 * device recorded (SAS_ERR_TIMEOUT expected).  Synchronises. */
sas_status sas_selftest_wait_timeout(int64_t limit_cycles, int32_t* host_status);

/* ===================================================================== decode
 *
 * SAS decode step (Alg. 2): one new token per sequence attends to its own
 * block B_0 plus the Top-K cached blocks chosen by the selector, without gate
 * bias.  Following the paper's inference implementation (Sec. 5), selection is
 * made once per query group: the G = Hq / Hkv query heads that share a KV head
 * share its kept blocks, and only those blocks' keys and values are read.
 *
 * Selector of a group (the library's reading; the paper does not describe
 * how a group forms its gate query):
 *   q~   = bf16(Wq_g [q_0; q_1; ...; q_{G-1}])   (the group's queries
 *          concatenated head by head, Wq_g of shape [d_sel, G*d]);
 *   K~_m = bf16(Wk_g mean(keys of block m))       (kept in a summary cache);
 *   s_m  = q~ . K~_m / sqrt(d_sel) for the C = floor((n-1)/64) historical
 *          blocks of a sequence of n tokens (the new token is position n-1).
 * With G = 1 this is the MEANPOOL_PROJ selector of sas_attention_fwd.
 * Top-K is exact-K with ties to the lower block; C <= K keeps every block.
 *
 * Paged cache (caller-owned device memory):
 *   K_cache, V_cache  bf16 [num_pages, Hkv, 64, d]: a page holds the 64 tokens
 *                     of one block for every KV head.
 *   block_table       int32 [B, max_blocks]: page of logical block m of
 *                     sequence b (entries of blocks a sequence has not reached
 *                     are never read).
 *   seq_lens          int32 [B]: tokens in the cache of each sequence AFTER
 *                     this step's token is added (1 <= n <= 64 * max_blocks).
 *   Ksum              bf16 [B, Hkv, max_blocks, d_sel]: block summaries K~_m
 *                     by logical block; entry m is valid once block m is full.
 * Lengths and page indices are read on the device, so a CUDA graph of a step
 * can be replayed while they change.  A length or page index out of range is
 * not read: that sequence is skipped and the device status word becomes
 * SAS_ERR_INVALID_ARG (see sas_decode_get_device_status). */

typedef struct {
    int32_t B;            /* sequences decoded together                               */
    int32_t Hq, Hkv;      /* query heads and KV heads; G = Hq / Hkv in {1, 2, 4, 8}     */
    int32_t d;            /* head dim, 64 or 128                                       */
    int32_t d_sel;        /* selector dim, 64 or 128; 0 selects d                      */
    int32_t block;        /* must be 64                                                */
    int32_t topk;         /* K kept blocks per group, 0 <= K <= 64                     */
    int32_t max_blocks;   /* block-table width: capacity of one sequence, <= 32768     */
    int32_t num_pages;    /* pages in K_cache / V_cache                                */
    float sm_scale;       /* scale on q.k; 0 selects 1/sqrt(d)                          */
    int32_t dense;        /* 1: attend to every cached block (no selector, no summaries:
                             the dense decode SAS is compared with)                      */
} sas_decode_config;

typedef struct sas_decode_handle sas_decode_handle;

/* Validates cfg and allocates the handle's workspace (gate queries, scores,
 * kept lists, split-attention partials, arrival counters, status word) on the
 * current device.  Synchronous. */
sas_status sas_decode_create(const sas_decode_config* cfg, sas_decode_handle** out);
void sas_decode_destroy(sas_decode_handle* h);

/* Fills the summary cache after a prefill: Ksum[b, g, m] = bf16(Wk[g] mean
 * of the 64 keys of block m) for every full block m < floor(seq_lens[b] / 64).
 *   K_cache    bf16 [num_pages, Hkv, 64, d]                           (in)
 *   block_table, seq_lens as above (here seq_lens counts cached tokens) (in)
 *   Wk         bf16 [Hkv, d_sel, d]                                   (in)
 *   Ksum       bf16 [B, Hkv, max_blocks, d_sel]                       (out) */
sas_status sas_decode_summarize(sas_decode_handle* h, const void* K_cache, const int32_t* block_table,
                                const int32_t* seq_lens, const void* Wk, void* Ksum, void* stream);

/* One decode step for every sequence of the batch (Alg. 2):
 *   1. appends k_new / v_new (bf16 [B, Hkv, d]; both NULL if the caller has
 *      already written position n-1 of the cache) at position n-1; when that
 *      position opens a new block (n-1 = 64c, c >= 1) the now full block c-1 is
 *      summarised into Ksum; computes each group's gate query from q;
 *   2. scores the C historical blocks of each group against Ksum and keeps
 *      the Top-K (ascending, written to sel_idx if given);
 *   3. attends every query head over its group's kept blocks plus the
 *      current block (positions 64c .. n-1).
 *   q        bf16 [B, Hq, d]; query head h belongs to KV head h / G   (in)
 *   Wq       bf16 [Hkv, d_sel, G*d]; Wk bf16 [Hkv, d_sel, d]          (in)
 *   Ksum     bf16 [B, Hkv, max_blocks, d_sel]                    (in/out)
 *   O        bf16 [B, Hq, d]                                         (out)
 *   LSE      fp32 [B, Hq] natural-log log-sum-exp of the logits, or NULL
 *   sel_idx  int32 [B, Hkv, topk] kept blocks, -1 padded, or NULL
 * In dense mode Wq, Wk and Ksum are not used (may be NULL) and sel_idx must be
 * NULL.  Three kernel launches, one per step above (two in dense mode), each
 * started early by programmatic dependent launch; no allocation, no
 * synchronisation, so the call can be captured in a CUDA graph. */
sas_status sas_decode_step(sas_decode_handle* h, const void* q, const void* k_new, const void* v_new,
                           void* K_cache, void* V_cache, const int32_t* block_table, const int32_t* seq_lens,
                           const void* Wq, const void* Wk, void* Ksum, void* O, float* LSE, int32_t* sel_idx,
                           void* stream);

/* Text of the last error recorded on this handle ("" if none). */
const char* sas_decode_last_error(const sas_decode_handle* h);

/* Reads and clears the handle's device status word (SAS_OK,
 * SAS_ERR_INVALID_ARG for an out-of-range length or page index,
 * SAS_ERR_TIMEOUT for a bounded wait that ran out).  Synchronises. */
sas_status sas_decode_get_device_status(sas_decode_handle* h, int32_t* out_status);

/* Event timing per kernel kind: sas_decode_set_timing(h, 1) starts recording
 * (clearing earlier records), (h, 0) stops and keeps them; sas_decode_get_timings
 * synchronises and sums launches and milliseconds per kind: 0 append + summary
 * + gate query, 1 scores + Top-K, 2 attention, 3 summary fill
 * (sas_decode_summarize).  n_kinds <= 4.  Steps recorded while a stream is
 * captured get external event nodes in the graph (which serialise the
 * kernels); each replay re-records them, and the timings then read the latest
 * replay. */
#define SAS_DECODE_NUM_KERNEL_KINDS 4
sas_status sas_decode_set_timing(sas_decode_handle* h, int32_t enable);
sas_status sas_decode_get_timings(sas_decode_handle* h, int64_t* launches, double* total_ms, int32_t n_kinds);

/* Kernels this handle has launched since creation. */
int64_t sas_decode_launch_count(const sas_decode_handle* h);

#ifdef __cplusplus
}
#endif

#endif /* SAS_H */
