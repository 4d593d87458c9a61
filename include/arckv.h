/*
 * arckv.h -- C ABI of the GB300 (sm_103a) ARC-KV per-context KV-cache
 * compaction library (libarckv.so).
 *
 * ARC-KV (arXiv 2609.36835) compacts, for every (layer, KV head) pair, a full
 * cache K, V in R^{T x d} into t entries (C_k, beta, C_v) such that the
 * compact operator
 *        O^(Q) = softmax(Q C_k^T + 1 beta^T) C_v           (Sec. 3.1, Eq. compact_attention)
 * approximates full attention softmax(Q K^T) V.  One call of arckv_compact
 * runs the four context-specific stages of Sec. 3.2 for all H_kv heads of one
 * layer:
 *   1. value-aware indexer scoring and top-t anchor selection
 *        (Sec. 3.3; App. A.1 Eqs. value_context, indexer_projection,
 *         pairwise_index_score; Sec. 3.3 Eq. indexer_pooling;
 *         App. A.6 Eq. persistent_support),
 *   2. response-profile assignment and convex-hull key merge
 *        (Sec. 3.4 Eqs. response_profile, anchor_assignment, mass_centroid,
 *         key_merge),
 *   3. attention-mass fit of beta (App. A.9 Eq. mass_fit),
 *   4. ridge fit of C_v (App. A.9 Eq. value_lstsq).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Pointers named in the signatures are DEVICE pointers on the current CUDA
 *   device, owned by the caller; the library allocates no device or host
 *   memory (apart from the fixed array inside libarckv.so that
 *   arckv_attend_static uses, described there).  Scratch space is the
 *   caller's workspace `ws` of at least the
 *   size returned by the matching *_workspace_bytes function, aligned to
 *   256 bytes.
 * - Arguments are checked on the host before anything is enqueued; a bad
 *   argument returns ARCKV_ERR_INVALID_ARG / ARCKV_ERR_SHAPE /
 *   ARCKV_ERR_WORKSPACE / ARCKV_ERR_UNSUPPORTED and enqueues nothing.
 * - All kernels are enqueued on `stream` in order, with one exception:
 *   arckv_compact's dual-form solves (t > n) run part of their kernels on a
 *   second stream that the library creates for each calling stream on its
 *   first such call (a non-blocking stream and two events, kept for the
 *   life of the process), forked from `stream` and joined back to it with
 *   events, so the call's work still begins after the work enqueued on
 *   `stream` before it and ends before the work enqueued after it.  These
 *   are the only resources the library creates itself.  Errors found on the
 *   device (a non-positive Cholesky pivot, a non-finite output) are recorded
 *   in a status word inside the workspace.  Without ARCKV_FLAG_NONBLOCKING
 *   the call synchronises `stream` and returns that status; with it the call
 *   returns ARCKV_OK after enqueueing and the status is read later with
 *   arckv_query_status (the call then performs no host synchronisation).
 * - Calls are reentrant as long as concurrent calls use distinct workspaces.
 * - bf16 means IEEE bfloat16 bit patterns (uint16); fp32 is IEEE binary32.
 * - All tensors are dense row-major with the listed shapes.
 */
#ifndef ARCKV_H_
#define ARCKV_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  ARCKV_OK = 0,
  ARCKV_ERR_INVALID_ARG = 1, /* null pointer, bad flag, bad scalar      */
  ARCKV_ERR_SHAPE = 2,       /* sizes out of range (e.g. t > T)         */
  ARCKV_ERR_WORKSPACE = 3,   /* workspace null, too small or misaligned */
  ARCKV_ERR_NOT_SPD = 4,     /* a fit's normal matrix lost definiteness */
  ARCKV_ERR_NONFINITE = 5,   /* NaN / Inf produced (or present in input)*/
  ARCKV_ERR_TIMEOUT = 6,     /* a bounded device wait gave up           */
  ARCKV_ERR_CUDA = 7,        /* a CUDA runtime call failed              */
  ARCKV_ERR_UNSUPPORTED = 8  /* valid but not implemented configuration */
} arckv_status;

/* Flags (arckv_config.flags). */
#define ARCKV_FLAG_NONBLOCKING 0x1u /* do not synchronise; see arckv_query_status */
#define ARCKV_FLAG_COMPACT_BF16 0x2u /* arckv_attend_joint: C_k, C_v are bf16, not fp32 */

/*
 * Problem description for one layer.  Sizes:
 *   H_kv  KV heads in the layer (>= 1)
 *   G     query heads per KV head (GQA group size, >= 1)
 *   T     cache length (>= 1)
 *   d     head dim (must be 128)
 *   n_pos reference positions; each KV head gets n = n_pos * G reference rows
 *   d_x   reference-activation width (multiple of 8)
 *   H_I   index heads (1..16), d_I index-head width (must be 128),
 *   d_A   value-attention width (must be 128)                       (App. A.1)
 *   t     anchor budget per head, 1 <= t <= T                       (Sec. 3.1)
 *   chunk_len  >= 0; 0 = one global top-t.  With chunk_len > 0 and T above
 *         10,000 the scores are cut into contiguous chunks of chunk_len (the
 *         last one shorter, at most 65535 chunks) and chunk c keeps its top
 *         t_c = clip_[1, T_c](round(t T_c / T)) positions, rounding exactly
 *         with halves to even; S is their union.  The realized anchor count
 *         t' = sum_c t_c (arckv_anchor_count) may differ slightly from t, and
 *         every [t] extent below is then t'.  Assignment, merge and fits stay
 *         global over the whole cache.                              (App. A.3)
 * Scalars:
 *   lambda_m  key-merging coefficient in [0, 1]                      (Eq. key_merge)
 *   logit_scale  factor on every model-attention logit q.k; the paper writes
 *             logits without the usual 1/sqrt(d) (Sec. 3.1), which callers
 *             pass here (0 selects 1/sqrt(d))
 *   ridge_w, ridge_v  >= 0: the beta and C_v normal matrices are solved as
 *             (Gram + lam I) with lam = ridge * trace(Gram) / t
 *   eps_w > 0, b_min <= b_max: the guards of Eq. mass_fit
 * Anchor scores: selector (below).
 */
typedef struct {
  int32_t H_kv, G, T, d, n_pos, d_x, H_I, d_I, d_A, t, chunk_len;
  float lambda_m, logit_scale, ridge_w, ridge_v, eps_w, b_min, b_max;
  uint32_t flags;
  int32_t selector;
} arckv_config;

/* arckv_config.selector: how anchors are scored before top-t.
 *   ARCKV_SELECTOR_INDEXER  the value-aware indexer (Sec. 3.3) -- ARC-KV
 *   ARCKV_SELECTOR_HA       highest attention: s_j = (mean_i p_ij^2)^(1/2),
 *                           p = softmax(logit_scale Q_ref K^T)          (App. B.1)
 *   ARCKV_SELECTOR_VI       value influence: s_j = (mean_i D_ij^2 / (||O_i||^2 + 1e-6))^(1/2),
 *                           D_ij = ||O_i - O_i^(-j)|| = p_ij / (1 - p_ij) ||v_j - O_i||,
 *                           O = p V; needs T >= 2                      (App. B.1)
 * HA and VI use no indexer weights and no X_ref (those pointers may be NULL);
 * the rest of the path (assignment, merge, fits) is unchanged. */
#define ARCKV_SELECTOR_INDEXER 0
#define ARCKV_SELECTOR_HA 1
#define ARCKV_SELECTOR_VI 2

/*
 * Frozen indexer parameters of the H_kv heads of one layer, bf16, stacked
 * over heads (App. A.1 Eqs. indexer_parameters, value_indexer_parameters):
 *   L_q, L_k, L_v [H_kv][H_I*d_I][d]     L_c [H_kv][H_I*d_I][d_A]
 *   L_x [H_kv][H_I][d_x]                 b_x [H_kv][H_I]
 *   U_q, U_k, U_v [H_kv][d_A][d]
 */
typedef struct {
  const void *L_q, *L_k, *L_x, *b_x, *U_q, *U_k, *U_v, *L_c, *L_v;
} arckv_indexer;

/* Number of timed stages reported through arckv_aux.stage_events. */
#define ARCKV_NUM_STAGES 11
/* Stage order: 0 indexer features (k_bar, value context, q_bar, w),
 * 1 index logits (one kernel), 2 row log-sum-exp, RMS pooling and top-t,
 * 3 reference attention (logits, row statistics, Y), 4 column statistics and
 * response profiles, 5 assignment (the argmax GEMM), 6 key merge, 7 the
 * products of the beta fit (compact logits, Phi_C, its Gram and right-hand
 * side), 8 the beta solve, 9 the products of the value fit, 10 the C_v solve.
 * With anchors_in, stages 0-2 are empty; with assign_in, stage 5 copies. */

/*
 * Optional inputs / outputs of arckv_compact (the pointer itself may be NULL;
 * every field may be NULL).
 *   scores     out fp32 [H_kv][T]  pooled indexer scores s (Eq. indexer_pooling)
 *   anchors    out int32 [H_kv][t] anchor positions S, ascending (t = t', above)
 *   assign     out int32 [H_kv][T] group index kappa(j) in [0, t)
 *   anchors_in in  int32 [H_kv][t] strictly ascending positions in [0, T):
 *              replaces indexer scoring and selection (the hard branch of
 *              Sec. 3.5 and stage-isolated testing); `scores` is then not written,
 *              and X_ref and the indexer weights are not read (they may be NULL)
 *   assign_in  in  int32 [H_kv][T] replaces the computed assignment; requires
 *              anchors_in and must satisfy assign_in[s_r] = r
 *   stage_events  cudaEvent_t[ARCKV_NUM_STAGES + 1] created by the caller; when
 *              non-NULL, event s is recorded on `stream` before stage s and the
 *              last one after the final stage
 *   launches   out: number of kernels this call enqueued
 */
typedef struct {
  float* scores;
  int32_t* anchors;
  int32_t* assign;
  const int32_t* anchors_in;
  const int32_t* assign_in;
  void* const* stage_events;
  int32_t* launches;
} arckv_aux;

/* Workspace bytes arckv_compact needs for `cfg` (0 if cfg is invalid).
 * Host-only; no CUDA call. */
size_t arckv_workspace_bytes(const arckv_config* cfg);

/* Realized anchors per head t' (App. A.3): t without chunking, else the sum
 * of the per-chunk budgets; 0 if cfg is invalid.  Host-only; no CUDA call.
 * C_k, beta, C_v, anchors and anchors_in have t' rows per head. */
int32_t arckv_anchor_count(const arckv_config* cfg);

/*
 * Compact one layer (all H_kv heads).
 *   K, V    bf16 [H_kv][T][d]         post-RoPE keys / values       (Sec. 3.1)
 *   Q_ref   bf16 [H_kv][n_pos][G][d]  reference queries; row i = r*G + g of a
 *                                     head pairs position r with query head g
 *   X_ref   bf16 [n_pos][d_x]         pre-query-projection activations, shared
 *                                     by the G rows of a position and by all
 *                                     heads of the layer           (App. A.1, A.5)
 *   idx     indexer weights (above)
 *   C_k     out fp32 [H_kv][t][d]     compact keys (row r <-> r-th anchor)
 *   beta    out fp32 [H_kv][t]        attention-mass bias
 *   C_v     out fp32 [H_kv][t][d]     compact values
 *   aux     optional (above)
 *   ws, ws_bytes  workspace
 *   stream  cudaStream_t (NULL = legacy default stream)
 */
arckv_status arckv_compact(const arckv_config* cfg, const void* K, const void* V,
                           const void* Q_ref, const void* X_ref, const arckv_indexer* idx,
                           float* C_k, float* beta, float* C_v, const arckv_aux* aux,
                           void* ws, size_t ws_bytes, void* stream);

/* Workspace bytes of arckv_attend (0 if the sizes are invalid). Host-only. */
size_t arckv_attend_workspace_bytes(int32_t H_kv, int32_t n, int32_t t, int32_t d);

/*
 * Attention against a compact cache (Sec. 3.1 Eq. compact_attention):
 *   O[h] = softmax(logit_scale * Q[h] C_k[h]^T + 1 beta[h]^T) C_v[h]
 *   Q bf16 [H_kv][n][d]; C_k, C_v fp32 [H_kv][t][d]; beta fp32 [H_kv][t];
 *   O out fp32 [H_kv][n][d].  n >= 1, 1 <= t, d == 128.
 * `flags` takes ARCKV_FLAG_NONBLOCKING.
 */
arckv_status arckv_attend(int32_t H_kv, int32_t n, int32_t t, int32_t d, float logit_scale,
                          const void* Q, const float* C_k, const float* beta, const float* C_v,
                          float* O, void* ws, size_t ws_bytes, uint32_t flags, void* stream);

/* Workspace bytes of arckv_attend_joint (0 if the sizes are invalid). Host-only. */
size_t arckv_attend_joint_workspace_bytes(int32_t H, int32_t n, int32_t t, int32_t F, int32_t d);

/*
 * Attention over a compact block followed by an uncompressed block (App. A.7
 * Eq. concatenated_attention_preservation):
 *   O[h] = softmax(logit_scale * Q[h] [C_k[h]; K_fixed[h]]^T + [beta[h]; 0_F]) [C_v[h]; V_fixed[h]]
 * for H independent heads (a decode batch folds into H: head = sequence x KV head).
 *   Q        bf16 [H][n][d]        n >= 1 query rows per head
 *   C_k, C_v [H][t][d] fp32, or bf16 with ARCKV_FLAG_COMPACT_BF16; beta fp32 [H][t]
 *   K_fixed, V_fixed  bf16 [H][F][d]  the uncompressed block (zero bias)
 *   O        out fp32 [H][n][d]
 * t >= 0, F >= 0, t + F >= 1, d == 128.  With t == 0 the compact arguments
 * may be NULL and the call is plain attention over K_fixed / V_fixed (the
 * full-cache baseline); with F == 0 it is the compact operator of
 * arckv_attend.  Every array pointer must be 16-byte aligned
 * (ARCKV_ERR_INVALID_ARG otherwise).  `flags` takes ARCKV_FLAG_NONBLOCKING
 * and ARCKV_FLAG_COMPACT_BF16; ws as for arckv_attend.
 */
arckv_status arckv_attend_joint(int32_t H, int32_t n, int32_t t, int32_t F, int32_t d, float logit_scale,
                                const void* Q, const void* C_k, const float* beta, const void* C_v,
                                const void* K_fixed, const void* V_fixed, float* O, void* ws, size_t ws_bytes,
                                uint32_t flags, void* stream);

/* Workspace bytes of arckv_truncated_error (0 if the sizes are invalid). Host-only. */
size_t arckv_truncated_error_workspace_bytes(int32_t H, int32_t n, int32_t T, int32_t t, int32_t d);

/*
 * Truncated-output error of anchor sets (App. B.1 Eq. background_truncated_error),
 * the held-out measure by which selectors are compared:
 *   p = softmax(logit_scale Q_eval[h] K[h]^T) over the full cache, O = p V,
 *   O~_i(S) = sum_{j in S[h]} p_ij v_j,
 *   E[h] = mean_i ||O_i - O~_i(S)|| / (||O_i|| + 1e-6)
 *   Q_eval bf16 [H][n][d]; K, V bf16 [H][T][d] (16-byte aligned);
 *   S int32 [H][t] distinct positions in [0, T) (t = 0: empty sets);
 *   E out fp32 [H].  d == 128.  `flags` takes ARCKV_FLAG_NONBLOCKING;
 *   out-of-range positions record ARCKV_ERR_INVALID_ARG (and are clamped).
 */
arckv_status arckv_truncated_error(int32_t H, int32_t n, int32_t T, int32_t t, int32_t d, float logit_scale,
                                   const void* Q_eval, const void* K, const void* V, const int32_t* S, float* E,
                                   void* ws, size_t ws_bytes, uint32_t flags, void* stream);

/*
 * Allocation-free compact attention.  The paper has no counterpart: this is a
 * deployment variant of arckv_attend for callers that cannot allocate device
 * memory when they call it -- for example an inference-engine plugin whose
 * execute step must not allocate, or a serving loop that has fixed its memory
 * budget up front and cannot risk an allocation failing or fragmenting memory
 * mid-request.  It computes exactly what arckv_attend computes, with the same
 * kernels, arguments (minus the workspace) and errors.
 *
 * Scratch: one fixed array of ARCKV_ATTEND_STATIC_MAX_FLOATS floats (32 MiB)
 * compiled into libarckv.so as a device global.  Every GPU on which the
 * library's device code is loaded holds it until the process exits.  A
 * problem needs arckv_attend_static_floats(H_kv, n, t, d) floats of it;
 * larger problems are rejected with ARCKV_ERR_WORKSPACE before anything is
 * enqueued.
 *
 * Set-up: the first call on a device (with that device current) looks up the
 * array's device address with cudaGetSymbolAddress and keeps it.  Under
 * CUDA's default lazy module loading that lookup is also when the driver
 * loads the module holding the array and so reserves its 32 MiB; with
 * CUDA_MODULE_LOADING=EAGER the reservation happens when the library is
 * loaded.  Make that first call during start-up -- before any stream capture
 * and before the phase in which nothing may allocate.  Every later call on
 * that device makes no allocation of any kind (no cudaMalloc, no cudaFree,
 * no allocating library routine).  If the device's primary context is reset
 * (cudaDeviceReset), the next call repeats the set-up in the new context.
 *
 * All calls share the one array and it keeps the previous call's contents
 * (each call clears what must start at zero): calls whose GPU work overlaps
 * -- on different streams, or from several host threads -- race on it, so
 * serialise them.  The call synchronises `stream` and returns the device
 * status.
 */
#define ARCKV_ATTEND_STATIC_MAX_FLOATS (8u << 20)
size_t arckv_attend_static_floats(int32_t H_kv, int32_t n, int32_t t, int32_t d);
arckv_status arckv_attend_static(int32_t H_kv, int32_t n, int32_t t, int32_t d, float logit_scale,
                                 const void* Q, const float* C_k, const float* beta, const float* C_v,
                                 float* O, void* stream);

/* Read (and clear) the device status word of a workspace after a
 * non-blocking call; synchronises `stream`. */
arckv_status arckv_query_status(void* ws, void* stream);

/* Diagnostic of the bounded device waits (the failure detection every
 * tensor-core kernel relies on): one CTA waits on an mbarrier that nothing
 * arrives on, with a wall-clock limit of limit_us microseconds (1 .. 10^6)
 * instead of the kernels' 2 s.  The wait gives up, records ARCKV_ERR_TIMEOUT
 * in the status word of `ws` (>= 256 bytes, 256-byte aligned) and the CTA
 * returns, so the call synchronises `stream` and returns ARCKV_ERR_TIMEOUT
 * with the CUDA context still usable.  ARCKV_ERR_INVALID_ARG for a limit out
 * of range, ARCKV_ERR_WORKSPACE for a missing or short workspace. */
arckv_status arckv_wait_probe(void* ws, size_t ws_bytes, uint32_t limit_us, void* stream);

/* Static description of a status code (never NULL). Host-only. */
const char* arckv_status_string(arckv_status s);

#ifdef __cplusplus
}
#endif
#endif /* ARCKV_H_ */
