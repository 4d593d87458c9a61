// Internal launchers of the ARC-KV stage kernels (host side).  Every launcher
// enqueues on `st` and returns the number of kernels it launched.
#pragma once
#include "common.cuh"

namespace arckv {

struct Dims {
  int H, G, T, d, n_pos, n, d_x, H_I, d_I, d_A, t, HD;
  int chunk;   // effective chunk length of the anchor selection (0: one global top-t)
};

// App. A.3 fixed chunking: with chunk length L > 0 and T_a = T above 10,000
// the scores are cut into contiguous chunks (the last one shorter) and chunk c
// keeps t_c = clip_[1, T_c](round(t T_c / T)) anchors, the rounding exact and
// half to even.  t is then the realized sum of the t_c.
constexpr int kChunkThreshold = 10000;
__host__ __device__ inline int chunk_budget(int T, int t, int Tc) {
  const long long num = (long long)t * Tc;
  long long q = num / T;
  const long long r = num % T;
  if (2 * r > T || (2 * r == T && (q & 1))) ++q;
  return (int)(q < 1 ? 1 : (q > Tc ? Tc : q));
}
// softmax(X) V products run fused (no probability triple in memory) when the
// fp32 logit rows can be tiled by TMA: T a multiple of 4
inline bool probs_fused(int T) { return (T & 3) == 0; }
inline int effective_chunk(int T, int chunk_len) { return (chunk_len > 0 && T > kChunkThreshold) ? chunk_len : 0; }
inline int realized_anchors(int T, int t, int chunk_len) {
  const int L = effective_chunk(T, chunk_len);
  if (L == 0) return t;
  int total = 0;
  for (int start = 0; start < T; start += L) total += chunk_budget(T, t, T - start < L ? T - start : L);
  return total;
}

constexpr int kSplitK = 8;   // grid slices per head some launches take (heads x slices ride in one grid dimension)

// Streaming multiprocessors of the current device (queried once per device).
int tc_gemm_sm_count();
// cudaFuncSetAttribute(kern, MaxDynamicSharedMemorySize, bytes), issued once
// per kernel and device (later calls with no larger size return at once).
cudaError_t set_dyn_smem(const void* kern, int bytes);
// Grid of a grid-stride kernel: enough CTAs for `count` elements at `per_cta`
// each, capped at `per_sm` resident CTAs on every SM of the device.
inline int stride_grid(long long count, int per_cta, int per_sm) {
  const long long want = (count + per_cta - 1) / per_cta;
  const long long cap = (long long)tc_gemm_sm_count() * per_sm;
  return (int)(want < 1 ? 1 : (want < cap ? want : cap));
}
constexpr int kCholNB = 64;  // Cholesky block size

// ---- indexer (Sec. 3.3, App. A.1) --------------------------------------
// k_bar = N(L_k k + L_v v) per d_I block, as a split-bf16 pair (one tcgen05
// GEMM over [K | V] against [L_k | L_v]).
int launch_query_proj_tc(const Dims& D, const bf16* Q, const bf16* L_q, const bf16* L_c, bf16* qcat, bf16* wcat,
                         bf16* qbar_hi, bf16* qbar_lo, DevStatus* stt, cudaStream_t st);
int launch_key_features_tc(const Dims& D, const bf16* K, const bf16* V, const bf16* L_k, const bf16* L_v,
                           bf16* kbar_hi, bf16* kbar_lo, DevStatus* stt, cudaStream_t st);
// Scratch of the query-side features.
struct QueryBufs {
  float *logits, *rshift, *rmul, *av;
  bf16 *q_h, *q_m, *q_l, *p_h, *p_m, *p_l;
  float2* part;        // per-(row, 128-column tile) softmax partials of the logits
  bf16 *qcat, *wcat;   // K-concatenated operands of the q_bar GEMM ([n][512], [HD][512])
  bf16 *vq3, *av3;     // bf16 triples of U_q q and A^V V (parts [H][n][128], one after another)
  bf16* ukt;           // U_k^T [H][d][d_A]
};
// value context c (Eq. value_context), q_bar (Eq. indexer_projection), w.
// VT is V transposed ([H][d][ldT] bf16, launch_transpose_v).  -1 on a TMA failure.
int launch_query_features(const Dims& D, const bf16* Q, const bf16* X, const bf16* K, const bf16* VT,
                          const bf16* U_q, const bf16* U_k, const bf16* U_v, const bf16* L_q, const bf16* L_c,
                          const bf16* L_x, const bf16* b_x, const QueryBufs& B, bf16* qbar_hi, bf16* qbar_lo,
                          float* wts, DevStatus* stt, cudaStream_t st);
// softmax products with fp32-grade split-3 operands (tc_attn.cu)
int launch_transpose_v(const Dims& D, const bf16* V, bf16* VT, cudaStream_t st);
// value logits [H][n][T] from the q'' triple and the bf16 keys, with row partials
int launch_value_logits_tc(const Dims& D, const bf16* q_h, const bf16* q_m, const bf16* q_l, const bf16* K,
                           float* logits, float2* part, DevStatus* stt, cudaStream_t st);
// out [H][n][128] = (exp(X - shift) * mul) V over rows of X [H][n][T].
int launch_probs_v_tc(const Dims& D, const float* X, const float* shift, const float* mul, bf16* p_h, bf16* p_m,
                      bf16* p_l, const bf16* VT, float* out, DevStatus* stt, cudaStream_t st,
                      const int* skip = nullptr);
// x (count floats) -> bf16 triple h + m + l
int launch_split3(const float* x, bf16* h, bf16* m, bf16* l, long long count, cudaStream_t st);
// I (Eq. pairwise_index_score) on tcgen05 with split-bf16 operands, and the
// per-(row, 128-column tile) softmax partials.  Returns launches, or -1 when a
// TMA descriptor cannot be encoded.
int launch_index_logits(const Dims& D, const bf16* qbar_hi, const bf16* qbar_lo, const bf16* kbar_hi,
                        const bf16* kbar_lo, const float* wts, float* I, float2* part, DevStatus* stt,
                        cudaStream_t st);
// row log-sum-exp and pooled s (Eq. indexer_pooling).
// Softmax partials of the index logits cover kIndexPartW columns each
// ([H][n][ceil(T / kIndexPartW)]); those of the value and reference logits
// kRowPartW columns each.
constexpr int kIndexPartW = 128;
constexpr int kRowPartW = 64;
int launch_index_pool(const Dims& D, const float* I, const float2* part, int ntiles, float* lse, float* s,
                      cudaStream_t st);

// ---- selection (Eq. persistent_support) ----------------------------------
// t_budget: the configured t (the per-chunk budgets derive from it); D.t is the realized count
int launch_top_t(const Dims& D, int t_budget, const float* s, int* anchors, DevStatus* stt, cudaStream_t st);
int launch_check_anchors(const Dims& D, int* anchors, DevStatus* stt, cudaStream_t st);

// ---- reference attention, assignment, merge (Sec. 3.4) ------------------
// l = scale Q K^T into `L` (tcgen05); z, m (row max / mass); Y = softmax(l) V
// (tcgen05, split-3 probabilities against VT); column statistics log phi,
// M_j and 1/||e^{l_:j - M_j}||.  -1 when a TMA descriptor cannot be encoded.
int launch_reference_attention(const Dims& D, float scale, const bf16* Q, const bf16* K, const bf16* VT,
                               float* L, float2* part, float* z, float* m, float* invm, bf16* p_h, bf16* p_m,
                               bf16* p_l, float* Y, DevStatus* stt, cudaStream_t st);
int launch_ref_logits_tc(const Dims& D, float scale, const bf16* Q, const bf16* K, float* L, float2* part,
                         DevStatus* stt, cudaStream_t st);
// Column statistics of the reference logits L: log phi [H][T] (mass weights of
// the merge) alone.
int launch_col_profiles(const Dims& D, const float* L, float* logphi, DevStatus* stt, cudaStream_t st);
// Assignment on tcgen05: column statistics (log phi written on the way) and
// the transposed split-bf16 profiles, the anchors' into the anchor rows S and
// the other keys' compacted into the first T - t rows of Ut (kmap: row -> key);
// then the argmax GEMM over the compacted rows (the anchors' own kappa(s_r) = r
// is set directly).
int launch_assign_prep(const Dims& D, const float* L, float* logphi, const int* anchors, bf16* Ut_hi, bf16* Ut_lo,
                       bf16* S_hi, bf16* S_lo, int* kmap, DevStatus* stt, cudaStream_t st);
int launch_assign_gemm(const Dims& D, const int* anchors, const bf16* Ut_hi, const bf16* Ut_lo, const bf16* S_hi,
                       const bf16* S_lo, const int* kmap, unsigned long long* best, int* kappa, DevStatus* stt,
                       cudaStream_t st);
int launch_check_assign(const Dims& D, int* kappa, const int* anchors, DevStatus* stt, cudaStream_t st);
// The counting sort of the merge runs over chunks of kSortChunk positions
// when a group histogram fits shared memory; its scratch (`cursor`) then
// holds sort_scratch_ints(H, T, t) ints.
constexpr int kSortChunk = 2048;
constexpr int kSortMaxT = 40 * 1024;
inline bool sort_chunked(int T, int t) { return t <= kSortMaxT && T > kSortChunk; }
inline long long sort_scratch_ints(int H, int T, int t) {
  const long long C = (T + kSortChunk - 1) / kSortChunk;
  return sort_chunked(T, t) ? (long long)H * t * (C + 1) : (long long)H * t;
}
int launch_merge(const Dims& D, float lambda_m, const bf16* K, const int* anchors, const int* kappa,
                 const float* logphi, int* perm, int* goff, int* cursor, float* C_k, cudaStream_t st);

// ---- fits (App. A.9) -----------------------------------------------------
struct FitBufs {
  float *LC, *Phi, *Gram, *Linv, *rhs, *wsol, *R, *Z;
  bf16 *PT_hi, *PT_lo, *YT_hi, *YT_lo;  // transposed split-bf16 operands ([t][ldn], [d][ldn])
  double *G64, *L64, *B64, *Z64, *X64;   // fp64 dual-form scratch (t > n only): [n][n], blocks, [n][d] x 3
  bf16* PT_mid;                         // middle part of the transposed triple of Phi_C ([t][ldn])
  bf16* ck3;                            // bf16 triple of C_k (parts [H][t][128], one after another)
  bf16 *Sl, *Sl2;                       // sliced operands of the dual fits (t > n only)
  int *eR, *eC;                         // their row exponents ([H][max(n, t)], [H][128])
  double *ir_u, *ir_sq, *ir_lam;        // refinement of the beta system: [H][n], [H][n], [H]
  bf16* Sl3;                            // right-hand-side slices of the dual solves (t > n only)
  int* eC2;
  double* cl_lam;                       // [H]
};
// Returns launches, or -1 when a TMA descriptor cannot be encoded.
// ev (nullable): events recorded before the beta solve, before the value
// products and before the C_v solve (stage events 8, 9, 10 of arckv_compact).
int launch_fits(const Dims& D, float scale, float ridge_w, float ridge_v, float eps_w, float b_min,
                float b_max, const bf16* Q, const float* C_k, const float* z, const float* m,
                const float* Y, const FitBufs& B, float* beta, float* C_v, DevStatus* stt, cudaStream_t st,
                cudaEvent_t const* ev = nullptr);
int launch_check_finite(const float* x, long long count, DevStatus* stt, cudaStream_t st);

// ---- fp64-grade products on the bf16 tensor pipe (tc_sliced.cu) ------------
// Operands are cut into S bf16 slices per row (S = 3, 4 or 5) with a power-of-two
// row scale; products of the sliced operands are exact up to ~2^-48 and
// returned in fp64 (or rounded to fp32).  K up to kSlicedMaxK.
constexpr int kSlicedMaxK = 26214;
bool sliced_supported(int K);
int sliced_last_failure();   // diagnostics: 1 map encoding, 100 + e attribute, 1000 + e launch (0: none)
size_t sliced_ld(int K);   // row pitch (elements) of a sliced operand with K columns
// X [H][R][K] (rows ldx apart, batches xbs apart) -> slices [S][H][R][sliced_ld(K)], exponents ex [H][R]
int launch_slice_rows(int S, const float* X, int R, int K, int ldx, long long xbs, int H, bf16* out, int* ex,
                      cudaStream_t st);
int launch_slice_rows(int S, const double* X, int R, int K, int ldx, long long xbs, int H, bf16* out, int* ex,
                      cudaStream_t st);
// the rows of X^T for X [H][K][R] (R contiguous): slices [S][H][R][sliced_ld(K)], exponents ex [H][R]
int launch_slice_cols(int S, const float* X, int K, int R, int ldx, long long xbs, int H, bf16* out, int* ex,
                      cudaStream_t st);
int launch_slice_cols(int S, const double* X, int K, int R, int ldx, long long xbs, int H, bf16* out, int* ex,
                      cudaStream_t st);
// C[b] (M x N, fp64, rows ldc apart, batches cbs apart) = A B^T, or C -= A B^T
// with `sub`; with `lower` only the tiles that reach C's lower triangle (M = N)
// (with 5 slices: nt0, nt1 select the 64-wide column tiles [nt0, nt1);
// max_ctas > 0 caps the persistent grid, leaving SMs to a concurrent stream)
int launch_sliced_f64(int S, const bf16* As, const int* eA, int M, const bf16* Bs, const int* eB, int N, int K, int H,
                      double* C, long long cbs, int ldc, bool lower, bool sub, DevStatus* stt, cudaStream_t st,
                      int nt0 = 0, int nt1 = 1 << 30, int max_ctas = 0);
// G[b] = X X^T (R x R, fp64) on the tiles that reach the lower triangle
int launch_sliced_gram_lower(int S, const bf16* Xs, const int* ex, int R, int K, int H, double* G, DevStatus* stt,
                             cudaStream_t st);
// C[b] (M x N, fp32, row stride ldc) = A B^T of sliced A [M][K], B [N][K]
int launch_sliced_product_f32(int S, const bf16* As, const int* eA, int M, const bf16* Bs, const int* eB, int N, int K,
                              int H, float* C, int ldc, DevStatus* stt, cudaStream_t st);

// ---- compact attention (Eq. compact_attention) ----------------------------
// Scratch of launch_attend: byte offsets from one 256-byte aligned base (the
// first 256 bytes are the status word) and the total size.
struct AttendLayout {
  size_t status, X, shift, mul, ck3, vt3, parts, p3, total;
};
AttendLayout attend_layout(int H, int n, int t);
// O [H][n][128] = softmax(scale Q C_k^T + beta) C_v on the tensor pipe; `ws` is
// the scratch base of attend_layout.  Returns launches or -1.
int launch_attend(int H, int n, int t, float scale, const bf16* Q, const float* C_k, const float* beta,
                  const float* C_v, float* O, char* ws, DevStatus* stt, cudaStream_t st);

// ---- HA / VI anchor scores (App. B.1) ----------------------------------
// E[h] = mean_i ||O_i - O~_i(S)|| / (||O_i|| + eps) (Eq. background_truncated_error);
// scratch inS [H][T] bytes, err [H][n].
int launch_truncated_error(int H, int n, int T, int t, float scale, float eps, const bf16* Q, const bf16* K,
                           const bf16* V, const int* S, float* E, unsigned char* inS, float* err, DevStatus* stt,
                           cudaStream_t st);
// Scratch of launch_vi_scores: per row amax, z2, mul2, Da, oo [H][n]; O^(-a) Om
// [H][n][128]; the split probabilities p_* [H][n][ldT] and Y's split y_*
// [H][n][128]; vv [H][T]; colpart [H][ceil(n/32)][T].
struct ViBufs {
  int* amax;
  float *z2, *mul2, *Da, *oo, *Om, *vv, *colpart;
  bf16 *p_h, *p_m, *p_l, *y_h, *y_m, *y_l;
};
// s [H][T] = VI scores from the reference logits L, row stats z, m, Y = softmax(L) V.
int launch_vi_scores(const Dims& D, const float* L, const float* z, const float* m, const float* Y, const bf16* V,
                     const bf16* VT, const ViBufs& B, float* s, float eps, DevStatus* stt, cudaStream_t st);

// ---- joint attention with an uncompressed block (App. A.7) -------------
// Key splits of the split-key pass (deterministic in H, n, t, F).
struct JointSplit {
  int per_split, nsplit;
};
JointSplit joint_split(int H, int n, int t, int F);
// O [H][n][128] fp32 = softmax(scale Q [C_k; K_f]^T + [beta; 0]) [C_v; V_f];
// C_k, C_v fp32 or (compact_bf16) bf16 [H][t][128]; K_f, V_f bf16 [H][F][128];
// scratch Opart [H][nsplit][n][128] fp32 and ml [H][nsplit][n].
int launch_attend_joint(int H, int n, int t, int F, float scale, const bf16* Q, const void* Ck, const float* beta,
                        const void* Cv, bool compact_bf16, const bf16* Kf, const bf16* Vf, float* O, float* Opart,
                        float2* ml, DevStatus* stt, cudaStream_t st);

// Shared small kernels.
int launch_part_stats(int H, int rows, int ntiles, const float2* part, float* shift, float* mul, float* sum,
                      cudaStream_t st);

}  // namespace arckv
