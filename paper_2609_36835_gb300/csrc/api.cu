// C ABI of libarckv: argument validation, workspace layout and the launch
// sequence of one layer's compaction.  Declarations and contracts are in
// include/arckv.h.
#include <string.h>

#include <algorithm>

#include <nvtx3/nvToolsExt.h>

#include "kernels.h"
#include "tc.cuh"

using namespace arckv;

namespace {

constexpr size_t kAlign = 256;

inline size_t up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

struct Layout {
  size_t status, kbar_hi, kbar_lo, vq, qpp, q_h, q_m, q_l, av, VT, p_h, p_m, p_l, vq3, av3, ukt, qbar_hi, qbar_lo, wts, NT, rA, rB, part, lse, s, anchors, z, m, invm, Y, logphi,
      qcat, wcat, Ut_hi, Ut_lo, S_hi, S_lo, best, kappa, kmap, perm, goff, cursor, LC, Phi, Gram, Linv, rhs, wsol, R, Z,
      ck3, YT_hi, YT_lo, G64, L64, B64, Z64, X64, Sl, Sl2, eR, eC, ir_u, ir_sq, ir_lam, Sl3, eC2, cl_lam, total;
};

Dims dims_of(const arckv_config& c) {
  Dims D;
  D.H = c.H_kv; D.G = c.G; D.T = c.T; D.d = c.d; D.n_pos = c.n_pos; D.n = c.n_pos * c.G; D.d_x = c.d_x;
  D.H_I = c.H_I; D.d_I = c.d_I; D.d_A = c.d_A; D.HD = c.H_I * c.d_I;
  D.chunk = effective_chunk(c.T, c.chunk_len);
  D.t = realized_anchors(c.T, c.t, c.chunk_len);   // = t without chunking
  return D;
}

arckv_status validate(const arckv_config* c) {
  if (!c) return ARCKV_ERR_INVALID_ARG;
  if (c->flags & ~ARCKV_FLAG_NONBLOCKING) return ARCKV_ERR_INVALID_ARG;
  if (c->H_kv < 1 || c->G < 1 || c->T < 1 || c->n_pos < 1 || c->t < 1 || c->t > c->T) return ARCKV_ERR_SHAPE;
  if (c->H_I < 1 || c->H_I > 16 || c->d_x < 8 || (c->d_x % 8) != 0) return ARCKV_ERR_SHAPE;
  if (c->d != 128 || c->d_I != 128 || c->d_A != 128) return ARCKV_ERR_UNSUPPORTED;
  if (c->chunk_len < 0) return ARCKV_ERR_INVALID_ARG;
  if (c->selector < ARCKV_SELECTOR_INDEXER || c->selector > ARCKV_SELECTOR_VI) return ARCKV_ERR_INVALID_ARG;
  if (c->selector == ARCKV_SELECTOR_VI && c->T < 2) return ARCKV_ERR_SHAPE;
  const int L = effective_chunk(c->T, c->chunk_len);
  if (L > 0 && (c->T + (long long)L - 1) / L > 65535) return ARCKV_ERR_SHAPE;   // chunks per head
  const long long tr = realized_anchors(c->T, c->t, c->chunk_len);
  // per-head element counts index with 32-bit ints inside the kernels
  const long long n = (long long)c->n_pos * c->G;
  if (n > (1 << 24) || (long long)c->T > (1 << 26) || n * c->T >= (1LL << 31) ||
      (long long)c->t * c->t >= (1LL << 31) || tr * tr >= (1LL << 31) || (long long)c->T * c->H_I * 128 >= (1LL << 31) ||
      (long long)c->H_kv * kSplitK > 65535)
    return ARCKV_ERR_SHAPE;
  if (!(c->lambda_m >= 0.f && c->lambda_m <= 1.f)) return ARCKV_ERR_INVALID_ARG;
  if (!(c->logit_scale >= 0.f) || !isfinite(c->logit_scale)) return ARCKV_ERR_INVALID_ARG;
  if (!(c->ridge_w >= 0.f) || !(c->ridge_v >= 0.f) || !isfinite(c->ridge_w) || !isfinite(c->ridge_v))
    return ARCKV_ERR_INVALID_ARG;
  if (!(c->eps_w > 0.f) || !(c->b_min <= c->b_max) || !isfinite(c->b_min) || !isfinite(c->b_max))
    return ARCKV_ERR_INVALID_ARG;
  return ARCKV_OK;
}

Layout plan(const arckv_config& c) {
  const Dims D = dims_of(c);
  const size_t H = D.H, T = D.T, n = D.n, t = D.t, HD = D.HD, f = 4;
  const size_t nblk = (t + kCholNB - 1) / kCholNB, ntile = (T + 63) / 64;   // softmax partials: 128 columns each, or kIndexPartW >= 64
  Layout L;
  size_t o = 0;
  auto take = [&](size_t bytes) { size_t r = o; o += up(bytes); return r; };
  L.status = take(sizeof(DevStatus));
  const size_t ldT = (T + 7) / 8 * 8;
  L.kbar_hi = take(H * T * HD * 2);
  L.kbar_lo = take(H * T * HD * 2);
  L.vq = take(H * n * 128 * f);    // VI selector scratch
  L.qpp = take(H * n * 128 * f);   // VI selector scratch
  L.q_h = take(H * n * 128 * 2);
  L.q_m = take(H * n * 128 * 2);
  L.q_l = take(H * n * 128 * 2);
  L.av = take(H * n * 128 * f);
  L.VT = take(H * 128 * ldT * 2);
  const size_t ptrip = probs_fused((int)T) ? 0 : H * n * ldT * 2;   // probability triple (unfused path only)
  L.p_h = take(ptrip);
  L.p_m = take(ptrip);
  L.p_l = take(ptrip);
  L.qcat = take(H * n * 512 * 2);
  L.vq3 = take(3 * H * n * 128 * 2);
  L.av3 = take(3 * H * n * 128 * 2);
  L.ukt = take(H * 128 * 128 * 2);
  L.wcat = take(H * HD * 512 * 2);
  L.qbar_hi = take(H * n * HD * 2);
  L.qbar_lo = take(H * n * HD * 2);
  L.wts = take(H * (size_t)D.n_pos * D.H_I * f);
  L.NT = take(H * n * T * f);
  L.rA = take(H * n * f);
  L.rB = take(H * n * f);
  L.part = take(H * n * ntile * 8);
  L.lse = take(H * n * f);
  L.s = take(H * T * f);
  L.anchors = take(H * t * 4);
  L.z = take(H * n * f);
  L.m = take(H * n * f);
  L.invm = take(H * n * f);
  L.Y = take(H * n * 128 * f);
  L.logphi = take(H * T * f);
  const size_t ldn = (n + 7) / 8 * 8;
  L.Ut_hi = take(H * T * ldn * 2);
  L.Ut_lo = take(H * T * ldn * 2);
  L.S_hi = take(H * t * ldn * 2);
  L.S_lo = take(H * t * ldn * 2);
  L.best = take(H * T * 8);
  L.kappa = take(H * T * 4);
  L.kmap = take(H * T * 4);
  L.perm = take(H * T * 4);
  L.goff = take(H * (t + 1) * 4);
  L.cursor = take((size_t)sort_scratch_ints((int)H, (int)T, (int)t) * 4);
  L.LC = take(H * n * (t > 128 ? t : 128) * f);   // also holds the n x d dual solution when t > n
  L.Phi = take(H * n * t * f);
  const bool dual = t > n;   // the fits run in their n x n dual form
  L.Gram = take(dual ? 0 : H * t * t * f);
  L.Linv = take(H * nblk * kCholNB * kCholNB * f);
  L.rhs = take(H * t * f);
  L.wsol = take(H * t * f);
  L.R = take(H * t * 128 * f);
  L.Z = take(H * t * 128 * f);
  L.ck3 = take(3 * H * t * 128 * 2);
  L.YT_hi = take(H * 128 * ldn * 2);
  L.YT_lo = take(H * 128 * ldn * 2);
  // fp64 dual-form scratch, only when t > n
  const size_t nd64 = t > n ? n : 0, nbn = (nd64 + kCholNB - 1) / kCholNB;
  L.G64 = take(H * nd64 * nd64 * 8);
  L.L64 = take(H * nbn * kCholNB * kCholNB * 8);
  L.B64 = take(H * nd64 * 128 * 8);
  L.Z64 = take(H * nd64 * 128 * 8);
  L.X64 = take(H * nd64 * 128 * 8);
  // sliced operands of the dual fits: up to 4 slices of Phi_C (or P^, P^^T)
  const size_t slrow = dual ? std::max(n * sliced_ld((int)t), t * sliced_ld((int)n)) : 0;
  // (the blocked dual Cholesky takes two 5-slice 64-column panel sets from it)
  L.Sl = take(std::max(4 * H * slrow, dual ? 2 * 5 * H * n * kCholNB : 0) * 2);
  L.Sl2 = take(dual ? std::max(4 * H * 128 * sliced_ld((int)n), 2 * 5 * H * kCholNB * kCholNB) * 2 : 0);
  L.eR = take(dual ? H * std::max(2 * n, t) * 4 : 0);
  L.eC = take(dual ? H * 128 * 4 : 0);
  L.ir_u = take(dual ? 0 : H * n * 8);
  L.ir_sq = take(dual ? 0 : H * n * 8);
  L.ir_lam = take(dual ? 0 : H * 8);
  // the blocked dual solves: 5-slice right-hand-side columns (up to 128 rows of K <= n)
  L.Sl3 = take(dual ? 5 * H * 128 * sliced_ld((int)n) * 2 : 0);
  L.eC2 = take(dual ? H * 128 * 4 : 0);
  L.cl_lam = take(dual ? H * 8 : 0);
  L.total = o;
  return L;
}

struct Launcher {
  int count = 0;
  cudaStream_t st;
};

arckv_status read_status(void* ws, cudaStream_t st) {
  unsigned int code = 0;
  if (cudaMemcpyAsync(&code, ws, sizeof(code), cudaMemcpyDeviceToHost, st) != cudaSuccess) return ARCKV_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return ARCKV_ERR_CUDA;
  return (arckv_status)code;
}

}  // namespace

extern "C" {

size_t arckv_workspace_bytes(const arckv_config* cfg) {
  if (validate(cfg) != ARCKV_OK) return 0;
  return plan(*cfg).total;
}

int32_t arckv_anchor_count(const arckv_config* cfg) {
  if (validate(cfg) != ARCKV_OK) return 0;
  return realized_anchors(cfg->T, cfg->t, cfg->chunk_len);
}

const char* arckv_status_string(arckv_status s) {
  switch (s) {
    case ARCKV_OK: return "ok";
    case ARCKV_ERR_INVALID_ARG: return "invalid argument";
    case ARCKV_ERR_SHAPE: return "shape out of range";
    case ARCKV_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    case ARCKV_ERR_NOT_SPD: return "normal matrix of a fit is not positive definite";
    case ARCKV_ERR_NONFINITE: return "non-finite value in inputs or results";
    case ARCKV_ERR_TIMEOUT: return "bounded device wait timed out";
    case ARCKV_ERR_CUDA: return "CUDA runtime error";
    case ARCKV_ERR_UNSUPPORTED: return "configuration not supported";
  }
  return "unknown status";
}

arckv_status arckv_query_status(void* ws, void* stream) {
  if (!ws) return ARCKV_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)stream;
  arckv_status s = read_status(ws, st);
  if (s == ARCKV_ERR_CUDA) return s;
  if (cudaMemsetAsync(ws, 0, sizeof(unsigned int), st) != cudaSuccess) return ARCKV_ERR_CUDA;
  return s;
}

// One CTA waits on an mbarrier that nothing arrives on, through the bounded
// wait of the tensor-core kernels with a limit of limit_ns: the wait gives up
// and records ARCKV_ERR_TIMEOUT in the status word, and the CTA returns.
__global__ void wait_probe_kernel(DevStatus* stt, unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);
    abort_flag = 0;
    tc::mbar_fence_init();
  }
  __syncthreads();
  volatile int* ab = &abort_flag;
  if (threadIdx.x == 0) tc::mbar_wait_for(&bar, 0, ab, stt, limit_ns);
  __syncthreads();
}

arckv_status arckv_wait_probe(void* ws, size_t ws_bytes, uint32_t limit_us, void* stream) {
  if (limit_us == 0 || limit_us > 1000000u) return ARCKV_ERR_INVALID_ARG;
  if (!ws || ws_bytes < sizeof(DevStatus) || ((uintptr_t)ws % kAlign) != 0) return ARCKV_ERR_WORKSPACE;
  cudaStream_t st = (cudaStream_t)stream;
  cudaGetLastError();
  DevStatus* stt = (DevStatus*)ws;
  if (cudaMemsetAsync(stt, 0, sizeof(DevStatus), st) != cudaSuccess) return ARCKV_ERR_CUDA;
  wait_probe_kernel<<<1, 32, 0, st>>>(stt, (unsigned long long)limit_us * 1000ull);
  if (cudaGetLastError() != cudaSuccess) return ARCKV_ERR_CUDA;
  return read_status(ws, st);
}

arckv_status arckv_compact(const arckv_config* cfg, const void* K, const void* V, const void* Q_ref,
                           const void* X_ref, const arckv_indexer* idx, float* C_k, float* beta, float* C_v,
                           const arckv_aux* aux, void* ws, size_t ws_bytes, void* stream) {
  arckv_status vs = validate(cfg);
  if (vs != ARCKV_OK) return vs;
  if (!K || !V || !Q_ref || !C_k || !beta || !C_v) return ARCKV_ERR_INVALID_ARG;
  const bool given_anchors = aux && aux->anchors_in;
  const bool given_assign = aux && aux->assign_in;
  if (given_assign && !given_anchors) return ARCKV_ERR_INVALID_ARG;
  const bool use_indexer = !given_anchors && cfg->selector == ARCKV_SELECTOR_INDEXER;
  if (use_indexer && (!idx || !X_ref || !idx->L_q || !idx->L_k || !idx->L_x || !idx->b_x || !idx->U_q || !idx->U_k ||
                         !idx->U_v || !idx->L_c || !idx->L_v))
    return ARCKV_ERR_INVALID_ARG;
  const Layout L = plan(*cfg);
  if (!ws || ws_bytes < L.total || ((uintptr_t)ws % kAlign) != 0) return ARCKV_ERR_WORKSPACE;

  const Dims D = dims_of(*cfg);
  cudaStream_t st = (cudaStream_t)stream;
  char* w = (char*)ws;
  auto F = [&](size_t off) { return (float*)(w + off); };
  auto I32 = [&](size_t off) { return (int*)(w + off); };
  DevStatus* stt = (DevStatus*)(w + L.status);
  const float scale = cfg->logit_scale > 0.f ? cfg->logit_scale : 1.0f / sqrtf((float)D.d);
  const bf16* Kb = (const bf16*)K;
  const bf16* Vb = (const bf16*)V;
  const bf16* Qb = (const bf16*)Q_ref;
  cudaEvent_t const* ev = (aux && aux->stage_events) ? (cudaEvent_t const*)aux->stage_events : nullptr;
  // stage boundaries: the caller's CUDA events, and one NVTX range per stage
  // (host-side enqueue spans, visible to Nsight; no cost without a tool attached)
  // (stages 7-10, whose boundaries lie inside launch_fits, share one range)
  static const char* const kStageNames[8] = {
      "arckv.indexer_features", "arckv.index_logits", "arckv.pool_top_t", "arckv.reference_attention",
      "arckv.column_profiles", "arckv.assignment", "arckv.merge", "arckv.fits"};
  int open_stage = -1;
  auto mark = [&](int s) {
    if (ev) cudaEventRecord(ev[s], st);
    if (open_stage >= 0) nvtxRangePop();
    open_stage = s < 8 ? s : -1;
    if (open_stage >= 0) nvtxRangePushA(kStageNames[s]);
  };
  nvtxRangePushA("arckv_compact");
  struct RangeGuard {
    int* open;
    ~RangeGuard() {
      if (*open >= 0) nvtxRangePop();
      nvtxRangePop();
    }
  } guard{&open_stage};
  int nl = 0;

  cudaGetLastError();  // clear a stale error from earlier, unrelated work
  if (cudaMemsetAsync(stt, 0, sizeof(DevStatus), st) != cudaSuccess) return ARCKV_ERR_CUDA;
  int* anchors = I32(L.anchors);
  auto B16 = [&](size_t off) { return (bf16*)(w + off); };
  mark(0);
  nl += launch_transpose_v(D, Vb, B16(L.VT), st);
  // the reference attention (a5) does not depend on S: with the HA / VI
  // selectors it runs first and its logits give the scores
  bool ref_done = false;
  auto reference_attention = [&]() -> int {
    ref_done = true;
    return launch_reference_attention(D, scale, Qb, Kb, B16(L.VT), F(L.NT), (float2*)(w + L.part), F(L.z), F(L.m),
                                      F(L.invm), B16(L.p_h), B16(L.p_m), B16(L.p_l), F(L.Y), stt, st);
  };
  if (!given_anchors && !use_indexer) {
    mark(1);
    mark(2);
    const int nlr0 = reference_attention();
    if (nlr0 < 0) return ARCKV_ERR_CUDA;
    nl += nlr0;
    if (cfg->selector == ARCKV_SELECTOR_HA) {
      // p = softmax(l): the same pooling as the index scores, on l's row partials
      nl += launch_index_pool(D, F(L.NT), (const float2*)(w + L.part), cdiv(D.T, kRowPartW), F(L.lse), F(L.s), st);
    } else {
      float* vq = F(L.vq);   // VI scratch: n-sized rows here, O^(-a) in L.qpp
      const size_t hn = (size_t)D.H * D.n;
      ViBufs VB{(int*)vq, vq + hn, vq + 2 * hn, vq + 3 * hn, vq + 4 * hn, F(L.qpp), F(L.best), F(L.Ut_hi),
                B16(L.p_h), B16(L.p_m), B16(L.p_l), B16(L.q_h), B16(L.q_m), B16(L.q_l)};
      const int nlv = launch_vi_scores(D, F(L.NT), F(L.z), F(L.m), F(L.Y), Vb, B16(L.VT), VB, F(L.s), 1e-6f, stt,
                                       st);
      if (nlv < 0) return ARCKV_ERR_CUDA;
      nl += nlv;
    }
    nl += launch_top_t(D, cfg->t, F(L.s), anchors, stt, st);
    nl += launch_check_anchors(D, anchors, stt, st);
  } else if (!given_anchors) {
    const int nlk = launch_key_features_tc(D, Kb, Vb, (const bf16*)idx->L_k, (const bf16*)idx->L_v, B16(L.kbar_hi),
                                           B16(L.kbar_lo), stt, st);
    if (nlk < 0) return ARCKV_ERR_CUDA;
    nl += nlk;
    QueryBufs QB{F(L.NT),    F(L.rA),    F(L.rB),    F(L.av),     B16(L.q_h),
                 B16(L.q_m), B16(L.q_l), B16(L.p_h), B16(L.p_m), B16(L.p_l),
                 (float2*)(w + L.part),  B16(L.qcat), B16(L.wcat), B16(L.vq3), B16(L.av3),
                 B16(L.ukt)};
    const int nlq = launch_query_features(D, Qb, (const bf16*)X_ref, Kb, B16(L.VT), (const bf16*)idx->U_q,
                                          (const bf16*)idx->U_k, (const bf16*)idx->U_v, (const bf16*)idx->L_q,
                                          (const bf16*)idx->L_c, (const bf16*)idx->L_x, (const bf16*)idx->b_x, QB,
                                          B16(L.qbar_hi), B16(L.qbar_lo), F(L.wts), stt, st);
    if (nlq < 0) return ARCKV_ERR_CUDA;
    nl += nlq;
    mark(1);
    const int nli = launch_index_logits(D, B16(L.qbar_hi), B16(L.qbar_lo), B16(L.kbar_hi), B16(L.kbar_lo),
                                        F(L.wts), F(L.NT), (float2*)(w + L.part), stt, st);
    if (nli < 0) return ARCKV_ERR_CUDA;
    nl += nli;
    mark(2);
    nl += launch_index_pool(D, F(L.NT), (const float2*)(w + L.part), cdiv(D.T, kIndexPartW), F(L.lse), F(L.s),
                            st);
    nl += launch_top_t(D, cfg->t, F(L.s), anchors, stt, st);
    nl += launch_check_anchors(D, anchors, stt, st);   // a selection fault becomes a status, not a stray index
  } else {
    mark(1);
    mark(2);
    cudaMemcpyAsync(anchors, aux->anchors_in, sizeof(int) * (size_t)D.H * D.t, cudaMemcpyDeviceToDevice, st);
    nl += launch_check_anchors(D, anchors, stt, st);
  }
  mark(3);
  if (!ref_done) {
    const int nlr = reference_attention();
    if (nlr < 0) return ARCKV_ERR_CUDA;
    nl += nlr;
  }
  int* kappa = I32(L.kappa);
  mark(4);
  if (!given_assign) {
    const int nla = launch_assign_prep(D, F(L.NT), F(L.logphi), anchors, B16(L.Ut_hi), B16(L.Ut_lo), B16(L.S_hi),
                                       B16(L.S_lo), I32(L.kmap), stt, st);
    if (nla < 0) return ARCKV_ERR_CUDA;
    mark(5);
    const int nlg = launch_assign_gemm(D, anchors, B16(L.Ut_hi), B16(L.Ut_lo), B16(L.S_hi), B16(L.S_lo),
                                       I32(L.kmap), (unsigned long long*)(w + L.best), kappa, stt, st);
    if (nlg < 0) return ARCKV_ERR_CUDA;
    nl += nla + nlg;
  } else {
    const int nlc = launch_col_profiles(D, F(L.NT), F(L.logphi), stt, st);   // log phi only
    if (nlc < 0) return ARCKV_ERR_CUDA;
    nl += nlc;
    mark(5);
    cudaMemcpyAsync(kappa, aux->assign_in, sizeof(int) * (size_t)D.H * D.T, cudaMemcpyDeviceToDevice, st);
    nl += launch_check_assign(D, kappa, anchors, stt, st);
  }
  mark(6);
  nl += launch_merge(D, cfg->lambda_m, Kb, anchors, kappa, F(L.logphi), I32(L.perm), I32(L.goff), I32(L.cursor),
                     C_k, st);
  mark(7);
  FitBufs B{F(L.LC),  F(L.Phi), F(L.Gram), F(L.Linv), F(L.rhs), F(L.wsol), F(L.R), F(L.Z),
            (bf16*)(w + L.S_hi), (bf16*)(w + L.S_lo), (bf16*)(w + L.YT_hi), (bf16*)(w + L.YT_lo),
            (double*)(w + L.G64), (double*)(w + L.L64), (double*)(w + L.B64), (double*)(w + L.Z64),
            (double*)(w + L.X64), (bf16*)(w + L.Ut_hi),   // Ut_hi [H][T][ldn] is free after the assignment
            (bf16*)(w + L.ck3), (bf16*)(w + L.Sl), (bf16*)(w + L.Sl2), I32(L.eR), I32(L.eC),
            (double*)(w + L.ir_u), (double*)(w + L.ir_sq), (double*)(w + L.ir_lam), (bf16*)(w + L.Sl3),
            I32(L.eC2), (double*)(w + L.cl_lam)};
  const int nlf = launch_fits(D, scale, cfg->ridge_w, cfg->ridge_v, cfg->eps_w, cfg->b_min, cfg->b_max, Qb, C_k,
                              F(L.z), F(L.m), F(L.Y), B, beta, C_v, stt, st, ev);
  if (nlf < 0) return ARCKV_ERR_CUDA;
  nl += nlf;
  nl += launch_check_finite(C_k, (long long)D.H * D.t * D.d, stt, st);
  nl += launch_check_finite(beta, (long long)D.H * D.t, stt, st);
  nl += launch_check_finite(C_v, (long long)D.H * D.t * D.d, stt, st);
  mark(ARCKV_NUM_STAGES);
  if (aux) {
    if (aux->scores && !given_anchors)
      cudaMemcpyAsync(aux->scores, F(L.s), sizeof(float) * (size_t)D.H * D.T, cudaMemcpyDeviceToDevice, st);
    if (aux->anchors)
      cudaMemcpyAsync(aux->anchors, anchors, sizeof(int) * (size_t)D.H * D.t, cudaMemcpyDeviceToDevice, st);
    if (aux->assign)
      cudaMemcpyAsync(aux->assign, kappa, sizeof(int) * (size_t)D.H * D.T, cudaMemcpyDeviceToDevice, st);
    if (aux->launches) *aux->launches = nl;
  }
  if (cudaGetLastError() != cudaSuccess) return ARCKV_ERR_CUDA;
  if (cfg->flags & ARCKV_FLAG_NONBLOCKING) return ARCKV_OK;
  return read_status(ws, st);
}

size_t arckv_attend_workspace_bytes(int32_t H_kv, int32_t n, int32_t t, int32_t d) {
  if (H_kv < 1 || n < 1 || t < 1 || d != 128) return 0;
  if ((long long)n * t >= (1LL << 31) || (long long)H_kv * n >= (1LL << 31) || (long long)H_kv * t * 128 >= (1LL << 31))
    return 0;
  return attend_layout(H_kv, n, t).total;
}

arckv_status arckv_attend(int32_t H_kv, int32_t n, int32_t t, int32_t d, float logit_scale, const void* Q,
                          const float* C_k, const float* beta, const float* C_v, float* O, void* ws,
                          size_t ws_bytes, uint32_t flags, void* stream) {
  if (flags & ~ARCKV_FLAG_NONBLOCKING) return ARCKV_ERR_INVALID_ARG;
  if (d != 128) return ARCKV_ERR_UNSUPPORTED;
  const size_t need = arckv_attend_workspace_bytes(H_kv, n, t, d);
  if (need == 0) return ARCKV_ERR_SHAPE;
  if (!Q || !C_k || !beta || !C_v || !O) return ARCKV_ERR_INVALID_ARG;
  if (!(logit_scale >= 0.f) || !isfinite(logit_scale)) return ARCKV_ERR_INVALID_ARG;
  if (!ws || ws_bytes < need || ((uintptr_t)ws % kAlign) != 0) return ARCKV_ERR_WORKSPACE;
  cudaStream_t st = (cudaStream_t)stream;
  char* w = (char*)ws;
  DevStatus* stt = (DevStatus*)w;
  const float scale = logit_scale > 0.f ? logit_scale : 1.0f / sqrtf((float)d);
  cudaGetLastError();
  if (cudaMemsetAsync(stt, 0, sizeof(DevStatus), st) != cudaSuccess) return ARCKV_ERR_CUDA;
  if (launch_attend(H_kv, n, t, scale, (const bf16*)Q, C_k, beta, C_v, O, w, stt, st) < 0) return ARCKV_ERR_CUDA;
  launch_check_finite(O, (long long)H_kv * n * d, stt, st);
  if (cudaGetLastError() != cudaSuccess) return ARCKV_ERR_CUDA;
  if (flags & ARCKV_FLAG_NONBLOCKING) return ARCKV_OK;
  return read_status(ws, st);
}

size_t arckv_attend_joint_workspace_bytes(int32_t H, int32_t n, int32_t t, int32_t F, int32_t d) {
  if (H < 1 || n < 1 || t < 0 || F < 0 || (long long)t + F < 1 || d != 128) return 0;
  if ((long long)t + F >= (1LL << 30) || (long long)H * n >= (1LL << 31) || cdiv(n, 4) > 65535 || H > 65535) return 0;
  const JointSplit js = joint_split(H, n, t, F);
  const size_t rows = (size_t)H * js.nsplit * n;
  return up(sizeof(DevStatus)) + up(rows * 128 * 4) + up(rows * 8);
}

arckv_status arckv_attend_joint(int32_t H, int32_t n, int32_t t, int32_t F, int32_t d, float logit_scale,
                                const void* Q, const void* C_k, const float* beta, const void* C_v,
                                const void* K_fixed, const void* V_fixed, float* O, void* ws, size_t ws_bytes,
                                uint32_t flags, void* stream) {
  if (flags & ~(ARCKV_FLAG_NONBLOCKING | ARCKV_FLAG_COMPACT_BF16)) return ARCKV_ERR_INVALID_ARG;
  if (d != 128) return ARCKV_ERR_UNSUPPORTED;
  const size_t need = arckv_attend_joint_workspace_bytes(H, n, t, F, d);
  if (need == 0) return ARCKV_ERR_SHAPE;
  if (!Q || !O || (t > 0 && (!C_k || !beta || !C_v)) || (F > 0 && (!K_fixed || !V_fixed)))
    return ARCKV_ERR_INVALID_ARG;
  // rows are read as 16-byte vectors
  auto misaligned = [](const void* p) { return p && ((uintptr_t)p % 16) != 0; };
  if (misaligned(C_k) || misaligned(C_v) || misaligned(K_fixed) || misaligned(V_fixed) || misaligned(O))
    return ARCKV_ERR_INVALID_ARG;
  if (!(logit_scale >= 0.f) || !isfinite(logit_scale)) return ARCKV_ERR_INVALID_ARG;
  if (!ws || ws_bytes < need || ((uintptr_t)ws % kAlign) != 0) return ARCKV_ERR_WORKSPACE;
  cudaStream_t st = (cudaStream_t)stream;
  char* w = (char*)ws;
  DevStatus* stt = (DevStatus*)w;
  const JointSplit js = joint_split(H, n, t, F);
  const size_t rows = (size_t)H * js.nsplit * n;
  float* Opart = (float*)(w + up(sizeof(DevStatus)));
  float2* ml = (float2*)(w + up(sizeof(DevStatus)) + up(rows * 128 * 4));
  const float scale = logit_scale > 0.f ? logit_scale : 1.0f / sqrtf((float)d);
  cudaGetLastError();
  if (cudaMemsetAsync(stt, 0, sizeof(DevStatus), st) != cudaSuccess) return ARCKV_ERR_CUDA;
  launch_attend_joint(H, n, t, F, scale, (const bf16*)Q, C_k, beta, C_v, (flags & ARCKV_FLAG_COMPACT_BF16) != 0,
                      (const bf16*)K_fixed, (const bf16*)V_fixed, O, Opart, ml, stt, st);
  launch_check_finite(O, (long long)H * n * d, stt, st);
  if (cudaGetLastError() != cudaSuccess) return ARCKV_ERR_CUDA;
  if (flags & ARCKV_FLAG_NONBLOCKING) return ARCKV_OK;
  return read_status(ws, st);
}

size_t arckv_truncated_error_workspace_bytes(int32_t H, int32_t n, int32_t T, int32_t t, int32_t d) {
  if (H < 1 || n < 1 || T < 1 || t < 0 || t > T || d != 128) return 0;
  if ((long long)H * T >= (1LL << 40) || (long long)H * n >= (1LL << 31) || cdiv(n, 4) > 65535 || H > 65535) return 0;
  return up(sizeof(DevStatus)) + up((size_t)H * T) + up((size_t)H * n * 4);
}

arckv_status arckv_truncated_error(int32_t H, int32_t n, int32_t T, int32_t t, int32_t d, float logit_scale,
                                   const void* Q_eval, const void* K, const void* V, const int32_t* S, float* E,
                                   void* ws, size_t ws_bytes, uint32_t flags, void* stream) {
  if (flags & ~ARCKV_FLAG_NONBLOCKING) return ARCKV_ERR_INVALID_ARG;
  if (d != 128) return ARCKV_ERR_UNSUPPORTED;
  const size_t need = arckv_truncated_error_workspace_bytes(H, n, T, t, d);
  if (need == 0) return ARCKV_ERR_SHAPE;
  if (!Q_eval || !K || !V || !E || (t > 0 && !S)) return ARCKV_ERR_INVALID_ARG;
  if ((((uintptr_t)K) % 16) || (((uintptr_t)V) % 16)) return ARCKV_ERR_INVALID_ARG;
  if (!(logit_scale >= 0.f) || !isfinite(logit_scale)) return ARCKV_ERR_INVALID_ARG;
  if (!ws || ws_bytes < need || ((uintptr_t)ws % kAlign) != 0) return ARCKV_ERR_WORKSPACE;
  cudaStream_t st = (cudaStream_t)stream;
  char* w = (char*)ws;
  DevStatus* stt = (DevStatus*)w;
  unsigned char* inS = (unsigned char*)(w + up(sizeof(DevStatus)));
  float* err = (float*)(w + up(sizeof(DevStatus)) + up((size_t)H * T));
  const float scale = logit_scale > 0.f ? logit_scale : 1.0f / sqrtf((float)d);
  cudaGetLastError();
  if (cudaMemsetAsync(stt, 0, sizeof(DevStatus), st) != cudaSuccess) return ARCKV_ERR_CUDA;
  launch_truncated_error(H, n, T, t, scale, 1e-6f, (const bf16*)Q_eval, (const bf16*)K, (const bf16*)V, S, E, inS,
                         err, stt, st);
  launch_check_finite(E, H, stt, st);
  if (cudaGetLastError() != cudaSuccess) return ARCKV_ERR_CUDA;
  if (flags & ARCKV_FLAG_NONBLOCKING) return ARCKV_OK;
  return read_status(ws, st);
}

}  // extern "C"
