// Value-aware indexer scoring (Sec. 3.3; App. A.1).
//
// Per KV head: k_bar_j,a = N((L_k k_j + L_v v_j)_a), Uk_j = U_k k_j,
// Uv_j = U_v v_j (key side, one pass over K and V);
// c_i = softmax_j((U_q q_i).(Uk_j)) Uv (Eq. value_context);
// q_bar_i,a = N((L_q q_i + L_c c_i)_a); w_i,a = (L_x x_r + b_x)_a
// (Eq. indexer_projection); I_ij = sum_a w_ia LeakyReLU_0.1(q_bar_ia.k_bar_ja / sqrt(d_I))
// (Eq. pairwise_index_score, in tc_index.cu); pi = row softmax of I and
// s_j = (mean_i pi_ij^2)^(1/2) (Eq. indexer_pooling).
#include "kernels.h"
#include "tc_gemm.cuh"

namespace arckv {

// w[b][r][a] = L_x[b][a] . x_r + b_x[b][a]: one CTA per (position, head).
__global__ void __launch_bounds__(512) index_weights_kernel(const bf16* X, const bf16* L_x, const bf16* b_x,
                                                            float* wts, int d_x, int H_I, int n_pos) {
  // one warp per index head a: w_ra = L_x[a] . x_r + b_x[a]
  const int r = blockIdx.x, b = blockIdx.y, a = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (a >= H_I) return;
  const bf16* x = X + (long long)r * d_x;
  const bf16* l = L_x + ((long long)b * H_I + a) * d_x;
  float acc = 0.f;
  if ((((uintptr_t)x | (uintptr_t)l) & 15) == 0) {   // rows are d_x % 8 == 0 elements long
    for (int k = lane * 8; k < d_x; k += 256) {
      const uint4 xv = *(const uint4*)(x + k), lv = *(const uint4*)(l + k);
      const __nv_bfloat162* xh = (const __nv_bfloat162*)&xv;
      const __nv_bfloat162* lh = (const __nv_bfloat162*)&lv;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 xf = __bfloat1622float2(xh[e]), lf = __bfloat1622float2(lh[e]);
        acc = fmaf(xf.x, lf.x, acc);
        acc = fmaf(xf.y, lf.y, acc);
      }
    }
  } else {
    for (int k = lane; k < d_x; k += 32) acc = fmaf(to_f32(x[k]), to_f32(l[k]), acc);
  }
  acc = warp_sum(acc);
  if (lane == 0) wts[((long long)b * n_pos + r) * H_I + a] = acc + to_f32(b_x[b * H_I + a]);
}

// out = A W^T for the n reference rows of every head, W [H][128][128] bf16
// (K-major), A either an exact bf16 input (A_m == nullptr: one MMA per
// product) or a bf16 triple (kSplit3A); the epilogue writes a bf16 triple.
static int gemm_rows128(const Dims& D, const bf16* A_h, const bf16* A_m, const bf16* A_l, const bf16* W,
                        const TcEpiSplit3& epi, DevStatus* stt, cudaStream_t st) {
  CUtensorMap mA, mA2, mA3, mB;
  if (!encode_bf16_map_3d(&mA, A_h, 128, D.n, D.H, 128) || !encode_bf16_map_3d(&mB, W, 128, 128, D.H, 128)) return -1;
  if (A_m == nullptr)
    return launch_tc_gemm<128, kPlain>(mA, mB, mA, mB, epi, D.H, D.n, 128, 128, 128, stt, st) == cudaSuccess ? 1 : -1;
  if (!encode_bf16_map_3d(&mA2, A_m, 128, D.n, D.H, 128) || !encode_bf16_map_3d(&mA3, A_l, 128, D.n, D.H, 128))
    return -1;
  return launch_tc_gemm<128, kSplit3A>(mA, mB, mA2, mA, epi, D.H, D.n, 128, 128, 128, stt, st, 0, &mA3) == cudaSuccess
             ? 1
             : -1;
}

int launch_query_features(const Dims& D, const bf16* Q, const bf16* X, const bf16* K, const bf16* VT,
                          const bf16* U_q, const bf16* U_k, const bf16* U_v, const bf16* L_q, const bf16* L_c,
                          const bf16* L_x, const bf16* b_x, const QueryBufs& B, bf16* qbar_hi, bf16* qbar_lo,
                          float* wts, DevStatus* stt, cudaStream_t st) {
  int nl = 0;
  const long long hn = (long long)D.H * D.n * 128, nd = (long long)D.n * 128;
  // vq = U_q q (exact products of bf16 inputs) and q'' = U_k^T vq, so that
  // (U_q q_i).(U_k k_j) = q''_i . k_j; both leave their GEMM as bf16 triples
  // (vq for the q'' product, q'' as the A operand of the value logits)
  Dims Dw = D;
  Dw.T = 128;
  nl += launch_transpose_v(Dw, U_k, B.ukt, st);   // U_k^T [H][d][d_A]
  bf16 *vq_h = B.vq3, *vq_m = B.vq3 + hn, *vq_l = B.vq3 + 2 * hn;
  int r = gemm_rows128(D, Q, nullptr, nullptr, U_q, TcEpiSplit3{vq_h, vq_m, vq_l, nd, 128}, stt, st);
  if (r < 0) return -1;
  nl += r;
  r = gemm_rows128(D, vq_h, vq_m, vq_l, B.ukt, TcEpiSplit3{B.q_h, B.q_m, B.q_l, nd, 128}, stt, st);
  if (r < 0) return -1;
  nl += r;
  // value-attention logits on the tensor cores, unscaled as printed in Eq. value_context
  r = launch_value_logits_tc(D, B.q_h, B.q_m, B.q_l, K, B.logits, B.part, stt, st);
  if (r < 0) return -1;
  nl += r;
  nl += launch_part_stats(D.H, D.n, cdiv(D.T, kRowPartW), B.part, B.rshift, B.rmul, nullptr, st);
  // A^V V on the tensor cores, then c = (A^V V) U_v^T = A^V (U_v V), written as
  // the bf16 triple that the q_bar GEMM reads (columns 128.. of its A operand)
  r = launch_probs_v_tc(D, B.logits, B.rshift, B.rmul, B.p_h, B.p_m, B.p_l, VT, B.av, stt, st);
  if (r < 0) return -1;
  nl += r;
  bf16 *av_h = B.av3, *av_m = B.av3 + hn, *av_l = B.av3 + 2 * hn;
  nl += launch_split3(B.av, av_h, av_m, av_l, hn, st);
  r = gemm_rows128(D, av_h, av_m, av_l, U_v, TcEpiSplit3{B.qcat + 128, B.qcat + 256, B.qcat + 384, nd * 4, 512}, stt,
                   st);
  if (r < 0) return -1;
  nl += r;
  // q_bar = N(L_q q + L_c c) per block, as a split-bf16 pair
  r = launch_query_proj_tc(D, Q, L_q, L_c, B.qcat, B.wcat, qbar_hi, qbar_lo, stt, st);
  if (r < 0) return -1;
  nl += r;
  index_weights_kernel<<<dim3(D.n_pos, D.H), 32 * D.H_I, 0, st>>>(X, L_x, b_x, wts, D.d_x, D.H_I, D.n_pos);
  ++nl;
  return nl;
}

// lse[b][i] = log sum_j exp(I_ij) from the column-tile partials; one warp per row.
__global__ void lse_reduce_kernel(const float2* part, float* lse, int n, int ntiles) {
  const int b = blockIdx.y, row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= n) return;
  const float2* p = part + ((long long)b * n + row) * ntiles;
  float mx = -INFINITY, sm = 0.f;
  for (int k = lane; k < ntiles; k += 32) lse_combine(mx, sm, p[k].x, p[k].y);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, mx, o), os = __shfl_xor_sync(0xffffffffu, sm, o);
    lse_combine(mx, sm, om, os);
  }
  if (lane == 0) lse[(long long)b * n + row] = mx + logf(sm);
}

// s_j = sqrt(mean_i exp(2 (I_ij - lse_i))).  A CTA owns 32 columns; warp w
// sums the rows i = w, w+8, ... of its column (four independent partial sums
// per thread) and the eight warp sums are added in warp order.
__global__ void __launch_bounds__(256) pool_kernel(const float* I, const float* lse, float* s, int n, int T) {
  const int b = blockIdx.y, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int j = blockIdx.x * 32 + lane;
  __shared__ float red[8][33];
  const float* Ib = I + (long long)b * n * T + j;
  const float* lb = lse + (long long)b * n;
  float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
  if (j < T) {
    int i = warp;
    for (; i + 24 < n; i += 32) {
      const float p0 = expf(Ib[(long long)i * T] - lb[i]);
      const float p1 = expf(Ib[(long long)(i + 8) * T] - lb[i + 8]);
      const float p2 = expf(Ib[(long long)(i + 16) * T] - lb[i + 16]);
      const float p3 = expf(Ib[(long long)(i + 24) * T] - lb[i + 24]);
      a0 = fmaf(p0, p0, a0);
      a1 = fmaf(p1, p1, a1);
      a2 = fmaf(p2, p2, a2);
      a3 = fmaf(p3, p3, a3);
    }
    for (; i < n; i += 8) {
      const float p0 = expf(Ib[(long long)i * T] - lb[i]);
      a0 = fmaf(p0, p0, a0);
    }
  }
  red[warp][lane] = (a0 + a1) + (a2 + a3);
  __syncthreads();
  if (warp == 0 && j < T) {
    float a = 0.f;
    for (int w = 0; w < 8; ++w) a += red[w][lane];
    s[(long long)b * T + j] = sqrtf(a / (float)n);
  }
}

// pool_kernel on 128 columns per CTA for T % 4 == 0: lane l owns columns
// 4l..4l+3 (16-byte loads), warp w the rows w, w+8, ... with four rows in
// flight, and pi^2 = e^{2 (I - lse)} = 2^(2 log2 e (I - lse)) is one MUFU op.
__global__ void __launch_bounds__(256) pool4_kernel(const float* I, const float* lse, float* s, int n, int T) {
  const int b = blockIdx.y, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int j = blockIdx.x * 128 + lane * 4;
  __shared__ float4 red[8][32];
  const float* Ib = I + (long long)b * n * T + j;
  const float* lb = lse + (long long)b * n;
  const float k2 = 2.0f * kLog2e;
  float4 a = make_float4(0.f, 0.f, 0.f, 0.f), c = a;
  if (j < T) {   // T % 4 == 0: all four columns are inside
    int i = warp;
    for (; i + 24 < n; i += 32) {
      const float4 x0 = *(const float4*)(Ib + (long long)i * T), x1 = *(const float4*)(Ib + (long long)(i + 8) * T);
      const float4 x2 = *(const float4*)(Ib + (long long)(i + 16) * T);
      const float4 x3 = *(const float4*)(Ib + (long long)(i + 24) * T);
      const float l0 = lb[i], l1 = lb[i + 8], l2 = lb[i + 16], l3 = lb[i + 24];
      a.x += ex2_approx((x0.x - l0) * k2) + ex2_approx((x2.x - l2) * k2);
      a.y += ex2_approx((x0.y - l0) * k2) + ex2_approx((x2.y - l2) * k2);
      a.z += ex2_approx((x0.z - l0) * k2) + ex2_approx((x2.z - l2) * k2);
      a.w += ex2_approx((x0.w - l0) * k2) + ex2_approx((x2.w - l2) * k2);
      c.x += ex2_approx((x1.x - l1) * k2) + ex2_approx((x3.x - l3) * k2);
      c.y += ex2_approx((x1.y - l1) * k2) + ex2_approx((x3.y - l3) * k2);
      c.z += ex2_approx((x1.z - l1) * k2) + ex2_approx((x3.z - l3) * k2);
      c.w += ex2_approx((x1.w - l1) * k2) + ex2_approx((x3.w - l3) * k2);
    }
    for (; i < n; i += 8) {
      const float4 x0 = *(const float4*)(Ib + (long long)i * T);
      const float l0 = lb[i];
      a.x += ex2_approx((x0.x - l0) * k2);
      a.y += ex2_approx((x0.y - l0) * k2);
      a.z += ex2_approx((x0.z - l0) * k2);
      a.w += ex2_approx((x0.w - l0) * k2);
    }
  }
  red[warp][lane] = make_float4(a.x + c.x, a.y + c.y, a.z + c.z, a.w + c.w);
  __syncthreads();
  if (warp == 0 && j < T) {
    float4 t4 = red[0][lane];
    for (int w = 1; w < 8; ++w) {
      const float4 u = red[w][lane];
      t4.x += u.x;
      t4.y += u.y;
      t4.z += u.z;
      t4.w += u.w;
    }
    const float inv = 1.0f / (float)n;
    *(float4*)(s + (long long)b * T + j) =
        make_float4(sqrtf(t4.x * inv), sqrtf(t4.y * inv), sqrtf(t4.z * inv), sqrtf(t4.w * inv));
  }
}

int launch_index_pool(const Dims& D, const float* I, const float2* part, int ntiles, float* lse, float* s,
                      cudaStream_t st) {
  lse_reduce_kernel<<<dim3(cdiv(D.n, 8), D.H), 256, 0, st>>>(part, lse, D.n, ntiles);
  if ((D.T & 3) == 0 && (((uintptr_t)I | (uintptr_t)s) & 15u) == 0)
    pool4_kernel<<<dim3(cdiv(D.T, 128), D.H), 256, 0, st>>>(I, lse, s, D.n, D.T);
  else
    pool_kernel<<<dim3(cdiv(D.T, 32), D.H), 256, 0, st>>>(I, lse, s, D.n, D.T);
  return 2;
}

}  // namespace arckv
