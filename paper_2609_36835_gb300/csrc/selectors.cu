// Attention-only and value-aware anchor scores of App. B.1
// (Eq. background_value_selectors), on the reference logits l = scale Q K^T
// of the full cache, p = softmax(l), O = p V:
//
//   HA: s_j = (mean_i p_ij^2)^(1/2)                      -- the pooling of Sec. 3.3
//                                                           applied to l instead of I;
//   VI: s_j = (mean_i D_ij^2 / (||O_i||^2 + eps))^(1/2),
//       D_ij = ||O_i - O_i^(-j)|| = p_ij / (1 - p_ij) ||v_j - O_i||.
//
// VI is evaluated without forming any n x T array beyond l itself:
//   * for j != a_i (a_i the first column holding row i's maximum z_i):
//       p/(1-p) = e / (m_i - e), e = e^{l_ij - z_i}, m_i = sum_u e^{l_iu - z_i}
//       (m_i - e >= 1 because column a_i contributes 1), and
//       ||v_j - O_i||^2 = ||v_j||^2 - 2 v_j.O_i + ||O_i||^2, with v_j.O_i = (Y V^T)_ij
//       from a split-3 tcgen05 GEMM whose epilogue forms the terms and sums
//       them over each warp's 32 rows with a transposing butterfly;
//   * for j = a_i, where p rounds to 1 and O_i to v_a, the same quantity is
//       p_a ||v_a - O_i^(-a)|| (exact algebra: O_i = p_a v_a + (1 - p_a) O_i^(-a)),
//       O_i^(-a) = softmax over the other keys (its own max shift z2_i) times V.
#include <climits>

#include "kernels.h"
#include "tc_gemm.cuh"

namespace arckv {

// Per row of l [H][n][T]: a_i, z2_i = max_{u != a_i} l_iu, mul2_i = 1 / sum_{u != a_i} e^{l_iu - z2_i}
// (0 when T = 1).  One warp per row.
__global__ void __launch_bounds__(256) vi_row_kernel(const float* L, int n, int T, int* amax, float* z2,
                                                     float* mul2) {
  const int b = blockIdx.y, row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= n) return;
  const long long r = (long long)b * n + row;
  const float* x = L + r * T;
  float mx = -INFINITY;
  int ai = INT_MAX;
  for (int j = lane; j < T; j += 32) {
    const float v = x[j];
    if (v > mx) {
      mx = v;
      ai = j;
    }
  }
  const float gmax = warp_max(mx);
  const int a = (int)__reduce_min_sync(0xffffffffu, (unsigned)(mx == gmax ? ai : INT_MAX));
  float m2 = -INFINITY, s2 = 0.f;
  for (int j = lane; j < T; j += 32)
    if (j != a) lse_combine(m2, s2, x[j], 1.f);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, m2, o), os = __shfl_xor_sync(0xffffffffu, s2, o);
    lse_combine(m2, s2, om, os);
  }
  if (lane == 0) {
    amax[r] = a;
    z2[r] = m2;
    mul2[r] = s2 > 0.f ? 1.0f / s2 : 0.f;
  }
}

// Per row: p_a = 1 / (1 + e^{z2 - z} / mul2), Da_i = p_a ||v_a - Om_i||, oo_i = ||Y_i||^2.
__global__ void __launch_bounds__(256) vi_rowfinish_kernel(const float* z, const int* amax, const float* z2,
                                                           const float* mul2, const bf16* V, const float* Om,
                                                           const float* Y, int n, int T, float* Da, float* oo) {
  const int b = blockIdx.y, row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= n) return;
  const long long r = (long long)b * n + row;
  const int a = amax[r];
  const float rest = mul2[r] > 0.f ? 1.0f / mul2[r] : 0.f;
  const float pa = 1.0f / (1.0f + rest * expf(z2[r] - z[r]));
  float dd = 0.f, yy = 0.f;
  for (int d = lane; d < 128; d += 32) {
    const float df = __bfloat162float(V[((long long)b * T + a) * 128 + d]) - Om[r * 128 + d];
    const float y = Y[r * 128 + d];
    dd = fmaf(df, df, dd);
    yy = fmaf(y, y, yy);
  }
  dd = warp_sum(dd);
  yy = warp_sum(yy);
  if (lane == 0) {
    Da[r] = pa * sqrtf(dd);
    oo[r] = yy;
  }
}

// out[k] = ||v_k||^2 for the cache rows V [rows][128] (one warp per row)
__global__ void __launch_bounds__(256) row_norm2_kernel(const bf16* V, long long rows, float* out) {
  const long long k = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (k >= rows) return;
  const uint2 u = *(const uint2*)(V + k * 128 + lane * 4);
  const float2 f0 = __bfloat1622float2(*(const __nv_bfloat162*)&u.x), f1 = __bfloat1622float2(*(const __nv_bfloat162*)&u.y);
  const float a = warp_sum(f0.x * f0.x + f0.y * f0.y + f1.x * f1.x + f1.y * f1.y);
  if (lane == 0) out[k] = a;
}

// Epilogue of G = Y V^T (row i, columns n0 + 32j + q): the VI terms
// D_ij^2 / (||O_i||^2 + eps), summed over the warp's 32 rows; lane q writes the
// column sum into part[b][row / 32][col].
struct TcEpiVI {
  const float* L;     // [H][n][T] reference logits
  const float* z;     // [H][n] row max
  const float* m;     // [H][n] sum_u e^{l_iu - z_i}
  const int* amax;    // [H][n]
  const float* Da;    // [H][n]
  const float* oo;    // [H][n] ||O_i||^2
  const float* vv;    // [H][T] ||v_j||^2
  float* part;        // [H][ceil(n / 32)][T]
  int n, T, nb;
  float eps;
  struct State {
    const float* lrow;
    const float* vvb;
    float* prow;
    float zi, mi, Dai2, ooi, inv;
    int ai, n0;
    bool row_ok, blk_ok;   // this row / this warp's 32-row block hold reference rows
  };
  __device__ __forceinline__ void init(State& s, int b, int row, int n0, int M, int) const {
    s.row_ok = row < M;
    s.blk_ok = (row & ~31) < M;
    const long long r = (long long)b * n + (s.row_ok ? row : 0);
    s.lrow = L + r * T + n0;
    s.vvb = vv + (long long)b * T + n0;
    s.prow = part + ((long long)b * nb + (s.blk_ok ? row / 32 : 0)) * T + n0;
    s.zi = z[r];
    s.mi = m[r];
    s.Dai2 = Da[r] * Da[r];
    s.ooi = oo[r];
    s.inv = 1.0f / (s.ooi + eps);
    s.ai = amax[r];
    s.n0 = n0;
  }
  __device__ __forceinline__ void consume(State& s, int, int j, float (&v)[32]) const {
    const int lane = threadIdx.x & 31;
    float t[32];
#pragma unroll
    for (int q = 0; q < 32; ++q) {
      const int col = s.n0 + j * 32 + q;
      float term = 0.f;
      if (s.row_ok && col < T) {
        float d2;
        if (col == s.ai) {
          d2 = s.Dai2;
        } else {
          const float e = expf(s.lrow[j * 32 + q] - s.zi);
          const float ratio = e / (s.mi - e);
          d2 = ratio * ratio * fmaxf(s.vvb[j * 32 + q] - 2.0f * v[q] + s.ooi, 0.f);
        }
        term = d2 * s.inv;
      }
      t[q] = term;
    }
    // transposing butterfly over the warp's 32 rows: lane q ends with column q's sum
#pragma unroll
    for (int w = 16; w >= 1; w >>= 1) {
      const bool up = lane & w;
#pragma unroll
      for (int q = 0; q < w; ++q) {
        const float mine = up ? t[w + q] : t[q], other = up ? t[q] : t[w + q];
        t[q] = mine + __shfl_xor_sync(0xffffffffu, other, w);
      }
    }
    // a warp's rows are 32 consecutive rows from a multiple of 32
    if (s.blk_ok && s.n0 + j * 32 + lane < T) s.prow[j * 32 + lane] = t[0];
  }
  __device__ __forceinline__ void finish(State&, int, int, int, int, int) const {}
};

// s_j = (sum_r part[r][j] / n)^(1/2)
__global__ void vi_reduce_kernel(const float* part, int nb, int n, int T, float* s) {
  const int b = blockIdx.y, j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= T) return;
  float a = 0.f;
  for (int r = 0; r < nb; ++r) a += part[((long long)b * nb + r) * T + j];
  s[(long long)b * T + j] = sqrtf(a / (float)n);
}

int launch_vi_scores(const Dims& D, const float* L, const float* z, const float* m, const float* Y, const bf16* V,
                     const bf16* VT, const ViBufs& B, float* s, float eps, DevStatus* stt, cudaStream_t st) {
  int nl = 0;
  vi_row_kernel<<<dim3(cdiv(D.n, 8), D.H), 256, 0, st>>>(L, D.n, D.T, B.amax, B.z2, B.mul2);
  ++nl;
  // O^(-a): softmax over the keys other than a_i, times V
  const int r = launch_probs_v_tc(D, L, B.z2, B.mul2, B.p_h, B.p_m, B.p_l, VT, B.Om, stt, st, B.amax);
  if (r < 0) return -1;
  nl += r;
  vi_rowfinish_kernel<<<dim3(cdiv(D.n, 8), D.H), 256, 0, st>>>(z, B.amax, B.z2, B.mul2, V, B.Om, Y, D.n, D.T, B.Da,
                                                              B.oo);
  row_norm2_kernel<<<cdiv((long long)D.H * D.T, 8), 256, 0, st>>>(V, (long long)D.H * D.T, B.vv);
  nl += 2;
  nl += launch_split3(Y, B.y_h, B.y_m, B.y_l, (long long)D.H * D.n * 128, st);
  CUtensorMap mA, mA2, mA3, mB;
  if (!encode_bf16_map_3d(&mA, B.y_h, 128, D.n, D.H, 128) || !encode_bf16_map_3d(&mA2, B.y_m, 128, D.n, D.H, 128) ||
      !encode_bf16_map_3d(&mA3, B.y_l, 128, D.n, D.H, 128) || !encode_bf16_map_3d(&mB, V, 128, D.T, D.H, 128))
    return -1;
  const int nb = cdiv(D.n, 32);
  TcEpiVI epi{L, z, m, B.amax, B.Da, B.oo, B.vv, B.colpart, D.n, D.T, nb, eps};
  if (launch_tc_gemm<128, kSplit3A>(mA, mB, mA2, mA, epi, D.H, D.n, D.T, 128, 128, stt, st, 0, &mA3) != cudaSuccess)
    return -1;
  vi_reduce_kernel<<<dim3(cdiv(D.T, 256), D.H), 256, 0, st>>>(B.colpart, nb, D.n, D.T, s);
  return nl + 2;
}

}  // namespace arckv
