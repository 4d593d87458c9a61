// Tensor-core stages of Sec. 3.4:
//   * reference logits l = scale Q K^T (bf16 operands are exact, one MMA per
//     product, fp32 accumulation);
//   * the anchor assignment kappa(j) = argmax_r u_j . u_{s_r}
//     (Eq. anchor_assignment) as a split-bf16 GEMM of the transposed profiles
//     U^T [T x n] against the anchor rows U_S^T [t x n] whose epilogue keeps
//     the row maximum (lowest r on ties) and merges it across column tiles
//     with a 64-bit atomicMax; the T x t similarity is never stored.
#include "kernels.h"
#include "tc_gemm.cuh"

namespace arckv {

struct TcEpiArgmax {
  unsigned long long* best;
  long long bbs;
  struct State {
    float bv;
    int bi, ncols, n0;
    bool row_ok;
  };
  __device__ __forceinline__ void init(State& s, int, int row, int n0, int M, int N) const {
    s.bv = -INFINITY;
    s.bi = -1;
    s.ncols = N - n0;
    s.n0 = n0;
    s.row_ok = row < M;
  }
  __device__ __forceinline__ void consume(State& s, int, int j, float (&v)[32]) const {
#pragma unroll
    for (int q = 0; q < 32; ++q)
      if (j * 32 + q < s.ncols && v[q] > s.bv) {
        s.bv = v[q];
        s.bi = s.n0 + j * 32 + q;
      }
  }
  __device__ __forceinline__ void finish(State& s, int b, int row, int, int, int) const {
    if (!s.row_ok || s.bi < 0) return;
    const unsigned long long key =
        ((unsigned long long)f32_ordered(s.bv) << 32) | (unsigned long long)(0xffffffffu - (unsigned int)s.bi);
    atomicMax(best + (long long)b * bbs + row, key);
  }
};

int launch_ref_logits_tc(const Dims& D, float scale, const bf16* Q, const bf16* K, float* L, float2* part,
                         DevStatus* stt, cudaStream_t st) {
  CUtensorMap mA, mB;
  if (!encode_bf16_map_3d(&mA, Q, D.d, D.n, D.H, 128) || !encode_bf16_map_3d(&mB, K, D.d, D.T, D.H, 128)) return -1;
  if (launch_tc_logits_rowpart<kPlain>(mA, mB, mA, mB, nullptr, L, scale, part, D.H, D.n, D.T, D.d, stt, st) !=
      cudaSuccess)
    return -1;
  return 1;
}

// Column statistics of the reference logits and the transposed response
// profiles (Sec. 3.4, Eq. response_profile), one CTA per (32 columns, head):
//   pass 1: per column the online (M_j, s1, s2) over the n rows, the 16 row
//     slices (warps) combined in slice order,
//       M_j = max_i l_ij,  s1 = sum_i e^{l_ij - M_j},  s2 = sum_i e^{2(l_ij - M_j)},
//       log phi_j = M_j + log s1 - log n  (the mass of Eq. mass_centroid),
//       invN_j = 1 / sqrt(s2);
//   pass 2 (Ut_hi given): U_ij = e^{l_ij - M_j} invN_j, re-read from L2 (the
//     strip was just streamed in), split into bf16 (hi, lo) and written
//     transposed, Ut[b][j][i] (row stride ldn >= n, a multiple of 8; the pad
//     columns n..ldn-1 are written as zeros).
// e^x is taken as 2^(x log2 e) after the subtraction.
__global__ void __launch_bounds__(512) col_profiles_kernel(const float* L, float* logphi, bf16* Ut_hi, bf16* Ut_lo,
                                                           int n, int T, int ldn) {
  const int b = blockIdx.y, lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int j0 = blockIdx.x * 32, j = j0 + lane;
  __shared__ float red[3][16][32];
  __shared__ float cstat[2][32];
  __shared__ float tile[64][33];
  const float* Lb = L + (long long)b * n * T + j;
  float mx = -INFINITY, s1 = 0.f, s2 = 0.f;
  if (j < T) {
    int i = w;
    for (; i + 48 < n; i += 64) {   // rows i, i + 16, i + 32, i + 48: one rescale per step
      const float v0 = Lb[(long long)i * T], v1 = Lb[(long long)(i + 16) * T];
      const float v2 = Lb[(long long)(i + 32) * T], v3 = Lb[(long long)(i + 48) * T];
      const float m4 = fmaxf(fmaxf(v0, v1), fmaxf(v2, v3));
      if (m4 > mx) {
        const float r = (mx == -INFINITY) ? 0.f : ex2_approx((mx - m4) * kLog2e);
        s1 *= r;
        s2 *= r * r;
        mx = m4;
      }
      const float e0 = ex2_approx((v0 - mx) * kLog2e), e1 = ex2_approx((v1 - mx) * kLog2e);
      const float e2 = ex2_approx((v2 - mx) * kLog2e), e3 = ex2_approx((v3 - mx) * kLog2e);
      s1 += (e0 + e1) + (e2 + e3);
      s2 += (e0 * e0 + e1 * e1) + (e2 * e2 + e3 * e3);
    }
    for (; i < n; i += 16) {
      const float v = Lb[(long long)i * T];
      if (v > mx) {
        const float r = (mx == -INFINITY) ? 0.f : ex2_approx((mx - v) * kLog2e);
        s1 = fmaf(s1, r, 1.f);
        s2 = fmaf(s2, r * r, 1.f);
        mx = v;
      } else {
        const float e = ex2_approx((v - mx) * kLog2e);
        s1 += e;
        s2 = fmaf(e, e, s2);
      }
    }
  }
  red[0][w][lane] = mx;
  red[1][w][lane] = s1;
  red[2][w][lane] = s2;
  __syncthreads();
  if (w == 0) {
    float M = -INFINITY;
    for (int q = 0; q < 16; ++q) M = fmaxf(M, red[0][q][lane]);
    float S1 = 0.f, S2 = 0.f;
    for (int q = 0; q < 16; ++q) {
      if (red[0][q][lane] == -INFINITY) continue;
      const float r = ex2_approx((red[0][q][lane] - M) * kLog2e);
      S1 = fmaf(red[1][q][lane], r, S1);
      S2 = fmaf(red[2][q][lane], r * r, S2);
    }
    if (j < T) logphi[(long long)b * T + j] = M + logf(S1) - logf((float)n);
    cstat[0][lane] = M;
    cstat[1][lane] = j < T ? 1.0f / sqrtf(S2) : 0.f;
  }
  __syncthreads();
  if (Ut_hi == nullptr) return;
  const float cm = cstat[0][lane], ci = cstat[1][lane];
  for (int i0 = 0; i0 < ldn; i0 += 64) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int r = w + 16 * k, i = i0 + r;
      tile[r][lane] = (i < n && j < T) ? ex2_approx((Lb[(long long)i * T] - cm) * kLog2e) * ci : 0.f;
    }
    __syncthreads();
    // warp w writes columns 2w and 2w + 1, lane l rows i0 + 2l and i0 + 2l + 1 (ldn even)
#pragma unroll
    for (int c = 2 * w; c < 2 * w + 2; ++c) {
      const int jj = j0 + c, i = i0 + 2 * lane;
      if (jj < T && i < ldn) {
        bf16 h0, l0, h1, l1;
        split_bf16(tile[2 * lane][c], h0, l0);
        split_bf16(tile[2 * lane + 1][c], h1, l1);
        const long long o = ((long long)b * T + jj) * ldn + i;
        *(__nv_bfloat162*)(Ut_hi + o) = __halves2bfloat162(h0, h1);
        *(__nv_bfloat162*)(Ut_lo + o) = __halves2bfloat162(l0, l1);
      }
    }
    __syncthreads();
  }
}

int launch_col_profiles(const Dims& D, const float* L, float* logphi, bf16* Ut_hi, bf16* Ut_lo, cudaStream_t st) {
  const int ldn = (D.n + 7) / 8 * 8;
  // each CTA re-reads its n x 32 strip from L2: with n > 1024 a shared-memory
  // reservation keeps at most two CTAs per SM so the live strips fit in L2
  const int smem = D.n > 1024 ? 80 * 1024 : 0;
  if (smem > 0 && cudaFuncSetAttribute(col_profiles_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
                      cudaSuccess)
    return -1;
  col_profiles_kernel<<<dim3(cdiv(D.T, 32), D.H), 512, smem, st>>>(L, logphi, Ut_hi, Ut_lo, D.n, D.T, ldn);
  return 1;
}

// UtS[b][r] = Ut[b][S_r] (hi and lo rows).
__global__ void gather_anchor_rows_kernel(const bf16* Ut_hi, const bf16* Ut_lo, const int* anchors, bf16* S_hi,
                                          bf16* S_lo, int T, int t, int ldn) {
  const int b = blockIdx.y, r = blockIdx.x;
  const int j = anchors[(long long)b * t + r];
  const long long src = ((long long)b * T + j) * ldn, dst = ((long long)b * t + r) * ldn;
  for (int i = threadIdx.x; i < ldn; i += blockDim.x) {
    S_hi[dst + i] = Ut_hi[src + i];
    S_lo[dst + i] = Ut_lo[src + i];
  }
}

__global__ void decode_assign_kernel2(const unsigned long long* best, int* kappa, long long count) {
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < count;
       k += (long long)gridDim.x * blockDim.x) {
    const unsigned long long v = best[k];
    kappa[k] = v ? (int)(0xffffffffu - (unsigned int)(v & 0xffffffffull)) : 0;
  }
}

__global__ void anchor_self_assign_kernel2(const int* anchors, int* kappa, int T, int t, int H) {
  const long long total = (long long)H * t;
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < total;
       k += (long long)gridDim.x * blockDim.x) {
    const long long b = k / t;
    kappa[b * T + anchors[k]] = (int)(k - b * t);
  }
}

int launch_assign_tc(const Dims& D, const float* L, float* logphi, const int* anchors, bf16* Ut_hi, bf16* Ut_lo,
                     bf16* S_hi, bf16* S_lo, unsigned long long* best, int* kappa, DevStatus* stt, cudaStream_t st) {
  const int ldn = (D.n + 7) / 8 * 8;
  if (launch_col_profiles(D, L, logphi, Ut_hi, Ut_lo, st) < 0) return -1;
  gather_anchor_rows_kernel<<<dim3(D.t, D.H), 128, 0, st>>>(Ut_hi, Ut_lo, anchors, S_hi, S_lo, D.T, D.t, ldn);
  cudaMemsetAsync(best, 0, sizeof(unsigned long long) * (size_t)D.H * D.T, st);
  CUtensorMap mA, mA2, mB, mB2;
  if (!encode_bf16_map_3d(&mA, Ut_hi, ldn, D.T, D.H, 128) || !encode_bf16_map_3d(&mA2, Ut_lo, ldn, D.T, D.H, 128) ||
      !encode_bf16_map_3d(&mB, S_hi, ldn, D.t, D.H, 128) || !encode_bf16_map_3d(&mB2, S_lo, ldn, D.t, D.H, 128))
    return -1;
  TcEpiArgmax epi{best, D.T};
  const int kfull = (ldn + 63) / 64 * 64;
  if (launch_tc_gemm<128, kSplit>(mA, mB, mA2, mB2, epi, D.H, D.T, D.t, ldn, kfull, stt, st) != cudaSuccess)
    return -1;
  const long long cnt = (long long)D.H * D.T;
  decode_assign_kernel2<<<min(cdiv(cnt, 256), 152 * 8), 256, 0, st>>>(best, kappa, cnt);
  anchor_self_assign_kernel2<<<cdiv((long long)D.H * D.t, 256), 256, 0, st>>>(anchors, kappa, D.T, D.t, D.H);
  return 5;
}

}  // namespace arckv
