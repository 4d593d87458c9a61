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

// One CTA per (64 rows i x 32 columns j of l, head): U_ij = exp(l_ij - M_j) * invN_j,
// split into bf16 (hi, lo) and written transposed, Ut[b][j][i] (row stride
// ldn >= n, a multiple of 8; the pad columns n..ldn-1 are written as zeros).
// Reads are 128-byte row segments; each warp writes 64 i-values of one j as
// bf16 pairs (128 bytes per tensor).
__global__ void __launch_bounds__(256) profiles_t_kernel(const float* L, const float* colM, const float* colInvN,
                                                         bf16* Ut_hi, bf16* Ut_lo, int n, int T, int ldn) {
  const int b = blockIdx.z, j0 = blockIdx.x * 32, i0 = blockIdx.y * 64;
  __shared__ float tile[64][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const float* Lb = L + (long long)b * n * T;
  const int j = j0 + tx;
  const float cm = j < T ? colM[(long long)b * T + j] : 0.f, ci = j < T ? colInvN[(long long)b * T + j] : 0.f;
  for (int r = ty; r < 64; r += 8) {
    const int i = i0 + r;
    float u = 0.f;
    if (i < n && j < T) u = expf(Lb[(long long)i * T + j] - cm) * ci;
    tile[r][tx] = u;
  }
  __syncthreads();
  for (int c = ty; c < 32; c += 8) {
    const int jj = j0 + c, i = i0 + 2 * tx;
    if (jj < T && i < ldn) {   // ldn even: i + 1 < ldn as well
      bf16 h0, l0, h1, l1;
      split_bf16(tile[2 * tx][c], h0, l0);
      split_bf16(tile[2 * tx + 1][c], h1, l1);
      const long long o = ((long long)b * T + jj) * ldn + i;
      *(__nv_bfloat162*)(Ut_hi + o) = __halves2bfloat162(h0, h1);
      *(__nv_bfloat162*)(Ut_lo + o) = __halves2bfloat162(l0, l1);
    }
  }
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

int launch_assign_tc(const Dims& D, const float* L, const float* colM, const float* colInvN, const int* anchors,
                     bf16* Ut_hi, bf16* Ut_lo, bf16* S_hi, bf16* S_lo, unsigned long long* best, int* kappa,
                     DevStatus* stt, cudaStream_t st) {
  const int ldn = (D.n + 7) / 8 * 8;
  profiles_t_kernel<<<dim3(cdiv(D.T, 32), cdiv(ldn, 64), D.H), 256, 0, st>>>(L, colM, colInvN, Ut_hi, Ut_lo, D.n,
                                                                             D.T, ldn);
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
