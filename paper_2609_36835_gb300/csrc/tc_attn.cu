// Softmax attention products on tcgen05 with fp32-grade accuracy:
//
//   value-attention logits (U_q q_i).(U_k k_j) = q''_i . k_j,
//       q''_i = U_k^T (U_q q_i)                       (Eq. value_context)
//   A V and softmax(l) V with A, softmax(l) row-stochastic and V the bf16 cache
//                                                     (Eq. value_context, Eq. value_lstsq's Y)
//
// In every product one operand is an exact bf16 input (K or V) and the other
// an fp32 value, which enters as a bf16 triple (h, m, l) summing to it within
// 2^-24; the kSplit3A GEMM issues h*B + m*B + l*B.
#include "kernels.h"
#include "tc_gemm.cuh"

namespace arckv {

__global__ void split3_kernel(const float* x, bf16* h, bf16* m, bf16* l, long long count) {
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < count;
       k += (long long)gridDim.x * blockDim.x)
    split3_bf16(x[k], h[k], m[k], l[k]);
}

// P = exp(X - shift_row) * mul_row as a bf16 triple [H][rows][ldc] (zero in the
// pad columns cols..ldc-1, and in column skip[row] when skip is given).
__global__ void probs_split3_kernel(const float* X, const float* shift, const float* mul, const int* skip, bf16* h,
                                    bf16* m, bf16* l, int rows, int cols, int ldc) {
  const int b = blockIdx.z, row = blockIdx.y;
  const long long rr = (long long)b * rows + row;
  const float sh = shift[rr], mu = mul[rr];
  const int sk = skip ? skip[rr] : -1;
  const float* x = X + rr * cols;
  const long long o = rr * ldc;
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < ldc; c += gridDim.x * blockDim.x) {
    const float p = (c < cols && c != sk) ? expf(x[c] - sh) * mu : 0.f;
    split3_bf16(p, h[o + c], m[o + c], l[o + c]);
  }
}

// VT[b][d][j] = V[b][j][d] (bf16), zero for T <= j < ldT.
__global__ void __launch_bounds__(256) transpose_v_kernel(const bf16* V, bf16* VT, int T, int ldT) {
  const int b = blockIdx.z, j0 = blockIdx.x * 32, d0 = blockIdx.y * 32;
  __shared__ bf16 tile[32][34];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const bf16 zero = __float2bfloat16_rn(0.f);
  for (int q = ty; q < 32; q += 8) {
    const int j = j0 + q;
    tile[q][tx] = (j < T) ? V[((long long)b * T + j) * 128 + d0 + tx] : zero;
  }
  __syncthreads();
  for (int q = ty; q < 32; q += 8) {
    const int j = j0 + tx;
    if (j < ldT) VT[((long long)b * 128 + d0 + q) * ldT + j] = tile[tx][q];
  }
}

// C[b] (rows x 128 or rows x N) = A3 B^T with A3 = (h, m, l) [H][rows][K] and B [H][N][K].
static int gemm_split3a(int H, int rows, int N, int K, int ldk, const bf16* h, const bf16* m, const bf16* l,
                        const bf16* B, float* C, int ldc, float alpha, DevStatus* stt, cudaStream_t st) {
  CUtensorMap mA, mA2, mA3, mB;
  if (!encode_bf16_map_3d(&mA, h, ldk, rows, H, 128) || !encode_bf16_map_3d(&mA2, m, ldk, rows, H, 128) ||
      !encode_bf16_map_3d(&mA3, l, ldk, rows, H, 128) || !encode_bf16_map_3d(&mB, B, ldk, N, H, 128))
    return -1;
  TcEpiStore epi{C, (long long)rows * ldc, ldc, alpha};
  const int kfull = (K + 63) / 64 * 64;
  if (launch_tc_gemm<128, kSplit3A>(mA, mB, mA2, mA, epi, H, rows, N, K, kfull, stt, st, 0, &mA3) != cudaSuccess)
    return -1;
  return 1;
}

int launch_value_logits_tc(const Dims& D, const float* qpp, bf16* q_h, bf16* q_m, bf16* q_l, const bf16* K,
                           float* logits, float2* part, DevStatus* stt, cudaStream_t st) {
  const long long cnt = (long long)D.H * D.n * 128;
  split3_kernel<<<min(cdiv(cnt, 256), 152 * 8), 256, 0, st>>>(qpp, q_h, q_m, q_l, cnt);
  CUtensorMap mA, mA2, mA3, mB;
  if (!encode_bf16_map_3d(&mA, q_h, 128, D.n, D.H, 128) || !encode_bf16_map_3d(&mA2, q_m, 128, D.n, D.H, 128) ||
      !encode_bf16_map_3d(&mA3, q_l, 128, D.n, D.H, 128) || !encode_bf16_map_3d(&mB, K, 128, D.T, D.H, 128))
    return -1;
  TcEpiStoreRowPart epi{{logits, (long long)D.n * D.T, D.T, 1.f}, part, cdiv(D.T, 128), 128};
  if (launch_tc_gemm<128, kSplit3A>(mA, mB, mA2, mA, epi, D.H, D.n, D.T, 128, 128, stt, st, 0, &mA3) != cudaSuccess)
    return -1;
  return 2;
}

int launch_split3(const float* x, bf16* h, bf16* m, bf16* l, long long count, cudaStream_t st) {
  split3_kernel<<<min(cdiv(count, 256), 152 * 8), 256, 0, st>>>(x, h, m, l, count);
  return 1;
}

int launch_transpose_v(const Dims& D, const bf16* V, bf16* VT, cudaStream_t st) {
  const int ldT = (D.T + 7) / 8 * 8;
  transpose_v_kernel<<<dim3(cdiv(ldT, 32), 4, D.H), 256, 0, st>>>(V, VT, D.T, ldT);
  return 1;
}

int launch_probs_v_tc(const Dims& D, const float* X, const float* shift, const float* mul, bf16* p_h, bf16* p_m,
                      bf16* p_l, const bf16* VT, float* out, DevStatus* stt, cudaStream_t st, const int* skip) {
  const int ldT = (D.T + 7) / 8 * 8;
  probs_split3_kernel<<<dim3(cdiv(ldT, 256 * 4), D.n, D.H), 256, 0, st>>>(X, shift, mul, skip, p_h, p_m, p_l, D.n,
                                                                          D.T, ldT);
  if (gemm_split3a(D.H, D.n, 128, ldT, ldT, p_h, p_m, p_l, VT, out, 128, 1.f, stt, st) < 0) return -1;
  return 2;
}

}  // namespace arckv
