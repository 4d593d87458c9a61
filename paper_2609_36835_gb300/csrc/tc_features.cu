// Key-side indexer features on tcgen05 (App. A.1 Eq. indexer_projection):
//
//   k_bar_j,a = N((L_k k_j + L_v v_j)_a),   Uk_j = U_k k_j,   Uv_j = U_v v_j
//
// as ONE GEMM of the concatenated cache rows [k_j | v_j] (K = 2d) against the
// per-head stacked weights
//   W = [[L_k | L_v];  [U_k | 0];  [0 | U_v]]        (H_I d_I + 2 d_A rows),
// so K and V are streamed from HBM once.  All operands are bf16 inputs, so one
// MMA per product with fp32 accumulation is exact up to the accumulation.
// Each 128-wide output tile of the first H_I d_I columns is one d_I block:
// the epilogue RMS-normalises it per row (N(z) = z / sqrt(|z|^2/d_I + 1e-6))
// and stores it as a split-bf16 pair for the index-logit GEMM.
#include "kernels.h"
#include "tc_gemm.cuh"

namespace arckv {

// W1 = [L_k; U_k; 0], W2 = [L_v; 0; U_v], each [H][HD + 2 d_A][d] bf16.
__global__ void stack_key_weights_kernel(const bf16* L_k, const bf16* L_v, const bf16* U_k, const bf16* U_v,
                                         bf16* W1, bf16* W2, int HD, int d) {
  const int b = blockIdx.y, row = blockIdx.x;
  const int NW = HD + 256;
  const bf16 zero = __float2bfloat16_rn(0.f);
  bf16* w1 = W1 + ((long long)b * NW + row) * d;
  bf16* w2 = W2 + ((long long)b * NW + row) * d;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    if (row < HD) {
      w1[c] = L_k[((long long)b * HD + row) * d + c];
      w2[c] = L_v[((long long)b * HD + row) * d + c];
    } else if (row < HD + 128) {
      w1[c] = U_k[((long long)b * 128 + row - HD) * d + c];
      w2[c] = zero;
    } else {
      w1[c] = zero;
      w2[c] = U_v[((long long)b * 128 + row - HD - 128) * d + c];
    }
  }
}

struct TcEpiKeyFeat {
  bf16* kbar_hi;
  bf16* kbar_lo;
  float* Uk;
  float* Uv;
  int T, HD;
  struct State {
    float acc[128];
    bool row_ok;
  };
  __device__ __forceinline__ void init(State& s, int, int row, int, int M, int) const { s.row_ok = row < M; }
  __device__ __forceinline__ void consume(State& s, int, int j, float (&v)[32]) const {
#pragma unroll
    for (int q = 0; q < 32; ++q) s.acc[j * 32 + q] = v[q];
  }
  __device__ __forceinline__ void finish(State& s, int b, int row, int n0, int, int) const {
    if (!s.row_ok) return;
    if (n0 < HD) {
      float ss = 0.f;
#pragma unroll
      for (int q = 0; q < 128; ++q) ss = fmaf(s.acc[q], s.acc[q], ss);
      const float sc = 1.0f / sqrtf(ss * (1.0f / 128.0f) + 1e-6f);
      const long long o = ((long long)b * T + row) * HD + n0;
#pragma unroll
      for (int q = 0; q < 128; q += 8) {
        __align__(16) bf16 hi[8], lo[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) split_bf16(s.acc[q + e] * sc, hi[e], lo[e]);
        *(uint4*)(kbar_hi + o + q) = *(const uint4*)hi;
        *(uint4*)(kbar_lo + o + q) = *(const uint4*)lo;
      }
    } else {
      float* dst = (n0 < HD + 128 ? Uk : Uv) + ((long long)b * T + row) * 128;
#pragma unroll
      for (int q = 0; q < 128; q += 4) *(float4*)(dst + q) = make_float4(s.acc[q], s.acc[q + 1], s.acc[q + 2], s.acc[q + 3]);
    }
  }
};

int launch_key_features_tc(const Dims& D, const bf16* K, const bf16* V, const bf16* L_k, const bf16* L_v,
                           const bf16* U_k, const bf16* U_v, bf16* W1, bf16* W2, bf16* kbar_hi, bf16* kbar_lo,
                           float* Uk, float* Uv, DevStatus* stt, cudaStream_t st) {
  const int NW = D.HD + 2 * D.d_A;
  stack_key_weights_kernel<<<dim3(NW, D.H), 128, 0, st>>>(L_k, L_v, U_k, U_v, W1, W2, D.HD, D.d);
  CUtensorMap mA, mA2, mB, mB2;
  if (!encode_bf16_map_3d(&mA, K, D.d, D.T, D.H, 128) || !encode_bf16_map_3d(&mA2, V, D.d, D.T, D.H, 128) ||
      !encode_bf16_map_3d(&mB, W1, D.d, NW, D.H, 128) || !encode_bf16_map_3d(&mB2, W2, D.d, NW, D.H, 128))
    return -1;
  TcEpiKeyFeat epi{kbar_hi, kbar_lo, Uk, Uv, D.T, D.HD};
  if (launch_tc_gemm<128, kConcat>(mA, mB, mA2, mB2, epi, D.H, D.T, NW, 2 * D.d, 2 * D.d, stt, st, D.d) !=
      cudaSuccess)
    return -1;
  return 2;
}

}  // namespace arckv
