// Key-side indexer features on tcgen05 (App. A.1 Eq. indexer_projection):
//
//   k_bar_j,a = N((L_k k_j + L_v v_j)_a)
//
// as ONE GEMM of the concatenated cache rows [k_j | v_j] (K = 2d) against the
// concatenated weights [L_k | L_v] (H_I d_I rows), so K and V are streamed
// from HBM once.  All operands are bf16 inputs, so one MMA per product with
// fp32 accumulation is exact up to the accumulation.  Each 128-wide output
// tile is one d_I block: the epilogue RMS-normalises it per row
// (N(z) = z / sqrt(|z|^2/d_I + 1e-6)) and stores it as a split-bf16 pair for
// the index-logit GEMM.
#include "kernels.h"
#include "tc_gemm.cuh"

namespace arckv {

struct TcEpiKeyFeat {
  bf16* kbar_hi;
  bf16* kbar_lo;
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
  }
};

int launch_key_features_tc(const Dims& D, const bf16* K, const bf16* V, const bf16* L_k, const bf16* L_v,
                           bf16* kbar_hi, bf16* kbar_lo, DevStatus* stt, cudaStream_t st) {
  CUtensorMap mA, mA2, mB, mB2;
  if (!encode_bf16_map_3d(&mA, K, D.d, D.T, D.H, 128) || !encode_bf16_map_3d(&mA2, V, D.d, D.T, D.H, 128) ||
      !encode_bf16_map_3d(&mB, L_k, D.d, D.HD, D.H, 128) || !encode_bf16_map_3d(&mB2, L_v, D.d, D.HD, D.H, 128))
    return -1;
  TcEpiKeyFeat epi{kbar_hi, kbar_lo, D.T, D.HD};
  if (launch_tc_gemm<128, kConcat>(mA, mB, mA2, mB2, epi, D.H, D.T, D.HD, 2 * D.d, 2 * D.d, stt, st, D.d) !=
      cudaSuccess)
    return -1;
  return 1;
}

}  // namespace arckv
