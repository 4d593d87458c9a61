// Indexer features on tcgen05 (App. A.1 Eq. indexer_projection):
//
//   k_bar_j,a = N((L_k k_j + L_v v_j)_a),   q_bar_i,a = N((L_q q_i + L_c c_i)_a)
//
// Key side:
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

// Block-normalised split-bf16 features: each 128-wide output tile is one
// d_I block, N(z) = z / sqrt(|z|^2 / 128 + 1e-6) per row, stored as (hi, lo)
// bf16 [H][rows][HD].  The row's sum of squares runs in eight independent
// chains; the four 32-row x 64-column boxes (hi and lo, two column halves)
// leave through 128-byte-swizzled staging and TMA stores (rows past `rows`
// fall outside the maps and are not written).
struct TcEpiBlockNorm {
  CUtensorMap map_hi, map_lo;   // [H][rows][HD] bf16, box {64, 32, 1}, 128-byte swizzle
  int rows;
  static constexpr int kStageBytes = 4 * 4096;
  struct State {
    float acc[128];
    uint8_t* stage;
    int b, y, n0;
  };
  __device__ __forceinline__ void init(State& s, int b, int row, int n0, int, int) const {
    s.b = b;
    s.y = row & ~31;
    s.n0 = n0;
  }
  __device__ __forceinline__ void attach(State& s, uint8_t* stage, int*) const { s.stage = stage; }
  __device__ __forceinline__ void consume(State& s, int, int j, float (&v)[32]) const {
#pragma unroll
    for (int q = 0; q < 32; ++q) s.acc[j * 32 + q] = v[q];
  }
  __device__ __forceinline__ void finish(State& s, int, int, int, int, int) const {
    float ss8[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) ss8[k] = 0.f;
#pragma unroll
    for (int q = 0; q < 128; ++q) ss8[q & 7] = fmaf(s.acc[q], s.acc[q], ss8[q & 7]);
    const float ss = ((ss8[0] + ss8[1]) + (ss8[2] + ss8[3])) + ((ss8[4] + ss8[5]) + (ss8[6] + ss8[7]));
    const float sc = 1.0f / sqrtf(ss * (1.0f / 128.0f) + 1e-6f);
    const int lane = threadIdx.x & 31;
    if (lane == 0) tc::bulk_wait_read<0>();   // the previous tile's boxes have left the staging buffers
    __syncwarp();
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      uint8_t* bh = s.stage + (2 * h) * 4096;
      uint8_t* bl = s.stage + (2 * h + 1) * 4096;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        __align__(16) bf16 hi[8], lo[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) split_bf16(s.acc[64 * h + 8 * k + e] * sc, hi[e], lo[e]);
        const int off = lane * 128 + ((k ^ (lane & 7)) << 4);
        *(uint4*)(bh + off) = *(const uint4*)hi;
        *(uint4*)(bl + off) = *(const uint4*)lo;
      }
    }
    tc::fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0 && s.y < rows) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        tc::tma_store_3d(&map_hi, s.stage + (2 * h) * 4096, s.n0 + 64 * h, s.y, s.b);
        tc::tma_store_3d(&map_lo, s.stage + (2 * h + 1) * 4096, s.n0 + 64 * h, s.y, s.b);
      }
      tc::bulk_commit();
    }
  }
};

static bool block_norm_epi(TcEpiBlockNorm& epi, bf16* hi, bf16* lo, int H, int rows, int HD) {
  epi.rows = rows;
  return encode_bf16_map_3d(&epi.map_hi, hi, HD, rows, H, 32) && encode_bf16_map_3d(&epi.map_lo, lo, HD, rows, H, 32);
}

int launch_key_features_tc(const Dims& D, const bf16* K, const bf16* V, const bf16* L_k, const bf16* L_v,
                           bf16* kbar_hi, bf16* kbar_lo, DevStatus* stt, cudaStream_t st) {
  CUtensorMap mA, mA2, mB, mB2;
  if (!encode_bf16_map_3d(&mA, K, D.d, D.T, D.H, 128) || !encode_bf16_map_3d(&mA2, V, D.d, D.T, D.H, 128) ||
      !encode_bf16_map_3d(&mB, L_k, D.d, D.HD, D.H, 128) || !encode_bf16_map_3d(&mB2, L_v, D.d, D.HD, D.H, 128))
    return -1;
  TcEpiBlockNorm epi{};
  if (!block_norm_epi(epi, kbar_hi, kbar_lo, D.H, D.T, D.HD)) return -1;
  if (launch_tc_gemm<128, kConcat>(mA, mB, mA2, mB2, epi, D.H, D.T, D.HD, 2 * D.d, 2 * D.d, stt, st, D.d) !=
      cudaSuccess)
    return -1;
  return 1;
}

// Query-side q_bar_i,a = N((L_q q_i + L_c c_i)_a) (Eq. indexer_projection) on
// tcgen05: the fp32 value context c enters as a bf16 triple, so the operands
// are concatenated along K as
//   A = [q | c_h | c_m | c_l]  [n][4 * 128],   B = [L_q | L_c | L_c | L_c]  [HD][4 * 128]
// and one plain GEMM gives L_q q + L_c (c_h + c_m + c_l) with exact bf16 products.
// The c triple is written into A by the GEMM that forms c; qcat_kernel adds q.
__global__ void __launch_bounds__(256) qcat_kernel(const bf16* Q, bf16* A, int n) {
  const int b = blockIdx.y, i = blockIdx.x * 16 + (threadIdx.x >> 4), k = (threadIdx.x & 15) * 8;
  if (i >= n) return;
  const long long r = (long long)b * n + i;
  *(uint4*)(A + r * 512 + k) = *(const uint4*)(Q + r * 128 + k);
}
__global__ void __launch_bounds__(256) wcat_kernel(const bf16* L_q, const bf16* L_c, bf16* W, long long rows) {
  const long long r = blockIdx.x * 2ll + (threadIdx.x >> 7);
  const int k = threadIdx.x & 127;
  if (r >= rows) return;
  bf16* w = W + r * 512;
  const bf16 c = L_c[r * 128 + k];
  w[k] = L_q[r * 128 + k];
  w[128 + k] = c;
  w[256 + k] = c;
  w[384 + k] = c;
}

int launch_query_proj_tc(const Dims& D, const bf16* Q, const bf16* L_q, const bf16* L_c, bf16* qcat, bf16* wcat,
                         bf16* qbar_hi, bf16* qbar_lo, DevStatus* stt, cudaStream_t st) {
  qcat_kernel<<<dim3(cdiv(D.n, 16), D.H), 256, 0, st>>>(Q, qcat, D.n);
  const long long wrows = (long long)D.H * D.HD;
  wcat_kernel<<<(unsigned)cdiv(wrows, 2), 256, 0, st>>>(L_q, L_c, wcat, wrows);
  CUtensorMap mA, mB;
  if (!encode_bf16_map_3d(&mA, qcat, 512, D.n, D.H, 128) || !encode_bf16_map_3d(&mB, wcat, 512, D.HD, D.H, 128))
    return -1;
  TcEpiBlockNorm epi{};
  if (!block_norm_epi(epi, qbar_hi, qbar_lo, D.H, D.n, D.HD)) return -1;
  if (launch_tc_gemm<128, kPlain>(mA, mB, mA, mB, epi, D.H, D.n, D.HD, 512, 512, stt, st) != cudaSuccess) return -1;
  return 3;
}

}  // namespace arckv
