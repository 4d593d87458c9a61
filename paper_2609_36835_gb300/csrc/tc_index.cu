// Index logits on tcgen05 (Sec. 3.3; App. A.1 Eq. pairwise_index_score):
//
//   I_ij = sum_a w_ia LeakyReLU_0.1(q_bar_ia . k_bar_ja / sqrt(d_I))
//
// as one split-bf16 tensor-core GEMM of q_bar [n x H_I d_I] against
// k_bar [T x H_I d_I] whose K dimension is consumed one index head (d_I = 128
// columns) at a time: every head's partial dot products land in their own
// TMEM accumulator and the epilogue folds them through the LeakyReLU and the
// row's head weight w_ia before the next head is added.  The epilogue then
// writes the row-softmax partials (max, sum of exp) of each kIndexPartW
// columns and the I tile.
#include "kernels.h"
#include "tc_gemm.cuh"

namespace arckv {

// Each epilogue thread folds one row of kW columns of a kBN-wide tile (kBN / kW
// warps per TMEM lane quarter: four epilogue warps for 128-wide tiles, eight
// for 256-wide ones) and writes their row-softmax partials,
// part[b][row][n0 / kW].  kTma: the I tile leaves through TMA stores staged in
// shared memory (32 x 32 boxes; two buffers per warp with four warps, one
// with eight); else each row writes its kW values.
template <bool kTma, int kW_, int kBN = 128>
struct TcEpiIndexT {
  static constexpr int kW = kW_;
  static constexpr int kEpiWarps = kBN / kW * 4;
  static constexpr int kNBuf = kEpiWarps == 4 ? 2 : 1;
  static constexpr int kStageBytes = kTma ? kNBuf * 32 * 128 : 0;
  const float* wts;  // [H][n_pos][H_I]
  float* I;          // [H][n][T]
  float2* part;      // [H][n][ntiles], ntiles = ceil(T / kW)
  int n, T, H_I, G, n_pos, ntiles;
  CUtensorMap map;   // kTma: I as [H][n][T], box {32, 32, 1}, 128-byte swizzle
  struct State {
    float acc[kW];
    const float* wrow;
    uint8_t* stage;
    int* stores;
    float w, wn;   // this head's weight / sqrt(d_I); the next head's weight (prefetched)
    bool row_ok;
  };
  __device__ __forceinline__ void init(State& s, int b, int row, int, int M, int) const {
    s.row_ok = row < M;
    s.wrow = wts + ((long long)b * n_pos + (s.row_ok ? row / G : 0)) * H_I;
    s.w = 0.f;
    s.wn = s.row_ok ? s.wrow[0] : 0.f;
#pragma unroll
    for (int q = 0; q < kW; ++q) s.acc[q] = 0.f;
  }
  __device__ __forceinline__ void attach(State& s, uint8_t* stage, int* stores) const {
    s.stage = stage;
    s.stores = stores;
  }
  __device__ __forceinline__ void consume(State& s, int chunk, int j, float (&v)[32]) const {
    // w LeakyReLU(v / sqrt(d_I)) = (w / sqrt(d_I)) max(v, 0.1 v)
    if (j == 0) {
      s.w = s.wn * 0.08838834764831845f;   // 1 / sqrt(d_I), d_I = 128
      s.wn = (s.row_ok && chunk + 1 < H_I) ? s.wrow[chunk + 1] : 0.f;
    }
#pragma unroll
    for (int q = 0; q < 32; ++q) s.acc[j * 32 + q] = fmaf(s.w, fmaxf(v[q], 0.1f * v[q]), s.acc[j * 32 + q]);
  }
  // the 256-wide tiles take their columns 16 at a time: with 128 running sums
  // per thread a 32-column load left the eight-warp epilogue spilling
  static constexpr bool kHalfLoads = kBN == 256;
  __device__ __forceinline__ void consume16(State& s, int chunk, int j, int h, float (&v)[16]) const {
    if (j == 0 && h == 0) {
      s.w = s.wn * 0.08838834764831845f;
      s.wn = (s.row_ok && chunk + 1 < H_I) ? s.wrow[chunk + 1] : 0.f;
    }
#pragma unroll
    for (int q = 0; q < 16; ++q)
      s.acc[j * 32 + h * 16 + q] = fmaf(s.w, fmaxf(v[q], 0.1f * v[q]), s.acc[j * 32 + h * 16 + q]);
  }
  __device__ __forceinline__ void finish(State& s, int b, int row, int n0, int, int N) const {
    const int nc = min(kW, N - n0);
    if (s.row_ok && nc > 0) {
      // eight independent max / sum chains over the half tile's columns
      float m8[8], a8[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) m8[k] = -INFINITY;
#pragma unroll
      for (int q = 0; q < kW; ++q)
        if (q < nc) m8[q & 7] = fmaxf(m8[q & 7], s.acc[q]);
      const float mx =
          fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])), fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7])));
      const float ml = mx * kLog2e;
#pragma unroll
      for (int k = 0; k < 8; ++k) a8[k] = 0.f;
#pragma unroll
      for (int q = 0; q < kW; ++q)
        if (q < nc) a8[q & 7] += ex2_approx(fmaf(s.acc[q], kLog2e, -ml));
      const float sm = ((a8[0] + a8[1]) + (a8[2] + a8[3])) + ((a8[4] + a8[5]) + (a8[6] + a8[7]));
      part[((long long)b * n + row) * ntiles + n0 / kW] = make_float2(mx, sm);
    }
    if constexpr (kTma) {
      // rows past n and columns past T fall outside the tensor map: not written
      const int y = row & ~31;
#pragma unroll
      for (int j = 0; j < kW / 32; ++j)
        staged_store_32x32<kNBuf>(&map, s.stage, s.stores, n0 + 32 * j, y, b, n, T, s.acc + 32 * j, 1.f);
    } else {
      if (!s.row_ok || nc <= 0) return;
      float* dst = I + ((long long)b * n + row) * T + n0;
      if ((T & 3) == 0 && nc == kW) {
#pragma unroll
        for (int q = 0; q < kW; q += 4)
          *(float4*)(dst + q) = make_float4(s.acc[q], s.acc[q + 1], s.acc[q + 2], s.acc[q + 3]);
      } else {
#pragma unroll
        for (int q = 0; q < kW; ++q)
          if (q < nc) dst[q] = s.acc[q];
      }
    }
  }
};

int launch_index_logits(const Dims& D, const bf16* qbar_hi, const bf16* qbar_lo, const bf16* kbar_hi,
                        const bf16* kbar_lo, const float* wts, float* I, float2* part, DevStatus* stt,
                        cudaStream_t st) {
  CUtensorMap mA, mA2, mB, mB2;
  // 128 x 256 tiles (M = 128, N = 256 MMAs: a quarter fewer operand bytes per
  // flop than 128 x 128) where T fills them; the key operand's box is 256 rows
  const bool wide = D.T >= 256;
  const int bB = wide ? 256 : 128;
  if (!encode_bf16_map_3d(&mA, qbar_hi, D.HD, D.n, D.H, 128) || !encode_bf16_map_3d(&mA2, qbar_lo, D.HD, D.n, D.H, 128) ||
      !encode_bf16_map_3d(&mB, kbar_hi, D.HD, D.T, D.H, bB) || !encode_bf16_map_3d(&mB2, kbar_lo, D.HD, D.T, D.H, bB))
    return -1;
  if ((D.T & 3) == 0 && ((uintptr_t)I & 15u) == 0) {
    if (wide) {
      TcEpiIndexT<true, kIndexPartW, 256> epi{wts, I, part, D.n, D.T, D.H_I, D.G, D.n_pos, cdiv(D.T, kIndexPartW), {}};
      if (!encode_f32_map_3d(&epi.map, I, D.T, D.n, D.H, 32, 32, D.T, (uint64_t)D.n * D.T, true)) return -1;
      if (launch_tc_gemm<256, kSplit>(mA, mB, mA2, mB2, epi, D.H, D.n, D.T, D.HD, 128, stt, st) != cudaSuccess)
        return -1;
      return 1;
    }
    TcEpiIndexT<true, kIndexPartW> epi{wts, I, part, D.n, D.T, D.H_I, D.G, D.n_pos, cdiv(D.T, kIndexPartW), {}};
    if (!encode_f32_map_3d(&epi.map, I, D.T, D.n, D.H, 32, 32, D.T, (uint64_t)D.n * D.T, true)) return -1;
    if (launch_tc_gemm<128, kSplit>(mA, mB, mA2, mB2, epi, D.H, D.n, D.T, D.HD, 128, stt, st) != cudaSuccess)
      return -1;
    return 1;
  }
  if (wide) {
    TcEpiIndexT<false, kIndexPartW, 256> epi{wts, I, part, D.n, D.T, D.H_I, D.G, D.n_pos, cdiv(D.T, kIndexPartW), {}};
    if (launch_tc_gemm<256, kSplit>(mA, mB, mA2, mB2, epi, D.H, D.n, D.T, D.HD, 128, stt, st) != cudaSuccess)
      return -1;
    return 1;
  }
  TcEpiIndexT<false, kIndexPartW> epi{wts, I, part, D.n, D.T, D.H_I, D.G, D.n_pos, cdiv(D.T, kIndexPartW), {}};
  if (launch_tc_gemm<128, kSplit>(mA, mB, mA2, mB2, epi, D.H, D.n, D.T, D.HD, 128, stt, st) != cudaSuccess) return -1;
  return 1;
}

}  // namespace arckv
