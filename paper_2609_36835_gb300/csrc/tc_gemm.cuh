// Warp-specialised tcgen05 GEMM for sm_103a:
//
//   D[b](m, n) = sum_k A[b](m, k) B[b](n, k)      (A, B bf16, K-major, D fp32 in TMEM)
//
// Persistent: one CTA per SM walks the 128 x BN output tiles (b, row tile,
// column tile; columns fastest) in a grid-stride loop.  With col_group > 0
// the column tiles are taken col_group at a time (b, column group, row tile,
// column tile in the group), so that the B operand of one group stays in L2
// while the A rows stream past it once per group.  Warp 0 streams 64-wide K slabs of A and B
// into a STAGES-deep ring of 128-byte-swizzled shared tiles with TMA; warp 1
// issues tcgen05.mma (M = 128, N = BN, K = 16) into one of two TMEM
// accumulators; warps 2..5 drain the accumulator with tcgen05.ld, one TMEM
// lane (= one output row) per thread, and hand it to the epilogue.
//
// MODE selects how the second pair of maps (mA2, mB2) is used:
//   kPlain  -- not used;
//   kSplit  -- each operand is a pair (hi, lo) of bf16 tensors with
//              x ~= hi + lo (hi = bf16(x), lo = bf16(x - hi)) and every K step
//              issues hi*hi + hi*lo + lo*hi: an fp32-accurate product on the
//              bf16 tensor pipe (the dropped lo*lo term is below 2^-16 relative);
//   kConcat -- the operands are concatenated along K: K < K1 comes from
//              (mA, mB), K >= K1 from (mA2, mB2) (K1 a multiple of 64);
//   kSplit3A -- A is a triple (h, m, l) of bf16 tensors with x = h + m + l to
//              within 2^-24 relative (mA, mA2, mA3) and B is exact bf16 (mB):
//              every K step issues h*B + m*B + l*B, fp32-grade products for an
//              fp32 operand against a bf16 input;
//   kSplit3S -- a Gram of one fp32 operand with itself: A and B are both the
//              triple (mA, mA2, mA3), read at rows m0 and n0, and every K step
//              issues hh + hm + mh + hl + lh + mm (the dropped ml, lm, ll terms
//              are below 2^-24 relative): fp32-grade X X^T on the bf16 pipe.
//
// K is consumed in chunks of `chunk_k` (a multiple of 64): each chunk gets a
// fresh accumulator and the epilogue sees every chunk separately, which lets
// a non-linearity act between chunks (the per-index-head LeakyReLU of
// Eq. pairwise_index_score).  The two TMEM buffers alternate between chunks,
// so the MMA of chunk c+1 overlaps the epilogue of chunk c -- also across
// tiles: the stage ring, the chunk counter and the accumulator alternation run
// on over a CTA's tiles, so a tile's last epilogue overlaps the next tile's
// first MMAs and no tile pays a prologue.
//
// Epilogue interface (all per thread = per output row):
//   struct State;                                     registers of one row
//   void init(State&, int b, int row, int n0, int M, int N);
//   void consume(State&, int chunk, int j, float (&v)[32]);  columns n0+32j..
//   void finish(State&, int b, int row, int n0, int M, int N);
// An epilogue that declares kEpiWarps = 8 gets two warps per TMEM lane
// quarter: warps 2..5 drain the first BN/2 columns and warps 6..9 the rest,
// and each sees a tile of BN/2 columns (init/finish get its first column;
// consume's j counts 32-column chunks within it).
// An epilogue that declares kStageBytes gets that much shared memory per
// epilogue warp (1024-byte aligned) through attach(State&, uint8_t*, int*)
// after init, for staging TMA stores, with a per-thread count of the stores
// issued so far (kept across tiles, so staging buffers alternate by issued
// store); the kernel waits for its bulk stores before it exits.
#pragma once
#include <algorithm>
#include <type_traits>

#include "tc.cuh"

namespace arckv {

enum TcMode { kPlain = 0, kSplit = 1, kConcat = 2, kSplit3A = 3, kSplit3S = 4 };

template <class E, class = void>
struct EpiWarps {
  static constexpr int value = 4;
};
template <class E>
struct EpiWarps<E, std::void_t<decltype(E::kEpiWarps)>> {
  static constexpr int value = E::kEpiWarps;
};

template <class E, class = void>
struct EpiStage {
  static constexpr int bytes = 0;
};
template <class E>
struct EpiStage<E, std::void_t<decltype(E::kStageBytes)>> {
  static constexpr int bytes = E::kStageBytes;
};

// An epilogue that declares kHalfLoads = true is fed 16 columns at a time
// through consume16(State&, int chunk, int j, int half, float (&v)[16]).
template <class E, class = void>
struct EpiHalfLoads {
  static constexpr bool value = false;
};
template <class E>
struct EpiHalfLoads<E, std::void_t<decltype(E::kHalfLoads)>> {
  static constexpr bool value = E::kHalfLoads;
};

template <int BN, int MODE>
struct TcCfg {
  static constexpr bool SPLIT = MODE == kSplit;
  static constexpr int TILE_A = 128 * 128;  // bytes: 128 rows x 64 bf16
  static constexpr int TILE_B = BN * 128;
  static constexpr int STAGE = MODE == kSplit     ? 2 * (TILE_A + TILE_B)
                               : MODE == kSplit3A ? 3 * TILE_A + TILE_B
                               : MODE == kSplit3S ? 3 * (TILE_A + TILE_B)
                                                  : TILE_A + TILE_B;
  static constexpr int STAGES_WANT = MODE == kSplit3S ? 2 : (MODE == kSplit || MODE == kSplit3A) ? 3 : 4;
  // as many of those as fit beside the epilogue staging (wide tiles take fewer)
  static constexpr int STAGES = STAGES_WANT * STAGE <= 200 * 1024 ? STAGES_WANT : (200 * 1024) / STAGE;
  static constexpr int SMEM = STAGES * STAGE + 1024;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
};

template <int BN, int MODE, class Epi>
__global__ void __launch_bounds__(64 + 32 * EpiWarps<Epi>::value, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap mA, const __grid_constant__ CUtensorMap mB,
                   const __grid_constant__ CUtensorMap mA2, const __grid_constant__ CUtensorMap mB2,
                   const __grid_constant__ CUtensorMap mA3, const __grid_constant__ Epi epi, int H, int M, int N, int K,
                   int chunk_k, int K1, DevStatus* stt, int col_group) {
  using C = TcCfg<BN, MODE>;
  constexpr int SB = EpiStage<Epi>::bytes;
  constexpr int NE = EpiWarps<Epi>::value;   // epilogue warps: 4 or 8
  constexpr int JG = BN / 32 / (NE / 4);     // 32-column chunks per epilogue warp
  static_assert(NE == 4 || NE == 8, "4 or 8 epilogue warps");
  constexpr bool SPLIT = C::SPLIT;
  constexpr int STAGES = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t full[STAGES], empty[STAGES], accf[2], acce[2], drain;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;
  const uint32_t raw = tc::smem_u32(smem_raw);
  uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nk = (K + 63) / 64;
  const int kpc = chunk_k / 64;
  const int nchunks = (nk + kpc - 1) / kpc;
  // persistent: CTA c takes tiles c, c + grid, ...; tile = (b, row tile, column tile), columns fastest
  const int Mt = (M + 127) / 128, Nt = (N + BN - 1) / BN;
  const int ntiles = H * Mt * Nt;
  const int Gc = col_group > 0 ? min(col_group, Nt) : Nt;   // column tiles per group
  auto tile_coords = [&](int tl, int& b, int& m0, int& n0) {
    b = tl / (Mt * Nt);
    int r = tl - b * (Mt * Nt);
    const int g = r / (Mt * Gc);                 // full groups of Mt x Gc tiles come first
    const int gw = min(Gc, Nt - g * Gc);         // the last group may be narrower
    r -= g * (Mt * Gc);
    m0 = (r / gw) * 128;
    n0 = (g * Gc + r % gw) * BN;
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&accf[i], 1);
      tc::mbar_init(&acce[i], NE);
    }
    tc::mbar_init(&drain, 1);
    abort_flag = 0;
    tc::mbar_fence_init();
  }
  if (warp == 1) tc::tmem_alloc(&tmem_slot, C::TMEM_COLS);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_slot;
  volatile int* abortp = &abort_flag;

  if (warp == 0) {
    if (lane == 0) {
      tc::tma_prefetch(&mA);
      tc::tma_prefetch(&mB);
      if (MODE == kSplit || MODE == kConcat) {
        tc::tma_prefetch(&mA2);
        tc::tma_prefetch(&mB2);
      }
      if (MODE == kSplit3A || MODE == kSplit3S) {
        tc::tma_prefetch(&mA2);
        tc::tma_prefetch(&mA3);
      }
      int g = 0;   // K slabs issued by this CTA (ring position across tiles)
      bool ok = true;
      for (int tl = blockIdx.x; tl < ntiles && ok; tl += gridDim.x) {
        int b, m0, n0;
        tile_coords(tl, b, m0, n0);
        for (int kb = 0; kb < nk; ++kb) {
          const int s = g % STAGES;
          if (g >= STAGES && !tc::mbar_wait(&empty[s], ((g / STAGES) - 1) & 1, abortp, stt)) {
            ok = false;
            break;
          }
          uint8_t* st = base + s * C::STAGE;
          tc::mbar_arrive_expect_tx(&full[s], C::STAGE);
          if (MODE == kConcat && kb * 64 >= K1) {
            tc::tma_load_3d(st, &mA2, kb * 64 - K1, m0, b, &full[s]);
            tc::tma_load_3d(st + C::TILE_A, &mB2, kb * 64 - K1, n0, b, &full[s]);
          } else if (MODE == kSplit3S) {
            // [A_h][B_h][A_m][B_m][A_l][B_l]
            const CUtensorMap* mp[3] = {&mA, &mA2, &mA3};
#pragma unroll
            for (int p = 0; p < 3; ++p) {
              tc::tma_load_3d(st + p * (C::TILE_A + C::TILE_B), mp[p], kb * 64, m0, b, &full[s]);
              tc::tma_load_3d(st + p * (C::TILE_A + C::TILE_B) + C::TILE_A, mp[p], kb * 64, n0, b, &full[s]);
            }
          } else {
            tc::tma_load_3d(st, &mA, kb * 64, m0, b, &full[s]);
            tc::tma_load_3d(st + C::TILE_A, &mB, kb * 64, n0, b, &full[s]);
          }
          if (SPLIT) {
            tc::tma_load_3d(st + C::TILE_A + C::TILE_B, &mA2, kb * 64, m0, b, &full[s]);
            tc::tma_load_3d(st + 2 * C::TILE_A + C::TILE_B, &mB2, kb * 64, n0, b, &full[s]);
          }
          if (MODE == kSplit3A) {
            tc::tma_load_3d(st + C::TILE_A + C::TILE_B, &mA2, kb * 64, m0, b, &full[s]);
            tc::tma_load_3d(st + 2 * C::TILE_A + C::TILE_B, &mA3, kb * 64, m0, b, &full[s]);
          }
          ++g;
        }
      }
      // every issued copy lands before the CTA may exit
      volatile int never = 0;
      for (int k = g > STAGES ? g - STAGES : 0; k < g; ++k)
        tc::mbar_wait(&full[k % STAGES], (k / STAGES) & 1, &never, stt);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = tc::idesc_bf16_f32(BN);
      bool ok = true;
      int g = 0, cg = 0;   // K slabs and chunks consumed by this CTA, across tiles
      for (int tl = blockIdx.x; tl < ntiles && ok; tl += gridDim.x) {
        for (int c = 0; c < nchunks && ok; ++c, ++cg) {
          const int buf = cg & 1;
          if (cg >= 2 && !tc::mbar_wait(&acce[buf], ((cg >> 1) - 1) & 1, abortp, stt)) {
            ok = false;
            break;
          }
          tc::fence_after_sync();
          const uint32_t d = tmem + (uint32_t)(buf * BN);
          const int kb0 = c * kpc, kb1 = min(nk, kb0 + kpc);
          for (int kb = kb0; kb < kb1; ++kb, ++g) {
            const int s = g % STAGES;
            if (!tc::mbar_wait(&full[s], (g / STAGES) & 1, abortp, stt)) {
              ok = false;
              break;
            }
            tc::fence_after_sync();
            const uint32_t a = tc::smem_u32(base + s * C::STAGE), bb = a + C::TILE_A;
#pragma unroll
            for (int ks = 0; ks < 4; ++ks) {
              const uint64_t ad = tc::sdesc_k128(a + ks * 32), bd = tc::sdesc_k128(bb + ks * 32);
              tc::mma_f16(d, ad, bd, idesc, (kb > kb0 || ks > 0) ? 1u : 0u);
              if (SPLIT) {
                const uint64_t ad2 = tc::sdesc_k128(a + C::TILE_A + C::TILE_B + ks * 32);
                const uint64_t bd2 = tc::sdesc_k128(bb + C::TILE_A + C::TILE_B + ks * 32);
                tc::mma_f16(d, ad, bd2, idesc, 1u);
                tc::mma_f16(d, ad2, bd, idesc, 1u);
              }
              if (MODE == kSplit3A) {
                const uint64_t am = tc::sdesc_k128(a + C::TILE_A + C::TILE_B + ks * 32);
                const uint64_t al = tc::sdesc_k128(a + 2 * C::TILE_A + C::TILE_B + ks * 32);
                tc::mma_f16(d, am, bd, idesc, 1u);
                tc::mma_f16(d, al, bd, idesc, 1u);
              }
              if (MODE == kSplit3S) {
                constexpr uint32_t P = C::TILE_A + C::TILE_B;
                const uint64_t am = tc::sdesc_k128(a + P + ks * 32), bm = tc::sdesc_k128(bb + P + ks * 32);
                const uint64_t al = tc::sdesc_k128(a + 2 * P + ks * 32), bl = tc::sdesc_k128(bb + 2 * P + ks * 32);
                tc::mma_f16(d, ad, bm, idesc, 1u);
                tc::mma_f16(d, am, bd, idesc, 1u);
                tc::mma_f16(d, ad, bl, idesc, 1u);
                tc::mma_f16(d, al, bd, idesc, 1u);
                tc::mma_f16(d, am, bm, idesc, 1u);
              }
            }
            tc::mma_commit(&empty[s]);
          }
          if (ok) tc::mma_commit(&accf[buf]);
        }
      }
      // all MMAs this thread issued have completed before teardown
      tc::mma_commit(&drain);
      volatile int never = 0;
      tc::mbar_wait(&drain, 0, &never, stt);
    }
  } else {
    const int q = warp & 3;              // TMEM lane quarter this warp may access
    const int cg = ((warp - 2) >> 2) * JG;   // first 32-column chunk of this warp
    const int row = q * 32 + lane;
    bool ok = true;
    int kc = 0;
    int stores = 0;   // staged stores issued by this warp (identical in all its lanes)
    for (int tl = blockIdx.x; tl < ntiles && ok; tl += gridDim.x) {
      int b, m0, n0;
      tile_coords(tl, b, m0, n0);
      typename Epi::State es;
      epi.init(es, b, m0 + row, n0 + cg * 32, M, N);
      if constexpr (SB > 0) epi.attach(es, base + STAGES * C::STAGE + (warp - 2) * SB, &stores);
      for (int c = 0; c < nchunks; ++c, ++kc) {
        const int buf = kc & 1;
        ok = tc::mbar_wait(&accf[buf], (kc >> 1) & 1, abortp, stt);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) break;
        tc::fence_after_sync();
#pragma unroll
        for (int j = 0; j < JG; ++j) {
          if constexpr (EpiHalfLoads<Epi>::value) {   // 16 columns at a time (fewer live registers)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              float v[16];
              tc::tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * BN + (cg + j) * 32 + h * 16), v);
              epi.consume16(es, c, j, h, v);
            }
          } else {
            float v[32];
            tc::tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * BN + (cg + j) * 32), v);
            epi.consume(es, c, j, v);
          }
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&acce[buf]);
      }
      if (ok) epi.finish(es, b, m0 + row, n0 + cg * 32, M, N);
    }
    if constexpr (SB > 0) {
      if (lane == 0) tc::bulk_wait_all();
      __syncwarp();
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// Resident CTAs of the persistent GEMM: one per SM (the stage ring takes most
// of the shared memory), looked up once per device.
int tc_gemm_sm_count();
cudaError_t set_dyn_smem(const void* kern, int bytes);

// Host: launch over H batches; maps are built by the caller (encode_bf16_map_3d,
// box rows 128 for A and BN for B).
template <int BN, int MODE, class Epi>
inline cudaError_t launch_tc_gemm(const CUtensorMap& mA, const CUtensorMap& mB, const CUtensorMap& mA2,
                                  const CUtensorMap& mB2, const Epi& epi, int H, int M, int N, int K, int chunk_k,
                                  DevStatus* stt, cudaStream_t st, int K1 = 0, const CUtensorMap* mA3 = nullptr,
                                  int col_group = 0) {
  using C = TcCfg<BN, MODE>;
  constexpr int NE = EpiWarps<Epi>::value;
  constexpr int smem = C::SMEM + NE * EpiStage<Epi>::bytes;
  static_assert(smem <= 227 * 1024, "stage ring and epilogue staging exceed shared memory");
  auto kern = tc_gemm_kernel<BN, MODE, Epi>;
  cudaError_t e = set_dyn_smem((const void*)kern, smem);
  if (e != cudaSuccess) return e;
  const long long ntiles = (long long)cdiv(N, BN) * cdiv(M, 128) * H;
  const int grid = (int)std::min<long long>(ntiles, tc_gemm_sm_count());
  kern<<<grid, 64 + 32 * NE, smem, st>>>(mA, mB, mA2, mB2, mA3 ? *mA3 : mA, epi, H, M, N, K, chunk_k, K1, stt,
                                         col_group);
  return cudaGetLastError();
}

// Plain fp32 store epilogue: C[b][row][col] = alpha * acc.
struct TcEpiStore {
  float* C;
  long long cbs;
  int ldc;
  float alpha;
  struct State {
    float* dst;
    bool row_ok, vec;
    int ncols;
  };
  __device__ __forceinline__ void init(State& s, int b, int row, int n0, int M, int N) const {
    s.dst = C + (long long)b * cbs + (long long)row * ldc + n0;
    s.row_ok = row < M;
    s.ncols = N - n0;
    s.vec = ((ldc & 3) == 0) && ((((uintptr_t)C) & 15) == 0) && ((cbs & 3) == 0) && ((n0 & 3) == 0);
  }
  __device__ __forceinline__ void consume(State& s, int, int j, float (&v)[32]) const {
    if (!s.row_ok) return;
    float* d = s.dst + j * 32;
    if (s.vec && j * 32 + 32 <= s.ncols) {
#pragma unroll
      for (int q = 0; q < 32; q += 4)
        *(float4*)(d + q) = make_float4(alpha * v[q], alpha * v[q + 1], alpha * v[q + 2], alpha * v[q + 3]);
    } else {
#pragma unroll
      for (int q = 0; q < 32; ++q)
        if (j * 32 + q < s.ncols) d[q] = alpha * v[q];
    }
  }
  __device__ __forceinline__ void finish(State&, int, int, int, int, int) const {}
};

// Transposed fp32 store: C[b][col][row] = alpha * acc (column stride ldc).
// A warp's 32 rows are 32 consecutive addresses of each output row.
struct TcEpiStoreT {
  float* C;
  long long cbs;
  int ldc;
  float alpha;
  struct State {
    float* base;
    int ncols;
    bool ok;
  };
  __device__ __forceinline__ void init(State& s, int b, int row, int n0, int M, int N) const {
    s.ok = row < M;
    s.ncols = N - n0;
    s.base = C + (long long)b * cbs + (long long)n0 * ldc + (s.ok ? row : 0);
  }
  __device__ __forceinline__ void consume(State& s, int, int j, float (&v)[32]) const {
    if (!s.ok) return;
#pragma unroll
    for (int q = 0; q < 32; ++q)
      if (j * 32 + q < s.ncols) s.base[(long long)(j * 32 + q) * ldc] = alpha * v[q];
  }
  __device__ __forceinline__ void finish(State&, int, int, int, int, int) const {}
};

// The fp32 result as a bf16 triple (h, m, l) (split3_bf16): element
// (b, row, col) of each part at b * bs + row * ldc + col, the operand format
// of a following kSplit3A product.
struct TcEpiSplit3 {
  bf16 *h, *m, *l;
  long long bs;
  int ldc;
  struct State {
    long long off;
    int ncols;
    bool ok;
  };
  __device__ __forceinline__ void init(State& s, int b, int row, int n0, int M, int N) const {
    s.ok = row < M;
    s.ncols = N - n0;
    s.off = (long long)b * bs + (long long)(s.ok ? row : 0) * ldc + n0;
  }
  __device__ __forceinline__ void consume(State& s, int, int j, float (&v)[32]) const {
    if (!s.ok) return;
#pragma unroll
    for (int q = 0; q < 32; q += 8) {
      const long long o = s.off + j * 32 + q;
      if (j * 32 + q + 8 <= s.ncols && (o & 7) == 0) {
        __align__(16) bf16 hh[8], mm[8], ll[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) split3_bf16(v[q + e], hh[e], mm[e], ll[e]);
        *(uint4*)(h + o) = *(const uint4*)hh;
        *(uint4*)(m + o) = *(const uint4*)mm;
        *(uint4*)(l + o) = *(const uint4*)ll;
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e)
          if (j * 32 + q + e < s.ncols) split3_bf16(v[q + e], h[o + e], m[o + e], l[o + e]);
      }
    }
  }
  __device__ __forceinline__ void finish(State&, int, int, int, int, int) const {}
};

// Staged TMA store of one warp's 32 rows x 32 columns at (x, y, b): the rows
// go into a 128-byte-swizzled staging buffer (conflict-free 16-byte stores)
// and one lane issues the tiled bulk store.  NBUF buffers of 4 KB rotate by
// issued store; before a buffer is rewritten, at most NBUF - 1 stores (the
// other buffers') may still be reading.  Boxes wholly outside [0, N) x [0, M)
// are skipped (warp-uniform).  v is scaled by alpha.
template <int NBUF = 2>
__device__ __forceinline__ void staged_store_32x32(const CUtensorMap* map, uint8_t* stage, int* stores, int x, int y,
                                                   int b, int M, int N, const float* v, float alpha) {
  if (y >= M || x >= N) return;
  const int lane = threadIdx.x & 31;
  uint8_t* buf = stage + (*stores % NBUF) * 4096;
  if (lane == 0) tc::bulk_wait_read<NBUF - 1>();
  __syncwarp();
#pragma unroll
  for (int k = 0; k < 8; ++k)
    *(float4*)(buf + lane * 128 + ((k ^ (lane & 7)) << 4)) =
        make_float4(alpha * v[4 * k], alpha * v[4 * k + 1], alpha * v[4 * k + 2], alpha * v[4 * k + 3]);
  tc::fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) {
    tc::tma_store_3d(map, buf, x, y, b);
    tc::bulk_commit();
  }
  ++*stores;
}

// fp32 store through shared memory and TMA (staged_store_32x32 per chunk,
// NBUF staging buffers per warp).  C is [H][M][N] with row stride ldc (a
// multiple of 4) in `map`.
template <int NBUF>
struct TcEpiStoreTmaT {
  CUtensorMap map;   // box {32, 32, 1}, 128-byte swizzle
  float alpha;
  int M, N;
  static constexpr int kStageBytes = NBUF * 32 * 128;
  struct State {
    uint8_t* stage;
    int* stores;
    int b, y, n0;
  };
  __device__ __forceinline__ void init(State& s, int b, int row, int n0, int, int) const {
    s.b = b;
    s.y = row & ~31;
    s.n0 = n0;
  }
  __device__ __forceinline__ void attach(State& s, uint8_t* stage, int* stores) const {
    s.stage = stage;
    s.stores = stores;
  }
  __device__ __forceinline__ void consume(State& s, int, int j, float (&v)[32]) const {
    staged_store_32x32<NBUF>(&map, s.stage, s.stores, s.n0 + 32 * j, s.y, s.b, M, N, v, alpha);
  }
  __device__ __forceinline__ void finish(State&, int, int, int, int, int) const {}
};

// A store epilogue (TcEpiStore or TcEpiStoreTma) that also writes each row's
// softmax partials over each kRowPartW = 64 columns: part[b][row][col / 64] =
// (max, sum exp(x - max)) of alpha * acc (exp as 2^(x log2 e) on the MUFU
// unit).  Eight epilogue warps, each draining 64 columns of a 128-wide tile.
template <class Store>
struct TcEpiRowPartT {
  Store st;
  float2* part;
  int ntiles, BNt;   // ntiles = ceil(N / 64), BNt = 64
  static constexpr int kEpiWarps = 8;
  static constexpr int kStageBytes = EpiStage<Store>::bytes;
  struct State {
    typename Store::State s;
    float mx, sm;
    long long prow;
    int ncols;
    bool row_ok;
  };
  __device__ __forceinline__ void init(State& s, int b, int row, int n0, int M, int N) const {
    st.init(s.s, b, row, n0, M, N);
    s.mx = -INFINITY;
    s.sm = 0.f;
    s.prow = ((long long)b * M + row) * ntiles + n0 / BNt;
    s.ncols = N - n0;
    s.row_ok = row < M;
  }
  __device__ __forceinline__ void attach(State& s, uint8_t* stage, int* stores) const {
    st.attach(s.s, stage, stores);
  }
  __device__ __forceinline__ void consume(State& s, int c, int j, float (&v)[32]) const {
    st.consume(s.s, c, j, v);
    const int nc = s.ncols - j * 32;   // columns of this chunk inside the matrix
    if (nc <= 0) return;
#pragma unroll
    for (int q = 0; q < 32; ++q) v[q] = (q < nc) ? st.alpha * v[q] : -INFINITY;
    // independent max / sum chains (a serial chain would stall the single
    // epilogue warp of each sub-partition on every dependent instruction)
    float m8[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) m8[k] = fmaxf(fmaxf(v[k], v[k + 8]), fmaxf(v[k + 16], v[k + 24]));
    const float m = fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])), fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7])));
    const float mn = fmaxf(s.mx, m);
    if (mn == -INFINITY) return;
    const float ml = mn * kLog2e;
    float a4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int q = 0; q < 32; ++q) a4[q & 3] += ex2_approx(fmaf(v[q], kLog2e, -ml));
    s.sm = fmaf(s.sm, ex2_approx(fmaf(s.mx, kLog2e, -ml)), (a4[0] + a4[1]) + (a4[2] + a4[3]));
    s.mx = mn;
  }
  __device__ __forceinline__ void finish(State& s, int, int, int, int, int) const {
    // a half tile that starts past the last column has no partial slot
    if (s.row_ok && s.ncols > 0) part[s.prow] = make_float2(s.mx, s.sm);
  }
};
using TcEpiStoreRowPart = TcEpiRowPartT<TcEpiStore>;
using TcEpiStoreRowPartTma = TcEpiRowPartT<TcEpiStoreTmaT<1>>;

// Row-partial logits L = alpha * (A B^T) [H][M][N] (row stride N) through the
// TMA-store epilogue when N is a multiple of 4 (row pitch on the 16-byte grid),
// else through plain stores.
template <int MODE>
inline cudaError_t launch_tc_logits_rowpart(const CUtensorMap& mA, const CUtensorMap& mB, const CUtensorMap& mA2,
                                            const CUtensorMap& mB2, const CUtensorMap* mA3, float* L, float alpha,
                                            float2* part, int H, int M, int N, int K, DevStatus* stt,
                                            cudaStream_t st) {
  const int ntiles = cdiv(N, 64);
  if ((N & 3) == 0 && (((uintptr_t)L) & 15u) == 0) {
    TcEpiStoreRowPartTma epi{};
    epi.st.alpha = alpha;
    epi.st.M = M;
    epi.st.N = N;
    epi.part = part;
    epi.ntiles = ntiles;
    epi.BNt = 64;
    if (!encode_f32_map_3d(&epi.st.map, L, N, M, H, 32, 32, N, (uint64_t)M * N, true))
      return cudaErrorInvalidValue;
    return launch_tc_gemm<128, MODE>(mA, mB, mA2, mB2, epi, H, M, N, K, K, stt, st, 0, mA3);
  }
  TcEpiStoreRowPart epi{{L, (long long)M * N, N, alpha}, part, ntiles, 64};
  return launch_tc_gemm<128, MODE>(mA, mB, mA2, mB2, epi, H, M, N, K, K, stt, st, 0, mA3);
}

}  // namespace arckv
