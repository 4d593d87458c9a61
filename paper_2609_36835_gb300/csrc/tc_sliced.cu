// fp64-grade products on the bf16 tensor pipe, for the ill-conditioned dual
// fits (App. A.9 Eqs. mass_fit, value_lstsq in their push-through form when
// t > n).
//
// Slices.  Row r of an operand X (fp32 or fp64) is scaled by 2^-e_r, where
// 2^e_r bounds the row's largest magnitude, and cut into S bf16 slices
//     X[r][k] = 2^e_r (x_1 + x_2 + ... + x_S) + residual,
//     x_i = I_i 2^(-8 i),  I_1 in [-256, 256],  I_i in [-128, 127] (i > 1):
// the balanced base-256 digits of Z = round(X[r][k] 2^(8 S - e_r)), so
// |residual| <= 2^(-8 S - 1) 2^e_r.  Every slice is an integer of at most 8
// significant bits times a power of two: exact in bf16.  The GB300's fp64
// pipe runs at a small fraction of its integer and fp32 rates, so the
// exponents, the rounding to Z and the digits are taken with integer
// operations on the operand's bits, and each fp64 result is one rounding
// conversion of a 64-bit integer sum with its power of two added to the
// exponent field (plus the subtraction of the `sub` mode).
//
// Products.  C = A B^T is the sum over all S^2 slice pairs (i, j).  A pair's
// products are integers times 2^(-8(i + j)), so the pairs of one level
// l = i + j add up exactly in fp32 while the integer sum stays below 2^24:
// with 128 terms of K that holds for l <= 4 (at most 128 (2 * 256 * 128 +
// 128^2) < 2^24).  Levels 2, 3 and 4 therefore run in fresh TMEM accumulators
// per 128-wide K chunk, and the epilogue converts each chunk's sums to
// integers and adds them up exactly (in 64-bit, for K <= 26214); the levels
// above 4 weigh at most 2^-24 of the total and accumulate in one fp32
// accumulator over the whole K.  The result (the exact levels in units of
// 2^-32 shifted to units of 2^-44, plus the fp32 levels rounded to that unit,
// in one 64-bit integer), rounded once to fp64 and scaled by 2^(e_m + f_n), is
// the exact product of the sliced operands up to ~2^-44 relative: the fp32
// arithmetic of the tensor pipe never meets a rounding that matters.
//
// Kernel layout (persistent, one CTA per SM): warp 0 streams 32-wide K slabs
// of the S slices of a 128-row A tile and a BN-row B tile with TMA (64-byte
// swizzle) into a shared ring; warp 1 issues the S^2 tcgen05 MMAs (M = 128,
// N = BN, K = 16) of every K step into the level accumulators; the epilogue
// warps (32 columns each) drain the exact levels after every chunk and
// assemble the tile.  With BN = 64 the accumulators are double-buffered (the
// exact levels of two alternating chunks, the higher levels of two
// alternating tiles: 512 TMEM columns), so a tile is assembled while the next
// one's MMAs run; with BN = 128 they fill the 512 columns once (SlShape).
#include <algorithm>

#include "kernels.h"
#include "tc.cuh"

namespace arckv {

namespace {

constexpr int kSlBM = 128, kSlBK = 32;   // tile rows, K slab
constexpr int kSlChunkSlabs = 4;                      // 128 K per exact chunk
constexpr int kSlTileA = kSlBM * kSlBK * 2;   // 8 KB

// Each epilogue warp stages its 32 rows x 16 columns of results (rows padded
// to 17 elements) in shared memory and writes them back row-contiguously, so
// that the stores (and the loads of the `sub` mode) are coalesced.
constexpr int kSlStageLd = 17;
constexpr int kSlStageBytes = 32 * kSlStageLd * 8;

// Tile shapes.  BN = 64: eight epilogue warps, the exact-level and the
// high-level accumulators double-buffered in TMEM (6 x 64 + 2 x 64 columns), the
// results staged per warp for coalesced stores; for the short-K block
// products of the Cholesky, where each tile's epilogue overlaps the next
// tile's MMAs.  BN = 128: each MMA reads as many operand bytes as its tensor
// time allows (an N = 64 MMA reads more per cycle than shared memory
// delivers), sixteen epilogue warps (32 columns each), single-buffered
// accumulators (3 x 128 + 128 columns) and plain stores; for the long-K Grams
// and back-projections, whose epilogue runs once per tile.
template <int BN_>
struct SlShape {
  static constexpr int BN = BN_;
  static constexpr int EW = BN == 64 ? 8 : 16;              // epilogue warps
  static constexpr int THREADS = 64 + 32 * EW;
  static constexpr int NBUF = BN == 64 ? 2 : 1;             // accumulator buffers
  static constexpr bool STAGED = BN == 64;
  static constexpr int TILE_B = BN * kSlBK * 2;
  static constexpr int COLT = kSlBM / BN;                   // column tiles per row tile (lower mode)
  static_assert(BN == 64 || BN == 128, "tile widths");
  static_assert(3 * NBUF * BN + NBUF * BN <= 512, "TMEM columns");
};

template <int S, int BN>
struct SlCfg {
  using Sh = SlShape<BN>;
  static constexpr int STAGE_BYTES = Sh::STAGED ? Sh::EW * kSlStageBytes : 0;
  static constexpr int STAGE = S * (kSlTileA + Sh::TILE_B);
  // the ring takes what the staging tiles, the 1 KB alignment slack and 1 KB
  // of static barriers leave of the 227 KB a CTA may hold
  static constexpr int RING = 227 * 1024 - 2048 - STAGE_BYTES;
  static constexpr int STAGES = std::min(6, RING / STAGE);
  static constexpr int SMEM = STAGES * STAGE + 1024 + STAGE_BYTES;
  static_assert(STAGES >= 2, "two ring stages at least");
};

// Marks an element whose sum met a non-finite operand (kept as NaN).
constexpr int kSlNaN = -0x40000000;

// T 2^ex rounded once to fp64: the conversion of T rounds (to nearest even),
// the scaling by 2^ex is an exact exponent adjustment; ldexp only outside the
// normal range (never for finite operands).
__device__ __forceinline__ double compose_f64(long long T, int ex) {
  if (ex == kSlNaN) return __longlong_as_double(0x7FF8000000000000ll);
  const double d = __ll2double_rn(T);
  const long long bits = __double_as_longlong(d);
  const int E = (int)((bits >> 52) & 0x7FF);
  if (E == 0) return d;   // zero (|T| >= 1 otherwise)
  const int E2 = E + ex;
  if (E2 <= 0 || E2 >= 2047) return ldexp(d, ex);
  return __longlong_as_double(bits + ((long long)ex << 52));
}

// T 2^ex rounded once to fp32.
__device__ __forceinline__ float compose_f32(long long T, int ex) {
  if (ex == kSlNaN) return __uint_as_float(0x7FC00000u);
  const float f = __ll2float_rn(T);           // the one rounding; the scaling below is exact
  const unsigned int b = __float_as_uint(f);
  const int E = (int)((b >> 23) & 0xFFu);
  if (E == 0) return f;                       // zero (T below 2^24 never rounds to a subnormal)
  const int E2 = E + ex;
  if (E2 <= 0 || E2 >= 255) return ldexpf(f, ex);
  return __uint_as_float((b & 0x807FFFFFu) | ((unsigned int)E2 << 23));
}

// A tile element: the integer T of its sum (units 2^-44 of the scaled
// operands) and the power of two that scales it back.
struct SlVal {
  long long T;
  int ex;
};

// Epilogue outputs: make() turns a tile element into the stored type; store()
// writes one element (row < M, col < N).
struct SlOutF64 {
  using Elem = double;
  double* C;
  long long cbs;
  int ldc;
  int sub;   // 0: C = A B^T; 1: C -= A B^T
  // `sub`: bring the 32 values this thread's row will update into L2 while
  // the tile's products run
  __device__ __forceinline__ void prefetch(int b, int row, int c0, int M, int N) const {
    if (!sub || row >= M) return;
    const double* d = C + (long long)b * cbs + (long long)row * ldc + c0;
    asm volatile("prefetch.global.L2 [%0];" ::"l"(d));
    if (c0 + 16 < N) asm volatile("prefetch.global.L2 [%0];" ::"l"(d + 16));
  }
  __device__ __forceinline__ double make(SlVal v) const { return compose_f64(v.T, v.ex); }
  __device__ __forceinline__ double* at(int b, int row, int col) const {
    return C + (long long)b * cbs + (long long)row * ldc + col;
  }
  __device__ __forceinline__ double old(const double* d) const { return sub ? __ldcg(d) : 0.0; }
  __device__ __forceinline__ void put(double* d, double old, double v) const { *d = sub ? old - v : v; }
};
struct SlOutF32 {
  using Elem = float;
  float* C;
  long long cbs;
  int ldc;
  __device__ __forceinline__ void prefetch(int, int, int, int, int) const {}
  __device__ __forceinline__ float make(SlVal v) const { return compose_f32(v.T, v.ex); }
  __device__ __forceinline__ float* at(int b, int row, int col) const {
    return C + (long long)b * cbs + (long long)row * ldc + col;
  }
  __device__ __forceinline__ float old(const float*) const { return 0.f; }
  __device__ __forceinline__ void put(float* d, float, float v) const { *d = v; }
};

// One warp's 32 rows (y0 + lane) x 16 columns (c0..) of results: each lane
// makes its row's values into the staging tile, then the warp writes the tile
// two rows per instruction (16 lanes per row: consecutive columns).
template <class Out, class F>
__device__ __forceinline__ void sl_store_rows(const Out& out, typename Out::Elem* stg, int lane, int b, int y0, int c0,
                                              int M, int N, F&& val) {
  using E = typename Out::Elem;
#pragma unroll
  for (int e = 0; e < 16; ++e) stg[lane * kSlStageLd + e] = out.make(val(e));
  __syncwarp();
  const int rr = lane >> 4, cc = lane & 15, col = c0 + cc;
  E* dst[16];
  E old[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) {   // all loads of the `sub` mode in flight before the stores
    const int row = y0 + 2 * i + rr;
    dst[i] = (row < M && col < N) ? out.at(b, row, col) : nullptr;
    old[i] = dst[i] ? out.old(dst[i]) : E(0);
  }
#pragma unroll
  for (int i = 0; i < 16; ++i)
    if (dst[i]) out.put(dst[i], old[i], stg[(2 * i + rr) * kSlStageLd + cc]);
  __syncwarp();
}

// The same 16 values of one row (row < M), written by their own thread.
template <class Out, class F>
__device__ __forceinline__ void sl_store_direct(const Out& out, int b, int row, int c0, int M, int N, F&& val) {
  if (row >= M) return;
#pragma unroll
  for (int e = 0; e < 16; ++e)
    if (c0 + e < N) {
      auto* d = out.at(b, row, c0 + e);
      out.put(d, out.old(d), out.make(val(e)));
    }
}

// Column tiles [nt0, row end) of row tile i: all of [nt0, nt1), or with
// `lower` only those that reach the lower triangle (column tile start <= row
// tile end) of a square product (ct column tiles per row tile).
__host__ __device__ __forceinline__ int sl_row_tiles(int i, int nt0, int nt1, bool lower, int ct) {
  const int e = lower ? (nt1 < ct * (i + 1) ? nt1 : ct * (i + 1)) : nt1;
  return e > nt0 ? e - nt0 : 0;
}
// Tile tl of the batch-major enumeration, column tiles fastest.
__device__ __forceinline__ void sl_tile(int tl, int Mt, int nt0, int nt1, bool lower, int ct, int per, int& b, int& mt,
                                        int& nt) {
  b = tl / per;
  int r = tl - b * per;
  if (!lower) {
    mt = r / (nt1 - nt0);
    nt = nt0 + (r - mt * (nt1 - nt0));
    return;
  }
  mt = 0;
  while (r >= sl_row_tiles(mt, nt0, nt1, true, ct)) {
    r -= sl_row_tiles(mt, nt0, nt1, true, ct);
    ++mt;
  }
  nt = nt0 + r;
}

template <int S, class Out, int BN>
__global__ void __launch_bounds__(SlShape<BN>::THREADS, 1)
    sliced_gemm_kernel(const __grid_constant__ CUtensorMap mA, const __grid_constant__ CUtensorMap mB, const Out out,
                       const int* __restrict__ eA, const int* __restrict__ eB, int H, int M, int N, int K, int lower,
                       int nt0, int nt1, DevStatus* stt) {
  using C = SlCfg<S, BN>;
  using Sh = SlShape<BN>;
  constexpr int STAGES = C::STAGES, EW = Sh::EW, NBUF = Sh::NBUF, TILE_B = Sh::TILE_B;
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t full[STAGES], empty[STAGES], accf[2], acce[2], l5f[2], l5e[2], drain;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;
  const uint32_t raw = tc::smem_u32(smem_raw);
  uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nk = (K + kSlBK - 1) / kSlBK;
  const int nchunks = (nk + kSlChunkSlabs - 1) / kSlChunkSlabs;
  const int Mt = (M + kSlBM - 1) / kSlBM;
  int per = 0;
  for (int i = 0; i < Mt; ++i) per += sl_row_tiles(i, nt0, nt1, lower != 0, Sh::COLT);
  const int ntiles = H * per;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&accf[i], 1);
      tc::mbar_init(&acce[i], EW);
      tc::mbar_init(&l5f[i], 1);
      tc::mbar_init(&l5e[i], EW);
    }
    tc::mbar_init(&drain, 1);
    abort_flag = 0;
    tc::mbar_fence_init();
  }
  // TMEM: exact levels 2..4 of two alternating chunks at columns (buf * 3 + lvl) * 64,
  // the levels above 4 of two alternating tiles at columns 384 + 64 (tile & 1)
  if (warp == 1) tc::tmem_alloc(&tmem_slot, 512);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_slot;
  volatile int* abortp = &abort_flag;

  if (warp == 0) {
    if (lane == 0) {
      tc::tma_prefetch(&mA);
      tc::tma_prefetch(&mB);
      int g = 0;
      bool ok = true;
      for (int tl = blockIdx.x; tl < ntiles && ok; tl += gridDim.x) {
        int b, mt, nt;
        sl_tile(tl, Mt, nt0, nt1, lower != 0, Sh::COLT, per, b, mt, nt);
        for (int kb = 0; kb < nk; ++kb) {
          const int s = g % STAGES;
          if (g >= STAGES && !tc::mbar_wait(&empty[s], ((g / STAGES) - 1) & 1, abortp, stt)) {
            ok = false;
            break;
          }
          uint8_t* st = base + s * C::STAGE;
          tc::mbar_arrive_expect_tx(&full[s], C::STAGE);
#pragma unroll
          for (int i = 0; i < S; ++i) {
            tc::tma_load_3d(st + i * kSlTileA, &mA, kb * kSlBK, mt * kSlBM, i * H + b, &full[s]);
            tc::tma_load_3d(st + S * kSlTileA + i * TILE_B, &mB, kb * kSlBK, nt * BN, i * H + b, &full[s]);
          }
          ++g;
        }
      }
      volatile int never = 0;
      for (int k = g > STAGES ? g - STAGES : 0; k < g; ++k)
        tc::mbar_wait(&full[k % STAGES], (k / STAGES) & 1, &never, stt);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = tc::idesc_bf16_f32(BN);
      bool ok = true;
      int g = 0, cg = 0, tcount = 0;
      for (int tl = blockIdx.x; tl < ntiles && ok; tl += gridDim.x, ++tcount) {
        // the level-5+ accumulator of this buffer must have been read (NBUF tiles ago)
        const int b5 = tcount % NBUF, u5 = tcount / NBUF;
        if (u5 >= 1 && !tc::mbar_wait(&l5e[b5], (u5 - 1) & 1, abortp, stt)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const uint32_t t5 = tmem + (uint32_t)((3 * NBUF + b5) * BN);
        bool started5 = false;
        for (int c = 0; c < nchunks && ok; ++c, ++cg) {
          const int buf = cg % NBUF, ub = cg / NBUF;
          if (ub >= 1 && !tc::mbar_wait(&acce[buf], (ub - 1) & 1, abortp, stt)) {
            ok = false;
            break;
          }
          tc::fence_after_sync();
          bool started[3] = {false, false, false};
          const int kb0 = c * kSlChunkSlabs, kb1 = min(nk, kb0 + kSlChunkSlabs);
          for (int kb = kb0; kb < kb1; ++kb, ++g) {
            const int s = g % STAGES;
            if (!tc::mbar_wait(&full[s], (g / STAGES) & 1, abortp, stt)) {
              ok = false;
              break;
            }
            tc::fence_after_sync();
            const uint32_t a = tc::smem_u32(base + s * C::STAGE), bb = a + S * kSlTileA;
#pragma unroll
            for (int ks = 0; ks < kSlBK / 16; ++ks) {
#pragma unroll
              for (int i = 0; i < S; ++i) {
                const uint64_t ad = tc::sdesc_k64(a + i * kSlTileA + ks * 32);
#pragma unroll
                for (int j = 0; j < S; ++j) {
                  const uint64_t bd = tc::sdesc_k64(bb + j * TILE_B + ks * 32);
                  const int lvl = i + j;   // 0-based: level l = lvl + 2
                  if (lvl <= 2) {
                    tc::mma_f16(tmem + (uint32_t)((buf * 3 + lvl) * BN), ad, bd, idesc, started[lvl] ? 1u : 0u);
                    started[lvl] = true;
                  } else {
                    tc::mma_f16(t5, ad, bd, idesc, started5 ? 1u : 0u);
                    started5 = true;
                  }
                }
              }
            }
            tc::mma_commit(&empty[s]);
          }
          if (ok) tc::mma_commit(&accf[buf]);
        }
        if (ok) tc::mma_commit(&l5f[b5]);
      }
      tc::mma_commit(&drain);
      volatile int never = 0;
      tc::mbar_wait(&drain, 0, &never, stt);
    }
  } else {
    const int q = warp & 3;                 // TMEM lane quarter
    const int part = (warp - 2) >> 2;       // 32-column part of the tile
    const int row_in = q * 32 + lane;
    bool ok = true;
    int kc = 0, tcount = 0;
    for (int tl = blockIdx.x; tl < ntiles && ok; tl += gridDim.x, ++tcount) {
      int b, mt, nt;
      sl_tile(tl, Mt, nt0, nt1, lower != 0, Sh::COLT, per, b, mt, nt);
      // exact running sum of levels 2..4 in units of 2^-32: level l contributes
      // its integer chunk sums shifted left by 8 (4 - l) bits (|sum| < 2^47)
      out.prefetch(b, mt * kSlBM + row_in, nt * BN + part * 32, M, N);
      long long acc[32];
#pragma unroll
      for (int e = 0; e < 32; ++e) acc[e] = 0;
      for (int c = 0; c < nchunks; ++c, ++kc) {
        const int buf = kc % NBUF;
        ok = tc::mbar_wait(&accf[buf], (kc / NBUF) & 1, abortp, stt);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) break;
        tc::fence_after_sync();
#pragma unroll
        for (int l = 0; l < 3; ++l) {
          // the chunk's level sum is an integer times 2^(-8 (l + 2)), below 2^24 in magnitude
          const float sc = l == 0 ? 65536.f : (l == 1 ? 16777216.f : 4294967296.f);
          const int sh = 16 - 8 * l;
#pragma unroll
          for (int p2 = 0; p2 < 2; ++p2) {
            float v[16];
            tc::tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)((buf * 3 + l) * BN + part * 32 + p2 * 16), v);
#pragma unroll
            for (int e = 0; e < 16; ++e) acc[p2 * 16 + e] += (long long)__float2int_rn(v[e] * sc) << sh;
          }
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&acce[buf]);
      }
      if (!ok) break;
      const int b5 = tcount % NBUF;
      ok = __all_sync(0xffffffffu, tc::mbar_wait(&l5f[b5], (tcount / NBUF) & 1, abortp, stt));
      if (!ok) break;
      tc::fence_after_sync();
      float v5[2][16];
      const uint32_t t5 = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)((3 * NBUF + b5) * BN + part * 32);
      tc::tmem_ld16(t5, v5[0]);
      tc::tmem_ld16(t5 + 16u, v5[1]);
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&l5e[b5]);
      const int row = mt * kSlBM + row_in;
      const int er = row < M ? eA[(long long)b * M + row] : 0;
      typename Out::Elem* stg =
          Sh::STAGED ? (typename Out::Elem*)(base + C::STAGES * C::STAGE + (warp - 2) * kSlStageBytes) : nullptr;
      const int* ecol = eB + (long long)b * N;
      // the sum in units of 2^-44: the exact levels (|acc| < 2^47 in units
      // of 2^-32) and the levels above 4 (|v5| < 2^-8) rounded to the unit,
      // taken as two fp32 halves of 22 bits (no 64-bit conversion)
      // (a non-finite operand leaves NaN in the levels above 4: every slice of
      // its row or column is NaN; such elements are marked in nanmask)
      unsigned nanmask = 0;
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        const float h = v5[e >> 4][e & 15] * 0x1p22f;   // exact
        if (h != h) nanmask |= 1u << e;
        const int hi = __float2int_rn(h);
        const int lo = __float2int_rn((h - (float)hi) * 0x1p22f);   // both steps exact
        acc[e] = acc[e] * 4096ll + (long long)hi * 4194304ll + lo;
      }
#pragma unroll
      for (int p2 = 0; p2 < 2; ++p2) {
        const int c0 = nt * BN + part * 32 + p2 * 16;
        int ec[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) ec[e] = c0 + e < N ? ecol[c0 + e] : 0;
        auto val = [&](int e) -> SlVal {
          if ((nanmask >> (p2 * 16 + e)) & 1u) return SlVal{0, kSlNaN};
          return SlVal{acc[p2 * 16 + e], er + ec[e] - 44};
        };
        if constexpr (Sh::STAGED)
          sl_store_rows(out, stg, lane, b, mt * kSlBM + q * 32, c0, M, N, val);
        else
          sl_store_direct(out, b, row, c0, M, N, val);
      }
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 512);
  }
}

// --------------------------------------------------------------- slicing

// Bits of |x|: for non-negative floats the bit patterns order like the values,
// so maxima of magnitudes are integer maxima.
__device__ __forceinline__ unsigned long long mag_bits(double x) {
  return (unsigned long long)__double_as_longlong(x) & 0x7FFFFFFFFFFFFFFFull;
}
__device__ __forceinline__ unsigned long long mag_bits(float x) { return __float_as_uint(x) & 0x7FFFFFFFu; }
__device__ __forceinline__ unsigned long long raw_bits(double x) { return (unsigned long long)__double_as_longlong(x); }
__device__ __forceinline__ unsigned long long raw_bits(float x) { return __float_as_uint(x); }

template <typename T>
struct FBits;
template <>
struct FBits<double> {
  static constexpr int kMant = 52, kBias = 1023, kExpMask = 0x7FF;
};
template <>
struct FBits<float> {
  static constexpr int kMant = 23, kBias = 127, kExpMask = 0xFF;
};

// Exponent of a row or column holding a non-finite value: its slices are NaN.
constexpr int kSlNonFinite = 0x40000000;

// Exponent e with |x| < 2^e for every |x| <= the magnitude whose bits are mb
// (frexp's exponent; 0 for 0, kSlNonFinite for a non-finite maximum).
template <typename T>
__device__ __forceinline__ int bound_exp_bits(unsigned long long mb) {
  using F = FBits<T>;
  if (mb == 0) return 0;
  const int E = (int)(mb >> F::kMant);
  if (E == F::kExpMask) return kSlNonFinite;
  if (E == 0) {   // subnormal: position of the leading mantissa bit
    const int lead = 63 - __clzll((long long)mb);
    return lead - F::kMant - F::kBias + 2;
  }
  return E - F::kBias + 1;
}

// Z = round(x 2^(8 S - e)) from the bits of x (|x| < 2^e): |Z| <= 2^(8 S).
template <int S, typename T>
__device__ __forceinline__ long long fixed_digits(T x, int e) {
  using F = FBits<T>;
  const unsigned long long mb = mag_bits(x);
  const int E = (int)(mb >> F::kMant);
  const unsigned long long m = (mb & ((1ull << F::kMant) - 1)) | (E ? (1ull << F::kMant) : 0ull);
  const int Ee = E ? E : 1;
  // x = m 2^(Ee - bias - mant); Z = m 2^-sh
  const int sh = F::kBias + F::kMant + e - 8 * S - Ee;
  long long Z;
  if (sh <= 0)
    Z = (long long)(m << (-sh));   // -sh <= 8 S - mant: no overflow
  else if (sh >= 63)
    Z = 0;
  else
    Z = (long long)((m + (1ull << (sh - 1))) >> sh);
  return (mag_bits(x) != raw_bits(x)) ? -Z : Z;   // sign bit set
}

// The S bf16 slices x_i = I_i 2^(-8 i) of Z 2^(-8 S): balanced base-256
// digits, I_S..I_2 in [-128, 127], I_1 = what remains (|I_1| <= 256).
// e = kSlNonFinite gives NaN slices.
template <int S, typename T>
__device__ __forceinline__ void digit_slices(T x, int e, bf16 (&o)[S]) {
  static_assert(S <= 5, "slice scales are built as normal fp32 powers of two");
  if (e == kSlNonFinite) {
#pragma unroll
    for (int i = 0; i < S; ++i) o[i] = __ushort_as_bfloat16((unsigned short)0x7FC0);
    return;
  }
  long long Z = fixed_digits<S>(x, e);
#pragma unroll
  for (int i = S - 1; i >= 1; --i) {
    const int d = (int)((Z + 128) & 255) - 128;
    Z = (Z - d) >> 8;
    o[i] = __float2bfloat16_rn((float)d * __uint_as_float((unsigned)(127 - 8 * (i + 1)) << 23));
  }
  o[0] = __float2bfloat16_rn((float)Z * 0x1p-8f);
}

// Row-sliced operand: X [H][R][K] (rows ldx apart, batches xbs apart) ->
// slices [S][H][R][ldo] bf16 and exponents [H][R].  One warp per row, four
// consecutive elements per lane and round, each plane's four slices written
// as one 8-byte store (ldo is a multiple of 8, so every plane row is 16-byte
// aligned).
template <int S, typename T>
__global__ void __launch_bounds__(256) slice_rows_kernel(const T* __restrict__ X, int R, int K, int ldx, long long xbs,
                                                         int H, bf16* __restrict__ out, int ldo,
                                                         int* __restrict__ ex) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long gr = (long long)blockIdx.x * 8 + warp;   // row over all batches
  if (gr >= (long long)H * R) return;
  const int b = (int)(gr / R), r = (int)(gr - (long long)b * R);
  const T* x = X + (long long)b * xbs + (long long)r * ldx;
  unsigned long long mb = 0;
  for (int k = 4 * lane; k < K; k += 128) {
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (k + u < K) mb = max(mb, mag_bits(x[k + u]));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mb = max(mb, __shfl_xor_sync(0xffffffffu, mb, o));
  const int e = bound_exp_bits<T>(mb);
  if (lane == 0) ex[gr] = e;
  const long long slice = (long long)H * R * ldo;
  bf16* o = out + gr * ldo;
  for (int k = 4 * lane; k < K; k += 128) {
    bf16 s[4][S];
#pragma unroll
    for (int u = 0; u < 4; ++u) digit_slices<S>(k + u < K ? x[k + u] : T(0), e, s[u]);
    if (k + 4 <= K) {
#pragma unroll
      for (int i = 0; i < S; ++i) {
        __nv_bfloat162 lo2, hi2;
        lo2.x = s[0][i];
        lo2.y = s[1][i];
        hi2.x = s[2][i];
        hi2.y = s[3][i];
        uint2 w;
        w.x = *reinterpret_cast<const unsigned int*>(&lo2);
        w.y = *reinterpret_cast<const unsigned int*>(&hi2);
        *reinterpret_cast<uint2*>(o + i * slice + k) = w;
      }
    } else {
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (k + u < K) {
#pragma unroll
          for (int i = 0; i < S; ++i) o[i * slice + k + u] = s[u][i];
        }
    }
  }
}

// Column maxima exponents of X [H][K][R] (R contiguous, rows ldx apart): ex [H][R].
// A CTA takes 32 columns (lane = column, coalesced rows); its 32 warps split
// the rows (four loads in flight each) and meet in shared memory.
template <typename T>
__global__ void __launch_bounds__(1024) col_exp_kernel(const T* __restrict__ X, int K, int R, int ldx, long long xbs,
                                                       int* __restrict__ ex) {
  __shared__ unsigned long long part[32][33];
  const int b = blockIdx.y, lane = threadIdx.x & 31, warp = threadIdx.x >> 5, r = blockIdx.x * 32 + lane;
  const T* x = X + (long long)b * xbs + r;
  unsigned long long m0 = 0, m1 = 0, m2 = 0, m3 = 0;
  if (r < R) {
    int k = warp;
    for (; k + 96 < K; k += 128) {
      m0 = max(m0, mag_bits(x[(long long)k * ldx]));
      m1 = max(m1, mag_bits(x[(long long)(k + 32) * ldx]));
      m2 = max(m2, mag_bits(x[(long long)(k + 64) * ldx]));
      m3 = max(m3, mag_bits(x[(long long)(k + 96) * ldx]));
    }
    for (; k < K; k += 32) m0 = max(m0, mag_bits(x[(long long)k * ldx]));
  }
  part[warp][lane] = max(max(m0, m1), max(m2, m3));
  __syncthreads();
  if (warp == 0 && r < R) {
    unsigned long long mb = part[0][lane];
#pragma unroll
    for (int w = 1; w < 32; ++w) mb = max(mb, part[w][lane]);
    ex[(long long)b * R + r] = bound_exp_bits<T>(mb);
  }
}

// Column-sliced operand (the rows of X^T): X [H][K][R] -> slices
// [S][H][R][ldo] of X^T with the exponents of col_exp_kernel; 32 x 32 tiles
// through shared memory.
template <int S, typename T>
__global__ void __launch_bounds__(256) slice_cols_kernel(const T* __restrict__ X, int K, int R, int ldx, long long xbs,
                                                         int H, const int* __restrict__ ex, bf16* __restrict__ out,
                                                         int ldo) {
  const int b = blockIdx.z, r0 = blockIdx.x * 32, k0 = blockIdx.y * 32;
  __shared__ T tile[32][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const T* xb = X + (long long)b * xbs;
  for (int q = ty; q < 32; q += 8) {
    const int k = k0 + q, r = r0 + tx;
    tile[q][tx] = (k < K && r < R) ? xb[(long long)k * ldx + r] : T(0);
  }
  __syncthreads();
  const long long slice = (long long)H * R * ldo;
  for (int q = ty; q < 32; q += 8) {
    const int r = r0 + q, k = k0 + tx;
    if (r < R && k < K) {
      bf16 s[S];
      digit_slices<S>(tile[tx][q], ex[(long long)b * R + r], s);
      const long long o = ((long long)b * R + r) * ldo + k;
#pragma unroll
      for (int i = 0; i < S; ++i) out[i * slice + o] = s[i];
    }
  }
}

int g_sliced_fail = 0;   // which step of the last failed launch_sliced gave up (diagnostics)

template <int S, int BN, class Out>
int launch_sliced(const bf16* As, const int* eA, int M, const bf16* Bs, const int* eB, int N, int K, int ldk, int H,
                  bool lower, const Out& out, DevStatus* stt, cudaStream_t st, int nt0 = 0, int nt1 = 1 << 30,
                  int max_ctas = 0) {
  CUtensorMap mA, mB;
  if (!encode_bf16_map_3d_sw64(&mA, As, K, M, (uint64_t)S * H, ldk, kSlBM) ||
      !encode_bf16_map_3d_sw64(&mB, Bs, K, N, (uint64_t)S * H, ldk, BN)) {
    g_sliced_fail = 1;
    return -1;
  }
  using C = SlCfg<S, BN>;
  using Sh = SlShape<BN>;
  auto kern = sliced_gemm_kernel<S, Out, BN>;
  const cudaError_t ea = set_dyn_smem((const void*)kern, C::SMEM);
  if (ea != cudaSuccess) {
    g_sliced_fail = 100 + (int)ea;
    return -1;
  }
  const int Mt = cdiv(M, kSlBM), Nt = cdiv(N, BN);
  nt1 = std::min(nt1, Nt);
  nt0 = std::max(nt0, 0);
  long long per = 0;
  for (int i = 0; i < Mt; ++i) per += sl_row_tiles(i, nt0, nt1, lower, Sh::COLT);
  if (per == 0) return 0;   // no tile in the column range
  int grid = (int)std::min<long long>(per * H, tc_gemm_sm_count());
  if (max_ctas > 0) grid = std::min(grid, max_ctas);
  kern<<<grid, Sh::THREADS, C::SMEM, st>>>(mA, mB, out, eA, eB, H, M, N, K, lower ? 1 : 0, nt0, nt1, stt);
  const cudaError_t el = cudaGetLastError();
  if (el != cudaSuccess) g_sliced_fail = 1000 + (int)el;
  return el == cudaSuccess ? 1 : -1;
}

}  // namespace

size_t sliced_ld(int K) { return (size_t)(K + 7) / 8 * 8; }

int sliced_last_failure() { return g_sliced_fail; }

bool sliced_supported(int K) { return K >= 1 && K <= kSlicedMaxK; }

template <typename T>
static int slice_rows_t(int S, const T* X, int R, int K, int ldx, long long xbs, int H, bf16* out, int* ex,
                        cudaStream_t st) {
  const int grid = cdiv((long long)H * R, 8), ldo = (int)sliced_ld(K);
  if (S == 3)
    slice_rows_kernel<3, T><<<grid, 256, 0, st>>>(X, R, K, ldx, xbs, H, out, ldo, ex);
  else if (S == 4)
    slice_rows_kernel<4, T><<<grid, 256, 0, st>>>(X, R, K, ldx, xbs, H, out, ldo, ex);
  else if (S == 5)
    slice_rows_kernel<5, T><<<grid, 256, 0, st>>>(X, R, K, ldx, xbs, H, out, ldo, ex);
  else
    return -1;
  return 1;
}

int launch_slice_rows(int S, const float* X, int R, int K, int ldx, long long xbs, int H, bf16* out, int* ex,
                      cudaStream_t st) {
  return slice_rows_t<float>(S, X, R, K, ldx, xbs, H, out, ex, st);
}

int launch_slice_rows(int S, const double* X, int R, int K, int ldx, long long xbs, int H, bf16* out, int* ex,
                      cudaStream_t st) {
  return slice_rows_t<double>(S, X, R, K, ldx, xbs, H, out, ex, st);
}

template <typename T>
static int slice_cols_t(int S, const T* X, int K, int R, int ldx, long long xbs, int H, bf16* out, int* ex,
                        cudaStream_t st) {
  const int ldo = (int)sliced_ld(K);
  col_exp_kernel<T><<<dim3(cdiv(R, 32), H), 1024, 0, st>>>(X, K, R, ldx, xbs, ex);
  const dim3 grid(cdiv(R, 32), cdiv(K, 32), H);
  if (S == 3)
    slice_cols_kernel<3, T><<<grid, 256, 0, st>>>(X, K, R, ldx, xbs, H, ex, out, ldo);
  else if (S == 4)
    slice_cols_kernel<4, T><<<grid, 256, 0, st>>>(X, K, R, ldx, xbs, H, ex, out, ldo);
  else if (S == 5)
    slice_cols_kernel<5, T><<<grid, 256, 0, st>>>(X, K, R, ldx, xbs, H, ex, out, ldo);
  else
    return -1;
  return 2;
}

int launch_slice_cols(int S, const float* X, int K, int R, int ldx, long long xbs, int H, bf16* out, int* ex,
                      cudaStream_t st) {
  return slice_cols_t<float>(S, X, K, R, ldx, xbs, H, out, ex, st);
}

int launch_slice_cols(int S, const double* X, int K, int R, int ldx, long long xbs, int H, bf16* out, int* ex,
                      cudaStream_t st) {
  return slice_cols_t<double>(S, X, K, R, ldx, xbs, H, out, ex, st);
}

int launch_sliced_gram_lower(int S, const bf16* Xs, const int* ex, int R, int K, int H, double* G, DevStatus* stt,
                             cudaStream_t st) {
  return launch_sliced_f64(S, Xs, ex, R, Xs, ex, R, K, H, G, (long long)R * R, R, true, false, stt, st);
}

// 128-wide tiles for the long-K products of up to four slices (the Grams and
// back-projections: the epilogue runs once per many chunks), 64-wide ones for
// the short-K block products of the Cholesky.
static bool sliced_wide(int S, int K) { return S <= 4 && K >= 256; }

int launch_sliced_f64(int S, const bf16* As, const int* eA, int M, const bf16* Bs, const int* eB, int N, int K, int H,
                      double* C, long long cbs, int ldc, bool lower, bool sub, DevStatus* stt, cudaStream_t st,
                      int nt0, int nt1, int max_ctas) {
  const int ldk = (int)sliced_ld(K);
  const SlOutF64 out{C, cbs, ldc, sub ? 1 : 0};
  const bool w = sliced_wide(S, K);
  if (S == 3)
    return w ? launch_sliced<3, 128>(As, eA, M, Bs, eB, N, K, ldk, H, lower, out, stt, st)
             : launch_sliced<3, 64>(As, eA, M, Bs, eB, N, K, ldk, H, lower, out, stt, st);
  if (S == 4)
    return w ? launch_sliced<4, 128>(As, eA, M, Bs, eB, N, K, ldk, H, lower, out, stt, st)
             : launch_sliced<4, 64>(As, eA, M, Bs, eB, N, K, ldk, H, lower, out, stt, st);
  if (S == 5) return launch_sliced<5, 64>(As, eA, M, Bs, eB, N, K, ldk, H, lower, out, stt, st, nt0, nt1, max_ctas);
  return -1;
}

int launch_sliced_product_f32(int S, const bf16* As, const int* eA, int M, const bf16* Bs, const int* eB, int N, int K,
                              int H, float* C, int ldc, DevStatus* stt, cudaStream_t st) {
  const int ldk = (int)sliced_ld(K);
  const SlOutF32 out{C, (long long)M * ldc, ldc};
  const bool w = sliced_wide(S, K);
  if (S == 3)
    return w ? launch_sliced<3, 128>(As, eA, M, Bs, eB, N, K, ldk, H, false, out, stt, st)
             : launch_sliced<3, 64>(As, eA, M, Bs, eB, N, K, ldk, H, false, out, stt, st);
  if (S == 4)
    return w ? launch_sliced<4, 128>(As, eA, M, Bs, eB, N, K, ldk, H, false, out, stt, st)
             : launch_sliced<4, 64>(As, eA, M, Bs, eB, N, K, ldk, H, false, out, stt, st);
  return -1;
}

}  // namespace arckv
