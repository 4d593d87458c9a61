// fp64-grade products on the bf16 tensor pipe, for the ill-conditioned dual
// fits (App. A.9 Eqs. mass_fit, value_lstsq in their push-through form when
// t > n).
//
// Slices.  Row r of an operand X (fp32 or fp64) is scaled by 2^-e_r, where
// 2^e_r bounds the row's largest magnitude, and cut into S bf16 slices
//     X[r][k] = 2^e_r (x_1 + x_2 + ... + x_S) + residual,
//     x_i = I_i 2^(-8 i),  I_1 in [-256, 256],  I_i in [-128, 128] (i > 1),
// each x_i the rounding of what the earlier slices left to the next 8 bits, so
// |residual| <= 2^(-8 S - 1) 2^e_r.  Every slice is an integer of at most 8
// significant bits times a power of two: exact in bf16.
//
// Products.  C = A B^T is the sum over all S^2 slice pairs (i, j).  A pair's
// products are integers times 2^(-8(i + j)), so the pairs of one level
// l = i + j add up exactly in fp32 while the integer sum stays below 2^24:
// with 128 terms of K that holds for l <= 4 (at most 128 (2 * 256 * 128 +
// 128^2) < 2^24).  Levels 2, 3 and 4 therefore run in fresh TMEM accumulators
// per 128-wide K chunk, and the epilogue converts each chunk's sums to
// integers and adds them up exactly (in 64-bit, for K <= 26214); the levels
// above 4 weigh at most 2^-24 of the total and accumulate in one fp32
// accumulator over the whole K.  The result, assembled in fp64 and scaled by
// 2^(e_m + f_n), is the exact product of the sliced operands up to the fp32
// rounding of the levels above 4 (~2^-48 relative): the fp32 arithmetic of the
// tensor pipe never meets a rounding that matters.
//
// Kernel layout (persistent, one CTA per SM): warp 0 streams 32-wide K slabs
// of the S slices of a 128-row A tile and a 64-row B tile with TMA (64-byte
// swizzle) into a shared ring; warp 1 issues the S^2 tcgen05 MMAs (M = 128,
// N = 64, K = 16) of every K step into the level accumulators; warps 2..9
// drain the exact levels after every chunk (two warps per TMEM lane quarter,
// 32 columns each) and assemble the tile.
#include <algorithm>

#include "kernels.h"
#include "tc.cuh"

namespace arckv {

namespace {

constexpr int kSlBM = 128, kSlBN = 64, kSlBK = 32;   // tile rows, columns, K slab
constexpr int kSlChunkSlabs = 4;                      // 128 K per exact chunk
constexpr int kSlEpiWarps = 8;
constexpr int kSlThreads = 64 + 32 * kSlEpiWarps;
constexpr int kSlTileA = kSlBM * kSlBK * 2, kSlTileB = kSlBN * kSlBK * 2;   // 8 KB, 4 KB

template <int S>
struct SlCfg {
  static constexpr int STAGE = S * (kSlTileA + kSlTileB);
  static constexpr int STAGES = std::min(6, (200 * 1024) / STAGE);
  static constexpr int SMEM = STAGES * STAGE + 1024;
};

// Epilogue outputs: 16 consecutive columns c0.. of one row, value e given by
// val(e) (evaluated once per element, in order, so no array of them is held).
struct SlOutF64 {
  double* C;
  long long cbs;
  int ldc;
  int sub;   // 0: C = A B^T; 1: C -= A B^T
  template <class F>
  __device__ __forceinline__ void put(int b, int row, int c0, int M, int N, F&& val) const {
    if (row >= M) return;
    double* d = C + (long long)b * cbs + (long long)row * ldc + c0;
    if (((((uintptr_t)d) & 15) == 0) && c0 + 16 <= N) {
#pragma unroll
      for (int q = 0; q < 16; q += 2) {
        const double x0 = val(q), x1 = val(q + 1);
        if (sub) {
          const double2 o = *(const double2*)(d + q);
          *(double2*)(d + q) = make_double2(o.x - x0, o.y - x1);
        } else {
          *(double2*)(d + q) = make_double2(x0, x1);
        }
      }
    } else {
#pragma unroll
      for (int q = 0; q < 16; ++q)
        if (c0 + q < N) d[q] = sub ? d[q] - val(q) : val(q);
    }
  }
};
struct SlOutF32 {
  float* C;
  long long cbs;
  int ldc;
  template <class F>
  __device__ __forceinline__ void put(int b, int row, int c0, int M, int N, F&& val) const {
    if (row >= M) return;
    float* d = C + (long long)b * cbs + (long long)row * ldc + c0;
    if (((((uintptr_t)d) & 15) == 0) && c0 + 16 <= N) {
#pragma unroll
      for (int q = 0; q < 16; q += 4) {
        const float x0 = (float)val(q), x1 = (float)val(q + 1), x2 = (float)val(q + 2), x3 = (float)val(q + 3);
        *(float4*)(d + q) = make_float4(x0, x1, x2, x3);
      }
    } else {
#pragma unroll
      for (int q = 0; q < 16; ++q)
        if (c0 + q < N) d[q] = (float)val(q);
    }
  }
};

// Tiles of one batch: all (row tile, column tile) pairs, or with `lower` only
// those that reach the lower triangle (column tile start <= row tile end) of a
// square product; column tiles fastest.
__device__ __forceinline__ void sl_tile(int tl, int Mt, int Nt, bool lower, int& b, int& mt, int& nt) {
  if (!lower) {
    b = tl / (Mt * Nt);
    const int r = tl - b * (Mt * Nt);
    mt = r / Nt;
    nt = r - mt * Nt;
    return;
  }
  int per = 0;
  for (int i = 0; i < Mt; ++i) per += min(Nt, 2 * (i + 1));
  b = tl / per;
  int r = tl - b * per;
  mt = 0;
  while (r >= min(Nt, 2 * (mt + 1))) {
    r -= min(Nt, 2 * (mt + 1));
    ++mt;
  }
  nt = r;
}

template <int S, class Out>
__global__ void __launch_bounds__(kSlThreads, 1)
    sliced_gemm_kernel(const __grid_constant__ CUtensorMap mA, const __grid_constant__ CUtensorMap mB, const Out out,
                       const int* __restrict__ eA, const int* __restrict__ eB, int H, int M, int N, int K, int lower,
                       DevStatus* stt) {
  using C = SlCfg<S>;
  constexpr int STAGES = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t full[STAGES], empty[STAGES], accf[2], acce[2], l5f, l5e, drain;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;
  const uint32_t raw = tc::smem_u32(smem_raw);
  uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nk = (K + kSlBK - 1) / kSlBK;
  const int nchunks = (nk + kSlChunkSlabs - 1) / kSlChunkSlabs;
  const int Mt = (M + kSlBM - 1) / kSlBM, Nt = (N + kSlBN - 1) / kSlBN;
  int per = 0;
  if (lower) {
    for (int i = 0; i < Mt; ++i) per += min(Nt, 2 * (i + 1));
  } else {
    per = Mt * Nt;
  }
  const int ntiles = H * per;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::mbar_init(&accf[i], 1);
      tc::mbar_init(&acce[i], kSlEpiWarps);
    }
    tc::mbar_init(&l5f, 1);
    tc::mbar_init(&l5e, kSlEpiWarps);
    tc::mbar_init(&drain, 1);
    abort_flag = 0;
    tc::mbar_fence_init();
  }
  // TMEM: exact levels 2..4 of two alternating chunks at columns (buf * 3 + lvl) * 64,
  // the levels above 4 at column 384
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
        sl_tile(tl, Mt, Nt, lower != 0, b, mt, nt);
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
            tc::tma_load_3d(st + S * kSlTileA + i * kSlTileB, &mB, kb * kSlBK, nt * kSlBN, i * H + b, &full[s]);
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
      constexpr uint32_t idesc = tc::idesc_bf16_f32(kSlBN);
      bool ok = true;
      int g = 0, cg = 0, tcount = 0;
      for (int tl = blockIdx.x; tl < ntiles && ok; tl += gridDim.x, ++tcount) {
        // the level-5+ accumulator of the previous tile must have been read
        if (tcount >= 1 && !tc::mbar_wait(&l5e, (tcount - 1) & 1, abortp, stt)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        bool started5 = false;
        for (int c = 0; c < nchunks && ok; ++c, ++cg) {
          const int buf = cg & 1;
          if (cg >= 2 && !tc::mbar_wait(&acce[buf], ((cg >> 1) - 1) & 1, abortp, stt)) {
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
                  const uint64_t bd = tc::sdesc_k64(bb + j * kSlTileB + ks * 32);
                  const int lvl = i + j;   // 0-based: level l = lvl + 2
                  if (lvl <= 2) {
                    tc::mma_f16(tmem + (uint32_t)((buf * 3 + lvl) * 64), ad, bd, idesc, started[lvl] ? 1u : 0u);
                    started[lvl] = true;
                  } else {
                    tc::mma_f16(tmem + 384u, ad, bd, idesc, started5 ? 1u : 0u);
                    started5 = true;
                  }
                }
              }
            }
            tc::mma_commit(&empty[s]);
          }
          if (ok) tc::mma_commit(&accf[buf]);
        }
        if (ok) tc::mma_commit(&l5f);
      }
      tc::mma_commit(&drain);
      volatile int never = 0;
      tc::mbar_wait(&drain, 0, &never, stt);
    }
  } else {
    const int q = warp & 3;                 // TMEM lane quarter
    const int half = (warp - 2) >> 2;       // 32-column half of the 64-wide tile
    const int row_in = q * 32 + lane;
    bool ok = true;
    int kc = 0, tcount = 0;
    for (int tl = blockIdx.x; tl < ntiles && ok; tl += gridDim.x, ++tcount) {
      int b, mt, nt;
      sl_tile(tl, Mt, Nt, lower != 0, b, mt, nt);
      // exact running sum of levels 2..4 in units of 2^-32: level l contributes
      // its integer chunk sums shifted left by 8 (4 - l) bits (|sum| < 2^47)
      long long acc[32];
#pragma unroll
      for (int e = 0; e < 32; ++e) acc[e] = 0;
      for (int c = 0; c < nchunks; ++c, ++kc) {
        const int buf = kc & 1;
        ok = tc::mbar_wait(&accf[buf], (kc >> 1) & 1, abortp, stt);
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
            tc::tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)((buf * 3 + l) * 64 + half * 32 + p2 * 16), v);
#pragma unroll
            for (int e = 0; e < 16; ++e) acc[p2 * 16 + e] += (long long)__float2int_rn(v[e] * sc) << sh;
          }
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&acce[buf]);
      }
      if (!ok) break;
      ok = __all_sync(0xffffffffu, tc::mbar_wait(&l5f, tcount & 1, abortp, stt));
      if (!ok) break;
      tc::fence_after_sync();
      float v5[2][16];
      tc::tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + 384u + (uint32_t)(half * 32), v5[0]);
      tc::tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + 384u + (uint32_t)(half * 32 + 16), v5[1]);
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&l5e);
      const int row = mt * kSlBM + row_in;
      const int er = row < M ? eA[(long long)b * M + row] : 0;
      const int* ecol = eB + (long long)b * N;
#pragma unroll
      for (int p2 = 0; p2 < 2; ++p2) {
        const int c0 = nt * kSlBN + half * 32 + p2 * 16;
        out.put(b, row, c0, M, N, [&](int e) -> double {
          const double t = (double)acc[p2 * 16 + e] * 0x1p-32 + (double)v5[p2][e];   // |acc| < 2^53: exact
          // 2^(er + ec) built from its bits (row and column exponents of finite
          // fp32 / fp64 data stay well inside the normal range)
          const int ex = er + ecol[c0 + e];   // only evaluated for columns below N
          return (ex > -1023 && ex < 1024) ? t * __longlong_as_double((long long)(1023 + ex) << 52) : ldexp(t, ex);
        });
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

// Exponent e with |x| <= 2^e for every x of magnitude <= mx (0 for mx = 0).
template <typename T>
__device__ __forceinline__ int bound_exp(T mx) {
  int e = 0;
  if (mx > T(0)) frexp((double)mx, &e);
  return e;
}

// x 2^p, exact (the scale 2^p alone may not be representable: a row of tiny
// fp32 values has p > 127).
__device__ __forceinline__ float scale2(float x, int p) { return ldexpf(x, p); }
__device__ __forceinline__ double scale2(double x, int p) { return ldexp(x, p); }

// Slices of value x (already scaled by 2^-e into [-1, 1]): x_i = I_i 2^(-8 i).
template <int S, typename T>
__device__ __forceinline__ void make_slices(T y, bf16 (&o)[S]) {
  T r = y;
  T sc = T(256);
#pragma unroll
  for (int i = 0; i < S; ++i) {
    const T a = rint(r * sc) / sc;   // exact: power-of-two scaling and rounding to an integer
    o[i] = __float2bfloat16_rn((float)a);
    r = r - a;                       // exact: the bits of y below slice i
    sc *= T(256);
  }
}

// Row-sliced operand: X [H][R][K] (rows ldx apart, batches xbs apart) ->
// slices [S][H][R][ldo] bf16 and exponents [H][R].  One warp per row.
template <int S, typename T>
__global__ void __launch_bounds__(256) slice_rows_kernel(const T* __restrict__ X, int R, int K, int ldx, long long xbs,
                                                         int H, bf16* __restrict__ out, int ldo,
                                                         int* __restrict__ ex) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long gr = (long long)blockIdx.x * 8 + warp;   // row over all batches
  if (gr >= (long long)H * R) return;
  const int b = (int)(gr / R), r = (int)(gr - (long long)b * R);
  const T* x = X + (long long)b * xbs + (long long)r * ldx;
  T mx = T(0);
  for (int k = lane; k < K; k += 32) mx = fmax(mx, fabs(x[k]));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmax(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  const int e = bound_exp(mx);
  if (lane == 0) ex[gr] = e;
  const long long slice = (long long)H * R * ldo;
  bf16* o = out + gr * ldo;
  for (int k = lane; k < K; k += 32) {
    bf16 s[S];
    make_slices<S>(scale2(x[k], -e), s);
#pragma unroll
    for (int i = 0; i < S; ++i) o[i * slice + k] = s[i];
  }
}

// Column maxima exponents of X [H][K][R] (R contiguous, rows ldx apart): ex [H][R].
// A CTA takes 32 columns (lane = column, coalesced rows); its 32 warps split
// the rows (four loads in flight each) and meet in shared memory.
template <typename T>
__global__ void __launch_bounds__(1024) col_exp_kernel(const T* __restrict__ X, int K, int R, int ldx, long long xbs,
                                                       int* __restrict__ ex) {
  __shared__ T part[32][33];
  const int b = blockIdx.y, lane = threadIdx.x & 31, warp = threadIdx.x >> 5, r = blockIdx.x * 32 + lane;
  const T* x = X + (long long)b * xbs + r;
  T m0 = T(0), m1 = T(0), m2 = T(0), m3 = T(0);
  if (r < R) {
    int k = warp;
    for (; k + 96 < K; k += 128) {
      m0 = fmax(m0, fabs(x[(long long)k * ldx]));
      m1 = fmax(m1, fabs(x[(long long)(k + 32) * ldx]));
      m2 = fmax(m2, fabs(x[(long long)(k + 64) * ldx]));
      m3 = fmax(m3, fabs(x[(long long)(k + 96) * ldx]));
    }
    for (; k < K; k += 32) m0 = fmax(m0, fabs(x[(long long)k * ldx]));
  }
  part[warp][lane] = fmax(fmax(m0, m1), fmax(m2, m3));
  __syncthreads();
  if (warp == 0 && r < R) {
    T mx = part[0][lane];
#pragma unroll
    for (int w = 1; w < 32; ++w) mx = fmax(mx, part[w][lane]);
    ex[(long long)b * R + r] = bound_exp(mx);
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
      make_slices<S>(scale2(tile[tx][q], -ex[(long long)b * R + r]), s);
      const long long o = ((long long)b * R + r) * ldo + k;
#pragma unroll
      for (int i = 0; i < S; ++i) out[i * slice + o] = s[i];
    }
  }
}

int g_sliced_fail = 0;   // which step of the last failed launch_sliced gave up (diagnostics)

template <int S, class Out>
int launch_sliced(const bf16* As, const int* eA, int M, const bf16* Bs, const int* eB, int N, int K, int ldk, int H,
                  bool lower, const Out& out, DevStatus* stt, cudaStream_t st) {
  CUtensorMap mA, mB;
  if (!encode_bf16_map_3d_sw64(&mA, As, K, M, (uint64_t)S * H, ldk, kSlBM) ||
      !encode_bf16_map_3d_sw64(&mB, Bs, K, N, (uint64_t)S * H, ldk, kSlBN)) {
    g_sliced_fail = 1;
    return -1;
  }
  using C = SlCfg<S>;
  auto kern = sliced_gemm_kernel<S, Out>;
  const cudaError_t ea = set_dyn_smem((const void*)kern, C::SMEM);
  if (ea != cudaSuccess) {
    g_sliced_fail = 100 + (int)ea;
    return -1;
  }
  const int Mt = cdiv(M, kSlBM), Nt = cdiv(N, kSlBN);
  long long per = 0;
  if (lower) {
    for (int i = 0; i < Mt; ++i) per += std::min(Nt, 2 * (i + 1));
  } else {
    per = (long long)Mt * Nt;
  }
  const int grid = (int)std::min<long long>(per * H, tc_gemm_sm_count());
  kern<<<grid, kSlThreads, C::SMEM, st>>>(mA, mB, out, eA, eB, H, M, N, K, lower ? 1 : 0, stt);
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

int launch_sliced_f64(int S, const bf16* As, const int* eA, int M, const bf16* Bs, const int* eB, int N, int K, int H,
                      double* C, long long cbs, int ldc, bool lower, bool sub, DevStatus* stt, cudaStream_t st) {
  const int ldk = (int)sliced_ld(K);
  const SlOutF64 out{C, cbs, ldc, sub ? 1 : 0};
  if (S == 3) return launch_sliced<3>(As, eA, M, Bs, eB, N, K, ldk, H, lower, out, stt, st);
  if (S == 4) return launch_sliced<4>(As, eA, M, Bs, eB, N, K, ldk, H, lower, out, stt, st);
  if (S == 5) return launch_sliced<5>(As, eA, M, Bs, eB, N, K, ldk, H, lower, out, stt, st);
  return -1;
}

int launch_sliced_product_f32(int S, const bf16* As, const int* eA, int M, const bf16* Bs, const int* eB, int N, int K,
                              int H, float* C, int ldc, DevStatus* stt, cudaStream_t st) {
  const int ldk = (int)sliced_ld(K);
  const SlOutF32 out{C, (long long)M * ldc, ldc};
  if (S == 3) return launch_sliced<3>(As, eA, M, Bs, eB, N, K, ldk, H, false, out, stt, st);
  if (S == 4) return launch_sliced<4>(As, eA, M, Bs, eB, N, K, ldk, H, false, out, stt, st);
  return -1;
}

}  // namespace arckv
