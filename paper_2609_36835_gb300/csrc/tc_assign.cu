// Tensor-core stages of Sec. 3.4:
//   * reference logits l = scale Q K^T (bf16 operands are exact, one MMA per
//     product, fp32 accumulation);
//   * the anchor assignment kappa(j) = argmax_r u_j . u_{s_r}
//     (Eq. anchor_assignment) as a split-bf16 GEMM of the transposed profiles
//     U^T [T x n] against the anchor rows U_S^T [t x n] whose epilogue keeps
//     the row maximum (lowest r on ties) and merges it across column tiles
//     with a 64-bit atomicMax; the T x t similarity is never stored.
#include <algorithm>

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

// The same with eight epilogue warps, two per TMEM lane quarter, for 256-wide
// tiles (each warp takes 128 columns).
struct TcEpiArgmax8 : TcEpiArgmax {
  static constexpr int kEpiWarps = 8;
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

// Where key j's profile row goes.  An anchor's (anchors[r] == j) to row r of
// the anchor rows U_S^T; every other key to row j - #{anchors < j} of the
// compacted key rows, the T - t rows the assignment GEMM takes as M: the
// anchors' own assignment is fixed, kappa(s_r) = r, so their GEMM rows would
// only be discarded.  ab: the head's anchors, ascending (checked upstream).
// The element offset of that row (an anchor row as -1 - offset), or
// kNoRow when invalid anchors (a caller's, already flagged
// ARCKV_ERR_INVALID_ARG) leave no valid row.
constexpr long long kNoRow = -(1ll << 62);
__device__ __forceinline__ long long profile_row(const int* ab, int t, int T, int b, int j, int ldn, int* kmap) {
  int lo = 0, hi = t;   // first index with ab[index] >= j
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (ab[mid] < j) lo = mid + 1;
    else hi = mid;
  }
  if (lo < t && ab[lo] == j) return -1 - ((long long)b * t + lo) * ldn;
  const int r = j - lo;
  if (r < 0 || r >= T - t) return kNoRow;
  kmap[(long long)b * T + r] = j;
  return ((long long)b * T + r) * ldn;
}

// Output rows of the profiles: key rows (Ut, compacted) or anchor rows (S),
// and the compacted row -> key map.
struct ProfileOut {
  bf16 *Ut_hi, *Ut_lo, *S_hi, *S_lo;
  int* kmap;           // [H][T]: key of compacted row c (c < T - t)
  const int* anchors;  // [H][t]
  int t;
};

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
__global__ void __launch_bounds__(512) col_profiles_kernel(const float* L, float* logphi, ProfileOut po, int n, int T,
                                                           int ldn) {
  const int b = blockIdx.y, lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int j0 = blockIdx.x * 32, j = j0 + lane;
  __shared__ float red[3][16][32];
  __shared__ float cstat[2][32];
  __shared__ float tile[64][33];
  __shared__ long long orow[32];   // element offset of each column's output row
  if (po.Ut_hi != nullptr && w == 0 && j < T)
    orow[lane] = profile_row(po.anchors + (long long)b * po.t, po.t, T, b, j, ldn, po.kmap);
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
  if (po.Ut_hi == nullptr) return;
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
      if (jj < T && i < ldn && orow[c] != kNoRow) {
        bf16 h0, l0, h1, l1;
        split_bf16(tile[2 * lane][c], h0, l0);
        split_bf16(tile[2 * lane + 1][c], h1, l1);
        const long long ro = orow[c];
        bf16* dh = ro >= 0 ? po.Ut_hi + ro : po.S_hi + (-1 - ro);
        bf16* dl = ro >= 0 ? po.Ut_lo + ro : po.S_lo + (-1 - ro);
        *(__nv_bfloat162*)(dh + i) = __halves2bfloat162(h0, h1);
        *(__nv_bfloat162*)(dl + i) = __halves2bfloat162(l0, l1);
      }
    }
    __syncthreads();
  }
}

// col_profiles_kernel with the n x W strip of l staged in shared memory by
// TMA (boxes of 256 rows x W columns, one mbarrier), so l crosses HBM once.
// Thread t owns column t % W and the rows congruent to t / W modulo 512 / W
// (the row phases are combined in order): pass 1 takes the column maxima,
// pass 2 overwrites the strip with e^{l - M_j} while summing s1 and s2, pass
// 3 scales by invN_j and writes the transposed split profiles.
template <int W>
__global__ void __launch_bounds__(512) col_profiles_tma_kernel(const __grid_constant__ CUtensorMap mL, float* logphi,
                                                               ProfileOut po, int n, int T, int ldn, int nbox,
                                                               DevStatus* stt) {
  constexpr int PH = 512 / W;   // row phases
  extern __shared__ uint8_t smem_raw[];
  const uint32_t r0 = tc::smem_u32(smem_raw);
  float* strip = (float*)(smem_raw + (((r0 + 127u) & ~127u) - r0));   // [nbox * 256][W], 128-byte aligned
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  __shared__ float red[3][PH][W];
  __shared__ float cstat[2][W];
  __shared__ float tile[64][W + 1];
  __shared__ long long orow[W];   // element offset of each column's output row (anchor rows: -1 - offset)
  const int b = blockIdx.y, j0 = blockIdx.x * W, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int c = tid % W, ph = tid / W, j = j0 + c;
  if (tid == 0) {
    tc::mbar_init(&bar, 1);
    abort_flag = 0;
    tc::mbar_fence_init();
  }
  __syncthreads();
  if (tid == 0) {
    tc::mbar_arrive_expect_tx(&bar, (uint32_t)(nbox * 256 * W * 4));
    for (int q = 0; q < nbox; ++q) tc::tma_load_3d(strip + q * 256 * W, &mL, j0, q * 256, b, &bar);
  }
  // the output rows of the CTA's keys (a binary search over the anchors)
  // while the strip is in flight
  if (po.Ut_hi != nullptr && tid >= 32 && tid < 32 + W && j0 + tid - 32 < T)
    orow[tid - 32] = profile_row(po.anchors + (long long)b * po.t, po.t, T, b, j0 + tid - 32, ldn, po.kmap);
  const bool ok = tc::mbar_wait(&bar, 0, &abort_flag, stt);
  if (!__syncthreads_and(ok)) {   // timed out: let the copies land (bounded) before leaving
    volatile int never = 0;
    if (tid == 0) tc::mbar_wait(&bar, 0, &never, stt);
    __syncthreads();
    return;
  }
  // pass 1: column maxima (four independent chains per thread)
  float m0 = -INFINITY, m1 = -INFINITY, m2 = -INFINITY, m3 = -INFINITY;
  if (j < T) {
    int i = ph;
    for (; i + 3 * PH < n; i += 4 * PH) {
      m0 = fmaxf(m0, strip[i * W + c]);
      m1 = fmaxf(m1, strip[(i + PH) * W + c]);
      m2 = fmaxf(m2, strip[(i + 2 * PH) * W + c]);
      m3 = fmaxf(m3, strip[(i + 3 * PH) * W + c]);
    }
    for (; i < n; i += PH) m0 = fmaxf(m0, strip[i * W + c]);
  }
  red[0][ph][c] = fmaxf(fmaxf(m0, m1), fmaxf(m2, m3));
  __syncthreads();
  if (tid < W) {
    float M = -INFINITY;
#pragma unroll 8
    for (int q = 0; q < PH; ++q) M = fmaxf(M, red[0][q][tid]);
    cstat[0][tid] = M;
  }
  __syncthreads();
  // pass 2: e_ij = e^{l_ij - M_j} replaces l in the strip; s1 = sum e, s2 = sum e^2
  {
    const float M = cstat[0][c];
    float a1 = 0.f, b1 = 0.f, a2 = 0.f, b2 = 0.f;
    if (j < T && M != -INFINITY) {
      int i = ph;
      for (; i + PH < n; i += 2 * PH) {
        const float e0 = ex2_approx((strip[i * W + c] - M) * kLog2e);
        const float e1 = ex2_approx((strip[(i + PH) * W + c] - M) * kLog2e);
        strip[i * W + c] = e0;
        strip[(i + PH) * W + c] = e1;
        a1 += e0;
        b1 += e1;
        a2 = fmaf(e0, e0, a2);
        b2 = fmaf(e1, e1, b2);
      }
      if (i < n) {
        const float e0 = ex2_approx((strip[i * W + c] - M) * kLog2e);
        strip[i * W + c] = e0;
        a1 += e0;
        a2 = fmaf(e0, e0, a2);
      }
    }
    red[1][ph][c] = a1 + b1;
    red[2][ph][c] = a2 + b2;
  }
  __syncthreads();
  if (tid < W) {
    float S1 = 0.f, S2 = 0.f;
#pragma unroll 8
    for (int q = 0; q < PH; ++q) {
      S1 += red[1][q][tid];
      S2 += red[2][q][tid];
    }
    if (j < T) logphi[(long long)b * T + j] = cstat[0][tid] + logf(S1) - logf((float)n);
    cstat[1][tid] = j < T ? 1.0f / sqrtf(S2) : 0.f;
  }
  __syncthreads();
  if (po.Ut_hi == nullptr) return;
  // pass 3: U_ij = e_ij invN_j, transposed through a padded tile 64 rows at a time
  constexpr int RPT = (64 + PH - 1) / PH;   // tile rows per thread: rows ph + k PH below 64
  const float inv = cstat[1][c];
  for (int i0 = 0; i0 < ldn; i0 += 64) {
#pragma unroll
    for (int k = 0; k < RPT; ++k) {
      const int r = ph + k * PH, i = i0 + r;
      if (r < 64) tile[r][c] = (i < n) ? strip[i * W + c] * inv : 0.f;
    }
    __syncthreads();
    // warp w writes columns w, w + 16, ...: lane l rows i0 + 2l and i0 + 2l + 1 (ldn even)
    for (int cc = warp; cc < W; cc += 16) {
      const int jj = j0 + cc, i = i0 + 2 * lane;
      if (jj < T && i < ldn && orow[cc] != kNoRow) {
        const float x0 = tile[2 * lane][cc], x1 = tile[2 * lane + 1][cc];
        const __nv_bfloat162 h = __floats2bfloat162_rn(x0, x1);
        const float2 hf = __bfloat1622float2(h);
        const long long ro = orow[cc];
        bf16* dh = ro >= 0 ? po.Ut_hi + ro : po.S_hi + (-1 - ro);
        bf16* dl = ro >= 0 ? po.Ut_lo + ro : po.S_lo + (-1 - ro);
        *(__nv_bfloat162*)(dh + i) = h;
        *(__nv_bfloat162*)(dl + i) = __floats2bfloat162_rn(x0 - hf.x, x1 - hf.y);
      }
    }
    __syncthreads();
  }
}

template <int W>
static int launch_col_profiles_tma(const Dims& D, const float* L, float* logphi, const ProfileOut& po, int ldn,
                                   int nbox, DevStatus* stt, cudaStream_t st) {
  CUtensorMap m;
  if (!encode_f32_map_3d(&m, L, D.T, D.n, D.H, W, 256)) return -1;
  const int smem = nbox * 256 * W * 4 + 128;
  if (set_dyn_smem((const void*)col_profiles_tma_kernel<W>, smem) !=
      cudaSuccess)
    return -1;
  col_profiles_tma_kernel<W><<<dim3(cdiv(D.T, W), D.H), 512, smem, st>>>(m, logphi, po, D.n, D.T, ldn, nbox, stt);
  return 1;
}

static int col_profiles(const Dims& D, const float* L, float* logphi, const ProfileOut& po, DevStatus* stt,
                        cudaStream_t st) {
  const int ldn = (D.n + 7) / 8 * 8;
  // staged strips of at most 64 KB (three CTAs per SM) when l is TMA-tileable
  const int nbox = cdiv(D.n, 256);
  if ((D.T & 3) == 0 && ((uintptr_t)L & 15u) == 0 && nbox <= 16) {
    if (nbox <= 4) return launch_col_profiles_tma<16>(D, L, logphi, po, ldn, nbox, stt, st);
    if (nbox <= 8) return launch_col_profiles_tma<8>(D, L, logphi, po, ldn, nbox, stt, st);
    return launch_col_profiles_tma<4>(D, L, logphi, po, ldn, nbox, stt, st);
  }
  // each CTA re-reads its n x 32 strip from L2: with n > 1024 a shared-memory
  // reservation keeps at most two CTAs per SM so the live strips fit in L2
  const int smem = D.n > 1024 ? 80 * 1024 : 0;
  if (smem > 0 && set_dyn_smem((const void*)col_profiles_kernel, smem) !=
                      cudaSuccess)
    return -1;
  col_profiles_kernel<<<dim3(cdiv(D.T, 32), D.H), 512, smem, st>>>(L, logphi, po, D.n, D.T, ldn);
  return 1;
}

int launch_col_profiles(const Dims& D, const float* L, float* logphi, DevStatus* stt, cudaStream_t st) {
  return col_profiles(D, L, logphi, ProfileOut{nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, D.t}, stt, st);
}

// kappa of the non-anchor keys from the argmax of their compacted rows
// (rows c < T - t of head b; kmap gives the key)
__global__ void decode_assign_kernel2(const unsigned long long* best, const int* kmap, int* kappa, int T, int Tm,
                                      long long count) {
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < count;
       k += (long long)gridDim.x * blockDim.x) {
    const long long b = k / Tm, o = b * T + (k - b * Tm);
    const unsigned long long v = best[o];
    const int j = kmap[o];
    if ((unsigned)j < (unsigned)T) kappa[b * T + j] = v ? (int)(0xffffffffu - (unsigned int)(v & 0xffffffffull)) : 0;
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

int launch_assign_prep(const Dims& D, const float* L, float* logphi, const int* anchors, bf16* Ut_hi, bf16* Ut_lo,
                       bf16* S_hi, bf16* S_lo, int* kmap, DevStatus* stt, cudaStream_t st) {
  return col_profiles(D, L, logphi, ProfileOut{Ut_hi, Ut_lo, S_hi, S_lo, kmap, anchors, D.t}, stt, st);
}

int launch_assign_gemm(const Dims& D, const int* anchors, const bf16* Ut_hi, const bf16* Ut_lo, const bf16* S_hi,
                       const bf16* S_lo, const int* kmap, unsigned long long* best, int* kappa, DevStatus* stt,
                       cudaStream_t st) {
  const int ldn = (D.n + 7) / 8 * 8;
  const int Tm = D.T - D.t;   // the non-anchor keys, compacted (none when t = T)
  int nl = 1;
  // every key gets an assignment in [0, t) even when invalid caller anchors
  // (flagged upstream) leave some compacted rows without a key
  cudaMemsetAsync(kappa, 0, sizeof(int) * (size_t)D.H * D.T, st);
  if (Tm > 0) {
    cudaMemsetAsync(best, 0, sizeof(unsigned long long) * (size_t)D.H * D.T, st);
    // 128 keys x 256 anchors per tile (M = 128, N = 256 MMAs): half the key-side
    // operand bytes per flop of a 128-wide tile.  The key map spans all T rows
    // of a head (its plane stride); the GEMM takes the first Tm.
    constexpr int BN = 256;
    CUtensorMap mA, mA2, mB, mB2;
    if (!encode_bf16_map_3d(&mA, Ut_hi, ldn, D.T, D.H, 128) || !encode_bf16_map_3d(&mA2, Ut_lo, ldn, D.T, D.H, 128) ||
        !encode_bf16_map_3d(&mB, S_hi, ldn, D.t, D.H, BN) || !encode_bf16_map_3d(&mB2, S_lo, ldn, D.t, D.H, BN))
      return -1;
    TcEpiArgmax8 epi;
    epi.best = best;
    epi.bbs = D.T;
    const int kfull = (ldn + 63) / 64 * 64;
    // anchor tiles in groups whose split profiles (BN rows x ldn x 4 bytes per
    // tile) take about 40 MB, so each group stays in L2 while the key profiles
    // stream past it (one pass over them per group instead of one per wave)
    const long long tile_bytes = (long long)BN * ldn * 4;
    const int group = (int)std::max<long long>(1, (40LL << 20) / tile_bytes);
    if (launch_tc_gemm<BN, kSplit>(mA, mB, mA2, mB2, epi, D.H, Tm, D.t, ldn, kfull, stt, st, 0, nullptr, group) !=
        cudaSuccess)
      return -1;
    const long long cnt = (long long)D.H * Tm;
    decode_assign_kernel2<<<stride_grid(cnt, 256, 8), 256, 0, st>>>(best, kmap, kappa, D.T, Tm, cnt);
    nl += 2;
  }
  anchor_self_assign_kernel2<<<cdiv((long long)D.H * D.t, 256), 256, 0, st>>>(anchors, kappa, D.T, D.t, D.H);
  return nl;
}

}  // namespace arckv
