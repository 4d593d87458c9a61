// Closed-form attention-mass and compact-value fits (App. A.9) and the
// compact attention operator (Sec. 3.1 Eq. compact_attention).
//
// beta:  Phi_C = exp(scale Q C_k^T - z), z_i = max_j scale q_i.k_j;
//        (Phi_C^T Phi_C + lam_w I) w = Phi_C^T (Phi_K 1);  w* = max(w, 0);
//        beta = clip(log max(w*, eps_w), b_min, b_max)          (Eq. mass_fit)
// C_v:   P^ = softmax(scale Q C_k^T + 1 beta^T);
//        (P^T P^ + lam_v I) C_v = P^T Y, Y = softmax(scale Q K^T) V   (Eq. value_lstsq)
// with lam = ridge * trace(Gram) / t.  Both systems are solved by a blocked
// right-looking Cholesky factorisation (64 x 64 blocks; each diagonal block
// is factored and inverted in shared memory) with the forward substitution
// fused into the trailing updates, then blocked back substitution, all in one
// cluster launch per system (chol_cluster_kernel).
#include <cooperative_groups.h>
#include <map>
#include <mutex>
#include <type_traits>

#include "kernels.h"
#include "tc_gemm.cuh"

namespace arckv {

constexpr int NB = kCholNB;

__global__ void phi_kernel(const float* LC, const float* z, float* Phi, int n, int t, long long count) {
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < count;
       k += (long long)gridDim.x * blockDim.x) {
    const long long row = k / t;  // = b * n + i
    Phi[k] = expf(LC[k] - z[row]);
  }
}

// rhs[b][r] = sum_i Phi[b][i][r] m[b][i]   (Phi_C^T Phi_K 1).  A CTA owns 32
// columns; warp w sums the rows i = w, w+8, ... (four partial sums) and the
// eight warp sums are added in warp order.
__global__ void __launch_bounds__(1024) mass_rhs_kernel(const float* Phi, const float* m, float* rhs, int n, int t) {
  // 32 columns per CTA, the rows split over 32 warps (four loads in flight each)
  const int b = blockIdx.y, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int r = blockIdx.x * 32 + lane;
  __shared__ float red[32][33];
  const float* P = Phi + (long long)b * n * t + r;
  const float* mb = m + (long long)b * n;
  float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
  if (r < t) {
    int i = warp;
    for (; i + 96 < n; i += 128) {
      a0 = fmaf(P[(long long)i * t], mb[i], a0);
      a1 = fmaf(P[(long long)(i + 32) * t], mb[i + 32], a1);
      a2 = fmaf(P[(long long)(i + 64) * t], mb[i + 64], a2);
      a3 = fmaf(P[(long long)(i + 96) * t], mb[i + 96], a3);
    }
    for (; i < n; i += 32) a0 = fmaf(P[(long long)i * t], mb[i], a0);
  }
  red[warp][lane] = (a0 + a1) + (a2 + a3);
  __syncthreads();
  if (warp == 0 && r < t) {
    float a = 0.f;
    for (int w = 0; w < 32; ++w) a += red[w][lane];
    rhs[(long long)b * t + r] = a;
  }
}

// ---------------------------------------------------------------------------
// Cluster Cholesky solver: (Gram + lam I) X = B for every head in ONE launch.
// One cluster of kCL CTAs (cluster_size) per head; the matrix, its factor and the right-hand
// sides live in global memory (L2-resident at these sizes) and are read with
// ld.global.cg so that no CTA sees a stale L1 line of another CTA's writes.
// Phases of each 64-wide block step k are separated by hardware cluster
// barriers (release / acquire at cluster scope):
//   trsm    L_ik = A_ik Linv_kk^T for block rows i > k (round robin);
//   update  A_ij -= L_ik L_jk^T (k < j <= i) and B_i -= L_ik (Linv_kk B_k);
//           the CTA that owns block k+1 updates the diagonal block first and
//           factors it at once, overlapping the serial factorisation with the
//           other CTAs' updates;
// then block back substitution X_k = Linv_kk^T (Linv_kk B_k + Z_k),
// Z_i -= L_ki^T X_k (i < k).  lam = ridge * trace(Gram) / tdiv is added to the
// diagonal as each diagonal block is factored (tdiv = t, or the primal size
// when the dual system is solved).
// fp32 systems run the trailing updates and (up to 128 right-hand sides) the
// back substitution as tcgen05 units of bf16-triple products; with one
// right-hand side rank 0 does the back substitution alone.  fp64 systems use
// SIMT tile products throughout.
// CTAs per cluster (one cluster per head): 4 up to 16 blocks (t <= 1024) --
// half the SMs of 8 at nearly the same latency, which leaves room for the
// concurrent layers -- and 8 for longer systems, whose tile work dominates.
constexpr int cluster_size(int t) { return (t + NB - 1) / NB > 16 ? 8 : 4; }
constexpr int kCT = 512;
// Shared tiles are [NB][NBP] with rows padded to a 16-byte multiple, so that
// mm64 can read them with vector loads.
template <typename R>
constexpr int NBP = NB + 16 / (int)sizeof(R);
template <typename R>
using Tile = R (*)[NBP<R>];
template <typename R>
constexpr int kTileF = NB * NBP<R>;

__device__ __forceinline__ float fma_r(float a, float b, float c) { return fmaf(a, b, c); }
__device__ __forceinline__ double fma_r(double a, double b, double c) { return fma(a, b, c); }
__device__ __forceinline__ float rcp_r(float x) { return __frcp_rn(x); }
__device__ __forceinline__ double rcp_r(double x) { return __drcp_rn(x); }

// Double-float arithmetic: a value hi + lo of two fp32 numbers (|lo| <= ulp(hi) / 2),
// ~48 significant bits.  The GB300's fp64 pipe issues at a small fraction of its
// fp32 rate, so the fp64 64 x 64 diagonal blocks of the dual Cholesky are
// factored in this arithmetic (each operation a short chain of fp32 operations:
// the error-free sum and product transformations of Dekker and Knuth, and one
// Newton step for the reciprocal and the square root), with the block read
// from and written back to fp64 storage.
struct df64 {
  float hi, lo;
  df64() = default;
  __device__ __forceinline__ df64(float h, float l) : hi(h), lo(l) {}
  __device__ __forceinline__ explicit df64(int v) : hi((float)v), lo(0.f) {}
};
__device__ __forceinline__ df64 df_fast2(float a, float b) {   // |a| >= |b| (or a = 0)
  const float s = a + b;
  return df64(s, b - (s - a));
}
__device__ __forceinline__ df64 df_two(float a, float b) {
  const float s = a + b, bb = s - a;
  return df64(s, (a - (s - bb)) + (b - bb));
}
__device__ __forceinline__ df64 operator+(df64 x, df64 y) {
  df64 s = df_two(x.hi, y.hi);
  const df64 t = df_two(x.lo, y.lo);
  s.lo += t.hi;
  s = df_fast2(s.hi, s.lo);
  s.lo += t.lo;
  return df_fast2(s.hi, s.lo);
}
__device__ __forceinline__ df64 operator-(df64 x) { return df64(-x.hi, -x.lo); }
__device__ __forceinline__ df64 operator-(df64 x, df64 y) { return x + (-y); }
__device__ __forceinline__ df64 operator*(df64 x, df64 y) {
  const float p = x.hi * y.hi;
  float e = fmaf(x.hi, y.hi, -p);
  e = fmaf(x.hi, y.lo, e);
  e = fmaf(x.lo, y.hi, e);
  return df_fast2(p, e);
}
__device__ __forceinline__ df64& operator*=(df64& x, df64 y) { return x = x * y; }
__device__ __forceinline__ bool operator>(df64 x, df64 y) { return x.hi > y.hi || (x.hi == y.hi && x.lo > y.lo); }
__device__ __forceinline__ bool finite_r(float x) { return isfinite(x); }
__device__ __forceinline__ bool finite_r(double x) { return isfinite(x); }
__device__ __forceinline__ bool finite_r(df64 x) { return isfinite(x.hi); }
__device__ __forceinline__ df64 fma_r(df64 a, df64 b, df64 c) { return a * b + c; }
__device__ __forceinline__ df64 rcp_r(df64 x) {   // r + r (1 - x r)
  const df64 r(__frcp_rn(x.hi), 0.f);
  return r + r * (df64(1) - x * r);
}
__device__ __forceinline__ float sqrt_r(float x) { return sqrtf(x); }
__device__ __forceinline__ double sqrt_r(double x) { return ::sqrt(x); }
__device__ __forceinline__ df64 sqrt_r(df64 x) {    // s + (x - s^2) / (2 s)
  if (!(x.hi > 0.f)) return df64(sqrtf(x.hi), 0.f);
  const float s = sqrtf(x.hi);
  const df64 r = x - df64(s, 0.f) * df64(s, 0.f);
  return df_fast2(s, r.hi * (0.5f / s));
}
// storage conversions (the block lives in fp64 in global memory)
template <typename R, typename G>
__device__ __forceinline__ R to_reg(G v) { return v; }
template <>
__device__ __forceinline__ df64 to_reg<df64, double>(double v) {
  const float h = __double2float_rn(v);
  return df64(h, __double2float_rn(v - (double)h));
}
template <typename G, typename R>
__device__ __forceinline__ G to_mem(R v) { return v; }
template <>
__device__ __forceinline__ double to_mem<double, df64>(df64 v) { return (double)v.hi + (double)v.lo; }
template <typename R>
__device__ __forceinline__ R warp_sum_r(R v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ unsigned cluster_rank() {
  unsigned r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// S[r][c] = G[(r0 + r) * ld + c0 + c] (or S[c][r] with `trans`), zero outside
// rows < rmax, cols < cmax of the source block.  Split into a fetch (eight
// loads per thread into registers) and a put (the shared stores), so that a
// caller loading two tiles issues all sixteen loads before its first store and
// pays the L2 latency once.  The transposed form maps a warp to 4 rows x 8
// columns, so its shared stores hit 32 distinct banks.
template <typename R>
struct TileRegs {
  static constexpr int NE = NB * NB / kCT;
  R v[NE];
  bool trans;
};
// element q of this thread: (row, col) of the source block
__device__ __forceinline__ void tile_pos(int q, bool trans, int& r, int& c) {
  const int e = threadIdx.x + q * kCT;
  if (!trans) {
    r = e / NB;
    c = e % NB;
  } else {
    const int lane = e & 31, w = e >> 5;
    c = (w & 7) * 8 + (lane & 7);
    r = (w >> 3) * 4 + (lane >> 3);
  }
}
template <typename R>
__device__ __forceinline__ void tile_fetch(TileRegs<R>& f, const R* G, long long ld, int r0, int c0, int rmax,
                                           int cmax, bool trans) {
  f.trans = trans;
#pragma unroll
  for (int q = 0; q < TileRegs<R>::NE; ++q) {
    int r, c;
    tile_pos(q, trans, r, c);
    f.v[q] = (r < rmax && c < cmax) ? __ldcg(G + (long long)(r0 + r) * ld + c0 + c) : R(0);
  }
}
template <typename R>
__device__ __forceinline__ void tile_put(Tile<R> S, const TileRegs<R>& f) {
#pragma unroll
  for (int q = 0; q < TileRegs<R>::NE; ++q) {
    int r, c;
    tile_pos(q, f.trans, r, c);
    if (f.trans) S[c][r] = f.v[q];
    else S[r][c] = f.v[q];
  }
}
template <typename R>
__device__ __forceinline__ void ld_tile(Tile<R> S, const R* G, long long ld, int r0, int c0, int rmax, int cmax,
                                        bool trans) {
  TileRegs<R> f;
  tile_fetch(f, G, ld, r0, c0, rmax, cmax, trans);
  tile_put(S, f);
}
// two tiles, one L2 round trip
template <typename R>
__device__ __forceinline__ void ld_tiles(Tile<R> S1, const R* G1, long long ld1, int r1, int c1, int rm1, int cm1,
                                         bool tr1, Tile<R> S2, const R* G2, long long ld2, int r2, int c2, int rm2,
                                         int cm2, bool tr2) {
  TileRegs<R> f1, f2;
  tile_fetch(f1, G1, ld1, r1, c1, rm1, cm1, tr1);
  tile_fetch(f2, G2, ld2, r2, c2, rm2, cm2, tr2);
  tile_put(S1, f1);
  tile_put(S2, f2);
}

// Thread tile of the 64 x 64 products: kTP rows x kTQ columns at (tile_ry, tile_cx).
// A warp covers 16 rows x 16 columns, so each k step of mm64 costs it one
// 16-byte load of the transposed left operand (4 rows) and one 8-byte load of
// the right one (2 columns): two shared wavefronts for 8 FMAs per thread.
constexpr int kTP = 4, kTQ = 2;
__device__ __forceinline__ int tile_ry() { return (threadIdx.x >> 7) * 16 + ((threadIdx.x >> 3) & 3) * 4; }
__device__ __forceinline__ int tile_cx() { return ((threadIdx.x >> 5) & 3) * 16 + (threadIdx.x & 7) * 2; }

// P[p*ld + q] -= acc[p][q] for p < pn, q < qn (all loads issued before the stores)
template <typename R>
__device__ __forceinline__ void rmw_sub(R* P, long long ld, int pn, int qn, const R (&acc)[kTP][kTQ]) {
  R old[kTP][kTQ];
#pragma unroll
  for (int p = 0; p < kTP; ++p)
#pragma unroll
    for (int q = 0; q < kTQ; ++q) old[p][q] = (p < pn && q < qn) ? __ldcg(P + p * ld + q) : R(0);
#pragma unroll
  for (int p = 0; p < kTP; ++p)
#pragma unroll
    for (int q = 0; q < kTQ; ++q)
      if (p < pn && q < qn) P[p * ld + q] = old[p][q] - acc[p][q];
}

__device__ __forceinline__ void lds2(float (&a)[2], const float* p) {
  const float2 v = *(const float2*)p;
  a[0] = v.x; a[1] = v.y;
}
__device__ __forceinline__ void lds4(float (&a)[4], const float* p) {
  const float4 v = *(const float4*)p;
  a[0] = v.x; a[1] = v.y; a[2] = v.z; a[3] = v.w;
}
__device__ __forceinline__ void lds2(double (&a)[2], const double* p) {
  const double2 v = *(const double2*)p;
  a[0] = v.x; a[1] = v.y;
}
__device__ __forceinline__ void lds4(double (&a)[4], const double* p) {
  const double2 v = *(const double2*)p, u = *(const double2*)(p + 2);
  a[0] = v.x; a[1] = v.y; a[2] = u.x; a[3] = u.y;
}

// acc[p][q] = sum_l XT[l][ry+p] Y[l][cx+q] (ry = tile_ry(), cx = tile_cx()): the left
// operand is held transposed so that each l takes one 4-wide and one 2-wide
// shared load.
template <typename R>
__device__ __forceinline__ void mm64(Tile<R> XT, Tile<R> Y, R (&acc)[kTP][kTQ]) {
  const int ry = tile_ry(), cx = tile_cx();
#pragma unroll
  for (int p = 0; p < kTP; ++p)
#pragma unroll
    for (int q = 0; q < kTQ; ++q) acc[p][q] = R(0);
#pragma unroll 8
  for (int l = 0; l < NB; ++l) {
    R a[4], c[2];
    lds4(a, &XT[l][ry]);
    lds2(c, &Y[l][cx]);
#pragma unroll
    for (int p = 0; p < kTP; ++p)
#pragma unroll
      for (int q = 0; q < kTQ; ++q) acc[p][q] = fma_r(a[p], c[q], acc[p][q]);
  }
}

// Load the lower part of A_kk + lam I into the tile L (identity beyond the
// matrix when kb < NB; zero above the diagonal).
template <typename R, typename G>
__device__ __forceinline__ void load_diag(Tile<R> L, const G* Ab, int t, int k0, int kb, G lam) {
  constexpr int NE = NB * NB / kCT;
  R v[NE];
#pragma unroll
  for (int q = 0; q < NE; ++q) {
    const int e = threadIdx.x + q * kCT, r = e / NB, c = e % NB;
    v[q] = (r < kb && c <= r) ? to_reg<R>(__ldcg(Ab + (long long)(k0 + r) * t + k0 + c) + (r == c ? lam : G(0)))
                              : (r == c ? R(1) : R(0));
  }
#pragma unroll
  for (int q = 0; q < NE; ++q) {
    const int e = threadIdx.x + q * kCT;
    L[e / NB][e % NB] = v[q];
  }
}

// Write L_kk (lower part, rows < kb) into A and the full tile Li into Linv[k].
template <typename R, typename G>
__device__ __forceinline__ void store_diag(Tile<R> L, Tile<R> Li, G* Ab, G* Lb, int t, int k, int kb) {
  G* Lo = Lb + (long long)k * NB * NB;
  const int k0 = k * NB;
  for (int e = threadIdx.x; e < NB * NB; e += kCT) {
    const int rr = e / NB, cc = e % NB;
    Lo[e] = cc <= rr ? to_mem<G>(Li[rr][cc]) : G(0);   // the inverse is lower triangular
    if (rr < kb && cc <= rr) Ab[(long long)(k0 + rr) * t + k0 + cc] = to_mem<G>(L[rr][cc]);
  }
}

// Factor diagonal block k (lower part of A_kk + lam I) in shared memory and
// invert the factor: L_kk goes into A and L_kk^-1 into Linv[k].  Blocked in
// four 16-wide panels, every phase on all warps:
//   panel p: factor its 16 x 16 diagonal block (unscaled right-looking, one
//            element per thread, one barrier per column; then the column
//            scaling by sqrt(a_cc)) and invert it (forward substitution by
//            columns, one barrier per row); L_panel = A_panel X_pp^T below it;
//            trailing update A -= L_panel L_panel^T;
//   inverse: off-diagonal 16 x 16 blocks X_ij = -X_ii sum_{m=j}^{i-1} L_im X_mj,
//            level by level (i - j = 1, 2, 3).
// Tiles: L (the block; pad column NB holds 1 / l_cc), Li (the inverse), T
// (scratch).  Pad rows beyond the matrix (kb < NB) are the identity.
template <typename R, typename G = R>
__device__ void factor_diag(G* Ab, G* Lb, int t, int k, G lam, Tile<R> L, Tile<R> Li, Tile<R> T, int* bad) {
  static_assert(kCT == 512 && NB == 64, "thread map of the 16-wide panels");
  const int tid = threadIdx.x, k0 = k * NB, kb = min(NB, t - k0);
  load_diag(L, Ab, t, k0, kb, lam);
  for (int e = tid; e < NB * NB; e += kCT) Li[e / NB][e % NB] = R(0);
  __syncthreads();
  const bool blk = tid < 256;
  const int er = (tid >> 4) & 15, ec = tid & 15;   // element of a 16 x 16 block (threads < 256)
  for (int p = 0; p < 4; ++p) {
    const int c0 = 16 * p;
    for (int j = 0; j < 15; ++j) {   // factor the diagonal block
      if (blk && ec > j && er >= ec) {
        R piv = L[c0 + j][c0 + j];
        if (!(piv > R(0)) || !finite_r(piv)) piv = R(1);
        L[c0 + er][c0 + ec] = fma_r(-L[c0 + er][c0 + j] * rcp_r(piv), L[c0 + ec][c0 + j], L[c0 + er][c0 + ec]);
      }
      __syncthreads();
    }
    R v = R(0);
    if (blk && er >= ec) {   // column scaling
      R pc = L[c0 + ec][c0 + ec];
      if (!(pc > R(0)) || !finite_r(pc)) {
        if (er == ec && c0 + ec < kb) *bad = 1;
        pc = R(1);
      }
      const R d = sqrt_r(pc);
      v = (er == ec) ? d : L[c0 + er][c0 + ec] * rcp_r(d);
    }
    __syncthreads();
    if (blk && er >= ec) {
      L[c0 + er][c0 + ec] = v;
      if (er == ec) {
        L[c0 + er][NB] = rcp_r(v);
        Li[c0 + er][c0 + er] = R(1);
      }
    }
    __syncthreads();
    for (int i = 0; i < 15; ++i) {   // Y = I; y_lj -= l_li y_ij / l_ii for l > i, j <= i
      if (blk && er > i && ec <= i)
        Li[c0 + er][c0 + ec] = fma_r(-L[c0 + er][c0 + i] * L[c0 + i][NB], Li[c0 + i][c0 + ec], Li[c0 + er][c0 + ec]);
      __syncthreads();
    }
    if (blk && ec <= er) Li[c0 + er][c0 + ec] *= L[c0 + er][NB];   // X_pp = diag(1 / l_rr) Y
    __syncthreads();
    if (p == 3) break;
    {  // panel below: L[r][c0 + c] = sum_m A[r][c0 + m] X_pp[c][m] (all reads before the writes)
      const int rows = NB - c0 - 16;
      R o[2];
      int pr[2], pcol[2];
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const int e = tid + q * kCT;
        pr[q] = -1;
        if (e < rows * 16) {
          const int r = c0 + 16 + e / 16, c = e % 16;
          R a = R(0);
          for (int m = 0; m <= c; ++m) a = fma_r(L[r][c0 + m], Li[c0 + c][c0 + m], a);
          o[q] = a;
          pr[q] = r;
          pcol[q] = c;
        }
      }
      __syncthreads();
#pragma unroll
      for (int q = 0; q < 2; ++q)
        if (pr[q] >= 0) L[pr[q]][c0 + pcol[q]] = o[q];
      __syncthreads();
    }
    {  // trailing update: L[r][c] -= sum_m L[r][c0 + m] L[c][c0 + m], c0 + 16 <= c <= r
      const int c1 = c0 + 16, wdt = NB - c1, ntri = wdt * (wdt + 1) / 2;
      for (int e = tid; e < ntri; e += kCT) {
        int r = (int)((sqrtf(8.f * e + 1.f) - 1.f) * 0.5f);
        while (r * (r + 1) / 2 > e) --r;
        while ((r + 1) * (r + 2) / 2 <= e) ++r;
        const int c = e - r * (r + 1) / 2;
        R a = L[c1 + r][c1 + c];
#pragma unroll
        for (int m = 0; m < 16; ++m) a = fma_r(-L[c1 + r][c0 + m], L[c1 + c][c0 + m], a);
        L[c1 + r][c1 + c] = a;
      }
      __syncthreads();
    }
  }
  for (int lv = 1; lv < 4; ++lv) {   // off-diagonal blocks of the inverse, level i - j = lv
    const int nbk = 4 - lv;
    for (int e = tid; e < nbk * 256; e += kCT) {
      const int j = e >> 8, i = j + lv, r = (e >> 4) & 15, c = e & 15;
      R a = R(0);
      for (int m = j; m < i; ++m)
#pragma unroll
        for (int q = 0; q < 16; ++q) a = fma_r(L[16 * i + r][16 * m + q], Li[16 * m + q][16 * j + c], a);
      T[16 * i + r][16 * j + c] = a;
    }
    __syncthreads();
    for (int e = tid; e < nbk * 256; e += kCT) {
      const int j = e >> 8, i = j + lv, r = (e >> 4) & 15, c = e & 15;
      R a = R(0);
      for (int q = 0; q <= r; ++q) a = fma_r(Li[16 * i + r][16 * i + q], T[16 * i + q][16 * j + c], a);
      Li[16 * i + r][16 * j + c] = -a;
    }
    __syncthreads();
  }
  store_diag(L, Li, Ab, Lb, t, k, kb);
  __syncthreads();
}

// S[r][c] = G1[(r0 + r) * ld + c0 + c] + G2[...] (zero outside rows < rmax, cols < cmax)
template <typename R>
__device__ __forceinline__ void ld_tile_sum(Tile<R> S, const R* G1, const R* G2, long long ld, int r0, int c0,
                                            int rmax, int cmax) {
  constexpr int NE = NB * NB / kCT;
  R v[NE], u[NE];
#pragma unroll
  for (int q = 0; q < NE; ++q) {
    const int e = threadIdx.x + q * kCT, r = e / NB, c = e % NB;
    const bool ok = r < rmax && c < cmax;
    const long long o = (long long)(r0 + r) * ld + c0 + c;
    v[q] = ok ? __ldcg(G1 + o) : R(0);
    u[q] = ok ? __ldcg(G2 + o) : R(0);
  }
#pragma unroll
  for (int q = 0; q < NE; ++q) {
    const int e = threadIdx.x + q * kCT;
    S[e / NB][e % NB] = v[q] + u[q];
  }
}

// P[p*ld + q] = acc[p][q] for p < pn, q < qn
template <typename R>
__device__ __forceinline__ void st_acc(R* P, long long ld, int pn, int qn, const R (&acc)[kTP][kTQ]) {
#pragma unroll
  for (int p = 0; p < kTP; ++p)
#pragma unroll
    for (int q = 0; q < kTQ; ++q)
      if (p < pn && q < qn) P[p * ld + q] = acc[p][q];
}

// Eight fp32 values of operand row r, K elements 8 ch .. 8 ch + 7, as bf16
// triples at their 128-byte-swizzled K-major positions (row r at r * 128
// bytes, 16-byte chunk ch at ch ^ (r % 8)) of the three part tiles.
__device__ __forceinline__ void put_split3_chunk(uint8_t* h, uint8_t* m, uint8_t* l, int r, int ch,
                                                 const float (&x)[8]) {
  __align__(16) bf16 hh[8], mm[8], ll[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) split3_bf16(x[e], hh[e], mm[e], ll[e]);
  const int off = r * 128 + ((ch ^ (r & 7)) << 4);
  *(uint4*)(h + off) = *(const uint4*)hh;
  *(uint4*)(m + off) = *(const uint4*)mm;
  *(uint4*)(l + off) = *(const uint4*)ll;
}

// Shared memory of the fp32 solver beyond its four tiles: the bf16 triples of
// the tensor-core update operands (A: 128 x 64, B: 64 x 64), 1024-byte aligned.
constexpr int kTcStageA = 128 * 128, kTcStageB = 64 * 128;
constexpr int kTcStageBytes = 3 * (kTcStageA + kTcStageB) + 1024;

template <typename R, int kCL>
__global__ void __cluster_dims__(kCL, 1, 1) __launch_bounds__(kCT, 1)
    chol_cluster_kernel(R* A, R* Linv, R* B, R* Z, R* X, int t, int nrhs, int ldb, long long bbs, R ridge, R tdiv,
                        DevStatus* stt) {
  namespace cg = cooperative_groups;
  extern __shared__ __align__(16) unsigned char smraw[];
  R* sm = (R*)smraw;
  Tile<R> S1 = (Tile<R>)sm;
  Tile<R> S2 = (Tile<R>)(sm + kTileF<R>);
  Tile<R> S3 = (Tile<R>)(sm + 2 * kTileF<R>);
  Tile<R> S4 = (Tile<R>)(sm + 3 * kTileF<R>);
  __shared__ R red[kCT / 32];
  __shared__ int bad, grab;
  __shared__ int ctr[2];   // rank 0's pair deals the tiles of alternate dynamic phases
  constexpr bool kTc = std::is_same<R, float>::value;   // tensor-core trailing updates (fp32 systems)
  __shared__ uint64_t mma_bar;
  __shared__ uint32_t tmem_slot;
  __shared__ int tc_abort;
  const int head = blockIdx.x / kCL;
  const int rank = (int)cluster_rank();
  const int tid = threadIdx.x;
  const int nblk = (t + NB - 1) / NB, nct = (nrhs + NB - 1) / NB;
  R* Ab = A + (long long)head * t * t;
  R* Lb = Linv + (long long)head * nblk * NB * NB;
  R* Bb = B + (long long)head * bbs;
  R* Zb = Z + (long long)head * bbs;
  R* Xb = X + (long long)head * bbs;
  const int ry = tile_ry(), cx = tile_cx();
  R acc[kTP][kTQ];
  int* ctr0 = cg::this_cluster().map_shared_rank(ctr, 0);
  // tensor-core update state: operand triples, a 64-column TMEM accumulator, its mbarrier
  uint8_t* stg = nullptr;
  uint32_t tmem = 0, mma_ph = 0;
  if constexpr (kTc) {
    const uint32_t s0 = tc::smem_u32(smraw), e0 = s0 + 4u * kTileF<R> * (uint32_t)sizeof(R);
    stg = smraw + (((e0 + 1023u) & ~1023u) - s0);
    if (tid == 0) {
      tc::mbar_init(&mma_bar, 1);
      tc_abort = 0;
      tc::mbar_fence_init();
    }
    if (tid < 32) tc::tmem_alloc(&tmem_slot, 64);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    tmem = tmem_slot;
  }
  auto tc_release = [&]() {   // every exit of a CTA that allocated TMEM
    if constexpr (kTc) {
      tc::fence_before_sync();
      __syncthreads();
      if (tid < 32) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, 64);
      }
    }
  };
  int ep = 0;   // dynamic phase number; phase ep draws from ctr0[ep & 1]
  // next tile of the current dynamic phase (block-uniform)
  auto next_tile = [&]() -> int {
    __syncthreads();
    if (tid == 0) grab = atomicAdd(ctr0 + (ep & 1), 1);
    __syncthreads();
    return grab;
  };
  // the same with the grab issued one draw ahead: next_tile_ahead() returns the
  // index grabbed by the previous call and already issues the following grab,
  // whose round trip to rank 0 then overlaps the caller's unit (thread 0 keeps
  // it in a register); start_ahead() issues the first grab of a phase
  int ahead = 0;
  auto start_ahead = [&]() {
    if (tid == 0) ahead = atomicAdd(ctr0 + (ep & 1), 1);
  };
  auto next_tile_ahead = [&]() -> int {
    __syncthreads();
    if (tid == 0) {
      grab = ahead;
      ahead = atomicAdd(ctr0 + (ep & 1), 1);
    }
    __syncthreads();
    return grab;
  };

  // lam = ridge * trace / t (every CTA forms it; the trace precedes all writes)
  R tr = R(0);
  for (int r = tid; r < t; r += kCT) tr += __ldcg(Ab + (long long)r * t + r);
  tr = warp_sum_r(tr);
  if ((tid & 31) == 0) red[tid >> 5] = tr;
  if (tid == 0) {
    bad = 0;
    ctr[0] = 0;
    ctr[1] = 0;
  }
  __syncthreads();
  if (tid < 32) {
    R v = tid < kCT / 32 ? red[tid] : R(0);
    v = warp_sum_r(v);
    if (tid == 0) red[0] = v;
  }
  __syncthreads();
  const R trace = red[0];
  const R lam = ridge * trace / tdiv;
  if (rank == 0 && tid == 0 && !isfinite(trace)) set_status(stt, ARCKV_ERR_NONFINITE);
  // zero Z (rows split over the cluster) and factor the first diagonal block
  for (long long e = (long long)rank * kCT + tid; e < (long long)t * ldb; e += (long long)kCL * kCT) Zb[e] = R(0);
  cluster_sync_all();   // everyone has read the unmodified diagonal for the trace; counters are set

  // trailing-update tiles of step k: x < ntri is the syrk tile (ii >= jj) of
  // the m trailing blocks, A_ij -= L_ik L_jk^T; the rest are rhs tiles
  // B_i -= L_ik Y_k with Y_k = Linv_kk B_k formed in the trsm phase
  // where tile x of step k reads its operands and writes its result
  struct UpdDesc {
    const R* Ga;   // L_ik (rows i0.., cols k0..), loaded transposed
    const R* Gb;   // L_jk (transposed) or Y_k (as is)
    R* dst;        // A_ij or B_i at the thread's first row / column
    long long ldb_, ldd;
    int i0, rb, br0, bc0, brm, bcm, pn, qn;
    bool btrans;
  };
  auto describe = [&](int k, int x, int ntri, UpdDesc& u) {
    const int k0 = k * NB;
    u.Ga = Ab;
    if (x < ntri) {
      int ii = (int)((sqrtf(8.f * x + 1.f) - 1.f) * 0.5f);
      while (ii * (ii + 1) / 2 > x) --ii;
      while ((ii + 1) * (ii + 2) / 2 <= x) ++ii;
      const int jj = x - ii * (ii + 1) / 2;
      const int i0 = (k + 1 + ii) * NB, j0 = (k + 1 + jj) * NB;
      u.i0 = i0;
      u.rb = min(NB, t - i0);
      const int cb = min(NB, t - j0);
      u.Gb = Ab; u.ldb_ = t; u.br0 = j0; u.bc0 = k0; u.brm = cb; u.bcm = NB; u.btrans = true;
      u.dst = Ab + (long long)(i0 + ry) * t + j0 + cx; u.ldd = t; u.pn = u.rb - ry; u.qn = cb - cx;
    } else {
      const int y = x - ntri, i = k + 1 + y / nct, c0 = (y % nct) * NB;
      const int i0 = i * NB, nc = min(NB, nrhs - c0);
      u.i0 = i0;
      u.rb = min(NB, t - i0);
      u.Gb = Bb; u.ldb_ = ldb; u.br0 = k0; u.bc0 = c0; u.brm = NB; u.bcm = nc; u.btrans = false;   // block k is full
      u.dst = Bb + (long long)(i0 + ry) * ldb + c0 + cx; u.ldd = ldb; u.pn = u.rb - ry; u.qn = nc - cx;
    }
  };
  // trailing-update tiles x0 and (when x1 < ntot) x1 of step k: all operand
  // loads in one L2 round trip, both products, both read-modify-writes
  auto update_tiles = [&](int k, int x0, int x1, int ntot, int ntri) {
    const int k0 = k * NB;
    const bool two = x1 < ntot;
    UpdDesc u0, u1;
    describe(k, x0, ntri, u0);
    if (two) describe(k, x1, ntri, u1);
    {
      TileRegs<R> fa0, fb0, fa1, fb1;
      tile_fetch(fa0, u0.Ga, t, u0.i0, k0, u0.rb, NB, true);
      tile_fetch(fb0, u0.Gb, u0.ldb_, u0.br0, u0.bc0, u0.brm, u0.bcm, u0.btrans);
      if (two) {
        tile_fetch(fa1, u1.Ga, t, u1.i0, k0, u1.rb, NB, true);
        tile_fetch(fb1, u1.Gb, u1.ldb_, u1.br0, u1.bc0, u1.brm, u1.bcm, u1.btrans);
      }
      tile_put(S1, fa0);
      tile_put(S2, fb0);
      if (two) {
        tile_put(S3, fa1);
        tile_put(S4, fb1);
      }
    }
    __syncthreads();
    mm64(S1, S2, acc);
    if (two) {
      R acc1[kTP][kTQ];
      mm64(S3, S4, acc1);
      rmw_sub(u0.dst, u0.ldd, u0.pn, u0.qn, acc);
      rmw_sub(u1.dst, u1.ldd, u1.pn, u1.qn, acc1);
    } else {
      rmw_sub(u0.dst, u0.ldd, u0.pn, u0.qn, acc);
    }
    __syncthreads();
  };


  // Tensor-core trailing update (fp32 systems).  Row i of step k holds the
  // syrk tiles A_ij -= L_ik L_jk^T (j = k+1 .. i) and then the rhs tiles
  // B_i -= L_ik Y_k; all share L_ik, so a unit takes two tiles of one row:
  //   D [128 x 64] = [X_1; X_2] L_ik^T,  X = L_jk (syrk) or Y_k^T (rhs),
  // D's rows m < 64 being tile 1 transposed and the rest tile 2.  Operands
  // enter as bf16 triples (hh, hm, mh, hl, lh, mm per 16-wide K step:
  // fp32-grade products); one thread issues the 24 MMAs into TMEM and every
  // warp then subtracts a 32-row x 16-column slice of D from its tile.
  // D [128 x 64] = A B^T from the staged triples (24 MMAs by one thread), then
  // wait for it; false when the wait gave up
  auto tc_mma = [&]() -> bool {
    uint8_t *Ah = stg, *Am = stg + kTcStageA, *Al = stg + 2 * kTcStageA;
    uint8_t *Bh = stg + 3 * kTcStageA, *Bm = Bh + kTcStageB, *Bl = Bh + 2 * kTcStageB;
    tc::fence_proxy_async_smem();
    __syncthreads();
    if (tid == 0) {
      tc::fence_after_sync();
      constexpr uint32_t idesc = tc::idesc_bf16_f32(64);
#pragma unroll
      for (int ks = 0; ks < 4; ++ks) {
        const uint32_t o = ks * 32;
        const uint64_t ah = tc::sdesc_k128(tc::smem_u32(Ah) + o), am = tc::sdesc_k128(tc::smem_u32(Am) + o),
                       al = tc::sdesc_k128(tc::smem_u32(Al) + o);
        const uint64_t bh = tc::sdesc_k128(tc::smem_u32(Bh) + o), bm = tc::sdesc_k128(tc::smem_u32(Bm) + o),
                       bl = tc::sdesc_k128(tc::smem_u32(Bl) + o);
        tc::mma_f16(tmem, ah, bh, idesc, ks > 0 ? 1u : 0u);
        tc::mma_f16(tmem, ah, bm, idesc, 1u);
        tc::mma_f16(tmem, am, bh, idesc, 1u);
        tc::mma_f16(tmem, ah, bl, idesc, 1u);
        tc::mma_f16(tmem, al, bh, idesc, 1u);
        tc::mma_f16(tmem, am, bm, idesc, 1u);
      }
      tc::mma_commit(&mma_bar);
    }
    volatile int* abp = &tc_abort;
    const bool ok = tc::mbar_wait(&mma_bar, mma_ph, abp, stt);
    mma_ph ^= 1u;
    tc::fence_after_sync();
    return ok;
  };
  // operand rows r < rows of a triple from a column-major source: element
  // (r, l) = G[l * ld + r] (+ G2[...] when given) for r < rvalid, l < kvalid,
  // zero elsewhere; consecutive threads take consecutive r (coalesced)
  auto stage_cols = [&](uint8_t* h, uint8_t* mm, uint8_t* l, int rows, const R* G, const R* G2, long long ld,
                        int rvalid, int kvalid) {
    for (int task = tid; task < rows * 8; task += kCT) {
      const int r = task % rows, ch = task / rows;
      float xv[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int kk = 8 * ch + q;
        float v = 0.f;
        if (r < rvalid && kk < kvalid) {
          v = (float)__ldcg(G + (long long)kk * ld + r);
          if (G2) v += (float)__ldcg(G2 + (long long)kk * ld + r);
        }
        xv[q] = v;
      }
      put_split3_chunk(h, mm, l, r, ch, xv);
    }
  };
  // D's slice of this warp: rows (TMEM lanes) 32 (w % 4) + lane, columns 16 (w / 4) ..
  auto tc_slice = [&](float (&v)[16], int& mrow, int& ncol) {
    const int warp = tid >> 5, lane = tid & 31, q = warp & 3, g = warp >> 2;
    tc::tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(g * 16), v);
    mrow = q * 32 + lane;
    ncol = g * 16;
  };
  // back substitution on the tensor cores (nrhs <= 128): rows m of D are the
  // right-hand-side columns, its columns n the rows of the block
  //   Z_i -= L_ki^T X_k:     D = X_k^T L_ki,         Z_i[n][m] -= D[m][n]
  //   X_k = Linv^T (Y + Z):  D = (Y_k + Z_k)^T Linv,  X_k[n][m] = D[m][n]
  auto tc_z_unit = [&](int k, int i) {
    const int k0 = k * NB, kb = min(NB, t - k0), i0 = i * NB;
    uint8_t* Ah = stg;
    uint8_t* Bh = stg + 3 * kTcStageA;
    stage_cols(Ah, Ah + kTcStageA, Ah + 2 * kTcStageA, 128, Xb + (long long)k0 * ldb, nullptr, ldb, nrhs, kb);
    stage_cols(Bh, Bh + kTcStageB, Bh + 2 * kTcStageB, 64, Ab + (long long)k0 * t + i0, nullptr, t, 64, kb);
    const bool ok = tc_mma();
    float v[16];
    int mrow, ncol;
    tc_slice(v, mrow, ncol);
    if (ok && mrow < nrhs) {   // block i < k is full
      R* dst = Zb + (long long)(i0 + ncol) * ldb + mrow;
      R old[16];
#pragma unroll
      for (int c = 0; c < 16; ++c) old[c] = __ldcg(dst + (long long)c * ldb);
#pragma unroll
      for (int c = 0; c < 16; ++c) dst[(long long)c * ldb] = old[c] - (R)v[c];
    }
    tc::fence_before_sync();
    __syncthreads();
  };
  auto tc_x_unit = [&](int k) {
    const int k0 = k * NB, kb = min(NB, t - k0);
    uint8_t* Ah = stg;
    uint8_t* Bh = stg + 3 * kTcStageA;
    stage_cols(Ah, Ah + kTcStageA, Ah + 2 * kTcStageA, 128, Bb + (long long)k0 * ldb, Zb + (long long)k0 * ldb, ldb,
               nrhs, kb);
    stage_cols(Bh, Bh + kTcStageB, Bh + 2 * kTcStageB, 64, Lb + (long long)k * NB * NB, nullptr, NB, 64, NB);
    const bool ok = tc_mma();
    float v[16];
    int mrow, ncol;
    tc_slice(v, mrow, ncol);
    if (ok && mrow < nrhs) {
      R* dst = Xb + (long long)(k0 + ncol) * ldb + mrow;
#pragma unroll
      for (int c = 0; c < 16; ++c)
        if (ncol + c < kb) dst[(long long)c * ldb] = (R)v[c];
    }
    tc::fence_before_sync();
    __syncthreads();
  };
  auto tc_units = [&](int m) {   // units of step k with m trailing blocks
    int u = 0;
    for (int ii = 0; ii < m; ++ii) u += (ii + 2 + nct) / 2;
    return u;
  };
  auto tc_update_unit = [&](int k, int m, int x) {
    const int k0 = k * NB;
    int ii = 0, rem = x;
    for (; ii < m; ++ii) {
      const int u = (ii + 2 + nct) / 2;
      if (rem < u) break;
      rem -= u;
    }
    const int i0 = (k + 1 + ii) * NB, len = ii + 1 + nct, e0 = 2 * rem;
    uint8_t *Ah = stg, *Am = stg + kTcStageA, *Al = stg + 2 * kTcStageA;
    uint8_t *Bh = stg + 3 * kTcStageA, *Bm = Bh + kTcStageB, *Bl = Bh + 2 * kTcStageB;
    // B operand: L_ik, rows i0 + n (zero past t), K = block k (full)
    for (int task = tid; task < 64 * 8; task += kCT) {
      const int n = task >> 3, ch = task & 7;
      float xv[8];
#pragma unroll
      for (int e = 0; e < 8; ++e)
        xv[e] = (i0 + n < t) ? (float)__ldcg(Ab + (long long)(i0 + n) * t + k0 + 8 * ch + e) : 0.f;
      put_split3_chunk(Bh, Bm, Bl, n, ch, xv);
    }
    // A operand: rows 64 h + r from tile e0 + h
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int e = e0 + h;
      if (e < ii + 1) {   // syrk: L_jk rows j0 + r
        const int j0 = (k + 1 + e) * NB;
        for (int task = tid; task < 64 * 8; task += kCT) {
          const int r = task >> 3, ch = task & 7;
          float xv[8];
#pragma unroll
          for (int q = 0; q < 8; ++q)
            xv[q] = (j0 + r < t) ? (float)__ldcg(Ab + (long long)(j0 + r) * t + k0 + 8 * ch + q) : 0.f;
          put_split3_chunk(Ah, Am, Al, 64 * h + r, ch, xv);
        }
      } else if (e < len) {   // rhs: Y_k^T, row r = column c0 + r of Y_k (zero past nrhs)
        const int c0 = (e - ii - 1) * NB;
        for (int task = tid; task < 64 * 8; task += kCT) {
          const int r = task & 63, ch = task >> 6;
          float xv[8];
#pragma unroll
          for (int q = 0; q < 8; ++q)
            xv[q] = (c0 + r < nrhs) ? (float)__ldcg(Bb + (long long)(k0 + 8 * ch + q) * ldb + c0 + r) : 0.f;
          put_split3_chunk(Ah, Am, Al, 64 * h + r, ch, xv);
        }
      } else {   // no second tile
        for (int task = tid; task < 64 * 8; task += kCT) {
          const float z[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
          put_split3_chunk(Ah, Am, Al, 64 * h + (task >> 3), task & 7, z);
        }
      }
    }
    tc::fence_proxy_async_smem();
    __syncthreads();
    if (tid == 0) {
      tc::fence_after_sync();
      constexpr uint32_t idesc = tc::idesc_bf16_f32(64);
#pragma unroll
      for (int ks = 0; ks < 4; ++ks) {
        const uint32_t o = ks * 32;
        const uint64_t ah = tc::sdesc_k128(tc::smem_u32(Ah) + o), am = tc::sdesc_k128(tc::smem_u32(Am) + o),
                       al = tc::sdesc_k128(tc::smem_u32(Al) + o);
        const uint64_t bh = tc::sdesc_k128(tc::smem_u32(Bh) + o), bm = tc::sdesc_k128(tc::smem_u32(Bm) + o),
                       bl = tc::sdesc_k128(tc::smem_u32(Bl) + o);
        tc::mma_f16(tmem, ah, bh, idesc, ks > 0 ? 1u : 0u);
        tc::mma_f16(tmem, ah, bm, idesc, 1u);
        tc::mma_f16(tmem, am, bh, idesc, 1u);
        tc::mma_f16(tmem, ah, bl, idesc, 1u);
        tc::mma_f16(tmem, al, bh, idesc, 1u);
        tc::mma_f16(tmem, am, bm, idesc, 1u);
      }
      tc::mma_commit(&mma_bar);
    }
    volatile int* abp = &tc_abort;
    const bool ok = tc::mbar_wait(&mma_bar, mma_ph, abp, stt);
    mma_ph ^= 1u;
    tc::fence_after_sync();
    // warp w: TMEM lanes 32 (w % 4) .. (rows of D), columns 16 (w / 4) ..
    const int warp = tid >> 5, lane = tid & 31, q = warp & 3, g = warp >> 2;
    float v[16];
    tc::tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(g * 16), v);
    const int h = q >> 1, r = (q & 1) * 32 + lane, e = e0 + h;
    if (ok && e < len) {
      R* dst;
      long long ld;
      bool col_ok;
      if (e < ii + 1) {   // A_ij[n][r] -= D[64 h + r][n]
        const int j0 = (k + 1 + e) * NB;
        dst = Ab + (long long)i0 * t + j0 + r;
        ld = t;
        col_ok = j0 + r < t;
      } else {            // B_i[n][c0 + r] -= D[64 h + r][n]
        const int c0 = (e - ii - 1) * NB;
        dst = Bb + (long long)i0 * ldb + c0 + r;
        ld = ldb;
        col_ok = c0 + r < nrhs;
      }
      if (col_ok) {
        R old[16];
#pragma unroll
        for (int c = 0; c < 16; ++c) {
          const int n = 16 * g + c;
          old[c] = (i0 + n < t) ? __ldcg(dst + (long long)n * ld) : R(0);
        }
#pragma unroll
        for (int c = 0; c < 16; ++c) {
          const int n = 16 * g + c;
          if (i0 + n < t) dst[(long long)n * ld] = old[c] - (R)v[c];
        }
      }
    }
    tc::fence_before_sync();
    __syncthreads();
  };

  // step k = -1 only factors the first diagonal block (one call site keeps the
  // register-resident factorisation inlined once)
  for (int k = -1; k < nblk; ++k) {
    const int m = nblk - k - 1, k0 = k * NB, kb = min(NB, t - k0);
    const R* Lk = Lb + (long long)k * NB * NB;
    // trsm phase: L_ik = A_ik Linv_kk^T (x < m) and Y_k = Linv_kk B_k, written over B_k
    for (int x = rank; k >= 0 && x < m + nct; x += kCL) {
      if (x < m) {
        const int i0 = (k + 1 + x) * NB, rb = min(NB, t - i0);
        ld_tiles(S1, Ab, t, i0, k0, rb, NB, true,                    // S1[l][r] = A_ik[r][l]
                 S2, Lk, (long long)NB, 0, 0, NB, NB, true);         // S2[l][c] = Linv[c][l]
        __syncthreads();
        mm64(S1, S2, acc);
        st_acc(Ab + (long long)(i0 + ry) * t + k0 + cx, t, rb - ry, NB, acc);
      } else {
        const int c0 = (x - m) * NB, nc = min(NB, nrhs - c0);
        ld_tiles(S1, Lk, (long long)NB, 0, 0, NB, NB, true,          // S1[l][r] = Linv[r][l]
                 S2, Bb, ldb, k0, c0, kb, nc, false);
        __syncthreads();
        mm64(S1, S2, acc);
        st_acc(Bb + (long long)(k0 + ry) * ldb + c0 + cx, ldb, kb - ry, nc - cx, acc);
      }
      __syncthreads();
    }
    if (k >= 0) {
      cluster_sync_all();
      if (m == 0) break;
    }
    // update phase: the owner of block k+1 updates and factors the diagonal
    // block first (overlapping the serial factorisation with the other CTAs'
    // updates); every CTA then draws the remaining tiles from the counter
    const int ntri = k >= 0 ? m * (m + 1) / 2 : 0, ntot = k >= 0 ? ntri + m * nct : 0;
    if (rank == 0 && tid == 0) ctr[(ep + 1) & 1] = 0;
    if constexpr (kTc) {
      // unit 0 holds the diagonal tile (k+1, k+1): its owner updates and factors it first
      const int nu = k >= 0 ? tc_units(m) : 0;
      if (rank == (k + 1) % kCL) {
        if (k >= 0) tc_update_unit(k, m, 0);
        factor_diag(Ab, Lb, t, k + 1, lam, S1, S2, S3, &bad);
      }
      start_ahead();
      for (;;) {
        const int x = 1 + next_tile_ahead();
        if (x >= nu) break;
        tc_update_unit(k, m, x);
      }
    } else {
      if (rank == (k + 1) % kCL) {
        if (k >= 0) update_tiles(k, 0, ntot, ntot, ntri);
        factor_diag(Ab, Lb, t, k + 1, lam, S1, S2, S3, &bad);
      }
      for (;;) {   // tiles are drawn two at a time
        const int x = 1 + 2 * next_tile();
        if (x >= ntot) break;
        update_tiles(k, x, x + 1, ntot, ntri);
      }
    }
    ++ep;
    cluster_sync_all();
  }

  // back substitution: X_k = Linv_kk^T (Y_k + Z_k) and Z_i -= L_ki^T X_k (i < k).
  // The owner of block k-1 applies X_k to Z_{k-1} first and forms X_{k-1} at
  // once; the other Z tiles are drawn from the counter.
  auto form_x = [&](int k) {
    const int k0 = k * NB, kb = min(NB, t - k0);
    for (int c0 = 0; c0 < nrhs; c0 += NB) {
      const int nc = min(NB, nrhs - c0);
      ld_tile(S1, Lb + (long long)k * NB * NB, NB, 0, 0, NB, NB, false);   // S1[l][r] = Linv[l][r]
      ld_tile_sum(S2, Bb, Zb, ldb, k0, c0, kb, nc);                        // Y_k + Z_k
      __syncthreads();
      mm64(S1, S2, acc);
      st_acc(Xb + (long long)(k0 + ry) * ldb + c0 + cx, ldb, kb - ry, nc - cx, acc);
      __syncthreads();
    }
  };
  auto z_tile = [&](int k, int i, int c0) {
    const int k0 = k * NB, kb = min(NB, t - k0), i0 = i * NB, nc = min(NB, nrhs - c0);
    ld_tiles(S1, Ab, t, k0, i0, kb, NB, false,     // S1[l][r] = L_ki[l][r]
             S2, Xb, ldb, k0, c0, kb, nc, false);  // X_k
    __syncthreads();
    mm64(S1, S2, acc);
    rmw_sub(Zb + (long long)(i0 + ry) * ldb + c0 + cx, ldb, NB - ry, nc - cx, acc);   // block i < k is full
    __syncthreads();
  };
  if (nrhs == 1 && t <= 2 * kTileF<R>) {
    // one right-hand side: the block steps are 64-long mat-vecs whose cost is
    // the barrier between them, so rank 0 runs them alone with CTA barriers
    // (Z in shared memory) and the other CTAs of the cluster leave
    if (rank == 0) {
      R* zs = &S3[0][0];   // Z [t] in S3 and S4 (free now: t <= 2 kTileF)
      R* vs = &S1[0][0];   // Y_k + Z_k [64]
      R* xs = &S1[1][0];   // X_k [64]
      for (int e = tid; e < t; e += kCT) zs[e] = R(0);
      __syncthreads();
      for (int k = nblk - 1; k >= 0; --k) {
        const int k0 = k * NB, kb = min(NB, t - k0);
        if (tid < NB) vs[tid] = tid < kb ? __ldcg(Bb + (long long)(k0 + tid) * ldb) + zs[k0 + tid] : R(0);
        __syncthreads();
        {  // X_k[c] = sum_l Linv_k[l][c] v[l]: eight threads per column, l = part, part + 8, ...
          const int c = tid >> 3, part = tid & 7;
          const R* Li = Lb + (long long)k * NB * NB;
          R a = R(0);
#pragma unroll
          for (int l = part; l < NB; l += 8) a = fma_r(__ldcg(Li + l * NB + c), vs[l], a);
          a += __shfl_xor_sync(0xffffffffu, a, 1);
          a += __shfl_xor_sync(0xffffffffu, a, 2);
          a += __shfl_xor_sync(0xffffffffu, a, 4);
          if (part == 0) {
            xs[c] = c < kb ? a : R(0);
            if (c < kb) Xb[(long long)(k0 + c) * ldb] = a;
          }
        }
        __syncthreads();
        // Z_j -= L_kj^T X_k for the columns before block k (one thread per column)
        for (int cc = tid; cc < k0; cc += kCT) {
          R a = R(0);
          for (int l = 0; l < kb; ++l) a = fma_r(__ldcg(Ab + (long long)(k0 + l) * t + cc), xs[l], a);
          zs[cc] -= a;
        }
        __syncthreads();
      }
    }
    if (tid == 0 && bad) set_status(stt, ARCKV_ERR_NOT_SPD);
    tc_release();
    return;
  }
  if constexpr (kTc) {
    if (nrhs <= 128) {
      if (rank == (nblk - 1) % kCL) tc_x_unit(nblk - 1);
      cluster_sync_all();
      for (int k = nblk - 1; k >= 1; --k) {
        if (rank == 0 && tid == 0) ctr[(ep + 1) & 1] = 0;
        if (rank == (k - 1) % kCL) {   // the owner of block k-1 finishes Z_{k-1} and forms X_{k-1}
          tc_z_unit(k, k - 1);
          tc_x_unit(k - 1);
        }
        start_ahead();
        for (;;) {
          const int i = next_tile_ahead();
          if (i >= k - 1) break;
          tc_z_unit(k, i);
        }
        ++ep;
        cluster_sync_all();
      }
      if (tid == 0 && bad) set_status(stt, ARCKV_ERR_NOT_SPD);
      tc_release();
      return;
    }
  }
  if (rank == (nblk - 1) % kCL) form_x(nblk - 1);
  cluster_sync_all();
  for (int k = nblk - 1; k >= 1; --k) {
    if (rank == 0 && tid == 0) ctr[(ep + 1) & 1] = 0;
    if (rank == (k - 1) % kCL) {
      for (int c0 = 0; c0 < nrhs; c0 += NB) z_tile(k, k - 1, c0);
      form_x(k - 1);
    }
    const int ntz = (k - 1) * nct;
    for (;;) {
      const int g = next_tile();
      if (g >= ntz) break;
      z_tile(k, g / nct, (g % nct) * NB);
    }
    ++ep;
    cluster_sync_all();
  }
  if (tid == 0 && bad) set_status(stt, ARCKV_ERR_NOT_SPD);
  tc_release();
}

template <typename R>
static int cholesky_solve(int H, int t, R* Gram, R* Linv, R* B, R* Z, R* X, int ldb, int nrhs, long long bbs,
                          float ridge, DevStatus* stt, cudaStream_t st, int tdiv = 0) {
  const int smem = 4 * kTileF<R> * (int)sizeof(R) + (std::is_same<R, float>::value ? kTcStageBytes : 0);
  const R td = (R)(tdiv > 0 ? tdiv : t);
  if (cluster_size(t) == 8) {
    set_dyn_smem((const void*)chol_cluster_kernel<R, 8>, smem);
    chol_cluster_kernel<R, 8><<<8 * H, kCT, smem, st>>>(Gram, Linv, B, Z, X, t, nrhs, ldb, bbs, (R)ridge, td, stt);
  } else {
    set_dyn_smem((const void*)chol_cluster_kernel<R, 4>, smem);
    chol_cluster_kernel<R, 4><<<4 * H, kCT, smem, st>>>(Gram, Linv, B, Z, X, t, nrhs, ldb, bbs, (R)ridge, td, stt);
  }
  return 1;
}

__global__ void beta_kernel(const float* w, float* beta, long long count, float eps_w, float b_min, float b_max) {
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < count;
       k += (long long)gridDim.x * blockDim.x) {
    const float ws = fmaxf(w[k], 0.f);
    beta[k] = fminf(fmaxf(logf(fmaxf(ws, eps_w)), b_min), b_max);
  }
}

// P[row] = softmax(LC[row] + beta), one warp per row (rows = H * n).
__global__ void softmax_bias_kernel(const float* LC, const float* beta, float* P, int n, int t) {
  const int b = blockIdx.y, row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= n) return;
  const float* x = LC + ((long long)b * n + row) * t;
  const float* be = beta + (long long)b * t;
  float* o = P + ((long long)b * n + row) * t;
  float mx = -INFINITY;
  for (int c = lane; c < t; c += 32) mx = fmaxf(mx, x[c] + be[c]);
  mx = warp_max(mx);
  float sm = 0.f;
  for (int c = lane; c < t; c += 32) sm += expf(x[c] + be[c] - mx);
  sm = warp_sum(sm);
  const float inv = 1.0f / sm;
  for (int c = lane; c < t; c += 32) o[c] = expf(x[c] + be[c] - mx) * inv;
}

// dst_hi/lo[b][c][r] = split(src[b][r][c]) for r < rows, zero for rows <= r < ldr:
// the transposed, K-major split-bf16 operand of the Gram GEMMs.
__global__ void __launch_bounds__(256) transpose_split_kernel(const float* src, int rows, int cols, bf16* dst_hi,
                                                              bf16* dst_lo, int ldr) {
  const int b = blockIdx.z, c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  __shared__ float tile[32][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const float* sb = src + (long long)b * rows * cols;
  for (int q = ty; q < 32; q += 8) {
    const int r = r0 + q, c = c0 + tx;
    tile[q][tx] = (r < rows && c < cols) ? sb[(long long)r * cols + c] : 0.f;
  }
  __syncthreads();
  for (int q = ty; q < 32; q += 8) {
    const int c = c0 + q, r = r0 + tx;
    if (c < cols && r < ldr) {
      bf16 hi, lo;
      split_bf16(tile[tx][q], hi, lo);
      const long long o = ((long long)b * cols + c) * ldr + r;
      dst_hi[o] = hi;
      dst_lo[o] = lo;
    }
  }
}

// Transposed bf16 triple of src [rows][cols] (fp32): dst_{h,m,l}[b][c][r]
// (row stride ldr >= rows; the pad r in [rows, ldr) is written as zeros).
__global__ void __launch_bounds__(256) transpose_split3_kernel(const float* src, int rows, int cols, bf16* dh, bf16* dm,
                                                               bf16* dl, int ldr) {
  const int b = blockIdx.z, c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  __shared__ float tile[32][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const float* sb = src + (long long)b * rows * cols;
  for (int q = ty; q < 32; q += 8) {
    const int r = r0 + q, c = c0 + tx;
    tile[q][tx] = (r < rows && c < cols) ? sb[(long long)r * cols + c] : 0.f;
  }
  __syncthreads();
  for (int q = ty; q < 32; q += 8) {
    const int c = c0 + q, r = r0 + tx;
    if (c < cols && r < ldr) {
      const long long o = ((long long)b * cols + c) * ldr + r;
      split3_bf16(tile[tx][q], dh[o], dm[o], dl[o]);
    }
  }
}

// C[b] (t x t, row stride t) = X^T X over the n reference rows, X^T given as a
// transposed bf16 triple [t][ldn]: the kSplit3S tensor-core Gram.
static int gram3_tc(int H, int t, int ldn, const bf16* Xh, const bf16* Xm, const bf16* Xl, float* C, DevStatus* stt,
                    cudaStream_t st) {
  CUtensorMap mA, mA2, mA3;
  if (!encode_bf16_map_3d(&mA, Xh, ldn, t, H, 128) || !encode_bf16_map_3d(&mA2, Xm, ldn, t, H, 128) ||
      !encode_bf16_map_3d(&mA3, Xl, ldn, t, H, 128))
    return -1;
  TcEpiStore epi{C, (long long)t * t, t, 1.f};
  const int kfull = (ldn + 63) / 64 * 64;
  if (launch_tc_gemm<128, kSplit3S>(mA, mA, mA2, mA2, epi, H, t, t, ldn, kfull, stt, st, 0, &mA3) != cudaSuccess)
    return -1;
  return 1;
}

// C[b] (M x N, row stride ldc) = X^T Z over the n reference rows, with X^T and
// Z^T given as transposed split-bf16 operands [M][ldn] and [N][ldn].
static int gram_tc(int H, int M, int N, int ldn, const bf16* Xh, const bf16* Xl, const bf16* Zh, const bf16* Zl,
                   float* C, int ldc, DevStatus* stt, cudaStream_t st) {
  CUtensorMap mA, mA2, mB, mB2;
  if (!encode_bf16_map_3d(&mA, Xh, ldn, M, H, 128) || !encode_bf16_map_3d(&mA2, Xl, ldn, M, H, 128) ||
      !encode_bf16_map_3d(&mB, Zh, ldn, N, H, 128) || !encode_bf16_map_3d(&mB2, Zl, ldn, N, H, 128))
    return -1;
  TcEpiStore epi{C, (long long)M * ldc, ldc, 1.f};
  const int kfull = (ldn + 63) / 64 * 64;
  if (launch_tc_gemm<128, kSplit>(mA, mB, mA2, mB2, epi, H, M, N, ldn, kfull, stt, st) != cudaSuccess) return -1;
  return 1;
}

// C[b] = X X^T in fp64 (X fp32 [rows][K]); 64 x 64 lower tiles, mirrored.
__global__ void __launch_bounds__(256) syrk64_kernel(const float* X, double* C, int rows, int K) {
  const int b = blockIdx.z, i0 = blockIdx.y * 64, j0 = blockIdx.x * 64;
  if (j0 > i0) return;
  const float* Xb = X + (long long)b * rows * K;
  double* Cb = C + (long long)b * rows * rows;
  __shared__ double As[16][65], Bs[16][65];
  const int ty = threadIdx.x >> 4, tx = threadIdx.x & 15;
  double acc[4][4];
#pragma unroll
  for (int p = 0; p < 4; ++p)
#pragma unroll
    for (int q = 0; q < 4; ++q) acc[p][q] = 0.0;
  for (int k0 = 0; k0 < K; k0 += 16) {
    for (int e = threadIdx.x; e < 64 * 16; e += 256) {
      const int r = e >> 4, kk = e & 15, k = k0 + kk;
      As[kk][r] = (i0 + r < rows && k < K) ? (double)Xb[(long long)(i0 + r) * K + k] : 0.0;
      Bs[kk][r] = (j0 + r < rows && k < K) ? (double)Xb[(long long)(j0 + r) * K + k] : 0.0;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      double a[4], c[4];
#pragma unroll
      for (int p = 0; p < 4; ++p) { a[p] = As[kk][ty * 4 + p]; c[p] = Bs[kk][tx * 4 + p]; }
#pragma unroll
      for (int p = 0; p < 4; ++p)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[p][q] = fma(a[p], c[q], acc[p][q]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int p = 0; p < 4; ++p)
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = i0 + ty * 4 + p, j = j0 + tx * 4 + q;
      if (i < rows && j < rows) {
        Cb[(long long)i * rows + j] = acc[p][q];
        Cb[(long long)j * rows + i] = acc[p][q];
      }
    }
}

__global__ void widen_kernel(const float* x, double* y, long long count) {
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < count;
       k += (long long)gridDim.x * blockDim.x)
    y[k] = (double)x[k];
}

// out[b][r][c] = sum_i X[b][i][r] Y[b][i][c] accumulated in fp64 (X fp32 [n][t],
// Y fp64 [n][ncol], out fp32 [t][ncol]); 64 x 32 output tiles.
__global__ void __launch_bounds__(256) xty64_kernel(const float* X, const double* Y, float* out, int n, int t,
                                                    int ncol) {
  const int b = blockIdx.z, r0 = blockIdx.x * 64, c0 = blockIdx.y * 32;
  const float* Xb = X + (long long)b * n * t;
  const double* Yb = Y + (long long)b * n * ncol;
  __shared__ double Xs[16][64], Ys[16][33];
  const int tr = threadIdx.x & 63, tc = threadIdx.x >> 6;   // 64 rows x 4 column groups of 8
  double acc[8];
#pragma unroll
  for (int q = 0; q < 8; ++q) acc[q] = 0.0;
  for (int i0 = 0; i0 < n; i0 += 16) {
    for (int e = threadIdx.x; e < 16 * 64; e += 256) {
      const int ii = e >> 6, r = e & 63;
      Xs[ii][r] = (i0 + ii < n && r0 + r < t) ? (double)Xb[(long long)(i0 + ii) * t + r0 + r] : 0.0;
    }
    for (int e = threadIdx.x; e < 16 * 32; e += 256) {
      const int ii = e >> 5, c = e & 31;
      Ys[ii][c] = (i0 + ii < n && c0 + c < ncol) ? Yb[(long long)(i0 + ii) * ncol + c0 + c] : 0.0;
    }
    __syncthreads();
#pragma unroll
    for (int ii = 0; ii < 16; ++ii) {
      const double xv = Xs[ii][tr];
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[q] = fma(xv, Ys[ii][tc * 8 + q], acc[q]);
    }
    __syncthreads();
  }
  const int r = r0 + tr;
  if (r >= t) return;
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const int c = c0 + tc * 8 + q;
    if (c < ncol) out[((long long)b * t + r) * ncol + c] = (float)acc[q];
  }
}

// ---------------------------------------------------------------------------
// Blocked Cholesky solve of the fp64 dual systems, (A + lam I) X = B with
// lam = ridge * trace(A) / tdiv, A [H][n][n] (lower part read, overwritten
// by L), B [H][n][nrhs] (overwritten by the forward solution Y = L^-1 B),
// X [H][n][nrhs].  Right-looking over 64-wide block columns; every block
// product runs on the tensor pipe as an exact product of 5-slice operands
// (2^-40 of each row's largest entry per operand, the same backward error as
// an fp64 factorisation to ~1e-12), and only the 64 x 64 diagonal factors
// and inverses (double-float, ~48 bits, from fp64 storage) and the block
// back substitution run on the SIMT pipes:
//   for k:  L_kk = chol(A_kk + lam I), Linv_kk = L_kk^-1        (double-float)
//           L_ik = A_ik Linv_kk^T                        i > k  (sliced)
//           A_ij -= L_ik L_jk^T                    j <= i, i > k  (sliced, lower tiles)
//           Y_k = Linv_kk B_k;  B_i -= L_ik Y_k         i > k  (sliced)
//   for k descending:  Z_k = sum_{i>k} L_ik^T X_i            (sliced)
//           X_k = Linv_kk^T (Y_k - Z_k)                         (fp64 SIMT)
// With one right-hand side both substitutions run in tri_solve_cluster_kernel.

constexpr int kCholSlices = 5;

__global__ void chol_lambda_kernel(const double* A, int n, double ridge, double tdiv, double* lam, DevStatus* stt) {
  __shared__ double red[8];
  const int b = blockIdx.x;
  const double* Ab = A + (long long)b * n * n;
  double a = 0.0;
  for (int r = threadIdx.x; r < n; r += 256) a += Ab[(long long)r * n + r];
  a = warp_sum_r(a);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = a;
  __syncthreads();
  if (threadIdx.x == 0) {
    double tr = 0.0;
    for (int w = 0; w < 8; ++w) tr += red[w];
    if (!isfinite(tr)) set_status(stt, ARCKV_ERR_NONFINITE);
    lam[b] = ridge * tr / tdiv;
  }
}

// Factor diagonal block k of every head (one CTA per head) in double-float
// arithmetic: L_kk into A, L_kk^-1 into Linv[k] (fp64 storage); a
// non-positive pivot records ARCKV_ERR_NOT_SPD.
__global__ void __launch_bounds__(kCT, 1) chol_diag_kernel(double* A, double* Linv, int n, int k, const double* lam,
                                                           DevStatus* stt) {
  extern __shared__ __align__(16) unsigned char smraw[];
  df64* sm = (df64*)smraw;
  Tile<df64> S1 = (Tile<df64>)sm;
  Tile<df64> S2 = (Tile<df64>)(sm + kTileF<df64>);
  Tile<df64> S3 = (Tile<df64>)(sm + 2 * kTileF<df64>);
  __shared__ int bad;
  const int b = blockIdx.x, nblk = (n + NB - 1) / NB;
  if (threadIdx.x == 0) bad = 0;
  __syncthreads();
  factor_diag<df64, double>(A + (long long)b * n * n, Linv + (long long)b * nblk * NB * NB, n, k, lam[b], S1, S2, S3,
                            &bad);
  if (threadIdx.x == 0 && bad) set_status(stt, ARCKV_ERR_NOT_SPD);
}

// X_k = Linv_kk^T (Y_k - Z_k) for block k of every head, 32 right-hand sides
// per CTA (grid: head x column group): V = Y_k - Z_k and Linv_kk go through
// shared memory, X[k0 + c][j] = sum_{l >= c} Linv_k[l][c] V[l][j].
__global__ void __launch_bounds__(256) chol_back_block_kernel(const double* Linv, const double* Y, const double* Z,
                                                              double* X, int n, int k, int nrhs, int useZ) {
  __shared__ double Ls[NB][NB + 1];
  __shared__ double Vs[NB][33];
  const int b = blockIdx.x, j0 = blockIdx.y * 32, nblk = (n + NB - 1) / NB, k0 = k * NB, kb = min(NB, n - k0);
  const int nj = min(32, nrhs - j0);
  const double* Li = Linv + ((long long)b * nblk + k) * NB * NB;
  const double* Yb = Y + ((long long)b * n + k0) * nrhs + j0;
  const double* Zb = Z + (long long)b * NB * nrhs + j0;
  double* Xb = X + ((long long)b * n + k0) * nrhs + j0;
  for (int e = threadIdx.x; e < NB * NB; e += 256) Ls[e / NB][e % NB] = Li[e];
  for (int e = threadIdx.x; e < NB * 32; e += 256) {
    const int l = e >> 5, j = e & 31;
    Vs[l][j] = (l < kb && j < nj) ? Yb[(long long)l * nrhs + j] - (useZ ? Zb[(long long)l * nrhs + j] : 0.0) : 0.0;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < kb * 32; e += 256) {
    const int c = e >> 5, j = e & 31;
    double a = 0.0;
    for (int l = c; l < kb; ++l) a = fma(Ls[l][c], Vs[l][j], a);
    if (j < nj) Xb[(long long)c * nrhs + j] = a;
  }
}

// w[b][r] = sum_i Phi[b][i][r] a[b][i] (Phi fp32 [n][t], a fp64): one thread
// per column r, the rows of the column read coalesced across the warp.  The
// terms cancel heavily (|a| |Phi| exceeds |w| by ~1e4 on 128K caches), so the
// sum runs in double-float arithmetic: each product Phi a_hi + Phi a_lo is
// formed exactly up to the lo part's rounding and added with an error-free
// sum; a is split into fp32 (hi, lo) pairs in shared memory, 1024 rows at a time.
__global__ void __launch_bounds__(256) phi_t_vec_kernel(const float* __restrict__ Phi, const double* __restrict__ a,
                                                        float* __restrict__ w, int n, int t) {
  __shared__ float ah[1024], al[1024];
  const int b = blockIdx.y, r = blockIdx.x * 256 + threadIdx.x;
  const float* p = Phi + (long long)b * n * t + min(r, t - 1);
  const double* ab = a + (long long)b * n;
  df64 sum(0.f, 0.f);
  for (int i0 = 0; i0 < n; i0 += 1024) {
    const int cnt = min(1024, n - i0);
    __syncthreads();
    for (int i = threadIdx.x; i < cnt; i += 256) {
      const double v = ab[i0 + i];
      const float h = __double2float_rn(v);
      ah[i] = h;
      al[i] = __double2float_rn(v - (double)h);
    }
    __syncthreads();
    if (r < t) {
      for (int i = 0; i < cnt; ++i) {
        const float x = p[(long long)(i0 + i) * t];
        const float ph = x * ah[i];
        const float pl = fmaf(x, al[i], fmaf(x, ah[i], -ph));
        df64 s2 = df_two(sum.hi, ph);
        s2.lo += sum.lo + pl;
        sum = df_fast2(s2.hi, s2.lo);
      }
    }
  }
  if (r < t) w[(long long)b * t + r] = sum.hi + sum.lo;
}

// Both substitutions of the single-right-hand-side dual beta system
// L L^T x = r (the fp64 factor in A's lower triangle, Linv the inverses of its
// 64 x 64 diagonal blocks) by a cluster of kTsCL CTAs per head: in each block
// step every rank sums its share of the off-diagonal blocks (block index
// j = rank mod kTsCL) into rank 0's shared memory, and rank 0 applies the
// diagonal block's inverse and publishes the block of the solution.  The fp64
// multiply-adds (n^2 per head) are spread over the cluster's SMs.  Every rank
// runs the same fixed trip counts, so every cluster barrier is reached by all.
constexpr int kTsCL = 8;
__global__ void __cluster_dims__(kTsCL, 1, 1) __launch_bounds__(256, 1)
    tri_solve_cluster_kernel(const double* __restrict__ A, const double* __restrict__ Linv,
                             const double* __restrict__ r, double* __restrict__ yd, double* __restrict__ x, int n) {
  namespace cg = cooperative_groups;
  __shared__ double red[kTsCL][NB];   // rank 0: the ranks' partial sums
  __shared__ double part[4][NB];
  __shared__ double v[NB];
  const int head = blockIdx.x / kTsCL, rank = (int)cluster_rank(), tid = threadIdx.x;
  const int nblk = (n + NB - 1) / NB;
  const double* Ab = A + (long long)head * n * n;
  const double* Lb = Linv + (long long)head * nblk * NB * NB;
  const double* rb = r + (long long)head * n;
  double* y = yd + (long long)head * n;
  double* xb = x + (long long)head * n;
  double* red0 = cg::this_cluster().map_shared_rank(&red[0][0], 0);
  // forward: y_k = Linv_kk (r_k - sum_{j<k} L_kj y_j)
  for (int k = 0; k < nblk; ++k) {
    const int k0 = k * NB, kb = min(NB, n - k0);
    {  // four threads per row of block k
      const int rr = tid >> 2, pt = tid & 3;
      double a0 = 0.0, a1 = 0.0;
      if (rr < kb) {
        const double* row = Ab + (long long)(k0 + rr) * n;
        for (int j = rank; j < k; j += kTsCL)
          for (int c = j * NB + pt; c < j * NB + NB; c += 8) {
            a0 = fma(__ldcg(row + c), __ldcg(y + c), a0);
            a1 = fma(__ldcg(row + c + 4), __ldcg(y + c + 4), a1);
          }
      }
      double a = a0 + a1;
      a += __shfl_xor_sync(0xffffffffu, a, 1);
      a += __shfl_xor_sync(0xffffffffu, a, 2);
      if (pt == 0) red0[rank * NB + rr] = a;
    }
    cluster_sync_all();
    if (rank == 0) {
      if (tid < NB) {
        double sum = 0.0;
#pragma unroll
        for (int q = 0; q < kTsCL; ++q) sum += red[q][tid];
        v[tid] = tid < kb ? rb[k0 + tid] - sum : 0.0;
      }
      __syncthreads();
      const int c = tid >> 2, pt = tid & 3;   // y_k[c] = sum_{l <= c} Linv_k[c][l] v[l]
      const double* Li = Lb + (long long)k * NB * NB + c * NB;
      double a = 0.0;
      for (int l = pt; l <= c; l += 4) a = fma(__ldcg(Li + l), v[l], a);
      a += __shfl_xor_sync(0xffffffffu, a, 1);
      a += __shfl_xor_sync(0xffffffffu, a, 2);
      if (pt == 0 && c < kb) y[k0 + c] = a;
    }
    cluster_sync_all();
  }
  // backward: x_k = Linv_kk^T (y_k - sum_{j>k} L_jk^T x_j)
  for (int k = nblk - 1; k >= 0; --k) {
    const int k0 = k * NB, kb = min(NB, n - k0);
    {  // column c of block k, four row groups
      const int c = tid & (NB - 1), pt = tid >> 6;
      double a0 = 0.0, a1 = 0.0;
      if (c < kb)
        for (int j = k + 1 + rank; j < nblk; j += kTsCL) {
          const int i1 = min(n, j * NB + NB);
          for (int i = j * NB + pt; i < i1; i += 8) {
            a0 = fma(__ldcg(Ab + (long long)i * n + k0 + c), __ldcg(xb + i), a0);
            if (i + 4 < i1) a1 = fma(__ldcg(Ab + (long long)(i + 4) * n + k0 + c), __ldcg(xb + i + 4), a1);
          }
        }
      part[pt][c] = a0 + a1;
    }
    __syncthreads();
    if (tid < NB) red0[rank * NB + tid] = (part[0][tid] + part[1][tid]) + (part[2][tid] + part[3][tid]);
    cluster_sync_all();
    if (rank == 0) {
      if (tid < NB) {
        double sum = 0.0;
#pragma unroll
        for (int q = 0; q < kTsCL; ++q) sum += red[q][tid];
        v[tid] = tid < kb ? y[k0 + tid] - sum : 0.0;
      }
      __syncthreads();
      const int c = tid >> 2, pt = tid & 3;   // x_k[c] = sum_{l >= c} Linv_k[l][c] v[l]
      const double* Li = Lb + (long long)k * NB * NB;
      double a = 0.0;
      for (int l = c + pt; l < NB; l += 4) a = fma(__ldcg(Li + (long long)l * NB + c), v[l], a);
      a += __shfl_xor_sync(0xffffffffu, a, 1);
      a += __shfl_xor_sync(0xffffffffu, a, 2);
      if (pt == 0 && c < kb) xb[k0 + c] = a;
    }
    cluster_sync_all();
  }
}

struct CholSlicedBufs {
  bf16 *sA, *sB, *sC;   // 5-slice operands: panel rows / columns, Linv_kk rows, right-hand-side columns
  int *eA, *eB, *eC;
  double *lam, *Z;      // [H], [H][64][nrhs]
};

// A second stream per calling stream (created on first use, kept for the
// process) and two events, for the look-ahead of the blocked dual Cholesky.
struct SideStream {
  cudaStream_t s;
  cudaEvent_t fork, join;
};
static bool side_stream(cudaStream_t main, SideStream& out) {
  static std::mutex mu;
  static std::map<std::pair<int, cudaStream_t>, SideStream> cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  std::lock_guard<std::mutex> g(mu);
  auto it = cache.find({dev, main});
  if (it != cache.end()) {
    out = it->second;
    return true;
  }
  SideStream ss{};
  if (cudaStreamCreateWithFlags(&ss.s, cudaStreamNonBlocking) != cudaSuccess) return false;
  if (cudaEventCreateWithFlags(&ss.fork, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&ss.join, cudaEventDisableTiming) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  cache[{dev, main}] = ss;
  out = ss;
  return true;
}

// Blocked right-looking Cholesky of the n x n systems with a look-ahead of
// one block: after step k's panel the trailing matrix is updated in two
// launches, first its leading 64-column block (block k + 1, all rows), then
// the rest of its lower triangle; the second runs on the calling stream
// while a side stream factors block k + 1, slices its inverse and forms and
// slices the panel below it, so the diagonal factor and the panel leave the
// critical path: the second update leaves kAheadSMs SMs free (its
// persistent grid is capped) and the side stream's panel product takes at
// most that many CTAs.  Slices of consecutive steps alternate between two
// buffers.
// The operations and their order per element are those of the plain blocked
// algorithm.
static int chol_solve_sliced(int H, int n, double* A, double* Linv, double* B, double* X, int nrhs, double ridge,
                             double tdiv, const CholSlicedBufs& W, DevStatus* stt, cudaStream_t st) {
  constexpr int S = kCholSlices;
  const int nblk = (n + NB - 1) / NB;
  const long long nn = (long long)n * n, nr = (long long)n * nrhs, lb = (long long)nblk * NB * NB;
  const int dsm = 3 * kTileF<df64> * (int)sizeof(df64);
  if (set_dyn_smem((const void*)chol_diag_kernel, dsm) != cudaSuccess)
    return -1;
  int nl = 0;
  auto ok = [&](int r) {
    if (r < 0) return false;
    nl += r;
    return true;
  };
  SideStream ss{};
  const bool ahead = nblk > 1 && side_stream(st, ss);
  constexpr int kAheadSMs = 16;
  const int main_ctas = ahead ? std::max(1, tc_gemm_sm_count() - kAheadSMs) : 0, side_ctas = ahead ? kAheadSMs : 0;
  const cudaStream_t sd = ahead ? ss.s : st;
  const long long sa_stride = (long long)S * H * n * NB, sb_stride = (long long)S * H * NB * NB;
  auto SA = [&](int k) { return W.sA + (k & 1) * sa_stride; };
  auto EA = [&](int k) { return W.eA + (k & 1) * (long long)H * n; };
  auto SB = [&](int k) { return W.sB + (k & 1) * sb_stride; };
  auto EB = [&](int k) { return W.eB + (k & 1) * (long long)H * NB; };
  // block k: its diagonal factor and inverse, the inverse's slices, the panel
  // L_ik = A_ik Linv_kk^T below it and the panel's slices (on stream s)
  auto diag_panel = [&](int k, cudaStream_t s) -> bool {
    const int k0 = k * NB, kb = std::min(NB, n - k0), m = n - k0 - kb;
    chol_diag_kernel<<<H, kCT, dsm, s>>>(A, Linv, n, k, W.lam, stt);
    ++nl;
    if (!ok(launch_slice_rows(S, Linv + (long long)k * NB * NB, kb, kb, NB, lb, H, SB(k), EB(k), s))) return false;
    if (m > 0) {
      double* panel = A + (long long)(k0 + kb) * n + k0;
      if (!ok(launch_slice_rows(S, panel, m, kb, n, nn, H, SA(k), EA(k), s))) return false;
      if (!ok(launch_sliced_f64(S, SA(k), EA(k), m, SB(k), EB(k), kb, kb, H, panel, nn, n, false, false, stt, s, 0,
                                1 << 30, s == st ? 0 : side_ctas)))
        return false;
      if (!ok(launch_slice_rows(S, panel, m, kb, n, nn, H, SA(k), EA(k), s))) return false;
    }
    return true;
  };
  chol_lambda_kernel<<<H, 256, 0, st>>>(A, n, ridge, tdiv, W.lam, stt);
  ++nl;
  if (!diag_panel(0, st)) return -1;
  for (int k = 0; k < nblk; ++k) {
    const int k0 = k * NB, kb = std::min(NB, n - k0), m = n - k0 - kb;
    if (m > 0) {
      // A_ij -= L_ik L_jk^T on the trailing lower triangle: block k + 1 first
      double* trail = A + (long long)(k0 + kb) * n + k0 + kb;
      if (!ok(launch_sliced_f64(S, SA(k), EA(k), m, SA(k), EA(k), m, kb, H, trail, nn, n, true, true, stt, st, 0, 1)))
        return -1;
      if (ahead) {
        cudaEventRecord(ss.fork, st);
        cudaStreamWaitEvent(sd, ss.fork, 0);
      }
      if (!diag_panel(k + 1, sd)) return -1;
      if (!ok(launch_sliced_f64(S, SA(k), EA(k), m, SA(k), EA(k), m, kb, H, trail, nn, n, true, true, stt, st, 1,
                                1 << 30, main_ctas)))
        return -1;
    }
    if (nrhs > 1) {
      // Y_k = Linv_kk B_k over B_k; B_i -= L_ik Y_k
      double* Bk = B + (long long)k0 * nrhs;
      if (!ok(launch_slice_cols(S, Bk, kb, nrhs, nrhs, nr, H, W.sC, W.eC, st))) return -1;
      if (!ok(launch_sliced_f64(S, SB(k), EB(k), kb, W.sC, W.eC, nrhs, kb, H, Bk, nr, nrhs, false, false, stt, st)))
        return -1;
      if (m > 0) {
        if (!ok(launch_slice_cols(S, Bk, kb, nrhs, nrhs, nr, H, W.sC, W.eC, st))) return -1;
        if (!ok(launch_sliced_f64(S, SA(k), EA(k), m, W.sC, W.eC, nrhs, kb, H, Bk + (long long)kb * nrhs, nr, nrhs,
                                  false, true, stt, st)))
          return -1;
      }
    }
    if (ahead && m > 0) {
      cudaEventRecord(ss.join, sd);
      cudaStreamWaitEvent(st, ss.join, 0);
    }
  }
  if (nrhs == 1) {
    // one right-hand side: both substitutions by a cluster per head (fp64,
    // n^2 multiply-adds spread over its SMs), the forward result left in W.Z
    tri_solve_cluster_kernel<<<H * kTsCL, 256, 0, st>>>(A, Linv, B, W.Z, X, n);
    return nl + 1;
  }
  for (int k = nblk - 1; k >= 0; --k) {
    const int k0 = k * NB, kb = std::min(NB, n - k0), m = n - k0 - kb;
    if (m > 0) {
      // Z_k = sum_{i>k} L_ik^T X_i: the columns of the panel against the columns of X below block k
      const double* panel = A + (long long)(k0 + kb) * n + k0;
      if (!ok(launch_slice_cols(S, panel, m, kb, n, nn, H, W.sA, W.eA, st))) return -1;
      if (!ok(launch_slice_cols(S, X + (long long)(k0 + kb) * nrhs, m, nrhs, nrhs, nr, H, W.sC, W.eC, st))) return -1;
      if (!ok(launch_sliced_f64(S, W.sA, W.eA, kb, W.sC, W.eC, nrhs, m, H, W.Z, (long long)NB * nrhs, nrhs, false,
                                false, stt, st)))
        return -1;
    }
    chol_back_block_kernel<<<dim3(H, cdiv(nrhs, 32)), 256, 0, st>>>(Linv, B, W.Z, X, n, k, nrhs, m > 0 ? 1 : 0);
    ++nl;
  }
  return nl;
}

// Dual (push-through) form of both ridge fits for t > n, where the primal
// t x t normal matrices have rank <= n:
//   (Phi^T Phi + lam I) w = Phi^T m   <=>   w = Phi^T a,  (Phi Phi^T + lam I) a = m
//   (P^T P + lam I) C_v = P^T Y       <=>   C_v = P^T A,  (P P^T + lam I) A = Y
// with the same lam = ridge * trace / t (trace(Phi^T Phi) = trace(Phi Phi^T)),
// so the solutions equal the primal ones; the systems are n x n.  These
// systems reach condition numbers ~1e8 on 128K caches (lam relative to t
// diagonal entries, n of them carrying the mass), and a Gram error that does
// not keep the Gram structure moves beta by up to cond x error: the n x n
// Grams are exact products of row-sliced Phi / P^ on the tensor cores (4
// slices: 32 bits of each row relative to its largest entry, a perturbation
// of the operand itself), the solves are fp64-grade (chol_solve_sliced),
// w = Phi^T a is summed in double-float and C_v = P^T A is a 4-slice
// tensor-core product (with 3 slices for P^ the held-out outputs of a 128K
// head drift by ~7e-3).  Beyond kSlicedMaxK the fp64 SIMT products serve.
static int fits_dual(const Dims& D, float ridge_w, float ridge_v, float eps_w, float b_min, float b_max,
                     const float* m, const float* Y, const FitBufs& B, float* beta, float* C_v, DevStatus* stt,
                     cudaStream_t st, cudaEvent_t const* ev) {
  auto mark = [&](int s) {
    if (ev) cudaEventRecord(ev[s], st);
  };
  const long long nt = (long long)D.n * D.t, nd = (long long)D.n * D.d;
  const bool sliced = sliced_supported(D.t) && sliced_supported(D.n);
  const dim3 sgrid(cdiv(D.n, 64), cdiv(D.n, 64), D.H);
  int nl = 0;
  auto gram = [&](int S) -> int {   // B.G64 = X X^T for X = B.Phi [n][t]
    if (!sliced) {
      syrk64_kernel<<<sgrid, 256, 0, st>>>(B.Phi, B.G64, D.n, D.t);
      return 1;
    }
    const int a = launch_slice_rows(S, B.Phi, D.n, D.t, D.t, nt, D.H, B.Sl, B.eR, st);
    const int g = launch_sliced_gram_lower(S, B.Sl, B.eR, D.n, D.t, D.H, B.G64, stt, st);
    return (a < 0 || g < 0) ? -1 : a + g;
  };
  // beta system
  int r = gram(4);
  if (r < 0) return -1;
  nl += r;
  const CholSlicedBufs CW{B.Sl, B.Sl2, B.Sl3, B.eR, B.eC, B.eC2, B.cl_lam, B.Z64};
  auto solve = [&](int nrhs, long long nrow, float ridge) -> int {
    if (sliced) return chol_solve_sliced(D.H, D.n, B.G64, B.L64, B.B64, B.X64, nrhs, ridge, D.t, CW, stt, st);
    return cholesky_solve<double>(D.H, D.n, B.G64, B.L64, B.B64, B.Z64, B.X64, nrhs, nrhs, nrow, ridge, stt, st, D.t);
  };
  mark(8);
  widen_kernel<<<cdiv((long long)D.H * D.n, 256), 256, 0, st>>>(m, B.B64, (long long)D.H * D.n);
  r = solve(1, D.n, ridge_w);
  if (r < 0) return -1;
  nl += 1 + r;
  phi_t_vec_kernel<<<dim3(cdiv(D.t, 256), D.H), 256, 0, st>>>(B.Phi, B.X64, B.rhs, D.n, D.t);   // w = Phi^T a
  const long long ht = (long long)D.H * D.t;
  beta_kernel<<<cdiv(ht, 256), 256, 0, st>>>(B.rhs, beta, ht, eps_w, b_min, b_max);
  softmax_bias_kernel<<<dim3(cdiv(D.n, 8), D.H), 256, 0, st>>>(B.LC, beta, B.Phi, D.n, D.t);
  nl += 3;
  // value system
  mark(9);
  r = gram(4);
  if (r < 0) return -1;
  nl += r;
  mark(10);
  widen_kernel<<<cdiv((long long)D.H * nd, 256), 256, 0, st>>>(Y, B.B64, (long long)D.H * nd);
  r = solve(D.d, nd, ridge_v);
  if (r < 0) return -1;
  nl += 1 + r;
  if (!sliced) {
    xty64_kernel<<<dim3(cdiv(D.t, 64), cdiv(D.d, 32), D.H), 256, 0, st>>>(B.Phi, B.X64, C_v, D.n, D.t, D.d);
    return nl + 1;
  }
  // C_v = P^T A: the rows of P^T (columns of P) and of A^T, 4 slices each
  const int a = launch_slice_cols(4, B.Phi, D.n, D.t, D.t, nt, D.H, B.Sl, B.eR, st);
  const int b = launch_slice_cols(4, B.X64, D.n, D.d, D.d, nd, D.H, B.Sl2, B.eC, st);
  const int c = launch_sliced_product_f32(4, B.Sl, B.eR, D.t, B.Sl2, B.eC, D.d, D.n, D.H, C_v, D.d, stt, st);
  if (a < 0 || b < 0 || c < 0) return -1;
  return nl + a + b + c;
}

// ---------------------------------------------------------------------------
// Iterative refinement of the beta system (t <= n; App. A.9 Eq. mass_fit).
// The tensor-core Gram and factor are fp32-grade; with condition numbers up to
// ~1e7 that leaves beta a few 1e-3 off on long caches.  Each step forms the
// residual of the normal equations against Phi itself in fp64,
//     r = Phi^T (m - Phi x) - lam x,   lam = ridge * sum_ir Phi_ir^2 / t,
// (the exact normal matrix of the fp32 Phi, no Gram rounding) and corrects
// x += (L L^T)^-1 r with the factor the solver left behind: L_kk and the
// off-diagonal blocks in the Gram's lower part, L_kk^-1 in Linv.

// u[b][i] = m_i - sum_r Phi_ir x_r (fp64); with sq, also sq[b][i] = sum_r Phi_ir^2.
// One warp per row.
__global__ void __launch_bounds__(256) ir_rows_kernel(const float* __restrict__ Phi, const float* __restrict__ m,
                                                      const float* __restrict__ x, double* __restrict__ u,
                                                      double* __restrict__ sq, int n, int t, int H) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long gr = (long long)blockIdx.x * 8 + warp;
  if (gr >= (long long)H * n) return;
  const int b = (int)(gr / n);
  const float* p = Phi + gr * t;
  const float* xb = x + (long long)b * t;
  double a = 0.0, q = 0.0;
  for (int r = lane; r < t; r += 32) {
    const double v = p[r];
    a = fma(v, (double)xb[r], a);
    if (sq) q = fma(v, v, q);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    a += __shfl_xor_sync(0xffffffffu, a, o);
    q += __shfl_xor_sync(0xffffffffu, q, o);
  }
  if (lane == 0) {
    u[gr] = (double)m[gr] - a;
    if (sq) sq[gr] = q;
  }
}

// lam[b] = ridge * sum_i sq[b][i] / t, summed in a fixed order (one CTA per head).
__global__ void __launch_bounds__(256) ir_lambda_kernel(const double* __restrict__ sq, double* __restrict__ lam, int n,
                                                        int t, double ridge) {
  __shared__ double red[8];
  const int b = blockIdx.x;
  double a = 0.0;
  for (int i = threadIdx.x; i < n; i += 256) a += sq[(long long)b * n + i];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(0xffffffffu, a, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = a;
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int w = 0; w < 8; ++w) s += red[w];
    lam[b] = ridge * s / t;
  }
}

// r[b][c] = sum_i Phi_ic u_i - lam x_c (fp64 sums, rounded to fp32 at the end).
// A CTA takes 32 columns (lane = column, coalesced rows) and its 8 warps
// split the rows, each with four independent partial sums; the warps' sums
// are added in warp order.
__global__ void __launch_bounds__(256) ir_cols_kernel(const float* __restrict__ Phi, const double* __restrict__ u,
                                                      const float* __restrict__ x, const double* __restrict__ lam,
                                                      float* __restrict__ r, int n, int t) {
  __shared__ double part[8][32];
  const int b = blockIdx.y, lane = threadIdx.x & 31, warp = threadIdx.x >> 5, c = blockIdx.x * 32 + lane;
  const float* p = Phi + (long long)b * n * t + c;
  const double* ub = u + (long long)b * n;
  double a0 = 0.0, a1 = 0.0, a2 = 0.0, a3 = 0.0;
  if (c < t) {
    int i = warp;
    for (; i + 24 < n; i += 32) {
      a0 = fma((double)p[(long long)i * t], ub[i], a0);
      a1 = fma((double)p[(long long)(i + 8) * t], ub[i + 8], a1);
      a2 = fma((double)p[(long long)(i + 16) * t], ub[i + 16], a2);
      a3 = fma((double)p[(long long)(i + 24) * t], ub[i + 24], a3);
    }
    for (; i < n; i += 8) a0 = fma((double)p[(long long)i * t], ub[i], a0);
  }
  part[warp][lane] = (a0 + a1) + (a2 + a3);
  __syncthreads();
  if (warp == 0 && c < t) {
    double a = part[0][lane];
#pragma unroll
    for (int w = 1; w < 8; ++w) a += part[w][lane];
    r[(long long)b * t + c] = (float)(a - lam[b] * (double)x[(long long)b * t + c]);
  }
}

// x += (L L^T)^-1 r for one head per CTA (512 threads): forward substitution
// y_k = Linv_kk (r_k - sum_{j<k} L_kj y_j), then x_k += Linv_kk^T (y_k -
// sum_{j>k} L_jk^T d_j).  y and the correction d live in `yd` ([H][t]).
// Used by the refinement steps of the primal beta solve.
template <typename R>
__global__ void __launch_bounds__(512) tri_solve_kernel(const R* __restrict__ A, const R* __restrict__ Linv,
                                                        const R* __restrict__ r, R* __restrict__ yd,
                                                        R* __restrict__ x, int t) {
  constexpr int NBk = kCholNB;
  __shared__ R v[NBk];
  __shared__ R part[8][NBk];
  const int b = blockIdx.x, tid = threadIdx.x;
  const int nblk = (t + NBk - 1) / NBk;
  const R* Ab = A + (long long)b * t * t;
  const R* Lb = Linv + (long long)b * nblk * NBk * NBk;
  const R* rb = r + (long long)b * t;
  R* y = yd + (long long)b * t;
  R* xb = x + (long long)b * t;
  // forward: 8 threads per row of block k sum L_kj y_j over the columns before k0
  for (int k = 0; k < nblk; ++k) {
    const int k0 = k * NBk, kb = min(NBk, t - k0);
    {
      const int rr = tid >> 3, pt = tid & 7;
      R a = R(0), a2 = R(0), a3 = R(0), a4 = R(0);
      if (rr < kb) {
        const R* row = Ab + (long long)(k0 + rr) * t;
        int c = pt;
        for (; c + 24 < k0; c += 32) {   // four independent chains: eight loads in flight together
          const R l0 = __ldcg(row + c), l1 = __ldcg(row + c + 8), l2 = __ldcg(row + c + 16), l3 = __ldcg(row + c + 24);
          const R y0 = __ldcg(y + c), y1 = __ldcg(y + c + 8), y2 = __ldcg(y + c + 16), y3 = __ldcg(y + c + 24);
          a = fma_r(l0, y0, a);
          a2 = fma_r(l1, y1, a2);
          a3 = fma_r(l2, y2, a3);
          a4 = fma_r(l3, y3, a4);
        }
        for (; c < k0; c += 8) a = fma_r(__ldcg(row + c), __ldcg(y + c), a);
      }
      a = (a + a2) + (a3 + a4);
      a += __shfl_xor_sync(0xffffffffu, a, 1);
      a += __shfl_xor_sync(0xffffffffu, a, 2);
      a += __shfl_xor_sync(0xffffffffu, a, 4);
      if (pt == 0) v[rr] = rr < kb ? rb[k0 + rr] - a : R(0);
    }
    __syncthreads();
    {  // y_k[c] = sum_{l <= c} Linv_k[c][l] v[l]
      const int c = tid >> 3, pt = tid & 7;
      const R* Li = Lb + (long long)k * NBk * NBk + c * NBk;
      R a = R(0);
      for (int l = pt; l <= c; l += 8) a = fma_r(__ldcg(Li + l), v[l], a);
      a += __shfl_xor_sync(0xffffffffu, a, 1);
      a += __shfl_xor_sync(0xffffffffu, a, 2);
      a += __shfl_xor_sync(0xffffffffu, a, 4);
      if (pt == 0 && c < kb) y[k0 + c] = a;
    }
    __threadfence_block();
    __syncthreads();
  }
  // backward: column c of block k, eight row parts; the correction d
  // overwrites y block by block (rows after k0 + kb already hold d)
  for (int k = nblk - 1; k >= 0; --k) {
    const int k0 = k * NBk, kb = min(NBk, t - k0);
    {
      const int c = tid & (NBk - 1), pt = tid >> 6;
      R a = R(0), a2 = R(0), a3 = R(0), a4 = R(0);
      if (c < kb) {
        const R* col = Ab + k0 + c;
        int rr = k0 + kb + pt;
        for (; rr + 24 < t; rr += 32) {
          const R l0 = __ldcg(col + (long long)rr * t), l1 = __ldcg(col + (long long)(rr + 8) * t);
          const R l2 = __ldcg(col + (long long)(rr + 16) * t), l3 = __ldcg(col + (long long)(rr + 24) * t);
          const R y0 = __ldcg(y + rr), y1 = __ldcg(y + rr + 8), y2 = __ldcg(y + rr + 16), y3 = __ldcg(y + rr + 24);
          a = fma_r(l0, y0, a);
          a2 = fma_r(l1, y1, a2);
          a3 = fma_r(l2, y2, a3);
          a4 = fma_r(l3, y3, a4);
        }
        for (; rr < t; rr += 8) a = fma_r(__ldcg(col + (long long)rr * t), __ldcg(y + rr), a);
      }
      part[pt][c] = (a + a2) + (a3 + a4);
    }
    __syncthreads();
    if (tid < NBk) {
      R a = R(0);
#pragma unroll
      for (int q = 0; q < 8; ++q) a += part[q][tid];
      v[tid] = tid < kb ? y[k0 + tid] - a : R(0);
    }
    __syncthreads();
    {  // d_k[c] = sum_{l >= c} Linv_k[l][c] v[l]
      const int c = tid >> 3, pt = tid & 7;
      const R* Li = Lb + (long long)k * NBk * NBk;
      R a = R(0);
      for (int l = c + pt; l < NBk; l += 8) a = fma_r(__ldcg(Li + (long long)l * NBk + c), v[l], a);
      a += __shfl_xor_sync(0xffffffffu, a, 1);
      a += __shfl_xor_sync(0xffffffffu, a, 2);
      a += __shfl_xor_sync(0xffffffffu, a, 4);
      if (pt == 0 && c < kb) {
        y[k0 + c] = a;
        xb[k0 + c] += a;
      }
    }
    __threadfence_block();
    __syncthreads();
  }
}

constexpr int kBetaRefineSteps = 2;

static int refine_beta(const Dims& D, float ridge_w, const float* m, const FitBufs& B, cudaStream_t st) {
  const long long hn = (long long)D.H * D.n;
  ir_rows_kernel<<<cdiv(hn, 8), 256, 0, st>>>(B.Phi, m, B.wsol, B.ir_u, B.ir_sq, D.n, D.t, D.H);
  ir_lambda_kernel<<<D.H, 256, 0, st>>>(B.ir_sq, B.ir_lam, D.n, D.t, (double)ridge_w);
  int nl = 2;
  for (int it = 0; it < kBetaRefineSteps; ++it) {
    if (it > 0) {
      ir_rows_kernel<<<cdiv(hn, 8), 256, 0, st>>>(B.Phi, m, B.wsol, B.ir_u, nullptr, D.n, D.t, D.H);
      ++nl;
    }
    ir_cols_kernel<<<dim3(cdiv(D.t, 32), D.H), 256, 0, st>>>(B.Phi, B.ir_u, B.wsol, B.ir_lam, B.rhs, D.n, D.t);
    tri_solve_kernel<float><<<D.H, 512, 0, st>>>(B.Gram, B.Linv, B.rhs, B.Z, B.wsol, D.t);
    nl += 2;
  }
  return nl;
}

int launch_fits(const Dims& D, float scale, float ridge_w, float ridge_v, float eps_w, float b_min,
                float b_max, const bf16* Q, const float* C_k, const float* z, const float* m,
                const float* Y, const FitBufs& B, float* beta, float* C_v, DevStatus* stt, cudaStream_t st,
                cudaEvent_t const* ev) {
  auto mark = [&](int s) {
    if (ev) cudaEventRecord(ev[s], st);
  };
  int nl = 0;
  const long long nt = (long long)D.n * D.t;
  // logits of the compact keys LC = scale Q C_k^T [n][t]: C_k enters as a bf16
  // triple, LC^T = C_k Q^T runs on the tensor cores and is stored transposed
  {
    const long long htd = (long long)D.H * D.t * D.d;
    bf16 *ck_h = B.ck3, *ck_m = B.ck3 + htd, *ck_l = B.ck3 + 2 * htd;
    nl += launch_split3(C_k, ck_h, ck_m, ck_l, htd, st);
    CUtensorMap mA, mA2, mA3, mB;
    if (!encode_bf16_map_3d(&mA, ck_h, D.d, D.t, D.H, 128) || !encode_bf16_map_3d(&mA2, ck_m, D.d, D.t, D.H, 128) ||
        !encode_bf16_map_3d(&mA3, ck_l, D.d, D.t, D.H, 128) || !encode_bf16_map_3d(&mB, Q, D.d, D.n, D.H, 128))
      return -1;
    if (launch_tc_gemm<128, kSplit3A>(mA, mB, mA2, mA, TcEpiStoreT{B.LC, nt, D.t, scale}, D.H, D.t, D.n, D.d, D.d,
                                      stt, st, 0, &mA3) != cudaSuccess)
      return -1;
    ++nl;
  }
  const long long cnt = (long long)D.H * nt;
  phi_kernel<<<stride_grid(cnt, 256, 16), 256, 0, st>>>(B.LC, z, B.Phi, D.n, D.t, cnt);
  ++nl;
  if (D.t > D.n) {
    const int nd = fits_dual(D, ridge_w, ridge_v, eps_w, b_min, b_max, m, Y, B, beta, C_v, stt, st, ev);
    return nd < 0 ? -1 : nl + nd;
  }
  // beta system: Gram = Phi_C^T Phi_C.  Its condition number reaches ~1e6 on
  // long caches, beyond what a split-bf16 pair (~1e-5 relative per entry)
  // resolves within tolerance: the operand enters as a bf16 triple and the
  // tensor-core Gram keeps every product term down to 2^-24 (kSplit3S).
  const int ldn = (D.n + 7) / 8 * 8;
  const dim3 tgrid(cdiv(D.t, 32), cdiv(ldn, 32), D.H);
  transpose_split3_kernel<<<tgrid, 256, 0, st>>>(B.Phi, D.n, D.t, B.PT_hi, B.PT_mid, B.PT_lo, ldn);
  if (gram3_tc(D.H, D.t, ldn, B.PT_hi, B.PT_mid, B.PT_lo, B.Gram, stt, st) < 0) return -1;
  nl += 2;
  mass_rhs_kernel<<<dim3(cdiv(D.t, 32), D.H), 1024, 0, st>>>(B.Phi, m, B.rhs, D.n, D.t);
  ++nl;
  mark(8);
  nl += cholesky_solve(D.H, D.t, B.Gram, B.Linv, B.rhs, B.Z, B.wsol, 1, 1, D.t, ridge_w, stt, st);
  nl += refine_beta(D, ridge_w, m, B, st);
  const long long ht = (long long)D.H * D.t;
  beta_kernel<<<cdiv(ht, 256), 256, 0, st>>>(B.wsol, beta, ht, eps_w, b_min, b_max);
  ++nl;
  // value system: P^ over the compact keys with the fitted bias; its Gram and
  // P^T Y on the tensor cores from transposed split-bf16 operands
  mark(9);
  softmax_bias_kernel<<<dim3(cdiv(D.n, 8), D.H), 256, 0, st>>>(B.LC, beta, B.Phi, D.n, D.t);
  ++nl;
  transpose_split_kernel<<<tgrid, 256, 0, st>>>(B.Phi, D.n, D.t, B.PT_hi, B.PT_lo, ldn);
  transpose_split_kernel<<<dim3(cdiv(D.d, 32), cdiv(ldn, 32), D.H), 256, 0, st>>>(Y, D.n, D.d, B.YT_hi, B.YT_lo,
                                                                                    ldn);
  nl += 2;
  if (gram_tc(D.H, D.t, D.t, ldn, B.PT_hi, B.PT_lo, B.PT_hi, B.PT_lo, B.Gram, D.t, stt, st) < 0) return -1;
  // R = P^T Y
  const long long td = (long long)D.t * D.d;
  if (gram_tc(D.H, D.t, D.d, ldn, B.PT_hi, B.PT_lo, B.YT_hi, B.YT_lo, B.R, D.d, stt, st) < 0) return -1;
  nl += 2;
  mark(10);
  nl += cholesky_solve(D.H, D.t, B.Gram, B.Linv, B.R, B.Z, C_v, D.d, D.d, td, ridge_v, stt, st);
  return nl;
}

__global__ void check_finite_kernel(const float* x, long long count, DevStatus* stt) {
  bool bad = false;
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < count;
       k += (long long)gridDim.x * blockDim.x)
    bad |= !isfinite(x[k]);
  if (__any_sync(0xffffffffu, bad) && (threadIdx.x & 31) == 0) set_status(stt, ARCKV_ERR_NONFINITE);
}

int launch_check_finite(const float* x, long long count, DevStatus* stt, cudaStream_t st) {
  check_finite_kernel<<<stride_grid(count, 256, 8), 256, 0, st>>>(x, count, stt);
  return 1;
}

// ---------------------------------------------------------------------------
// Compact attention (Sec. 3.1 Eq. compact_attention) on the tensor pipe:
//   X = scale Q C_k^T + 1 beta^T   (C_k as a bf16 triple against the exact bf16
//                                   queries; transposed store; beta added with
//                                   the row statistics)
//   O = softmax(X) C_v = sum_p softmax(X) C_v,p over the bf16 triple
//       (h, m, l) of C_v: three fused softmax-V products (fp32-grade
//       probabilities formed on the fly), added in a fixed order.

// x += beta over each row, then shift = max, mul = 1 / sum exp(x - shift); one
// warp per row of X [H][n][t].
__global__ void __launch_bounds__(256) bias_rowstats_kernel(float* X, const float* beta, float* shift, float* mul,
                                                            int n, int t) {
  const int b = blockIdx.y, row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= n) return;
  float* x = X + ((long long)b * n + row) * t;
  const float* be = beta + (long long)b * t;
  float mx = -INFINITY;
  for (int c = lane; c < t; c += 32) {
    const float v = x[c] + be[c];
    x[c] = v;
    mx = fmaxf(mx, v);
  }
  mx = warp_max(mx);
  float sm = 0.f;
  for (int c = lane; c < t; c += 32) sm += expf(x[c] - mx);
  sm = warp_sum(sm);
  if (lane == 0) {
    shift[(long long)b * n + row] = mx;
    mul[(long long)b * n + row] = 1.0f / sm;
  }
}

// O[e] = P0[e] + P1[e] + P2[e]
__global__ void sum3_kernel(const float* P, float* O, long long count) {
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < count;
       k += (long long)gridDim.x * blockDim.x)
    O[k] = (P[k] + P[count + k]) + P[2 * count + k];
}

AttendLayout attend_layout(int H, int n, int t) {
  AttendLayout L{};
  const size_t h = H, ldt = (size_t)(t + 7) / 8 * 8;
  size_t o = 0;
  auto take = [&](size_t bytes) { const size_t r = o; o += (bytes + 255) / 256 * 256; return r; };
  L.status = take(256);
  L.X = take(h * n * t * 4);
  L.shift = take(h * n * 4);
  L.mul = take(h * n * 4);
  L.ck3 = take(3 * h * t * 128 * 2);
  L.vt3 = take(3 * h * 128 * ldt * 2);
  L.parts = take(3 * h * n * 128 * 4);
  L.p3 = take(probs_fused(t) ? 0 : 3 * h * n * ldt * 2);
  L.total = o;
  return L;
}

int launch_attend(int H, int n, int t, float scale, const bf16* Q, const float* C_k, const float* beta,
                  const float* C_v, float* O, char* ws, DevStatus* stt, cudaStream_t st) {
  const AttendLayout L = attend_layout(H, n, t);
  const long long htd = (long long)H * t * 128, ldt = (t + 7) / 8 * 8;
  float* X = (float*)(ws + L.X);
  float* shift = (float*)(ws + L.shift);
  float* mul = (float*)(ws + L.mul);
  bf16* ck = (bf16*)(ws + L.ck3);
  bf16* vt = (bf16*)(ws + L.vt3);
  float* parts = (float*)(ws + L.parts);
  bf16* p3 = (bf16*)(ws + L.p3);
  int nl = launch_split3(C_k, ck, ck + htd, ck + 2 * htd, htd, st);
  {  // X^T = C_k Q^T, stored transposed as X [H][n][t] and scaled
    CUtensorMap mA, mA2, mA3, mB;
    if (!encode_bf16_map_3d(&mA, ck, 128, t, H, 128) || !encode_bf16_map_3d(&mA2, ck + htd, 128, t, H, 128) ||
        !encode_bf16_map_3d(&mA3, ck + 2 * htd, 128, t, H, 128) || !encode_bf16_map_3d(&mB, Q, 128, n, H, 128))
      return -1;
    if (launch_tc_gemm<128, kSplit3A>(mA, mB, mA2, mA, TcEpiStoreT{X, (long long)n * t, t, scale}, H, t, n, 128, 128,
                                      stt, st, 0, &mA3) != cudaSuccess)
      return -1;
    ++nl;
  }
  bias_rowstats_kernel<<<dim3(cdiv(n, 8), H), 256, 0, st>>>(X, beta, shift, mul, n, t);
  // C_v^T as a bf16 triple [H][128][ldt] (zero pad)
  transpose_split3_kernel<<<dim3(cdiv(128, 32), cdiv(ldt, 32), H), 256, 0, st>>>(
      C_v, t, 128, vt, vt + (long long)H * 128 * ldt, vt + 2LL * H * 128 * ldt, (int)ldt);
  nl += 2;
  Dims D{};
  D.H = H;
  D.n = n;
  D.T = t;
  D.d = 128;
  const long long hnd = (long long)H * n * 128, pl = (long long)H * n * ldt;
  for (int p = 0; p < 3; ++p) {
    const int r = launch_probs_v_tc(D, X, shift, mul, p3, p3 + pl, p3 + 2 * pl, vt + p * (long long)H * 128 * ldt,
                                    parts + p * hnd, stt, st);
    if (r < 0) return -1;
    nl += r;
  }
  sum3_kernel<<<stride_grid(hnd, 256, 8), 256, 0, st>>>(parts, O, hnd);
  return nl + 1;
}

}  // namespace arckv
