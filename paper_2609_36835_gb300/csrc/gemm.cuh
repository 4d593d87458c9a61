// Register-tiled fp32 SIMT GEMM template used by the dense stages.
//
//   C[b](m, n) = sum_{k in [kb, ke)} A[b](m, k) * B[b](n, k)
//
// A CTA of 256 threads owns a 128 x 128 tile of C; each thread accumulates an
// 8 x 8 register micro-tile (rows ty*4 + {0..3} and 64 + ty*4 + {0..3},
// columns tx*4 + {0..3} and 64 + tx*4 + {0..3}).  K is walked in slabs of 16,
// double-buffered through registers into K-major shared tiles.  Operands are
// described by small loader structs (row-K, column-K) that convert bf16 or
// fp32 inputs to fp32 on the fly and zero-fill every element outside
// [0, M|N) x [kb, ke).
#pragma once
#include "common.cuh"

namespace arckv {

constexpr int GBM = 128, GBN = 128, GBK = 16, GNT = 256, GSST = GBM + 4;

// Row-K operand: element (r, k) = p[b * bs + r * ld + k].
template <typename T>
struct RowK {
  const T* p;
  long long bs;
  int ld;
  const T* base;
  int r0, R;
  bool vec;
  __device__ __forceinline__ void bind(int b, int r0_, int R_) {
    base = p + (long long)b * bs;
    r0 = r0_;
    R = R_;
    const int align = 16 / (int)sizeof(T);
    vec = ((ld % align) == 0) && ((bs % align) == 0) && (((uintptr_t)p & 15) == 0);
  }
  // thread piece: row r0 + (tid & 127), k = k0 + (tid >> 7) * 8 + q, q < 8
  __device__ __forceinline__ void fetch(int k0, int kend, float (&v)[8]) const {
    const int r = r0 + (threadIdx.x & 127);
    const int k = k0 + (threadIdx.x >> 7) * 8;
    const T* src = base + (long long)r * ld + k;
    if (r < R && k + 8 <= kend && vec) {
      if (sizeof(T) == 4) {
        float4 x0 = *(const float4*)(src), x1 = *(const float4*)(src + 4);
        v[0] = x0.x; v[1] = x0.y; v[2] = x0.z; v[3] = x0.w;
        v[4] = x1.x; v[5] = x1.y; v[6] = x1.z; v[7] = x1.w;
      } else {
        uint4 x = *(const uint4*)(src);
        const bf16* h = (const bf16*)&x;
#pragma unroll
        for (int q = 0; q < 8; ++q) v[q] = to_f32(h[q]);
      }
    } else {
#pragma unroll
      for (int q = 0; q < 8; ++q) v[q] = (r < R && k + q < kend) ? to_f32(src[q]) : 0.f;
    }
  }
  __device__ __forceinline__ int row() const { return r0 + (threadIdx.x & 127); }
  __device__ __forceinline__ void store(float* S, const float (&v)[8]) const {
    const int r = threadIdx.x & 127, kq = (threadIdx.x >> 7) * 8;
#pragma unroll
    for (int q = 0; q < 8; ++q) S[(kq + q) * GSST + r] = v[q];
  }
};

// Column-K operand: element (r, k) = p[b * bs + k * ld + r].
template <typename T>
struct ColK {
  const T* p;
  long long bs;
  int ld;
  const T* base;
  int r0, R;
  bool vec;
  __device__ __forceinline__ void bind(int b, int r0_, int R_) {
    base = p + (long long)b * bs;
    r0 = r0_;
    R = R_;
    const int align = 16 / (int)sizeof(T);
    vec = ((ld % align) == 0) && ((bs % align) == 0) && (((uintptr_t)p & 15) == 0);
  }
  // thread piece: k = k0 + (tid >> 4), r = r0 + (tid & 15) * 8 + q
  __device__ __forceinline__ void fetch(int k0, int kend, float (&v)[8]) const {
    const int k = k0 + (threadIdx.x >> 4);
    const int r = r0 + (threadIdx.x & 15) * 8;
    const T* src = base + (long long)k * ld + r;
    if (k < kend && r + 8 <= R && vec) {
      if (sizeof(T) == 4) {
        float4 x0 = *(const float4*)(src), x1 = *(const float4*)(src + 4);
        v[0] = x0.x; v[1] = x0.y; v[2] = x0.z; v[3] = x0.w;
        v[4] = x1.x; v[5] = x1.y; v[6] = x1.z; v[7] = x1.w;
      } else {
        uint4 x = *(const uint4*)(src);
        const bf16* h = (const bf16*)&x;
#pragma unroll
        for (int q = 0; q < 8; ++q) v[q] = to_f32(h[q]);
      }
    } else {
#pragma unroll
      for (int q = 0; q < 8; ++q) v[q] = (k < kend && r + q < R) ? to_f32(src[q]) : 0.f;
    }
  }
  __device__ __forceinline__ void store(float* S, const float (&v)[8]) const {
    float* d = S + (threadIdx.x >> 4) * GSST + (threadIdx.x & 15) * 8;
    *(float4*)d = make_float4(v[0], v[1], v[2], v[3]);
    *(float4*)(d + 4) = make_float4(v[4], v[5], v[6], v[7]);
  }
};

__device__ __forceinline__ int tile_row(int i) { return (threadIdx.x >> 4) * 4 + (i & 3) + (i >> 2) * 64; }

template <class LA, class LB>
__device__ __forceinline__ void gemm_mainloop(LA& la, LB& lb, int kb, int ke, float (&acc)[8][8],
                                              float* sA, float* sB) {
  if (kb >= ke) return;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float ra[8], rb[8];
  la.fetch(kb, ke, ra);
  lb.fetch(kb, ke, rb);
  la.store(sA, ra);
  lb.store(sB, rb);
  __syncthreads();
  int buf = 0;
  for (int k0 = kb; k0 < ke; k0 += GBK) {
    const bool more = k0 + GBK < ke;
    if (more) {
      la.fetch(k0 + GBK, ke, ra);
      lb.fetch(k0 + GBK, ke, rb);
    }
    const float* A = sA + buf * GBK * GSST;
    const float* B = sB + buf * GBK * GSST;
#pragma unroll
    for (int kk = 0; kk < GBK; ++kk) {
      const float4 a0 = *(const float4*)(A + kk * GSST + ty * 4);
      const float4 a1 = *(const float4*)(A + kk * GSST + 64 + ty * 4);
      const float4 b0 = *(const float4*)(B + kk * GSST + tx * 4);
      const float4 b1 = *(const float4*)(B + kk * GSST + 64 + tx * 4);
      const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    if (more) {
      la.store(sA + (buf ^ 1) * GBK * GSST, ra);
      lb.store(sB + (buf ^ 1) * GBK * GSST, rb);
    }
    __syncthreads();
    buf ^= 1;
  }
}

// ------------------------------------------------------------- epilogues

// C[b * cbs + sp * sbs + m * ldc + n] = alpha * acc (sp = split-K slice).
// With `sym`, an off-diagonal tile is also written transposed (lower-tile
// launches of a symmetric product).
struct EpiStore {
  float* C;
  long long cbs, sbs;
  int ldc;
  float alpha;
  bool sym;
  __device__ __forceinline__ void apply(int b, int sp, int m0, int n0, int M, int N, float (&acc)[8][8],
                                        float*) const {
    float* base = C + (long long)b * cbs + (long long)sp * sbs;
    const bool vec = ((ldc & 3) == 0) && ((((uintptr_t)base) & 15) == 0);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int m = m0 + tile_row(i);
      if (m >= M) continue;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int n = n0 + (threadIdx.x & 15) * 4 + h * 64;
        float* dst = base + (long long)m * ldc + n;
        const float v0 = alpha * acc[i][h * 4 + 0], v1 = alpha * acc[i][h * 4 + 1];
        const float v2 = alpha * acc[i][h * 4 + 2], v3 = alpha * acc[i][h * 4 + 3];
        if (vec && n + 4 <= N) {
          *(float4*)dst = make_float4(v0, v1, v2, v3);
        } else {
          if (n + 0 < N) dst[0] = v0;
          if (n + 1 < N) dst[1] = v1;
          if (n + 2 < N) dst[2] = v2;
          if (n + 3 < N) dst[3] = v3;
        }
        if (sym && m0 != n0) {
          const float vv[4] = {v0, v1, v2, v3};
#pragma unroll
          for (int q = 0; q < 4; ++q)
            if (n + q < N) base[(long long)(n + q) * ldc + m] = vv[q];
        }
      }
    }
  }
};

template <class LA, class LB, class EPI, bool LOWER>
__global__ void __launch_bounds__(GNT) gemm_kernel(LA la, LB lb, EPI epi, int M, int N, int K, int splits) {
  __shared__ __align__(16) float sA[2 * GBK * GSST];
  __shared__ __align__(16) float sB[2 * GBK * GSST];
  const int z = blockIdx.z, b = z / splits, sp = z - b * splits;
  const int m0 = blockIdx.y * GBM, n0 = blockIdx.x * GBN;
  if (LOWER && n0 > m0) return;
  const int kper = ((K + splits - 1) / splits + GBK - 1) / GBK * GBK;
  const int kb = sp * kper, ke = min(K, kb + kper);
  la.bind(b, m0, M);
  lb.bind(b, n0, N);
  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
  gemm_mainloop(la, lb, kb, ke, acc, sA, sB);
  epi.apply(b, sp, m0, n0, M, N, acc, sA);
}

template <bool LOWER = false, class LA, class LB, class EPI>
inline void launch_gemm(const LA& la, const LB& lb, const EPI& epi, int H, int M, int N, int K, int splits,
                        cudaStream_t st) {
  dim3 grid(cdiv(N, GBN), cdiv(M, GBM), H * splits);
  gemm_kernel<LA, LB, EPI, LOWER><<<grid, GNT, 0, st>>>(la, lb, epi, M, N, K, splits);
}

}  // namespace arckv
