// Attention over a compact block followed by an uncompressed block (App. A.7
// Eq. concatenated_attention_preservation):
//
//   O_i = sum_j e^{a_ij} v_j / sum_j e^{a_ij},   a_ij = scale q_i.k_j + b_j,
//   k, v, b = [C_k; K_fixed], [C_v; V_fixed], [beta; 0_F]
//
// for H independent heads of n query rows (a decode batch folds into H).
// The operation streams every key and value once and does ~2 FMA per byte of
// bf16 cache: it is HBM-bound, so it runs on the SIMT pipes as a split-key
// ("flash-decoding") pass, not as a GEMM:
//   attend_split_kernel: CTA (key split, 4-row block, head); per 64-key tile
//     - logits: thread (key tid/4, 32-dim quarter tid%4) loads its slice of the
//       key straight from HBM (16-byte vectors, a warp reads 8 whole rows),
//       dots it with the 4 query rows held in shared memory, and the 4
//       quarters are combined with two shuffles;
//     - online softmax per row (running max m, running sum l);
//     - values: warp w takes keys w, w+8, ... of the tile, lane l dims
//       4l..4l+3, so a warp reads whole value rows; the accumulators are
//       rescaled by e^{m_old - m_new};
//   attend_combine_kernel: per (head, row) merges the splits' (m, l, o).
// t = 0 gives plain attention over the uncompressed block (the full-cache
// baseline of the decode measurement); F = 0 the compact operator of Sec. 3.1.
//
// bf16 caches (both blocks bf16) take attend_bulk_kernel instead: one thread
// streams each 64-key tile of K and V (16 KB each, contiguous rows) into a
// 3-stage shared-memory ring with cp.async.bulk, so that every CTA keeps up
// to 64 KB in flight, and the warps read the tiles two keys per instruction
// (512 contiguous bytes: no bank conflicts).  Lane l holds query dims
// 8 (l%16) .. +7 of the 4 rows in registers; the 16 partial dot products of a
// lane (4 keys x 4 rows) are summed over the 16 lanes of each half-warp by a
// transposing butterfly (15 shuffles).
#include <algorithm>

#include "kernels.h"
#include "tc.cuh"

namespace arckv {

constexpr int kJR = 4;        // query rows per CTA
constexpr int kJTile = 64;    // keys per tile
constexpr int kJThreads = 256;

__device__ __forceinline__ void load32(const float* p, float (&x)[32]) {
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const float4 v = __ldg((const float4*)p + q);
    x[4 * q] = v.x; x[4 * q + 1] = v.y; x[4 * q + 2] = v.z; x[4 * q + 3] = v.w;
  }
}
__device__ __forceinline__ void load32(const bf16* p, float (&x)[32]) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint4 v = __ldg((const uint4*)p + q);
    const __nv_bfloat162* h = (const __nv_bfloat162*)&v;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 f = __bfloat1622float2(h[e]);
      x[8 * q + 2 * e] = f.x;
      x[8 * q + 2 * e + 1] = f.y;
    }
  }
}
__device__ __forceinline__ void load4(const float* p, float (&x)[4]) {
  const float4 v = __ldg((const float4*)p);
  x[0] = v.x; x[1] = v.y; x[2] = v.z; x[3] = v.w;
}
__device__ __forceinline__ void load4(const bf16* p, float (&x)[4]) {
  const uint2 v = __ldg((const uint2*)p);
  const float2 a = __bfloat1622float2(*(const __nv_bfloat162*)&v.x), b = __bfloat1622float2(*(const __nv_bfloat162*)&v.y);
  x[0] = a.x; x[1] = a.y; x[2] = b.x; x[3] = b.y;
}

// sum_q qv[q] k[q] over a 32-dim slice held as loaded (fp32, or packed bf16 pairs)
struct KSlice32F {
  float x[32];
  __device__ __forceinline__ void load(const float* p) { load32(p, x); }
  __device__ __forceinline__ void zero() {
#pragma unroll
    for (int q = 0; q < 32; ++q) x[q] = 0.f;
  }
  __device__ __forceinline__ float dot(const float4* qv) const {
    float a = 0.f;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const float4 y = qv[q];
      a = fmaf(y.x, x[4 * q], a);
      a = fmaf(y.y, x[4 * q + 1], a);
      a = fmaf(y.z, x[4 * q + 2], a);
      a = fmaf(y.w, x[4 * q + 3], a);
    }
    return a;
  }
};
struct KSlice32H {
  uint4 x[4];
  __device__ __forceinline__ void load(const bf16* p) {
#pragma unroll
    for (int q = 0; q < 4; ++q) x[q] = __ldg((const uint4*)p + q);
  }
  __device__ __forceinline__ void zero() {
#pragma unroll
    for (int q = 0; q < 4; ++q) x[q] = make_uint4(0u, 0u, 0u, 0u);
  }
  __device__ __forceinline__ float dot(const float4* qv) const {
    float a = 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const __nv_bfloat162* h = (const __nv_bfloat162*)&x[q];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const float2 f0 = __bfloat1622float2(h[2 * e]), f1 = __bfloat1622float2(h[2 * e + 1]);
        const float4 y = qv[2 * q + e];
        a = fmaf(y.x, f0.x, a);
        a = fmaf(y.y, f0.y, a);
        a = fmaf(y.z, f1.x, a);
        a = fmaf(y.w, f1.y, a);
      }
    }
    return a;
  }
};
template <typename TC> struct KSliceOf { using type = KSlice32F; };
template <> struct KSliceOf<bf16> { using type = KSlice32H; };

// The tiles of keys [jlo, jhi) of one block: key j is row j - koff of Kb / Vb,
// with bias[j] (bias == nullptr: zero).  Updates the running (m, l) in sM / sL
// and the per-thread accumulators acc.
template <typename KT>
__device__ __forceinline__ void attend_tiles(const KT* Kb, const KT* Vb, const float* bias, int jlo, int jhi,
                                             int koff, float (*sQ)[128], float (*sP)[kJTile], float* sM, float* sL,
                                             float* sF, float (&acc)[kJR][4]) {
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  for (int j0 = jlo; j0 < jhi; j0 += kJTile) {
    {  // logits of the tile
      const int jj = tid >> 2, p = tid & 3, j = j0 + jj;
      typename KSliceOf<KT>::type k;
      if (j < jhi) k.load(Kb + (long long)(j - koff) * 128 + p * 32);
      else k.zero();
      float part[kJR];
#pragma unroll
      for (int r = 0; r < kJR; ++r) {
        float a = k.dot((const float4*)&sQ[r][p * 32]);
        a += __shfl_xor_sync(0xffffffffu, a, 1);
        a += __shfl_xor_sync(0xffffffffu, a, 2);
        part[r] = a;
      }
      if (p == 0) {
        const float b = (j < jhi && bias) ? __ldg(bias + j) : 0.f;
#pragma unroll
        for (int r = 0; r < kJR; ++r) sP[r][jj] = (j < jhi) ? part[r] + b : -INFINITY;
      }
    }
    __syncthreads();
    if (w < kJR) {  // online softmax of row w over the tile (at least one key is valid)
      const float a0 = sP[w][lane], a1 = sP[w][lane + 32];
      const float mold = sM[w], mnew = fmaxf(mold, warp_max(fmaxf(a0, a1)));
      const float e0 = expf(a0 - mnew), e1 = expf(a1 - mnew);
      sP[w][lane] = e0;
      sP[w][lane + 32] = e1;
      const float ssum = warp_sum(e0 + e1);
      if (lane == 0) {
        const float f = expf(mold - mnew);   // 0 on the first tile (mold = -inf)
        sF[w] = f;
        sL[w] = sL[w] * f + ssum;
        sM[w] = mnew;
      }
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < kJR; ++r) {
      const float f = sF[r];
#pragma unroll
      for (int q = 0; q < 4; ++q) acc[r][q] *= f;
    }
#pragma unroll 4
    for (int i = 0; i < kJTile / 8; ++i) {
      const int jj = w + 8 * i, j = j0 + jj;
      if (j < jhi) {
        float v[4];
        load4(Vb + (long long)(j - koff) * 128 + lane * 4, v);
#pragma unroll
        for (int r = 0; r < kJR; ++r) {
          const float pr = sP[r][jj];
#pragma unroll
          for (int q = 0; q < 4; ++q) acc[r][q] = fmaf(pr, v[q], acc[r][q]);
        }
      }
    }
    __syncthreads();
  }
}

// Partial results of key split sp: Opart[h][sp][i][:] = sum_j e^{a_ij - m} v_j
// (unnormalised) and ml[h][sp][i] = (m, l = sum_j e^{a_ij - m}).  The split's
// key range is cut at t so that every tile holds one block's keys.
template <typename TC>
__global__ void __launch_bounds__(kJThreads, 3) attend_split_kernel(const bf16* Q, int n, const TC* Ck, const float* beta,
                                                                    const TC* Cv, int t, const bf16* Kf, const bf16* Vf,
                                                                    int F, float scale, int per_split, int nsplit,
                                                                    float* Opart, float2* ml) {
  const int h = blockIdx.z, r0 = blockIdx.y * kJR, sp = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const int L = t + F, jb = sp * per_split, je = min(L, jb + per_split);
  __shared__ __align__(16) float sQ[kJR][128];
  __shared__ float sP[kJR][kJTile];
  __shared__ float sM[kJR], sL[kJR], sF[kJR];
  __shared__ __align__(16) float sAcc[kJThreads / 32][kJR][128];
  for (int e = tid; e < kJR * 128; e += kJThreads) {
    const int r = e >> 7, dd = e & 127;
    sQ[r][dd] = (r0 + r < n) ? scale * __bfloat162float(Q[((long long)h * n + r0 + r) * 128 + dd]) : 0.f;
  }
  if (tid < kJR) {
    sM[tid] = -INFINITY;
    sL[tid] = 0.f;
  }
  float acc[kJR][4];
#pragma unroll
  for (int r = 0; r < kJR; ++r)
#pragma unroll
    for (int q = 0; q < 4; ++q) acc[r][q] = 0.f;
  __syncthreads();
  if (jb < t)
    attend_tiles<TC>(Ck + (long long)h * t * 128, Cv + (long long)h * t * 128, beta + (long long)h * t, jb,
                     min(je, t), 0, sQ, sP, sM, sL, sF, acc);
  if (je > t)
    attend_tiles<bf16>(Kf + (long long)h * F * 128, Vf + (long long)h * F * 128, nullptr, max(jb, t), je, t, sQ, sP,
                       sM, sL, sF, acc);
#pragma unroll
  for (int r = 0; r < kJR; ++r) *(float4*)&sAcc[w][r][lane * 4] = make_float4(acc[r][0], acc[r][1], acc[r][2], acc[r][3]);
  __syncthreads();
  for (int e = tid; e < kJR * 128; e += kJThreads) {
    const int r = e >> 7, dd = e & 127;
    if (r0 + r >= n) continue;
    float o = 0.f;
#pragma unroll
    for (int q = 0; q < kJThreads / 32; ++q) o += sAcc[q][r][dd];
    const long long row = ((long long)h * nsplit + sp) * n + r0 + r;
    Opart[row * 128 + dd] = o;
    if (dd == 0) ml[row] = make_float2(sM[r], sL[r]);
  }
}

constexpr int kBStages = 3;
constexpr int kBTileBytes = kJTile * 128 * 2;   // one bf16 tile of K (or V)

// Partial results of key split sp as in attend_split_kernel, for bf16 blocks.
__global__ void __launch_bounds__(kJThreads, 2) attend_bulk_kernel(const bf16* Q, int n, const bf16* Ck,
                                                                   const float* beta, const bf16* Cv, int t,
                                                                   const bf16* Kf, const bf16* Vf, int F, float scale,
                                                                   int per_split, int nsplit, float* Opart,
                                                                   float2* ml, DevStatus* stt) {
  extern __shared__ __align__(128) unsigned char smraw[];
  bf16* sK = (bf16*)smraw;                                       // [stage][64][128]
  bf16* sV = (bf16*)(smraw + kBStages * kBTileBytes);            // [stage][64][128]
  __shared__ __align__(8) uint64_t bar[kBStages];
  __shared__ float sP[kJR][kJTile];
  __shared__ float sM[kJR], sL[kJR], sF[kJR];
  __shared__ int abort_flag;
  const int h = blockIdx.z, r0 = blockIdx.y * kJR, sp = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5, hl = lane & 15, hh = lane >> 4;
  const int L = t + F, jb = sp * per_split, je = min(L, jb + per_split);
  // tiles: the compact keys [jb, min(je, t)) then the uncompressed ones [max(jb, t), je)
  const int c_lo = jb, c_hi = min(je, t), f_lo = max(jb, t), f_hi = je;
  const int n1 = c_hi > c_lo ? (c_hi - c_lo + kJTile - 1) / kJTile : 0;
  const int ntile = n1 + (f_hi > f_lo ? (f_hi - f_lo + kJTile - 1) / kJTile : 0);
  const bf16* Ckh = Ck + (long long)h * t * 128;
  const bf16* Cvh = Cv + (long long)h * t * 128;
  const bf16* Kfh = Kf + (long long)h * F * 128;
  const bf16* Vfh = Vf + (long long)h * F * 128;
  const float* bh = beta + (long long)h * t;
  // tile i -> (first key j0, keys nk, compact?)
  auto tile_of = [&](int i, int& j0, int& nk, bool& comp) {
    comp = i < n1;
    j0 = comp ? c_lo + i * kJTile : f_lo + (i - n1) * kJTile;
    nk = min(kJTile, (comp ? c_hi : f_hi) - j0);
  };
  auto issue = [&](int i) {   // one thread: both tiles of tile i into stage i % S
    int j0, nk;
    bool comp;
    tile_of(i, j0, nk, comp);
    const int s = i % kBStages;
    const uint32_t bytes = (uint32_t)nk * 256u;
    tc::mbar_arrive_expect_tx(&bar[s], 2 * bytes);
    const long long row = comp ? j0 : (long long)(j0 - t);
    tc::bulk_load(sK + (size_t)s * kJTile * 128, (comp ? Ckh : Kfh) + row * 128, bytes, &bar[s]);
    tc::bulk_load(sV + (size_t)s * kJTile * 128, (comp ? Cvh : Vfh) + row * 128, bytes, &bar[s]);
  };
  if (tid == 0) {
    for (int s = 0; s < kBStages; ++s) tc::mbar_init(&bar[s], 1);
    tc::mbar_fence_init();
    abort_flag = 0;
  }
  if (tid < kJR) {
    sM[tid] = -INFINITY;
    sL[tid] = 0.f;
  }
  __syncthreads();
  if (tid == 0)
    for (int i = 0; i < min(kBStages, ntile); ++i) issue(i);
  // the 4 query rows at dims 8 hl .. 8 hl + 7, pre-scaled
  float q[kJR][8];
#pragma unroll
  for (int r = 0; r < kJR; ++r)
#pragma unroll
    for (int e = 0; e < 8; ++e)
      q[r][e] = (r0 + r < n) ? scale * __bfloat162float(Q[((long long)h * n + r0 + r) * 128 + hl * 8 + e]) : 0.f;
  float acc[kJR][8];
#pragma unroll
  for (int r = 0; r < kJR; ++r)
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[r][e] = 0.f;
  int done = 0;   // tiles consumed
  for (int i = 0; i < ntile; ++i) {
    int j0, nk;
    bool comp;
    tile_of(i, j0, nk, comp);
    const int s = i % kBStages;
    const bool ok = tc::mbar_wait(&bar[s], (uint32_t)((i / kBStages) & 1), &abort_flag, stt);
    if (__syncthreads_or(!ok)) break;
    const bf16* Kt = sK + (size_t)s * kJTile * 128;
    const bf16* Vt = sV + (size_t)s * kJTile * 128;
    {  // logits: warp w takes keys 8w .. 8w+7, two per load (lane half hh)
      float v[16];
#pragma unroll
      for (int qq = 0; qq < 4; ++qq) {
        const int kk = 8 * w + 2 * qq + hh;
        const uint4 raw = *(const uint4*)(Kt + kk * 128 + hl * 8);
        const __nv_bfloat162* h2 = (const __nv_bfloat162*)&raw;
        float k8[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __bfloat1622float2(h2[e]);
          k8[2 * e] = f.x;
          k8[2 * e + 1] = f.y;
        }
#pragma unroll
        for (int r = 0; r < kJR; ++r) {
          float a = 0.f;
#pragma unroll
          for (int e = 0; e < 8; ++e) a = fmaf(q[r][e], k8[e], a);
          v[qq * 4 + r] = a;
        }
      }
      // transposing butterfly over the 16 lanes of the half-warp: lane hl ends
      // with the sum of entry hl (key 2 (hl >> 2) + hh of the warp, row hl & 3)
#pragma unroll
      for (int i8 = 0; i8 < 8; ++i8) {
        const bool up = hl & 8;
        const float mine = up ? v[8 + i8] : v[i8], other = up ? v[i8] : v[8 + i8];
        v[i8] = mine + __shfl_xor_sync(0xffffffffu, other, 8);
      }
#pragma unroll
      for (int i4 = 0; i4 < 4; ++i4) {
        const bool up = hl & 4;
        const float mine = up ? v[4 + i4] : v[i4], other = up ? v[i4] : v[4 + i4];
        v[i4] = mine + __shfl_xor_sync(0xffffffffu, other, 4);
      }
#pragma unroll
      for (int i2 = 0; i2 < 2; ++i2) {
        const bool up = hl & 2;
        const float mine = up ? v[2 + i2] : v[i2], other = up ? v[i2] : v[2 + i2];
        v[i2] = mine + __shfl_xor_sync(0xffffffffu, other, 2);
      }
      {
        const bool up = hl & 1;
        const float mine = up ? v[1] : v[0], other = up ? v[0] : v[1];
        v[0] = mine + __shfl_xor_sync(0xffffffffu, other, 1);
      }
      const int kk = 8 * w + 2 * (hl >> 2) + hh, r = hl & 3;
      const bool valid = kk < nk;
      const float b = (valid && comp) ? __ldg(bh + j0 + kk) : 0.f;
      sP[r][kk] = valid ? v[0] + b : -INFINITY;
    }
    __syncthreads();
    if (w < kJR) {  // online softmax of row w over the tile (at least one key is valid)
      const float a0 = sP[w][lane], a1 = sP[w][lane + 32];
      const float mold = sM[w], mnew = fmaxf(mold, warp_max(fmaxf(a0, a1)));
      const float e0 = expf(a0 - mnew), e1 = expf(a1 - mnew);
      sP[w][lane] = e0;
      sP[w][lane + 32] = e1;
      const float ssum = warp_sum(e0 + e1);
      if (lane == 0) {
        const float f = expf(mold - mnew);   // 0 on the first tile (mold = -inf)
        sF[w] = f;
        sL[w] = sL[w] * f + ssum;
        sM[w] = mnew;
      }
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < kJR; ++r) {
      const float f = sF[r];
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[r][e] *= f;
    }
#pragma unroll
    for (int qq = 0; qq < 4; ++qq) {   // values: the same keys, dims 8 hl .. 8 hl + 7
      const int kk = 8 * w + 2 * qq + hh;
      if (kk < nk) {
        const uint4 raw = *(const uint4*)(Vt + kk * 128 + hl * 8);
        const __nv_bfloat162* h2 = (const __nv_bfloat162*)&raw;
        float v8[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __bfloat1622float2(h2[e]);
          v8[2 * e] = f.x;
          v8[2 * e + 1] = f.y;
        }
#pragma unroll
        for (int r = 0; r < kJR; ++r) {
          const float pr = sP[r][kk];
#pragma unroll
          for (int e = 0; e < 8; ++e) acc[r][e] = fmaf(pr, v8[e], acc[r][e]);
        }
      }
    }
    __syncthreads();   // stage s and sP are free
    done = i + 1;
    if (tid == 0 && i + kBStages < ntile) issue(i + kBStages);
  }
  if (done < ntile) {
    // a wait gave up (status recorded): let the copies already issued land
    // (bounded) before the CTA's shared memory goes away, and write nothing
    if (tid == 0) {
      const unsigned long long t0 = tc::globaltimer();
      for (int i = done; i < min(ntile, done + kBStages); ++i)
        while (!tc::mbar_try_wait(&bar[i % kBStages], (uint32_t)((i / kBStages) & 1)) &&
               tc::globaltimer() - t0 < tc::kWaitLimitNs) {
        }
    }
    __syncthreads();
    return;
  }
  // lanes l and l ^ 16 hold the same dims over different keys
#pragma unroll
  for (int r = 0; r < kJR; ++r)
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[r][e] += __shfl_xor_sync(0xffffffffu, acc[r][e], 16);
  float* sAcc = (float*)smraw;   // [8 warps][kJR][128], over the drained stages
  if (hh == 0) {
#pragma unroll
    for (int r = 0; r < kJR; ++r) {
      *(float4*)&sAcc[(w * kJR + r) * 128 + hl * 8] = make_float4(acc[r][0], acc[r][1], acc[r][2], acc[r][3]);
      *(float4*)&sAcc[(w * kJR + r) * 128 + hl * 8 + 4] = make_float4(acc[r][4], acc[r][5], acc[r][6], acc[r][7]);
    }
  }
  __syncthreads();
  for (int e = tid; e < kJR * 128; e += kJThreads) {
    const int r = e >> 7, dd = e & 127;
    if (r0 + r >= n) continue;
    float o = 0.f;
#pragma unroll
    for (int q8 = 0; q8 < kJThreads / 32; ++q8) o += sAcc[(q8 * kJR + r) * 128 + dd];
    const long long row = ((long long)h * nsplit + sp) * n + r0 + r;
    Opart[row * 128 + dd] = o;
    if (dd == 0) ml[row] = make_float2(sM[r], sL[r]);
  }
}

// O[h][i] = sum_s e^{m_s - m} Opart_s / sum_s e^{m_s - m} l_s (one warp per row, lane dims 4l..4l+3)
__global__ void __launch_bounds__(256) attend_combine_kernel(const float* Opart, const float2* ml, int n, int nsplit,
                                                             long long rows, float* O) {
  const long long g = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (g >= rows) return;
  const long long h = g / n, i = g % n;
  float m = -INFINITY;
  for (int s = 0; s < nsplit; ++s) m = fmaxf(m, ml[(h * nsplit + s) * n + i].x);
  float l = 0.f, o0 = 0.f, o1 = 0.f, o2 = 0.f, o3 = 0.f;
  for (int s = 0; s < nsplit; ++s) {
    const long long row = (h * nsplit + s) * n + i;
    const float2 v = ml[row];
    const float f = expf(v.x - m);
    l = fmaf(v.y, f, l);
    const float4 op = *(const float4*)(Opart + row * 128 + lane * 4);
    o0 = fmaf(f, op.x, o0);
    o1 = fmaf(f, op.y, o1);
    o2 = fmaf(f, op.z, o2);
    o3 = fmaf(f, op.w, o3);
  }
  const float inv = 1.0f / l;
  *(float4*)(O + g * 128 + lane * 4) = make_float4(o0 * inv, o1 * inv, o2 * inv, o3 * inv);
}

// ---------------------------------------------------------------------------
// Truncated-output error of an anchor set (App. B.1 Eq. background_truncated_error):
//   O_i = sum_j p_ij v_j, O~_i(S) = sum_{j in S} p_ij v_j (p over the full cache),
//   err_i = ||O_i - O~_i|| / (||O_i|| + eps).
// One CTA per (4-row block, head) makes one pass over the keys: the logits and
// online softmax of attend_tiles, and two value accumulators (all keys; keys in S).
__global__ void __launch_bounds__(kJThreads) trunc_err_kernel(const bf16* Q, int n, const bf16* K, const bf16* V,
                                                              int T, const unsigned char* inS, float scale, float eps,
                                                              float* err) {
  const int h = blockIdx.y, r0 = blockIdx.x * kJR;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  __shared__ __align__(16) float sQ[kJR][128];
  __shared__ float sP[kJR][kJTile];
  __shared__ float sM[kJR], sL[kJR], sF[kJR];
  __shared__ __align__(16) float sAcc[2][kJThreads / 32][kJR][128];
  const bf16* Kh = K + (long long)h * T * 128;
  const bf16* Vh = V + (long long)h * T * 128;
  const unsigned char* mh = inS + (long long)h * T;
  for (int e = tid; e < kJR * 128; e += kJThreads) {
    const int r = e >> 7, dd = e & 127;
    sQ[r][dd] = (r0 + r < n) ? scale * __bfloat162float(Q[((long long)h * n + r0 + r) * 128 + dd]) : 0.f;
  }
  if (tid < kJR) {
    sM[tid] = -INFINITY;
    sL[tid] = 0.f;
  }
  float acc[kJR][4], accs[kJR][4];
#pragma unroll
  for (int r = 0; r < kJR; ++r)
#pragma unroll
    for (int q = 0; q < 4; ++q) acc[r][q] = accs[r][q] = 0.f;
  __syncthreads();
  for (int j0 = 0; j0 < T; j0 += kJTile) {
    {
      const int jj = tid >> 2, p = tid & 3, j = j0 + jj;
      KSlice32H k;
      if (j < T) k.load(Kh + (long long)j * 128 + p * 32);
      else k.zero();
      float part[kJR];
#pragma unroll
      for (int r = 0; r < kJR; ++r) {
        float a = k.dot((const float4*)&sQ[r][p * 32]);
        a += __shfl_xor_sync(0xffffffffu, a, 1);
        a += __shfl_xor_sync(0xffffffffu, a, 2);
        part[r] = a;
      }
      if (p == 0) {
#pragma unroll
        for (int r = 0; r < kJR; ++r) sP[r][jj] = (j < T) ? part[r] : -INFINITY;
      }
    }
    __syncthreads();
    if (w < kJR) {
      const float a0 = sP[w][lane], a1 = sP[w][lane + 32];
      const float mold = sM[w], mnew = fmaxf(mold, warp_max(fmaxf(a0, a1)));
      const float e0 = expf(a0 - mnew), e1 = expf(a1 - mnew);
      sP[w][lane] = e0;
      sP[w][lane + 32] = e1;
      const float ssum = warp_sum(e0 + e1);
      if (lane == 0) {
        const float f = expf(mold - mnew);
        sF[w] = f;
        sL[w] = sL[w] * f + ssum;
        sM[w] = mnew;
      }
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < kJR; ++r) {
      const float f = sF[r];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        acc[r][q] *= f;
        accs[r][q] *= f;
      }
    }
    for (int i = 0; i < kJTile / 8; ++i) {
      const int jj = w + 8 * i, j = j0 + jj;
      if (j < T) {
        float v[4];
        load4(Vh + (long long)j * 128 + lane * 4, v);
        const bool in = mh[j] != 0;
#pragma unroll
        for (int r = 0; r < kJR; ++r) {
          const float pr = sP[r][jj];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            acc[r][q] = fmaf(pr, v[q], acc[r][q]);
            if (in) accs[r][q] = fmaf(pr, v[q], accs[r][q]);
          }
        }
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int r = 0; r < kJR; ++r) {
    *(float4*)&sAcc[0][w][r][lane * 4] = make_float4(acc[r][0], acc[r][1], acc[r][2], acc[r][3]);
    *(float4*)&sAcc[1][w][r][lane * 4] = make_float4(accs[r][0], accs[r][1], accs[r][2], accs[r][3]);
  }
  __syncthreads();
  if (w < kJR && r0 + w < n) {   // warp r: row r's norms over its 128 dims
    const int r = w;
    const float inv = 1.0f / sL[r];
    float dd = 0.f, oo = 0.f;
    for (int c = lane; c < 128; c += 32) {
      float o = 0.f, os = 0.f;
#pragma unroll
      for (int q = 0; q < kJThreads / 32; ++q) {
        o += sAcc[0][q][r][c];
        os += sAcc[1][q][r][c];
      }
      o *= inv;
      os *= inv;
      dd = fmaf(o - os, o - os, dd);
      oo = fmaf(o, o, oo);
    }
    dd = warp_sum(dd);
    oo = warp_sum(oo);
    if (lane == 0) err[(long long)h * n + r0 + r] = sqrtf(dd) / (sqrtf(oo) + eps);
  }
}

// inS[h][j] = 1 for the anchors S[h][:] (clamped into [0, T); out-of-range entries record INVALID_ARG)
__global__ void anchor_mask_kernel(const int* S, int t, int T, int H, unsigned char* inS, DevStatus* stt) {
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < (long long)H * t;
       k += (long long)gridDim.x * blockDim.x) {
    const long long h = k / t;
    int j = S[k];
    if (j < 0 || j >= T) {
      set_status(stt, ARCKV_ERR_INVALID_ARG);
      j = min(max(j, 0), T - 1);
    }
    inS[h * T + j] = 1;
  }
}

// E[h] = mean_i err[h][i] (fixed order)
__global__ void row_mean_kernel(const float* err, int n, int H, float* E) {
  const int h = blockIdx.x * blockDim.x + threadIdx.x;
  if (h >= H) return;
  float a = 0.f;
  for (int i = 0; i < n; ++i) a += err[(long long)h * n + i];
  E[h] = a / (float)n;
}

int launch_truncated_error(int H, int n, int T, int t, float scale, float eps, const bf16* Q, const bf16* K,
                           const bf16* V, const int* S, float* E, unsigned char* inS, float* err, DevStatus* stt,
                           cudaStream_t st) {
  cudaMemsetAsync(inS, 0, (size_t)H * T, st);
  if (t > 0)
    anchor_mask_kernel<<<stride_grid((long long)H * t, 256, 4), 256, 0, st>>>(S, t, T, H, inS, stt);
  trunc_err_kernel<<<dim3(cdiv(n, kJR), H), kJThreads, 0, st>>>(Q, n, K, V, T, inS, scale, eps, err);
  row_mean_kernel<<<cdiv(H, 128), 128, 0, st>>>(err, n, H, E);
  return 3;
}

JointSplit joint_split(int H, int n, int t, int F) {
  JointSplit s;
  const int L = t + F, rb = cdiv(n, kJR);
  const long long ctas = (long long)H * rb;
  const int want = (int)std::max<long long>(1, ((long long)tc_gemm_sm_count() * 8 + ctas - 1) / ctas);   // about 8 CTAs per SM
  const int ntiles = cdiv(L, kJTile);
  const int nsp = std::min(want, ntiles);
  s.per_split = cdiv(ntiles, nsp) * kJTile;
  s.nsplit = cdiv(L, s.per_split);
  return s;
}

int launch_attend_joint(int H, int n, int t, int F, float scale, const bf16* Q, const void* Ck, const float* beta,
                        const void* Cv, bool compact_bf16, const bf16* Kf, const bf16* Vf, float* O, float* Opart,
                        float2* ml, DevStatus* stt, cudaStream_t st) {
  const JointSplit s = joint_split(H, n, t, F);
  const dim3 grid(s.nsplit, cdiv(n, kJR), H);
  if (compact_bf16 || t == 0) {
    const int smem = 2 * kBStages * kBTileBytes;
    set_dyn_smem((const void*)attend_bulk_kernel, smem);
    attend_bulk_kernel<<<grid, kJThreads, smem, st>>>(Q, n, (const bf16*)Ck, beta, (const bf16*)Cv, t, Kf, Vf, F,
                                                      scale, s.per_split, s.nsplit, Opart, ml, stt);
  } else
    attend_split_kernel<float><<<grid, kJThreads, 0, st>>>(Q, n, (const float*)Ck, beta, (const float*)Cv, t, Kf, Vf,
                                                           F, scale, s.per_split, s.nsplit, Opart, ml);
  const long long rows = (long long)H * n;
  attend_combine_kernel<<<(unsigned)cdiv(rows, 8), 256, 0, st>>>(Opart, ml, n, s.nsplit, rows, O);
  return 2;
}

}  // namespace arckv
