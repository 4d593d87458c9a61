// Softmax attention products on tcgen05 with fp32-grade accuracy:
//
//   value-attention logits (U_q q_i).(U_k k_j) = q''_i . k_j,
//       q''_i = U_k^T (U_q q_i)                       (Eq. value_context)
//   A V and softmax(l) V with A, softmax(l) row-stochastic and V the bf16 cache
//                                                     (Eq. value_context, Eq. value_lstsq's Y)
//
// In every product one operand is an exact bf16 input (K or V) and the other
// an fp32 value, which enters as a bf16 triple (h, m, l) summing to it within
// 2^-24; the kSplit3A GEMM issues h*B + m*B + l*B.
#include "kernels.h"
#include "tc_gemm.cuh"

namespace arckv {

__global__ void split3_kernel(const float* x, bf16* h, bf16* m, bf16* l, long long count) {
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < count;
       k += (long long)gridDim.x * blockDim.x)
    split3_bf16(x[k], h[k], m[k], l[k]);
}

// P = exp(X - shift_row) * mul_row as a bf16 triple [H][rows][ldc] (zero in the
// pad columns cols..ldc-1, and in column skip[row] when skip is given).
__global__ void probs_split3_kernel(const float* X, const float* shift, const float* mul, const int* skip, bf16* h,
                                    bf16* m, bf16* l, int rows, int cols, int ldc) {
  const int b = blockIdx.z, row = blockIdx.y;
  const long long rr = (long long)b * rows + row;
  const float sh = shift[rr], mu = mul[rr];
  const int sk = skip ? skip[rr] : -1;
  const float* x = X + rr * cols;
  const long long o = rr * ldc;
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < ldc; c += gridDim.x * blockDim.x) {
    const float p = (c < cols && c != sk) ? expf(x[c] - sh) * mu : 0.f;
    split3_bf16(p, h[o + c], m[o + c], l[o + c]);
  }
}

// VT[b][d][j] = V[b][j][d] (bf16), zero for T <= j < ldT.
__global__ void __launch_bounds__(256) transpose_v_kernel(const bf16* V, bf16* VT, int T, int ldT) {
  const int b = blockIdx.z, j0 = blockIdx.x * 32, d0 = blockIdx.y * 32;
  __shared__ bf16 tile[32][34];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const bf16 zero = __float2bfloat16_rn(0.f);
  for (int q = ty; q < 32; q += 8) {
    const int j = j0 + q;
    tile[q][tx] = (j < T) ? V[((long long)b * T + j) * 128 + d0 + tx] : zero;
  }
  __syncthreads();
  for (int q = ty; q < 32; q += 8) {
    const int j = j0 + tx;
    if (j < ldT) VT[((long long)b * 128 + d0 + q) * ldT + j] = tile[tx][q];
  }
}

// C[b] (rows x 128 or rows x N) = A3 B^T with A3 = (h, m, l) [H][rows][K] and B [H][N][K].
static int gemm_split3a(int H, int rows, int N, int K, int ldk, const bf16* h, const bf16* m, const bf16* l,
                        const bf16* B, float* C, int ldc, float alpha, DevStatus* stt, cudaStream_t st) {
  CUtensorMap mA, mA2, mA3, mB;
  if (!encode_bf16_map_3d(&mA, h, ldk, rows, H, 128) || !encode_bf16_map_3d(&mA2, m, ldk, rows, H, 128) ||
      !encode_bf16_map_3d(&mA3, l, ldk, rows, H, 128) || !encode_bf16_map_3d(&mB, B, ldk, N, H, 128))
    return -1;
  TcEpiStore epi{C, (long long)rows * ldc, ldc, alpha};
  const int kfull = (K + 63) / 64 * 64;
  if (launch_tc_gemm<128, kSplit3A>(mA, mB, mA2, mA, epi, H, rows, N, K, kfull, stt, st, 0, &mA3) != cudaSuccess)
    return -1;
  return 1;
}

int launch_value_logits_tc(const Dims& D, const bf16* q_h, const bf16* q_m, const bf16* q_l, const bf16* K,
                           float* logits, float2* part, DevStatus* stt, cudaStream_t st) {
  CUtensorMap mA, mA2, mA3, mB;
  if (!encode_bf16_map_3d(&mA, q_h, 128, D.n, D.H, 128) || !encode_bf16_map_3d(&mA2, q_m, 128, D.n, D.H, 128) ||
      !encode_bf16_map_3d(&mA3, q_l, 128, D.n, D.H, 128) || !encode_bf16_map_3d(&mB, K, 128, D.T, D.H, 128))
    return -1;
  if (launch_tc_logits_rowpart<kSplit3A>(mA, mB, mA2, mA, &mA3, logits, 1.f, part, D.H, D.n, D.T, 128, stt, st) !=
      cudaSuccess)
    return -1;
  return 1;
}

int launch_split3(const float* x, bf16* h, bf16* m, bf16* l, long long count, cudaStream_t st) {
  split3_kernel<<<stride_grid(count, 256, 8), 256, 0, st>>>(x, h, m, l, count);
  return 1;
}

int launch_transpose_v(const Dims& D, const bf16* V, bf16* VT, cudaStream_t st) {
  const int ldT = (D.T + 7) / 8 * 8;
  transpose_v_kernel<<<dim3(cdiv(ldT, 32), 4, D.H), 256, 0, st>>>(V, VT, D.T, ldT);
  return 1;
}

// ---------------------------------------------------------------------------
// Fused O = P V with P = exp(X - shift_row) * mul_row, X the fp32 logits
// [H][rows][T] and V the bf16 cache (as V^T [H][128][ldT]).  P never reaches
// memory: TMA streams 128 x 64 slabs of X into a raw ring; sixteen converter
// warps form P there (e^x as 2^(x log2 e), one MUFU op per element), split it into the bf16 triple (h, m, l) and write the
// three operand tiles straight into the 128-byte-swizzled K-major layout the
// MMA reads; one thread issues h V + m V + l V per 16-wide K step into a
// 128 x 128 fp32 TMEM accumulator; a fifth warp streams the V^T slabs.  The
// products are those of the unfused split-3 GEMM, in the same order.
//
// CTA = (row tile of 128, K split); with two K splits the halves are added
// into a zeroed output with fp32 atomics (two addends onto 0: the sum does not
// depend on their order).
namespace {
constexpr int kPvRawBytes = 128 * 64 * 4;   // one fp32 slab of X
constexpr int kPvTile = 128 * 128;          // one bf16 128 x 64 operand tile
constexpr int kPvRS = 3;                    // raw ring depth
constexpr int kPvOS = 2;                    // operand ring depth (h, m, l, V^T)
constexpr int kPvOpBytes = 4 * kPvTile;
constexpr int kPvConv = 16;                 // converter warps 2..17, 8 rows each
constexpr int kPvThreads = 32 * (kPvConv + 3);
constexpr int kPvSmem = kPvRS * kPvRawBytes + kPvOS * kPvOpBytes + 1024;
}  // namespace

template <bool kSkip>
__global__ void __launch_bounds__(kPvThreads, 1)
    probs_v_kernel(const __grid_constant__ CUtensorMap mX, const __grid_constant__ CUtensorMap mVT,
                   const float* shift, const float* mul, const int* skip, float* O, int rows, int T, int splits,
                   DevStatus* stt) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ uint64_t rfull[kPvRS], rempty[kPvRS], vfull[kPvOS], ofull[kPvOS], oempty[kPvOS], accf, drain;
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_flag;
  const uint32_t r0 = tc::smem_u32(smem_raw);
  uint8_t* rbase = smem_raw + (((r0 + 1023u) & ~1023u) - r0);
  uint8_t* obase = rbase + kPvRS * kPvRawBytes;   // 1024-byte aligned: the ring is a multiple of 1 KB
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = (rows + 127) / 128;
  const int tile = blockIdx.x / splits, sp = blockIdx.x - tile * splits;
  const int b = tile / mt, m0 = (tile - b * mt) * 128;
  const int nk = (T + 63) / 64;
  const int kb0 = (int)((long long)nk * sp / splits), kb1 = (int)((long long)nk * (sp + 1) / splits);
  const int nkb = kb1 - kb0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kPvRS; ++s) {
      tc::mbar_init(&rfull[s], 1);
      tc::mbar_init(&rempty[s], kPvConv);
    }
    for (int s = 0; s < kPvOS; ++s) {
      tc::mbar_init(&vfull[s], 1);
      tc::mbar_init(&ofull[s], kPvConv);
      tc::mbar_init(&oempty[s], 1);
    }
    tc::mbar_init(&accf, 1);
    tc::mbar_init(&drain, 1);
    abort_flag = 0;
    tc::mbar_fence_init();
  }
  if (warp == 1) tc::tmem_alloc(&tmem_slot, 128);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_slot;
  volatile int* abortp = &abort_flag;

  if (warp == 0) {
    // X slabs
    if (lane == 0) {
      tc::tma_prefetch(&mX);
      int g = 0;
      for (; g < nkb; ++g) {
        const int s = g % kPvRS;
        if (g >= kPvRS && !tc::mbar_wait(&rempty[s], ((g / kPvRS) - 1) & 1, abortp, stt)) break;
        tc::mbar_arrive_expect_tx(&rfull[s], kPvRawBytes);
        tc::tma_load_3d(rbase + s * kPvRawBytes, &mX, (kb0 + g) * 64, m0, b, &rfull[s]);
      }
      volatile int never = 0;
      for (int k = g > kPvRS ? g - kPvRS : 0; k < g; ++k) tc::mbar_wait(&rfull[k % kPvRS], (k / kPvRS) & 1, &never, stt);
    }
  } else if (warp == kPvConv + 2) {
    // V^T slabs
    if (lane == 0) {
      tc::tma_prefetch(&mVT);
      int g = 0;
      for (; g < nkb; ++g) {
        const int s = g % kPvOS;
        if (g >= kPvOS && !tc::mbar_wait(&oempty[s], ((g / kPvOS) - 1) & 1, abortp, stt)) break;
        tc::mbar_arrive_expect_tx(&vfull[s], kPvTile);
        tc::tma_load_3d(obase + s * kPvOpBytes + 3 * kPvTile, &mVT, (kb0 + g) * 64, 0, b, &vfull[s]);
      }
      volatile int never = 0;
      for (int k = g > kPvOS ? g - kPvOS : 0; k < g; ++k) tc::mbar_wait(&vfull[k % kPvOS], (k / kPvOS) & 1, &never, stt);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = tc::idesc_bf16_f32(128);
      bool ok = true;
      for (int g = 0; g < nkb && ok; ++g) {
        const int s = g % kPvOS;
        const uint32_t ph = (g / kPvOS) & 1;
        if (!tc::mbar_wait(&vfull[s], ph, abortp, stt) || !tc::mbar_wait(&ofull[s], ph, abortp, stt)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const uint32_t a = tc::smem_u32(obase + s * kPvOpBytes), bv = a + 3 * kPvTile;
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
          const uint64_t bd = tc::sdesc_k128(bv + ks * 32);
#pragma unroll
          for (int part = 0; part < 3; ++part)
            tc::mma_f16(tmem, tc::sdesc_k128(a + part * kPvTile + ks * 32), bd, idesc,
                        (g > 0 || ks > 0 || part > 0) ? 1u : 0u);
        }
        tc::mma_commit(&oempty[s]);
      }
      if (ok) tc::mma_commit(&accf);
      tc::mma_commit(&drain);
      volatile int never = 0;
      tc::mbar_wait(&drain, 0, &never, stt);
    }
  } else {
    // converters: warp cw owns rows 8 cw .. 8 cw + 7 of the tile, two rows per
    // step (lanes 0-15 the first, 16-31 the second), four columns per lane
    const int cw = warp - 2, hl = lane >> 4, cl = lane & 15;
    float zl[4], mu[4];   // per step: shift * log2 e and scale of this lane's row (0, 0 past the end: P = 0)
    int sk[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int row = m0 + cw * 8 + 2 * u + hl;
      zl[u] = 0.f;
      mu[u] = 0.f;
      sk[u] = -1;
      if (row < rows) {
        const long long rr = (long long)b * rows + row;
        zl[u] = shift[rr] * kLog2e;
        mu[u] = mul[rr];
        if (kSkip) sk[u] = skip[rr];
      }
    }
    bool ok = true;
    for (int g = 0; g < nkb; ++g) {
      const int rs = g % kPvRS, os = g % kPvOS;
      ok = tc::mbar_wait(&rfull[rs], (g / kPvRS) & 1, abortp, stt);
      if (ok && g >= kPvOS) ok = tc::mbar_wait(&oempty[os], ((g / kPvOS) - 1) & 1, abortp, stt);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      const float* R = (const float*)(rbase + rs * kPvRawBytes);
      uint8_t* A = obase + os * kPvOpBytes;
      const int c = (kb0 + g) * 64 + 4 * cl;   // this lane's first column
      const bool edge = kSkip || c + 4 > T;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int r = cw * 8 + 2 * u + hl;
        const float4 x = *(const float4*)(R + r * 64 + 4 * cl);
        float p[4] = {ex2_approx(fmaf(x.x, kLog2e, -zl[u])) * mu[u], ex2_approx(fmaf(x.y, kLog2e, -zl[u])) * mu[u],
                      ex2_approx(fmaf(x.z, kLog2e, -zl[u])) * mu[u], ex2_approx(fmaf(x.w, kLog2e, -zl[u])) * mu[u]};
        if (edge) {
#pragma unroll
          for (int e = 0; e < 4; ++e)
            if (c + e >= T || c + e == sk[u]) p[e] = 0.f;
        }
        __nv_bfloat162 h0, m0_, l0, h1, m1, l1;
        split3_bf16x2(p[0], p[1], h0, m0_, l0);
        split3_bf16x2(p[2], p[3], h1, m1, l1);
        // 128-byte swizzle: 16-byte chunk cl / 2 of row r sits at chunk (cl / 2) ^ (r % 8)
        const uint32_t off = (uint32_t)r * 128u + ((((uint32_t)cl >> 1) ^ ((uint32_t)r & 7u)) << 4) +
                             (((uint32_t)cl & 1u) << 3);
        *(uint2*)(A + off) = make_uint2(*(uint32_t*)&h0, *(uint32_t*)&h1);
        *(uint2*)(A + kPvTile + off) = make_uint2(*(uint32_t*)&m0_, *(uint32_t*)&m1);
        *(uint2*)(A + 2 * kPvTile + off) = make_uint2(*(uint32_t*)&l0, *(uint32_t*)&l1);
      }
      tc::fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        tc::mbar_arrive(&rempty[rs]);
        tc::mbar_arrive(&ofull[os]);
      }
    }
    if (ok) ok = tc::mbar_wait(&accf, 0, abortp, stt);
    ok = __all_sync(0xffffffffu, ok);
    if (ok) {
      tc::fence_after_sync();
      const int qd = warp & 3, cg = cw >> 2;   // TMEM lane quarter; 32-column group
      const int row = m0 + qd * 32 + lane;
      float v[32];
      tc::tmem_ld32(tmem + ((uint32_t)(qd * 32) << 16) + (uint32_t)(cg * 32), v);
      if (row < rows) {
        float* d = O + ((long long)b * rows + row) * 128 + cg * 32;
        if (splits > 1) {
#pragma unroll
          for (int e = 0; e < 32; ++e) atomicAdd(d + e, v[e]);
        } else {
#pragma unroll
          for (int e = 0; e < 32; e += 4) *(float4*)(d + e) = make_float4(v[e], v[e + 1], v[e + 2], v[e + 3]);
        }
      }
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 128);
  }
}

// The fused product (probs_fused(T): X rows tileable by TMA); returns the
// launches issued or -1 (also for base pointers off the 16-byte grid).
static int launch_probs_v_fused(const Dims& D, const float* X, const float* shift, const float* mul, const int* skip,
                                const bf16* VT, float* out, DevStatus* stt, cudaStream_t st) {
  if (((uintptr_t)X & 15u) != 0 || ((uintptr_t)out & 15u) != 0) return -1;
  const int ldT = (D.T + 7) / 8 * 8;
  CUtensorMap mX, mVT;
  if (!encode_f32_map_3d(&mX, X, D.T, D.n, D.H, 64, 128) || !encode_bf16_map_3d(&mVT, VT, ldT, 128, D.H, 128))
    return -1;
  const int tiles = D.H * cdiv(D.n, 128), nk = cdiv(D.T, 64);
  const int splits = (2 * tiles <= tc_gemm_sm_count() && nk >= 2) ? 2 : 1;
  auto kern = skip ? probs_v_kernel<true> : probs_v_kernel<false>;
  if (set_dyn_smem((const void*)kern, kPvSmem) != cudaSuccess) return -1;
  if (splits > 1 && cudaMemsetAsync(out, 0, sizeof(float) * (size_t)D.H * D.n * 128, st) != cudaSuccess) return -1;
  kern<<<tiles * splits, kPvThreads, kPvSmem, st>>>(mX, mVT, shift, mul, skip, out, D.n, D.T, splits, stt);
  return cudaGetLastError() == cudaSuccess ? 1 : -1;
}

int launch_probs_v_tc(const Dims& D, const float* X, const float* shift, const float* mul, bf16* p_h, bf16* p_m,
                      bf16* p_l, const bf16* VT, float* out, DevStatus* stt, cudaStream_t st, const int* skip) {
  if (probs_fused(D.T)) return launch_probs_v_fused(D, X, shift, mul, skip, VT, out, stt, st);
  // X rows not TMA-tileable: P as a bf16 triple in memory, then the split-3 GEMM
  const int ldT = (D.T + 7) / 8 * 8;
  probs_split3_kernel<<<dim3(cdiv(ldT, 256 * 4), D.n, D.H), 256, 0, st>>>(X, shift, mul, skip, p_h, p_m, p_l, D.n,
                                                                          D.T, ldT);
  if (gemm_split3a(D.H, D.n, 128, ldT, ldT, p_h, p_m, p_l, VT, out, 128, 1.f, stt, st) < 0) return -1;
  return 2;
}

}  // namespace arckv
