// Top-t anchor selection (App. A.6 Eq. persistent_support) and small shared
// row / reduction kernels.
#include "kernels.h"

namespace arckv {

// Exclusive prefix sum over a 1024-thread block; `sc` holds 32 ints.
__device__ __forceinline__ int block_excl_scan_1024(int v, int* sc, int& total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sc[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = sc[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    sc[lane] = w;
  }
  __syncthreads();
  const int off = warp > 0 ? sc[warp - 1] : 0;
  total = sc[31];
  __syncthreads();
  return off + x - v;
}

// One 1024-thread CTA per (chunk, head).  MSB-first radix select (8-bit
// digits) of the t_c-th largest score of the chunk on the ordered bit
// patterns, then an order-preserving compaction: every position with a larger
// score, plus the lowest-position ones among those equal to the threshold
// (ties -> lower position), written in ascending position order after the
// anchors of the chunks before it.  L = 0: one chunk, the whole cache, t_c = t.
constexpr int kSelE = 8;   // consecutive scores per thread per round

__global__ void __launch_bounds__(1024) top_t_kernel(const float* s, int Tall, int tb, int L, int tp, int* anchors,
                                                     DevStatus* stt) {
  const int b = blockIdx.y, c = blockIdx.x, tid = threadIdx.x;
  int cstart = 0, T = Tall, t = tb, off = 0;   // chunk start, length, budget, output offset
  if (L > 0) {
    cstart = c * L;
    T = min(L, Tall - cstart);
    t = chunk_budget(Tall, tb, T);
    for (int q = 0; q < c; ++q) off += chunk_budget(Tall, tb, min(L, Tall - q * L));
  }
  const float* sb = s + (long long)b * Tall + cstart;
  int* out = anchors + (long long)b * tp + off;
  __shared__ int hist[256];
  __shared__ int sc[32];
  __shared__ unsigned int sh_prefix;
  __shared__ int sh_rem;
  unsigned int prefix = 0u, mask = 0u;
  int rem = t;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    if (tid < 256) hist[tid] = 0;
    __syncthreads();
    for (int j0 = tid * kSelE; j0 < T; j0 += 1024 * kSelE) {   // kSelE consecutive scores per thread
      float v[kSelE];
#pragma unroll
      for (int q = 0; q < kSelE; ++q) v[q] = j0 + q < T ? sb[j0 + q] : 0.f;
#pragma unroll
      for (int q = 0; q < kSelE; ++q) {
        if (j0 + q >= T) break;
        if (pass == 0 && !isfinite(v[q])) set_status(stt, ARCKV_ERR_NONFINITE);
        const unsigned int key = f32_ordered(v[q]);
        if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1);
      }
    }
    __syncthreads();
    if (tid == 0) {
      int cum = 0, D = 0;
      for (int dg = 255; dg >= 0; --dg) {
        if (cum + hist[dg] >= rem) { D = dg; break; }
        cum += hist[dg];
      }
      sh_prefix = prefix | ((unsigned int)D << shift);
      sh_rem = rem - cum;
    }
    __syncthreads();
    prefix = sh_prefix;
    rem = sh_rem;
    mask |= 0xffu << shift;
  }
  // compaction, kSelE consecutive positions per thread per round: threads in
  // order, each thread's positions in order, so the output stays ascending
  int base = 0, eqseen = 0;
  for (int r0 = 0; r0 < T; r0 += 1024 * kSelE) {
    const int jb = r0 + tid * kSelE;
    unsigned int key[kSelE];
    int neq = 0;
#pragma unroll
    for (int q = 0; q < kSelE; ++q) {
      key[q] = jb + q < T ? f32_ordered(sb[jb + q]) : 0u;
      neq += (jb + q < T && key[q] == prefix) ? 1 : 0;
    }
    int eqtot, tot;
    int eqrank = block_excl_scan_1024(neq, sc, eqtot) + eqseen;
    unsigned int take = 0u;
#pragma unroll
    for (int q = 0; q < kSelE; ++q) {
      const bool in = jb + q < T, eq = in && key[q] == prefix;
      if (in && (key[q] > prefix || (eq && eqrank < rem))) take |= 1u << q;
      eqrank += eq ? 1 : 0;
    }
    int pos = block_excl_scan_1024(__popc(take), sc, tot) + base;
#pragma unroll
    for (int q = 0; q < kSelE; ++q)
      if ((take >> q) & 1u) {
        if (pos < t) out[pos] = cstart + jb + q;
        ++pos;
      }
    base += tot;
    eqseen += eqtot;
  }
  if (tid == 0 && base != t) set_status(stt, ARCKV_ERR_INVALID_ARG);
}

int launch_top_t(const Dims& D, int t_budget, const float* s, int* anchors, DevStatus* stt, cudaStream_t st) {
  const int nch = D.chunk > 0 ? cdiv(D.T, D.chunk) : 1;
  top_t_kernel<<<dim3(nch, D.H), 1024, 0, st>>>(s, D.T, D.chunk > 0 ? t_budget : D.t, D.chunk, D.t, anchors, stt);
  return 1;
}

// Caller-supplied anchors (copied into the workspace) must be strictly
// ascending positions in [0, T).  A violation is recorded as
// ARCKV_ERR_INVALID_ARG and every entry is clamped to [0, T) so that later
// kernels never index outside the cache.  One CTA per head.
__global__ void check_anchors_kernel(int* anchors, int T, int t, DevStatus* stt) {
  int* a = anchors + (long long)blockIdx.x * t;
  bool bad = false;
  for (int r = threadIdx.x; r < t; r += blockDim.x) {
    const int v = a[r];
    bad |= (v < 0 || v >= T || (r > 0 && a[r - 1] >= v));
  }
  __syncthreads();
  for (int r = threadIdx.x; r < t; r += blockDim.x) a[r] = min(max(a[r], 0), T - 1);
  if (bad) set_status(stt, ARCKV_ERR_INVALID_ARG);
}

int launch_check_anchors(const Dims& D, int* anchors, DevStatus* stt, cudaStream_t st) {
  check_anchors_kernel<<<D.H, 256, 0, st>>>(anchors, D.T, D.t, stt);
  return 1;
}

// Row statistics from per-tile softmax partials part[b][row][tile] = (max, sum):
// shift = max, sum = total sum of exp(x - shift), mul = 1 / sum.  One warp per row.
__global__ void part_stats_kernel(const float2* part, float* shift, float* mul, float* sum, int rows, int ntiles) {
  const int b = blockIdx.y, row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= rows) return;
  const float2* p = part + ((long long)b * rows + row) * ntiles;
  float mx = -INFINITY, sm = 0.f;
  for (int k = lane; k < ntiles; k += 32) lse_combine(mx, sm, p[k].x, p[k].y);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, mx, o), os = __shfl_xor_sync(0xffffffffu, sm, o);
    lse_combine(mx, sm, om, os);
  }
  if (lane == 0) {
    const long long k = (long long)b * rows + row;
    shift[k] = mx;
    if (mul) mul[k] = 1.0f / sm;
    if (sum) sum[k] = sm;
  }
}

int launch_part_stats(int H, int rows, int ntiles, const float2* part, float* shift, float* mul, float* sum,
                      cudaStream_t st) {
  part_stats_kernel<<<dim3(cdiv(rows, 8), H), 256, 0, st>>>(part, shift, mul, sum, rows, ntiles);
  return 1;
}


}  // namespace arckv
