// Full-cache reference attention, response-profile assignment and the
// convex-hull key merge (Sec. 3.4).
//
// The paper's profiles u_j and mass weights phi_j use one global shift
// z_merge = max_ij l_ij (Eq. response_profile, Eq. mass_centroid).  Both u_j
// (a normalised column) and the ratios phi_j / sum_{G_r} phi_j are invariant to
// any per-column shift, so the kernels shift column j by its own maximum M_j,
// which keeps every column representable in fp32 when the logit range
// exceeds the fp32 exponent range (column statistics and profiles: the
// col_profiles kernel of the assignment stage).
#include "kernels.h"

namespace arckv {

int launch_reference_attention(const Dims& D, float scale, const bf16* Q, const bf16* K, const bf16* VT,
                               float* L, float2* part, float* z, float* m, float* invm, bf16* p_h, bf16* p_m,
                               bf16* p_l, float* Y, DevStatus* stt, cudaStream_t st) {
  // l = scale * Q K^T on the tensor cores, with per-tile row softmax partials
  if (launch_ref_logits_tc(D, scale, Q, K, L, part, stt, st) < 0) return -1;
  // z_i = max_j l_ij (z^fit of Eq. mass_fit), m_i = sum_j e^{l_ij - z_i} = (Phi_K 1)_i
  launch_part_stats(D.H, D.n, cdiv(D.T, kRowPartW), part, z, invm, m, st);
  // Y = softmax(l) V
  const int r = launch_probs_v_tc(D, L, z, invm, p_h, p_m, p_l, VT, Y, stt, st);
  if (r < 0) return -1;
  return 2 + r;
}

// Caller-supplied assignment (copied into the workspace): values in [0, t)
// and kappa(s_r) = r.  A violation is recorded as ARCKV_ERR_INVALID_ARG and
// out-of-range entries are clamped to [0, t).  Runs after the anchors check,
// so anchors are already inside [0, T).  Two kernels: the anchor rows are
// read only after every clamp has landed.
__global__ void check_assign_range_kernel(int* kappa, int t, long long total, DevStatus* stt) {
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < total;
       k += (long long)gridDim.x * blockDim.x) {
    const int v = kappa[k];
    if (v < 0 || v >= t) {
      set_status(stt, ARCKV_ERR_INVALID_ARG);
      kappa[k] = min(max(v, 0), t - 1);
    }
  }
}

__global__ void check_assign_anchor_kernel(const int* kappa, const int* anchors, int T, int t, int H, DevStatus* stt) {
  const long long ta = (long long)H * t;
  for (long long k = blockIdx.x * (long long)blockDim.x + threadIdx.x; k < ta;
       k += (long long)gridDim.x * blockDim.x) {
    const long long b = k / t;
    if (kappa[b * T + anchors[k]] != (int)(k - b * t)) set_status(stt, ARCKV_ERR_INVALID_ARG);
  }
}

int launch_check_assign(const Dims& D, int* kappa, const int* anchors, DevStatus* stt, cudaStream_t st) {
  const long long total = (long long)D.H * D.T;
  check_assign_range_kernel<<<stride_grid(total, 256, 8), 256, 0, st>>>(kappa, D.t, total, stt);
  check_assign_anchor_kernel<<<stride_grid((long long)D.H * D.t, 256, 8), 256, 0, st>>>(kappa, anchors, D.T, D.t,
                                                                                     D.H, stt);
  return 2;
}

__device__ __forceinline__ int block_excl_scan_1024_m(int v, int* sc, int& total) {
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

// Stable counting sort of positions by group (one 1024-thread CTA per head):
// perm lists the members of G_0, G_1, ... each in ascending position order;
// goff[r] .. goff[r+1] delimits G_r.
__global__ void __launch_bounds__(1024) group_sort_kernel(const int* kappa, int T, int t, int* perm, int* goff,
                                                          int* cursor) {
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int* kb = kappa + (long long)b * T;
  int* pb = perm + (long long)b * T;
  int* gb = goff + (long long)b * (t + 1);
  int* cb = cursor + (long long)b * t;
  __shared__ int sc[32];
  for (int r = tid; r < t; r += 1024) cb[r] = 0;
  __syncthreads();
  for (int j = tid; j < T; j += 1024) atomicAdd(&cb[min(max(kb[j], 0), t - 1)], 1);   // (in range by construction)
  __syncthreads();
  int base = 0;
  for (int r0 = 0; r0 < t; r0 += 1024) {
    const int r = r0 + tid;
    const int c = (r < t) ? cb[r] : 0;
    int tot;
    const int ex = block_excl_scan_1024_m(c, sc, tot) + base;
    if (r < t) { gb[r] = ex; cb[r] = ex; }
    base += tot;
  }
  if (tid == 0) gb[t] = base;
  __syncthreads();
  const unsigned int lt = (1u << lane) - 1u;
  for (int j0 = 0; j0 < T; j0 += 1024) {
    const int j = j0 + tid;
    const int key = (j < T) ? min(max(kb[j], 0), t - 1) : -1;
    const unsigned int peers = __match_any_sync(0xffffffffu, key);
    const int rank = __popc(peers & lt);
    const bool leader = (__ffs(peers) - 1) == lane;
    int pos = 0;
    for (int w = 0; w < 32; ++w) {
      if (warp == w) {
        if (key >= 0) pos = cb[key] + rank;
        __syncwarp();
        if (key >= 0 && leader) cb[key] += __popc(peers);
      }
      __syncthreads();
    }
    if (key >= 0) pb[pos] = j;
  }
}

// The same stable counting sort over many CTAs: the positions are cut into
// chunks of kSortChunk; each chunk counts its members per group (a
// shared-memory histogram), the counts give every (group, chunk) its first
// slot in group-major, chunk-minor order, and each chunk then scatters its
// positions in ascending order from those slots.  perm and goff come out
// identical to group_sort_kernel's.  cnt is [H][t][C], C = ceil(T / kSortChunk).
__global__ void __launch_bounds__(1024) sort_hist_kernel(const int* __restrict__ kappa, int T, int t, int C,
                                                         int* __restrict__ cnt) {
  extern __shared__ int hist[];
  const int c = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  for (int g = tid; g < t; g += 1024) hist[g] = 0;
  __syncthreads();
  const int* kb = kappa + (long long)b * T;
  const int j1 = min(T, (c + 1) * kSortChunk);
  // (assignments are in [0, t) by construction and by launch_check_assign;
  // the clamp keeps the shared-memory index in bounds regardless)
  for (int j = c * kSortChunk + tid; j < j1; j += 1024) atomicAdd(&hist[min(max(kb[j], 0), t - 1)], 1);
  __syncthreads();
  int* cb = cnt + (long long)b * t * C + c;
  for (int g = tid; g < t; g += 1024) cb[(long long)g * C] = hist[g];
}

// tot[b][g] = sum over chunks of cnt[b][g][.]
__global__ void __launch_bounds__(256) sort_totals_kernel(const int* __restrict__ cnt, int t, int C, int H,
                                                          int* __restrict__ tot) {
  const long long gi = (long long)blockIdx.x * 256 + threadIdx.x;
  if (gi >= (long long)H * t) return;
  const int* row = cnt + gi * C;
  int a = 0;
  for (int c = 0; c < C; ++c) a += row[c];
  tot[gi] = a;
}

// goff[b] = exclusive scan of tot[b] (one CTA per head); goff[b][t] = T
__global__ void __launch_bounds__(1024) sort_scan_kernel(const int* __restrict__ tot, int t, int* __restrict__ goff) {
  __shared__ int sc[32];
  const int b = blockIdx.x, tid = threadIdx.x;
  const int* tb = tot + (long long)b * t;
  int* gb = goff + (long long)b * (t + 1);
  int base = 0;
  for (int r0 = 0; r0 < t; r0 += 1024) {
    const int r = r0 + tid;
    int total;
    const int ex = block_excl_scan_1024_m(r < t ? tb[r] : 0, sc, total) + base;
    if (r < t) gb[r] = ex;
    base += total;
  }
  if (tid == 0) gb[t] = base;
}

// cnt[b][g][c] <- the first slot of chunk c's members of group g
__global__ void __launch_bounds__(256) sort_slots_kernel(int* __restrict__ cnt, const int* __restrict__ goff, int t,
                                                         int C, int H) {
  const long long gi = (long long)blockIdx.x * 256 + threadIdx.x;
  if (gi >= (long long)H * t) return;
  const int b = (int)(gi / t), g = (int)(gi - (long long)b * t);
  int* row = cnt + gi * C;
  int run = goff[(long long)b * (t + 1) + g];
  for (int c = 0; c < C; ++c) {
    const int k = row[c];
    row[c] = run;
    run += k;
  }
}

// each chunk's positions, ascending, to their groups' slots
__global__ void __launch_bounds__(1024) sort_scatter_kernel(const int* __restrict__ kappa, int T, int t, int C,
                                                            const int* __restrict__ cnt, int* __restrict__ perm) {
  extern __shared__ int cur[];
  const int c = blockIdx.x, b = blockIdx.y, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int* cb = cnt + (long long)b * t * C + c;
  for (int g = tid; g < t; g += 1024) cur[g] = cb[(long long)g * C];
  __syncthreads();
  const int* kb = kappa + (long long)b * T;
  int* pb = perm + (long long)b * T;
  const unsigned int lt = (1u << lane) - 1u;
  const int j1 = min(T, (c + 1) * kSortChunk);
  for (int j0 = c * kSortChunk; j0 < j1; j0 += 1024) {
    const int j = j0 + tid;
    const int key = (j < j1) ? min(max(kb[j], 0), t - 1) : -1;
    const unsigned int peers = __match_any_sync(0xffffffffu, key);
    const int rank = __popc(peers & lt);
    const bool leader = (__ffs(peers) - 1) == lane;
    int pos = 0;
    for (int w = 0; w < 32; ++w) {   // warps in order: ascending positions within the chunk
      if (warp == w) {
        if (key >= 0) pos = cur[key] + rank;
        __syncwarp();
        if (key >= 0 && leader) cur[key] += __popc(peers);
      }
      __syncthreads();
    }
    if (key >= 0) pb[pos] = j;
  }
}

constexpr int kMergeWarpMax = 128;

// Groups of more than kMergeWarpMax members (this launch skips the others),
// one CTA per group with the member layout of group_merge_kernel in each of
// its eight warps (32 members in flight); the warps' partial sums are added in
// warp order, so the result does not depend on scheduling.
__global__ void __launch_bounds__(256) group_merge_cta_kernel(const bf16* K, const int* anchors, const int* perm,
                                                              const int* goff, const float* logphi, float lambda_m,
                                                              float* C_k, int T, int t) {
  const int b = blockIdx.y, r = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int* pb = perm + (long long)b * T;
  const int* gb = goff + (long long)b * (t + 1);
  const float* lp = logphi + (long long)b * T;
  const bf16* Kb = K + (long long)b * T * 128;
  const int beg = gb[r], end = gb[r + 1];
  if (end - beg <= kMergeWarpMax) return;
  __shared__ float red[8][129];
  __shared__ float gmax_s[8];
  float gm = -INFINITY;
  for (int q = beg + threadIdx.x; q < end; q += 256) gm = fmaxf(gm, lp[pb[q]]);
  gm = warp_max(gm);
  if (lane == 0) gmax_s[warp] = gm;
  __syncthreads();
  gm = gmax_s[0];
  for (int w = 1; w < 8; ++w) gm = fmaxf(gm, gmax_s[w]);
  const int slot = lane >> 3, d0 = (lane & 7) * 16;
  float acc[16], ws = 0.f;
#pragma unroll
  for (int e = 0; e < 16; ++e) acc[e] = 0.f;
  for (int q = beg + warp * 4 + slot; q < end; q += 32) {
    const int j = pb[q];
    const float om = ex2_approx((lp[j] - gm) * kLog2e);
    const uint4* src = (const uint4*)(Kb + (long long)j * 128 + d0);
    const uint4 u0 = src[0], u1 = src[1];
    const __nv_bfloat162* h0 = (const __nv_bfloat162*)&u0;
    const __nv_bfloat162* h1 = (const __nv_bfloat162*)&u1;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 f0 = __bfloat1622float2(h0[e]), f1 = __bfloat1622float2(h1[e]);
      acc[2 * e] = fmaf(om, f0.x, acc[2 * e]);
      acc[2 * e + 1] = fmaf(om, f0.y, acc[2 * e + 1]);
      acc[8 + 2 * e] = fmaf(om, f1.x, acc[8 + 2 * e]);
      acc[8 + 2 * e + 1] = fmaf(om, f1.y, acc[8 + 2 * e + 1]);
    }
    ws += om;
  }
#pragma unroll
  for (int o = 8; o < 32; o <<= 1) {
#pragma unroll
    for (int e = 0; e < 16; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);
    ws += __shfl_xor_sync(0xffffffffu, ws, o);
  }
  if (lane < 8) {
#pragma unroll
    for (int e = 0; e < 16; ++e) red[warp][d0 + e] = acc[e];
    if (lane == 0) red[warp][128] = ws;
  }
  __syncthreads();
  if (threadIdx.x >= 128) return;
  const int dcol = threadIdx.x;
  float a = 0.f, wsum = 0.f;
  for (int w = 0; w < 8; ++w) {
    a += red[w][dcol];
    wsum += red[w][128];
  }
  const int s = anchors[(long long)b * t + r];
  const float k = to_f32(Kb[(long long)s * 128 + dcol]);
  C_k[((long long)b * t + r) * 128 + dcol] = fmaf(lambda_m, a * (1.0f / wsum) - k, k);
}

// Groups of up to kMergeWarpMax members, one warp per group r:
// mu_r = sum_{G_r} w_j k_j / sum_{G_r} w_j with
// w_j = e^{log phi_j - max_{G_r} log phi} (Eq. mass_centroid).  The members
// j = perm[goff[r] .. goff[r+1]) are read four at a time (eight lanes per
// member, sixteen dimensions per lane, two 16-byte loads); each of the four
// member slots sums its members in ascending order and the slots are combined
// by a fixed shuffle tree, so the result does not depend on scheduling.
// c_r = k_{s_r} + lambda_m (mu_r - k_{s_r}), which is (1 - lambda_m) k_{s_r} +
// lambda_m mu_r of Eq. key_merge.  Groups hold ~10 members, so one warp per
// group avoids the block barriers and idle warps of a CTA per group.
__global__ void __launch_bounds__(256) group_merge_kernel(const bf16* K, const int* anchors, const int* perm,
                                                          const int* goff, const float* logphi, float lambda_m,
                                                          float* C_k, int T, int t) {
  const int b = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * 8 + warp;
  if (r >= t) return;
  const int* pb = perm + (long long)b * T;
  const int* gb = goff + (long long)b * (t + 1);
  const float* lp = logphi + (long long)b * T;
  const bf16* Kb = K + (long long)b * T * 128;
  const int beg = gb[r], end = gb[r + 1];
  if (end - beg > kMergeWarpMax) return;   // group_merge_cta_kernel
  float gm = -INFINITY;
  for (int q = beg + lane; q < end; q += 32) gm = fmaxf(gm, lp[pb[q]]);
  gm = warp_max(gm);
  const int slot = lane >> 3, d0 = (lane & 7) * 16;
  float acc[16], ws = 0.f;
#pragma unroll
  for (int e = 0; e < 16; ++e) acc[e] = 0.f;
  for (int q = beg + slot; q < end; q += 4) {
    const int j = pb[q];
    const float om = ex2_approx((lp[j] - gm) * kLog2e);
    const uint4* src = (const uint4*)(Kb + (long long)j * 128 + d0);
    const uint4 u0 = src[0], u1 = src[1];
    const __nv_bfloat162* h0 = (const __nv_bfloat162*)&u0;
    const __nv_bfloat162* h1 = (const __nv_bfloat162*)&u1;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 f0 = __bfloat1622float2(h0[e]), f1 = __bfloat1622float2(h1[e]);
      acc[2 * e] = fmaf(om, f0.x, acc[2 * e]);
      acc[2 * e + 1] = fmaf(om, f0.y, acc[2 * e + 1]);
      acc[8 + 2 * e] = fmaf(om, f1.x, acc[8 + 2 * e]);
      acc[8 + 2 * e + 1] = fmaf(om, f1.y, acc[8 + 2 * e + 1]);
    }
    ws += om;
  }
#pragma unroll
  for (int o = 8; o < 32; o <<= 1) {
#pragma unroll
    for (int e = 0; e < 16; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);
    ws += __shfl_xor_sync(0xffffffffu, ws, o);
  }
  if (lane < 8) {
    const int s = anchors[(long long)b * t + r];
    const float inv = 1.0f / ws;
    const bf16* ks = Kb + (long long)s * 128 + d0;
    float* dst = C_k + ((long long)b * t + r) * 128 + d0;
#pragma unroll
    for (int e = 0; e < 16; e += 4) {
      float o4[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float k = to_f32(ks[e + u]);
        o4[u] = fmaf(lambda_m, acc[e + u] * inv - k, k);
      }
      *(float4*)(dst + e) = make_float4(o4[0], o4[1], o4[2], o4[3]);
    }
  }
}

int launch_merge(const Dims& D, float lambda_m, const bf16* K, const int* anchors, const int* kappa,
                 const float* logphi, int* perm, int* goff, int* cursor, float* C_k, cudaStream_t st) {
  int nl = 2;
  const int C = cdiv(D.T, kSortChunk), hb = (int)cdiv((long long)D.H * D.t, 256);
  const int hsm = D.t * (int)sizeof(int);
  if (sort_chunked(D.T, D.t) && set_dyn_smem((const void*)sort_hist_kernel, hsm) == cudaSuccess &&
      set_dyn_smem((const void*)sort_scatter_kernel, hsm) == cudaSuccess) {
    // cursor: the chunk counts [H][t][C], then the group totals [H][t]
    int* tot = cursor + (long long)D.H * D.t * C;
    sort_hist_kernel<<<dim3(C, D.H), 1024, hsm, st>>>(kappa, D.T, D.t, C, cursor);
    sort_totals_kernel<<<hb, 256, 0, st>>>(cursor, D.t, C, D.H, tot);
    sort_scan_kernel<<<D.H, 1024, 0, st>>>(tot, D.t, goff);
    sort_slots_kernel<<<hb, 256, 0, st>>>(cursor, goff, D.t, C, D.H);
    sort_scatter_kernel<<<dim3(C, D.H), 1024, hsm, st>>>(kappa, D.T, D.t, C, cursor, perm);
    nl += 5;
  } else {
    group_sort_kernel<<<D.H, 1024, 0, st>>>(kappa, D.T, D.t, perm, goff, cursor);
    ++nl;
  }
  group_merge_kernel<<<dim3(cdiv(D.t, 8), D.H), 256, 0, st>>>(K, anchors, perm, goff, logphi, lambda_m, C_k, D.T,
                                                              D.t);
  group_merge_cta_kernel<<<dim3(D.t, D.H), 256, 0, st>>>(K, anchors, perm, goff, logphi, lambda_m, C_k, D.T, D.t);
  return nl;
}

}  // namespace arckv
