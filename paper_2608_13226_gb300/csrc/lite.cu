// K6-K8: CoverPrune-Lite (Sec. 4.1, Eqs. lite_group, lite_select; Sec. 4.2,
// Eqs. blk_plan, blk_ot).
#include "common.cuh"
#include "bf16_dot.cuh"

namespace cp {

// Spread the low 10 bits of q so that bit i lands on bit 3i.
__device__ __forceinline__ uint32_t spread3(uint32_t q) {
  q &= 0x3FFu;
  q = (q | (q << 16)) & 0x030000FFu;
  q = (q | (q << 8)) & 0x0300F00Fu;
  q = (q | (q << 4)) & 0x030C30C3u;
  q = (q | (q << 2)) & 0x09249249u;
  return q;
}

// Voxel cell of one coordinate: floor((x - lo) / voxel) in fp32 with each
// operation rounded once, clamped to [0, 1023].
__device__ __forceinline__ uint32_t voxel_cell(float x, float lo, float voxel) {
  float cell = floorf(__fdiv_rn(__fsub_rn(x, lo), voxel));
  cell = fminf(fmaxf(cell, 0.0f), 1023.0f);
  return (uint32_t)cell;
}

// K6: Morton code per token and the order by (code, index).  One block per
// scene; the (code, index) keys are sorted bitonically in shared memory.
__global__ void __launch_bounds__(1024) k_morton(const float* __restrict__ pos_all,
                                                 const SceneStats* __restrict__ stats, float voxel,
                                                 int N, int L, int32_t* __restrict__ perm_all) {
  extern __shared__ unsigned long long mk[];  // [L]
  const int b = blockIdx.x;
  const float* X = pos_all + (size_t)b * N * 3;
  const float lx = stats[b].bbox_min[0], ly = stats[b].bbox_min[1], lz = stats[b].bbox_min[2];
  for (int j = threadIdx.x; j < L; j += blockDim.x) {
    if (j < N) {
      const uint32_t code = spread3(voxel_cell(X[3 * j], lx, voxel)) |
                            (spread3(voxel_cell(X[3 * j + 1], ly, voxel)) << 1) |
                            (spread3(voxel_cell(X[3 * j + 2], lz, voxel)) << 2);
      mk[j] = ((unsigned long long)code << 32) | (uint32_t)j;
    } else {
      mk[j] = ~0ull;
    }
  }
  __syncthreads();
  for (int size = 2; size <= L; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < (L >> 1); i += blockDim.x) {
        const int a = 2 * i - (i & (stride - 1));
        const int c = a + stride;
        const bool up = (a & size) == 0;
        const unsigned long long x = mk[a], y = mk[c];
        if ((x > y) == up) { mk[a] = y; mk[c] = x; }
      }
      __syncthreads();
    }
  }
  for (int p = threadIdx.x; p < N; p += blockDim.x)
    perm_all[(size_t)b * N + p] = (int32_t)(mk[p] & 0xFFFFFFFFull);
}

int launch_morton(const float* pos, const SceneStats* stats, const DevParams& P, int64_t B, int64_t N,
                  int32_t* perm, cudaStream_t s) {
  int L = 2;
  while (L < N) L <<= 1;
  const size_t smem = sizeof(unsigned long long) * (size_t)L;
  if (smem > 48 * 1024 &&
      cuda_status(cudaFuncSetAttribute(k_morton, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem),
                  "launch_morton: smem attribute") != CP_OK)
    return CP_ECUDA;
  k_morton<<<(unsigned)B, 1024, smem, s>>>(pos, stats, P.voxel, (int)N, L, perm);
  return last_launch_status();
}

// Block-wide inclusive scans over blockDim.x == 1024 values.
__device__ __forceinline__ unsigned long long block_incl_sum_u64(unsigned long long x,
                                                                 unsigned long long* s_w,
                                                                 unsigned long long* total) {
  const int l = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    unsigned long long y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (l >= o) x += y;
  }
  if (l == 31) s_w[w] = x;
  __syncthreads();
  if (w == 0) {
    unsigned long long y = s_w[l];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      unsigned long long z = __shfl_up_sync(0xFFFFFFFFu, y, o);
      if (l >= o) y += z;
    }
    s_w[l] = y;
  }
  __syncthreads();
  const unsigned long long r = x + (w > 0 ? s_w[w - 1] : 0ull);
  *total = s_w[31];
  __syncthreads();
  return r;
}

__device__ __forceinline__ int block_incl_max_int(int x, int* s_w, int* total) {
  const int l = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (l >= o) x = max(x, y);
  }
  if (l == 31) s_w[w] = x;
  __syncthreads();
  if (w == 0) {
    int y = s_w[l];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int z = __shfl_up_sync(0xFFFFFFFFu, y, o);
      if (l >= o) y = max(y, z);
    }
    s_w[l] = y;
  }
  __syncthreads();
  const int r = w > 0 ? max(x, s_w[w - 1]) : x;
  *total = s_w[31];
  __syncthreads();
  return r;
}

// K7: capacity-guided grouping of Eq. lite_group in exact integers.
//   Q_j = rint(v_j 2^40); P(p) = inclusive running mass in Morton order;
//   ideal start of group q >= 1: 1 + min{p : P(p) K >= q P(N-1)};
//   b_q = q + min(N - K, max_{q' <= q} (ideal_q' - q')), b_0 = 0, b_K = N.
// One block of 1024 threads per scene.
__global__ void __launch_bounds__(1024) k_groups(const float* __restrict__ v_all,
                                                 const int32_t* __restrict__ perm_all, int N, int K,
                                                 unsigned long long* __restrict__ prefix_all,
                                                 int32_t* __restrict__ gs_all) {
  __shared__ unsigned long long s_w[32];
  __shared__ int s_wi[32];
  const int b = blockIdx.x;
  const float* v = v_all + (size_t)b * N;
  const int32_t* perm = perm_all + (size_t)b * N;
  unsigned long long* P = prefix_all + (size_t)b * N;
  int32_t* gs = gs_all + (size_t)b * (K + 1);
  unsigned long long carry = 0ull;
  for (int c0 = 0; c0 < N; c0 += 1024) {
    const int p = c0 + threadIdx.x;
    unsigned long long q = 0ull;
    if (p < N) {
      const float vj = v[perm[p]];
      q = vj > 0.0f ? __double2ull_rn((double)vj * 1099511627776.0) : 0ull;  // 2^40
    }
    unsigned long long tot;
    const unsigned long long incl = block_incl_sum_u64(q, s_w, &tot);
    if (p < N) P[p] = carry + incl;
    carry += tot;
  }
  __syncthreads();
  const unsigned long long total = carry;
  // ideal_q - q for q = 1..K-1, staged in gs[q]
  for (int q = 1 + threadIdx.x; q < K; q += 1024) {
    const unsigned __int128 target = (unsigned __int128)q * total;
    int lo = 0, hi = N - 1;  // smallest p with P[p] * K >= target (exists: P[N-1]*K >= target)
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if ((unsigned __int128)__ldcg(P + mid) * (unsigned)K >= target) hi = mid; else lo = mid + 1;
    }
    gs[q] = (lo + 1) - q;
  }
  __syncthreads();
  int run = INT32_MIN;
  for (int c0 = 1; c0 < K; c0 += 1024) {
    const int q = c0 + threadIdx.x;
    const int d = q < K ? gs[q] : INT32_MIN;
    int tot;
    const int m = max(run, block_incl_max_int(d, s_wi, &tot));
    if (q < K) gs[q] = q + min(N - K, m);
    run = max(run, tot);
  }
  if (threadIdx.x == 0) {
    gs[0] = 0;
    gs[K] = N;
  }
}

int launch_groups(const float* v, const int32_t* perm, int64_t B, int64_t N, int64_t K,
                  uint64_t* prefix, int32_t* gs, cudaStream_t s) {
  k_groups<<<(unsigned)B, 1024, 0, s>>>(v, perm, (int)N, (int)K,
                                        reinterpret_cast<unsigned long long*>(prefix), gs);
  return last_launch_status();
}

// K8: prototype of each group (Eq. lite_select):
//   s_q = argmin_{t in G_q} sum_{j in G_q} v_j C(t, j), lowest index on ties,
// with C exactly as in the cost kernels.
//
// Scores of the members a = w, w + nwarps, ... of a group (warp w), each a
// full-width dot product per pair; the sum over targets runs in group
// order.  Keeps the warp's best (score, token).
template <typename T>
__device__ __forceinline__ void lite_proto_simt(const T* F, const float* inv, const float* X,
                                                const int32_t* TAU, const float* v,
                                                const int32_t* mem, int sz, const SceneNorms& nm,
                                                const DevParams& P, int D, int w, int lane,
                                                int nwarps, float& best, int& best_t) {
  constexpr int V = Vec16<T>::n;
  for (int a = w; a < sz; a += nwarps) {
    const int t = mem[a];
    const T* ft = F + (size_t)t * D;
    const float xt = X[3 * t], yt = X[3 * t + 1], zt = X[3 * t + 2];
    const int tt = TAU[t];
    const float inv_t = inv[t];
    float sc = 0.0f;
    for (int c = 0; c < sz; ++c) {
      const int j = mem[c];
      const T* fj = F + (size_t)j * D;
      float dot = 0.0f;
      for (int d = lane * V; d < D; d += 32 * V) {
        float x[V], y[V];
        Vec16<T>::load(ft + d, x);
        Vec16<T>::load(fj + d, y);
#pragma unroll
        for (int i = 0; i < V; ++i) dot = fmaf(x[i], y[i], dot);
      }
      dot = warp_sum(dot);
      float cosv = clamp_cos(dot * inv_t * inv[j]);
      if (t == j && inv_t > 0.0f) cosv = 1.0f;
      const float d2 = sqdist_rn(xt, yt, zt, X[3 * j], X[3 * j + 1], X[3 * j + 2]);
      sc += v[j] * fst_cost_from(cosv, d2, tt, TAU[j], nm, P);
    }
    if (sc < best || (sc == best && t < best_t)) {
      best = sc;
      best_t = t;
    }
  }
}

// One block per group, one warp per candidate (fp32 features, and bf16
// groups of more than LP_MAXG members).
template <typename T>
__global__ void __launch_bounds__(256) k_lite_proto(
    const T* __restrict__ F_all, const float* __restrict__ inv_all, const float* __restrict__ pos_all,
    const int32_t* __restrict__ frame_all, const SceneNorms* __restrict__ norms,
    const float* __restrict__ v_all, const int32_t* __restrict__ perm_all,
    const int32_t* __restrict__ gs_all, DevParams P, int N, int D, int K,
    int32_t* __restrict__ proto, double* __restrict__ score) {
  const int q = blockIdx.x, b = blockIdx.y;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int32_t* gs = gs_all + (size_t)b * (K + 1);
  const int sz = gs[q + 1] - gs[q];
  float best = INFINITY;
  int best_t = INT32_MAX;
  lite_proto_simt<T>(F_all + (size_t)b * N * D, inv_all + (size_t)b * N,
                     pos_all + (size_t)b * N * 3, frame_all + (size_t)b * N,
                     v_all + (size_t)b * N, perm_all + (size_t)b * N + gs[q], sz, norms[b], P, D,
                     w, lane, 8, best, best_t);
  __shared__ float s_sc[8];
  __shared__ int s_t[8];
  if (lane == 0) {
    s_sc[w] = best;
    s_t[w] = best_t;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 1; i < 8; ++i)
      if (s_sc[i] < best || (s_sc[i] == best && s_t[i] < best_t)) {
        best = s_sc[i];
        best_t = s_t[i];
      }
    proto[(size_t)b * K + q] = best_t;
    score[(size_t)b * K + q] = (double)best;
  }
}

// bf16 features: the group's feature Gram on the tensor cores (mma.sync
// m16n8k16, fp32 accumulate).  Members are taken in 16-row blocks and the
// 16 x 16 tiles (bi <= bj) of X X^T are computed one after the other, the
// feature width split over the block's 4 warps (warp w takes the 32-column
// chunks w, w + 4, ...) and the four partial tiles added in warp order.  In
// a chunk each lane loads 16 bytes of each of its rows (columns 8 (lane %
// 4) ..): those 8 values feed two k16 steps, the columns' order along k
// being the same for A and for B, so the dot products are unchanged.  A
// block against itself reuses its A registers as B.  The tiles land, both
// ways for bi < bj, in a shared-memory Gram, from which the scores read
// every pair's dot product once.  Groups of more than LP_MAXG members
// (rare: capacity-balanced groups are small) take the full-width loop.
constexpr int LP_MAXG = 64, LP_WARPS = 4;
__device__ __forceinline__ uint4 ld_row16(const __nv_bfloat16* row, int col, int D) {
  return (row != nullptr && col < D) ? __ldg(reinterpret_cast<const uint4*>(row + col))
                                     : make_uint4(0u, 0u, 0u, 0u);
}
// ld_row16 as an asynchronous copy into shared memory (zeros where it gives
// zeros: no bytes are read then, and F itself stands in as the source)
__device__ __forceinline__ void cp_row16(uint4* dst, const __nv_bfloat16* row, int col, int D,
                                         const void* any) {
  const bool ok = row != nullptr && col < D;
  cp_async16_zfill(dst, ok ? (const void*)(row + col) : any, ok);
}
constexpr int LP_STAGES = 4;  // chunks of a warp in flight (diagonal tiles)
__global__ void __launch_bounds__(32 * LP_WARPS) k_lite_proto_tc(
    const __nv_bfloat16* __restrict__ F_all, const float* __restrict__ inv_all,
    const float* __restrict__ pos_all, const int32_t* __restrict__ frame_all,
    const SceneNorms* __restrict__ norms, const float* __restrict__ v_all,
    const int32_t* __restrict__ perm_all, const int32_t* __restrict__ gs_all, DevParams P, int N,
    int D, int K, int32_t* __restrict__ proto, double* __restrict__ score) {
  __shared__ float s_dot[LP_MAXG][LP_MAXG + 1];
  __shared__ float s_part[LP_WARPS][16][17];
  // diagonal tiles: each lane's two 16-byte pieces of a chunk, LP_STAGES deep
  __shared__ __align__(16) uint4 s_stg[LP_WARPS][LP_STAGES][2][32];
  __shared__ float s_inv[LP_MAXG], s_v[LP_MAXG], s_x[LP_MAXG][3];
  __shared__ int s_mem[LP_MAXG], s_tau[LP_MAXG];
  __shared__ float s_sc[LP_WARPS];
  __shared__ int s_t[LP_WARPS];
  const int q = blockIdx.x, b = blockIdx.y;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const __nv_bfloat16* F = F_all + (size_t)b * N * D;
  const float* inv = inv_all + (size_t)b * N;
  const float* X = pos_all + (size_t)b * N * 3;
  const int32_t* TAU = frame_all + (size_t)b * N;
  const float* v = v_all + (size_t)b * N;
  const int32_t* gs = gs_all + (size_t)b * (K + 1);
  const int32_t* mem = perm_all + (size_t)b * N + gs[q];
  const int sz = gs[q + 1] - gs[q];
  const SceneNorms nm = norms[b];
  float best = INFINITY;
  int best_t = INT32_MAX;
  if (sz > LP_MAXG) {
    lite_proto_simt<__nv_bfloat16>(F, inv, X, TAU, v, mem, sz, nm, P, D, w, lane, LP_WARPS, best,
                                   best_t);
  } else {
    for (int a = threadIdx.x; a < sz; a += blockDim.x) {
      const int t = mem[a];
      s_mem[a] = t;
      s_inv[a] = inv[t];
      s_v[a] = v[t];
      s_x[a][0] = X[3 * t];
      s_x[a][1] = X[3 * t + 1];
      s_x[a][2] = X[3 * t + 2];
      s_tau[a] = TAU[t];
    }
    __syncthreads();
    const int g = lane >> 2, tg = lane & 3;
    const int nb = (sz + 15) >> 4;
    for (int bi = 0; bi < nb; ++bi) {
      for (int bj = bi; bj < nb; ++bj) {
        const int ra0 = 16 * bi + g, ra1 = ra0 + 8, rb0 = 16 * bj + g, rb1 = rb0 + 8;
        const __nv_bfloat16* pa0 = ra0 < sz ? F + (size_t)s_mem[ra0] * D : nullptr;
        const __nv_bfloat16* pa1 = ra1 < sz ? F + (size_t)s_mem[ra1] * D : nullptr;
        const __nv_bfloat16* pb0 = rb0 < sz ? F + (size_t)s_mem[rb0] * D : nullptr;
        const __nv_bfloat16* pb1 = rb1 < sz ? F + (size_t)s_mem[rb1] * D : nullptr;
        float d0[4] = {0.f, 0.f, 0.f, 0.f}, d1[4] = {0.f, 0.f, 0.f, 0.f};
        if (bi == bj) {
          // diagonal tile (B rows are A's): the same chunks and MMAs as the
          // loop below, the rows brought in by asynchronous copies
          // LP_STAGES chunks ahead (each lane reads back only its own copies)
          const int nch = (D - 32 * w + 32 * LP_WARPS - 1) / (32 * LP_WARPS);
          auto issue = [&](int i) {
            const int col = 32 * w + 32 * LP_WARPS * i + 8 * tg;
            cp_row16(&s_stg[w][i % LP_STAGES][0][lane], pa0, col, D, F);
            cp_row16(&s_stg[w][i % LP_STAGES][1][lane], pa1, col, D, F);
          };
#pragma unroll
          for (int i = 0; i < LP_STAGES - 1; ++i) {
            if (i < nch) issue(i);
            cp_commit();
          }
          for (int i = 0; i < nch; ++i) {
            if (i + LP_STAGES - 1 < nch) issue(i + LP_STAGES - 1);
            cp_commit();
            cp_wait<LP_STAGES - 1>();  // chunk i has landed
            const uint4 x0 = s_stg[w][i % LP_STAGES][0][lane];
            const uint4 x1 = s_stg[w][i % LP_STAGES][1][lane];
            mma_bf16_16816(d0, x0.x, x1.x, x0.y, x1.y, x0.x, x0.y);
            mma_bf16_16816(d1, x0.x, x1.x, x0.y, x1.y, x1.x, x1.y);
            mma_bf16_16816(d0, x0.z, x1.z, x0.w, x1.w, x0.z, x0.w);
            mma_bf16_16816(d1, x0.z, x1.z, x0.w, x1.w, x1.z, x1.w);
          }
          cp_wait<0>();
        }
        // off-diagonal tiles (groups of more than 16): A and B rows loaded
#pragma unroll 2
        for (int c0 = 32 * w; bi != bj && c0 < D; c0 += 32 * LP_WARPS) {
          const int col = c0 + 8 * tg;
          const uint4 x0 = ld_row16(pa0, col, D), x1 = ld_row16(pa1, col, D);
          const uint4 y0 = ld_row16(pb0, col, D), y1 = ld_row16(pb1, col, D);
          // k16 step over columns 8 tg + {0..3} of every lane, then + {4..7}
          mma_bf16_16816(d0, x0.x, x1.x, x0.y, x1.y, y0.x, y0.y);
          mma_bf16_16816(d1, x0.x, x1.x, x0.y, x1.y, y1.x, y1.y);
          mma_bf16_16816(d0, x0.z, x1.z, x0.w, x1.w, y0.z, y0.w);
          mma_bf16_16816(d1, x0.z, x1.z, x0.w, x1.w, y1.z, y1.w);
        }
        // d0: tile rows g (d0[0..1]) and g + 8 (d0[2..3]), columns 2 tg + {0, 1};
        // d1: the same rows, columns 8 + 2 tg + {0, 1}
        s_part[w][g][2 * tg] = d0[0];
        s_part[w][g][2 * tg + 1] = d0[1];
        s_part[w][g + 8][2 * tg] = d0[2];
        s_part[w][g + 8][2 * tg + 1] = d0[3];
        s_part[w][g][8 + 2 * tg] = d1[0];
        s_part[w][g][9 + 2 * tg] = d1[1];
        s_part[w][g + 8][8 + 2 * tg] = d1[2];
        s_part[w][g + 8][9 + 2 * tg] = d1[3];
        __syncthreads();
        for (int e = threadIdx.x; e < 256; e += blockDim.x) {
          const int r = e >> 4, c = e & 15;
          const int rr = 16 * bi + r, cc = 16 * bj + c;
          if (rr < sz && cc < sz) {
            const float x = ((s_part[0][r][c] + s_part[1][r][c]) + s_part[2][r][c]) +
                            s_part[3][r][c];
            s_dot[rr][cc] = x;
            if (bi != bj) s_dot[cc][rr] = x;
          }
        }
        __syncthreads();  // s_part is reused by the next tile
      }
    }
    for (int a = w; a < sz; a += LP_WARPS) {
      const int t = s_mem[a];
      const float inv_t = s_inv[a];
      float sc = 0.0f;
      for (int c = lane; c < sz; c += 32) {
        float cosv = clamp_cos(s_dot[a][c] * inv_t * s_inv[c]);
        if (c == a && inv_t > 0.0f) cosv = 1.0f;
        const float d2 = sqdist_rn(s_x[a][0], s_x[a][1], s_x[a][2], s_x[c][0], s_x[c][1],
                                   s_x[c][2]);
        sc += s_v[c] * fst_cost_from(cosv, d2, s_tau[a], s_tau[c], nm, P);
      }
      sc = warp_sum(sc);
      if (sc < best || (sc == best && t < best_t)) {
        best = sc;
        best_t = t;
      }
    }
  }
  if (lane == 0) {
    s_sc[w] = best;
    s_t[w] = best_t;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 1; i < LP_WARPS; ++i)
      if (s_sc[i] < best || (s_sc[i] == best && s_t[i] < best_t)) {
        best = s_sc[i];
        best_t = s_t[i];
      }
    proto[(size_t)b * K + q] = best_t;
    score[(size_t)b * K + q] = (double)best;
  }
}

// Lite objective: sum of the group scores, fp64, fixed order.
__global__ void __launch_bounds__(256) k_sum_scores(const double* __restrict__ score, int K,
                                                    double* __restrict__ objective) {
  const int b = blockIdx.x;
  double acc = 0.0;
  for (int q = threadIdx.x; q < K; q += blockDim.x) acc += score[(size_t)b * K + q];
  acc = warp_sum(acc);
  __shared__ double s[8];
  if ((threadIdx.x & 31) == 0) s[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int i = 0; i < 8; ++i) t += s[i];
    objective[b] = t;
  }
}

int launch_lite_proto(const void* feats, int dtype, const float* inv, const float* pos,
                      const int32_t* frame, const SceneNorms* norms, const float* v,
                      const int32_t* perm, const int32_t* gs, const DevParams& P, int64_t B,
                      int64_t N, int64_t D, int64_t K, int32_t* proto, double* score,
                      double* objective, cudaStream_t s) {
  dim3 grid((unsigned)K, (unsigned)B);
  if (dtype == CP_BF16)
    k_lite_proto_tc<<<grid, 32 * LP_WARPS, 0, s>>>((const __nv_bfloat16*)feats, inv, pos, frame,
                                                   norms, v, perm, gs, P, (int)N, (int)D, (int)K,
                                                   proto, score);
  else
    k_lite_proto<float><<<grid, 256, 0, s>>>((const float*)feats, inv, pos, frame, norms, v, perm,
                                             gs, P, (int)N, (int)D, (int)K, proto, score);
  int st = last_launch_status();
  if (st != CP_OK || !objective) return st;
  k_sum_scores<<<(unsigned)B, 256, 0, s>>>(score, (int)K, objective);
  return last_launch_status();
}

}  // namespace cp
