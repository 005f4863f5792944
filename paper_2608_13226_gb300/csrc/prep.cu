// K0 (scene statistics, inverse feature norms), K1 (3D nearest neighbours and
// scene diameter) and the min-max normalisers of Sec. 3.3.
#include "common.cuh"
#include "bf16_dot.cuh"

namespace cp {

// ---------------------------------------------------------------------------
// K0a: frame range (0 when frame is NULL) and bounding-box minimum per scene;
// initialises the fields that later kernels reduce into atomically.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(512) k_scene_stats(const float* __restrict__ pos,
                                                     const int32_t* __restrict__ frame,
                                                     int N, SceneStats* stats) {
  const int b = blockIdx.x;
  const float* X = pos + (size_t)b * N * 3;
  const int32_t* T = frame ? frame + (size_t)b * N : nullptr;  // may be absent
  int tmin = INT32_MAX, tmax = INT32_MIN;
  float lo[3] = {INFINITY, INFINITY, INFINITY};
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    const int t = T ? T[j] : 0;
    tmin = min(tmin, t);
    tmax = max(tmax, t);
#pragma unroll
    for (int a = 0; a < 3; ++a) lo[a] = fminf(lo[a], X[3 * j + a]);
  }
  __shared__ int s_tmin[16], s_tmax[16];
  __shared__ float s_lo[3][16];
  for (int o = 16; o > 0; o >>= 1) {
    tmin = min(tmin, __shfl_xor_sync(0xFFFFFFFFu, tmin, o));
    tmax = max(tmax, __shfl_xor_sync(0xFFFFFFFFu, tmax, o));
#pragma unroll
    for (int a = 0; a < 3; ++a) lo[a] = fminf(lo[a], __shfl_xor_sync(0xFFFFFFFFu, lo[a], o));
  }
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  if (l == 0) {
    s_tmin[w] = tmin;
    s_tmax[w] = tmax;
    for (int a = 0; a < 3; ++a) s_lo[a][w] = lo[a];
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const int nw = blockDim.x >> 5;
    for (int i = 1; i < nw; ++i) {
      tmin = min(tmin, s_tmin[i]);
      tmax = max(tmax, s_tmax[i]);
      for (int a = 0; a < 3; ++a) lo[a] = fminf(lo[a], s_lo[a][i]);
    }
    SceneStats st;
    st.cos_max_key = 0u;           // below every real key
    st.cos_min_key = 0xFFFFFFFFu;  // above every real key
    st.d2_max_bits = 0u;           // d^2 >= 0: float bits order like the values
    st.tau_min = tmin;
    st.tau_max = tmax;
    for (int a = 0; a < 3; ++a) st.bbox_min[a] = lo[a];
    for (int i = 0; i < 8; ++i) st.pad[i] = 0u;
    stats[b] = st;
  }
}

int launch_scene_stats(const float* pos, const int32_t* frame, int64_t B, int64_t N,
                       SceneStats* stats, cudaStream_t s) {
  k_scene_stats<<<(unsigned)B, 512, 0, s>>>(pos, frame, (int)N, stats);
  return last_launch_status();
}

// ---------------------------------------------------------------------------
// K0b: inv[j] = 1 / ||f_j|| (0 for a zero feature), one warp per token.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) k_inv_norms(const T* __restrict__ F,
                                                   const float* __restrict__ pos, int64_t rows,
                                                   int D, float* __restrict__ inv,
                                                   float4* __restrict__ tok) {
  const int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const T* f = F + row * D;
  constexpr int V = Vec16<T>::n;
  float acc = 0.0f;
  if constexpr (V == 8) {  // bf16: the same products and order, no widening
    for (int d = lane * V; d < D; d += 32 * V) {
      const uint4 x = __ldg(reinterpret_cast<const uint4*>(f + d));
      acc = dot8_bf16(x, x, acc);
    }
  } else {
    for (int d = lane * V; d < D; d += 32 * V) {
      float x[V];
      Vec16<T>::load(f + d, x);
#pragma unroll
      for (int i = 0; i < V; ++i) acc = fmaf(x[i], x[i], acc);
    }
  }
  acc = warp_sum(acc);
  if (lane == 0) {
    const float iv = acc > 0.0f ? 1.0f / sqrtf(acc) : 0.0f;
    inv[row] = iv;
    if (tok) tok[row] = make_float4(pos[3 * row], pos[3 * row + 1], pos[3 * row + 2], iv);
  }
}

int launch_inv_norms(const void* feats, int dtype, const float* pos, int64_t B, int64_t N,
                     int64_t D, float* inv, float4* tok, cudaStream_t s) {
  const int64_t rows = B * N;
  const unsigned grid = (unsigned)((rows + 7) / 8);
  if (dtype == CP_BF16)
    k_inv_norms<__nv_bfloat16><<<grid, 256, 0, s>>>((const __nv_bfloat16*)feats, pos, rows,
                                                     (int)D, inv, tok);
  else
    k_inv_norms<float><<<grid, 256, 0, s>>>((const float*)feats, pos, rows, (int)D, inv, tok);
  return last_launch_status();
}

// ---------------------------------------------------------------------------
// K1: for token j, its kk nearest other tokens ordered by (fp32 d^2, index)
// (capacity set N_n of Eq. fst_capacity_score and SGS neighbourhood M_g of
// Eq. local_neighbor), and the largest squared distance of the row (for the
// spatial normaliser).  One block per token; the N keys live in shared
// memory; the kk-th smallest key is found by bisection on its bit pattern
// (d^2 >= 0, so float bits order like the values), the winners are collected
// in index order and sorted by (key, index).
// ---------------------------------------------------------------------------
constexpr int KNN_THREADS = 256;

__device__ __forceinline__ int block_sum_int(int v, int* s_red) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) s_red[w] = v;
  __syncthreads();
  int t = 0;
  for (int i = 0; i < KNN_THREADS / 32; ++i) t += s_red[i];
  return t;
}

__global__ void __launch_bounds__(KNN_THREADS) k_knn(const float* __restrict__ pos, int N, int kk,
                                                     int list_len, int32_t* __restrict__ nbr,
                                                     SceneStats* stats) {
  extern __shared__ __align__(16) unsigned char smem[];
  unsigned long long* list = reinterpret_cast<unsigned long long*>(smem);  // [list_len]
  uint32_t* key = reinterpret_cast<uint32_t*>(list + list_len);            // [N]
  __shared__ int s_red[KNN_THREADS / 32];
  __shared__ uint32_t s_redu[KNN_THREADS / 32];
  __shared__ int s_wcnt[2][KNN_THREADS / 32];

  const int j = blockIdx.x, b = blockIdx.y;
  const float* X = pos + (size_t)b * N * 3;
  const float xj = X[3 * j], yj = X[3 * j + 1], zj = X[3 * j + 2];
  uint32_t dmax = 0u;
  for (int k = threadIdx.x; k < N; k += KNN_THREADS) {
    float d2 = sqdist_rn(xj, yj, zj, X[3 * k], X[3 * k + 1], X[3 * k + 2]);
    uint32_t bits = __float_as_uint(d2);
    dmax = max(dmax, bits);
    key[k] = (k == j) ? 0xFFFFFFFFu : bits;
  }
  for (int o = 16; o > 0; o >>= 1) dmax = max(dmax, __shfl_xor_sync(0xFFFFFFFFu, dmax, o));
  if ((threadIdx.x & 31) == 0) s_redu[threadIdx.x >> 5] = dmax;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 1; i < KNN_THREADS / 32; ++i) dmax = max(dmax, s_redu[i]);
    atomicMax(&stats[b].d2_max_bits, dmax);
  }
  if (kk <= 0) return;

  // bisection: smallest T with #{key <= T} >= kk
  uint32_t lo = 0u, hi = 0xFFFFFFFEu;
  while (lo < hi) {
    const uint32_t mid = lo + ((hi - lo) >> 1);
    int c = 0;
    for (int k = threadIdx.x; k < N; k += KNN_THREADS) c += key[k] <= mid;
    c = block_sum_int(c, s_red);
    if (c >= kk) hi = mid; else lo = mid + 1;
  }
  const uint32_t T = lo;
  int less = 0;
  for (int k = threadIdx.x; k < N; k += KNN_THREADS) less += key[k] < T;
  less = block_sum_int(less, s_red);
  const int need_eq = kk - less;

  // collect in index order: every key < T, and the first need_eq keys == T
  for (int i = threadIdx.x; i < list_len; i += KNN_THREADS) list[i] = ~0ull;
  __syncthreads();
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  int base = 0, eq_taken = 0;
  for (int c0 = 0; c0 < N; c0 += KNN_THREADS) {
    const int k = c0 + threadIdx.x;
    const uint32_t kv = k < N ? key[k] : 0xFFFFFFFFu;
    const bool is_eq = kv == T && k < N;
    // rank among equal keys of this chunk, in index order
    const unsigned beq = __ballot_sync(0xFFFFFFFFu, is_eq);
    if (l == 0) s_wcnt[0][w] = __popc(beq);
    __syncthreads();
    int eq_before = 0, eq_total = 0;
    for (int i = 0; i < KNN_THREADS / 32; ++i) {
      eq_before += i < w ? s_wcnt[0][i] : 0;
      eq_total += s_wcnt[0][i];
    }
    const int rank_eq = eq_taken + eq_before + __popc(beq & ((1u << l) - 1u));
    const bool take = (kv < T && k < N) || (is_eq && rank_eq < need_eq);
    const unsigned bt = __ballot_sync(0xFFFFFFFFu, take);
    if (l == 0) s_wcnt[1][w] = __popc(bt);
    __syncthreads();
    int t_before = 0, t_total = 0;
    for (int i = 0; i < KNN_THREADS / 32; ++i) {
      t_before += i < w ? s_wcnt[1][i] : 0;
      t_total += s_wcnt[1][i];
    }
    if (take) {
      const int p = base + t_before + __popc(bt & ((1u << l) - 1u));
      list[p] = ((unsigned long long)kv << 32) | (unsigned)k;
    }
    base += t_total;
    eq_taken += eq_total;
    __syncthreads();
  }
  // bitonic sort of list[0, list_len) ascending by (key, index)
  for (int size = 2; size <= list_len; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < (list_len >> 1); i += KNN_THREADS) {
        const int a = 2 * i - (i & (stride - 1));
        const int c = a + stride;
        const bool up = (a & size) == 0;
        const unsigned long long x = list[a], y = list[c];
        if ((x > y) == up) { list[a] = y; list[c] = x; }
      }
      __syncthreads();
    }
  }
  int32_t* out = nbr + ((size_t)b * N + j) * kk;
  for (int q = threadIdx.x; q < kk; q += KNN_THREADS) out[q] = (int32_t)(list[q] & 0xFFFFFFFFu);
}

// K1 for kk <= 32: one warp per token.  Each lane scans every 32nd candidate
// and keeps its KK smallest (d^2 bits, index) keys in registers, sorted; the
// warp then merges the 32 lists by repeated warp-wide minimum.  The keys are
// the same total order as the block kernel's, so the lists are identical.
template <int KK>
__global__ void __launch_bounds__(256) k_knn_warp(const float* __restrict__ pos, int N, int kk,
                                                  int32_t* __restrict__ nbr, SceneStats* stats) {
  const int j = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int b = blockIdx.y;
  const int lane = threadIdx.x & 31;
  const float* X = pos + (size_t)b * N * 3;
  uint32_t dmax = 0u;
  if (j < N) {
    const float xj = X[3 * j], yj = X[3 * j + 1], zj = X[3 * j + 2];
    unsigned long long best[KK];
#pragma unroll
    for (int i = 0; i < KK; ++i) best[i] = ~0ull;
    for (int k = lane; k < N; k += 32) {
      const float d2 = sqdist_rn(xj, yj, zj, __ldg(X + 3 * k), __ldg(X + 3 * k + 1),
                                 __ldg(X + 3 * k + 2));
      const uint32_t bits = __float_as_uint(d2);
      dmax = max(dmax, bits);
      const unsigned long long key = ((unsigned long long)bits << 32) | (uint32_t)k;
      if (k != j && key < best[KK - 1]) {
        best[KK - 1] = key;
#pragma unroll
        for (int i = KK - 1; i > 0; --i) {
          if (best[i] < best[i - 1]) {
            const unsigned long long t = best[i];
            best[i] = best[i - 1];
            best[i - 1] = t;
          }
        }
      }
    }
    int32_t* out = nbr + ((size_t)b * N + j) * kk;
    for (int q = 0; q < kk; ++q) {
      const unsigned long long m = warp_min_u64(best[0]);
      if (lane == 0) out[q] = (int32_t)(m & 0xFFFFFFFFull);
      if (best[0] == m) {  // keys are unique: exactly one lane pops its head
#pragma unroll
        for (int i = 0; i < KK - 1; ++i) best[i] = best[i + 1];
        best[KK - 1] = ~0ull;
      }
    }
  }
  for (int o = 16; o > 0; o >>= 1) dmax = max(dmax, __shfl_xor_sync(0xFFFFFFFFu, dmax, o));
  __shared__ uint32_t s_dmax[8];
  if (lane == 0) s_dmax[threadIdx.x >> 5] = dmax;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t m = s_dmax[0];
    for (int i = 1; i < 8; ++i) m = max(m, s_dmax[i]);
    atomicMax(&stats[b].d2_max_bits, m);
  }
}

// K1 for kk <= 8, two tokens per warp, 16 per block: the block stages the
// candidate positions in shared-memory tiles of 2048 (from the float4 token
// table when one is given, else from the xyz array), so each position is
// read from L2 once per 16 query rows; the quick test on the d^2 bits skips
// the 64-bit key compare for almost every candidate.  Same keys, same lists
// as k_knn_warp.
constexpr int KNN_TILE = 2048;

template <int KK, bool TOK>
__global__ void __launch_bounds__(256) k_knn_pair(const float* __restrict__ pos,
                                                  const float4* __restrict__ tok, int N, int kk,
                                                  int32_t* __restrict__ nbr, SceneStats* stats) {
  __shared__ float4 s_p[KNN_TILE];
  const int j0 = (blockIdx.x * 8 + (threadIdx.x >> 5)) * 2;
  const int b = blockIdx.y;
  const int lane = threadIdx.x & 31;
  const float* X = pos + (size_t)b * N * 3;
  const float4* T = TOK ? tok + (size_t)b * N : nullptr;
  const bool active = j0 < N;
  const bool two = j0 + 1 < N;
  const int j1 = two ? j0 + 1 : j0;
  float ax = 0.f, ay = 0.f, az = 0.f, bx = 0.f, by = 0.f, bz = 0.f;
  if (active) {
    ax = X[3 * j0]; ay = X[3 * j0 + 1]; az = X[3 * j0 + 2];
    bx = X[3 * j1]; by = X[3 * j1 + 1]; bz = X[3 * j1 + 2];
  }
  uint32_t dmax = 0u;
  unsigned long long best0[KK], best1[KK];
#pragma unroll
  for (int i = 0; i < KK; ++i) best0[i] = best1[i] = ~0ull;
  for (int base = 0; base < N; base += KNN_TILE) {
    const int n = min(KNN_TILE, N - base);
    __syncthreads();  // the previous tile is consumed
    for (int i = threadIdx.x; i < n; i += 256) {
      if (TOK) {
        s_p[i] = __ldg(T + base + i);
      } else {
        const int k = base + i;
        s_p[i] = make_float4(__ldg(X + 3 * k), __ldg(X + 3 * k + 1), __ldg(X + 3 * k + 2), 0.f);
      }
    }
    __syncthreads();
    if (!active) continue;
    for (int i = lane; i < n; i += 32) {
      const int k = base + i;
      const float4 p = s_p[i];
      const uint32_t ba = __float_as_uint(sqdist_rn(ax, ay, az, p.x, p.y, p.z));
      const uint32_t bb = __float_as_uint(sqdist_rn(bx, by, bz, p.x, p.y, p.z));
      dmax = max(dmax, max(ba, bb));
      if (ba <= (uint32_t)(best0[KK - 1] >> 32) && k != j0) {
        const unsigned long long key = ((unsigned long long)ba << 32) | (uint32_t)k;
        if (key < best0[KK - 1]) {
          best0[KK - 1] = key;
#pragma unroll
          for (int t = KK - 1; t > 0; --t)
            if (best0[t] < best0[t - 1]) {
              const unsigned long long x = best0[t];
              best0[t] = best0[t - 1];
              best0[t - 1] = x;
            }
        }
      }
      if (bb <= (uint32_t)(best1[KK - 1] >> 32) && k != j1) {
        const unsigned long long key = ((unsigned long long)bb << 32) | (uint32_t)k;
        if (key < best1[KK - 1]) {
          best1[KK - 1] = key;
#pragma unroll
          for (int t = KK - 1; t > 0; --t)
            if (best1[t] < best1[t - 1]) {
              const unsigned long long x = best1[t];
              best1[t] = best1[t - 1];
              best1[t - 1] = x;
            }
        }
      }
    }
  }
  if (active && nbr) {
    int32_t* out0 = nbr + ((size_t)b * N + j0) * kk;
    for (int q = 0; q < kk; ++q) {
      const unsigned long long m = warp_min_u64(best0[0]);
      if (lane == 0) out0[q] = (int32_t)(m & 0xFFFFFFFFull);
      if (best0[0] == m) {  // keys are unique: exactly one lane pops its head
#pragma unroll
        for (int i = 0; i < KK - 1; ++i) best0[i] = best0[i + 1];
        best0[KK - 1] = ~0ull;
      }
    }
    if (two) {
      int32_t* out1 = nbr + ((size_t)b * N + j1) * kk;
      for (int q = 0; q < kk; ++q) {
        const unsigned long long m = warp_min_u64(best1[0]);
        if (lane == 0) out1[q] = (int32_t)(m & 0xFFFFFFFFull);
        if (best1[0] == m) {
#pragma unroll
          for (int i = 0; i < KK - 1; ++i) best1[i] = best1[i + 1];
          best1[KK - 1] = ~0ull;
        }
      }
    }
  }
  for (int o = 16; o > 0; o >>= 1) dmax = max(dmax, __shfl_xor_sync(0xFFFFFFFFu, dmax, o));
  __shared__ uint32_t s_dmax[8];
  if (lane == 0) s_dmax[threadIdx.x >> 5] = dmax;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t m = s_dmax[0];
    for (int i = 1; i < 8; ++i) m = max(m, s_dmax[i]);
    atomicMax(&stats[b].d2_max_bits, m);
  }
}

int launch_knn(const float* pos, const float4* tok, int64_t B, int64_t N, int kk, int32_t* nbr,
               SceneStats* stats, cudaStream_t s) {
  if (kk <= 8) {
    dim3 grid((unsigned)((N + 15) / 16), (unsigned)B);
    if (tok)
      k_knn_pair<8, true><<<grid, 256, 0, s>>>(pos, tok, (int)N, kk, nbr, stats);
    else
      k_knn_pair<8, false><<<grid, 256, 0, s>>>(pos, nullptr, (int)N, kk, nbr, stats);
    return last_launch_status();
  }
  if (kk <= 32) {
    dim3 grid((unsigned)((N + 7) / 8), (unsigned)B);
    if (kk <= 16)
      k_knn_warp<16><<<grid, 256, 0, s>>>(pos, (int)N, kk, nbr, stats);
    else
      k_knn_warp<32><<<grid, 256, 0, s>>>(pos, (int)N, kk, nbr, stats);
    return last_launch_status();
  }
  int list_len = 1;
  while (list_len < kk) list_len <<= 1;
  if (list_len < 2) list_len = 2;
  const size_t smem = sizeof(unsigned long long) * list_len + sizeof(uint32_t) * (size_t)N;
  if (smem > 48 * 1024 &&
      cuda_status(cudaFuncSetAttribute(k_knn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem),
                  "launch_knn: smem attribute") != CP_OK)
    return CP_ECUDA;
  dim3 grid((unsigned)N, (unsigned)B);
  k_knn<<<grid, KNN_THREADS, smem, s>>>(pos, (int)N, kk, list_len, nbr, stats);
  return last_launch_status();
}

// ---------------------------------------------------------------------------
// K1 through a uniform grid (kk <= kKnnGridMax): exact, with the same keys and lists
// as the brute-force kernels, but each query visits only the cells around
// it.  The scene's bounding box is cut into cubic cells of side h =
// (largest extent) / G with G = the least integer such that 4 G^3 >= N, so
// at most G^3 cells; points are counting-sorted by cell.  A query scans the
// shells of cells at Chebyshev distance r = 0, 1, 2, ... from its own cell;
// every point outside the first r shells is more than r h away along some
// axis, so once the kk-th best squared distance is below ((r - 1/1024) h)^2
// (the margin covers the rounding of the cell coordinates) no later point
// can enter the list.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int grid_side(int N) {
  int G = 1;
  while (4 * G * G * G < N) ++G;
  return G;
}

// One block per scene: bounding box, cell size, counting sort by cell.
__global__ void __launch_bounds__(1024) k_grid_build(const float* __restrict__ pos, int N,
                                                     int gmax, GridInfo* __restrict__ info,
                                                     int32_t* __restrict__ cell_start,
                                                     float4* __restrict__ sorted) {
  extern __shared__ int s_cnt[];  // [gmax + 1]
  __shared__ float s_red[6][32];
  const int b = blockIdx.x;
  const float* X = pos + (size_t)b * N * 3;
  float lo[3] = {INFINITY, INFINITY, INFINITY}, hi[3] = {-INFINITY, -INFINITY, -INFINITY};
  for (int j = threadIdx.x; j < N; j += blockDim.x)
#pragma unroll
    for (int a = 0; a < 3; ++a) {
      lo[a] = fminf(lo[a], X[3 * j + a]);
      hi[a] = fmaxf(hi[a], X[3 * j + a]);
    }
  for (int o = 16; o > 0; o >>= 1)
#pragma unroll
    for (int a = 0; a < 3; ++a) {
      lo[a] = fminf(lo[a], __shfl_xor_sync(0xFFFFFFFFu, lo[a], o));
      hi[a] = fmaxf(hi[a], __shfl_xor_sync(0xFFFFFFFFu, hi[a], o));
    }
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  if (l == 0)
    for (int a = 0; a < 3; ++a) {
      s_red[a][w] = lo[a];
      s_red[3 + a][w] = hi[a];
    }
  for (int c = threadIdx.x; c <= gmax; c += blockDim.x) s_cnt[c] = 0;
  __syncthreads();
  __shared__ GridInfo s_g;
  if (threadIdx.x == 0) {
    const int nw = blockDim.x >> 5;
    for (int i = 1; i < nw; ++i)
      for (int a = 0; a < 3; ++a) {
        s_red[a][0] = fminf(s_red[a][0], s_red[a][i]);
        s_red[3 + a][0] = fmaxf(s_red[3 + a][0], s_red[3 + a][i]);
      }
    const int G = grid_side(N);
    float ext = 0.0f;
    for (int a = 0; a < 3; ++a) ext = fmaxf(ext, s_red[3 + a][0] - s_red[a][0]);
    GridInfo g;
    g.h = ext > 0.0f ? ext / (float)G : 1.0f;
    g.inv_h = 1.0f / g.h;
    int nc = 1;
    for (int a = 0; a < 3; ++a) {
      g.lo[a] = s_red[a][0];
      const float e = s_red[3 + a][0] - s_red[a][0];
      int d = (int)ceilf(e * g.inv_h);
      d = d < 1 ? 1 : (d > G ? G : d);
      g.dims[a] = d;
      nc *= d;
    }
    g.ncells = nc;
    s_g = g;
    info[b] = g;
  }
  __syncthreads();
  const GridInfo g = s_g;
  for (int j = threadIdx.x; j < N; j += blockDim.x) atomicAdd(&s_cnt[grid_cell(g, X + 3 * j)], 1);
  __syncthreads();
  if (threadIdx.x == 0) {  // exclusive scan; cells <= G^3 <= 13824
    int run = 0;
    for (int c = 0; c < g.ncells; ++c) {
      const int n = s_cnt[c];
      s_cnt[c] = run;
      run += n;
    }
    s_cnt[g.ncells] = run;
  }
  __syncthreads();
  int32_t* cs = cell_start + (size_t)b * (gmax + 1);
  for (int c = threadIdx.x; c <= g.ncells; c += blockDim.x) cs[c] = s_cnt[c];
  __syncthreads();
  float4* out = sorted + (size_t)b * N;
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    const int slot = atomicAdd(&s_cnt[grid_cell(g, X + 3 * j)], 1);
    out[slot] = make_float4(X[3 * j], X[3 * j + 1], X[3 * j + 2], __int_as_float(j));
  }
}

// One thread per query token.  The KK best keys are kept unsorted with the
// position of the worst: a closer point overwrites the worst (a select per
// slot, so the list stays in registers) and the worst is found again; the
// list is sorted once at the end.  Keys are (d^2 bits, index), as in the
// brute-force kernels.
template <int KK>
__global__ void __launch_bounds__(128) k_knn_grid(const float* __restrict__ pos, int N, int kk,
                                                  int gmax, const GridInfo* __restrict__ info,
                                                  const int32_t* __restrict__ cell_start,
                                                  const float4* __restrict__ sorted,
                                                  int32_t* __restrict__ nbr) {
  // thread jj takes the jj-th token in cell order: a warp's queries share
  // their cells, so its lanes scan the same candidate cells together
  const int jj = blockIdx.x * blockDim.x + threadIdx.x;
  const int b = blockIdx.y;
  if (jj >= N) return;
  const GridInfo g = info[b];
  const int32_t* cs = cell_start + (size_t)b * (gmax + 1);
  const float4* P = sorted + (size_t)b * N;
  const float4 qp = P[jj];
  const int j = __float_as_int(qp.w);
  const float qx = qp.x, qy = qp.y, qz = qp.z;
  const int cx = grid_coord(g, qx, 0), cy = grid_coord(g, qy, 1), cz = grid_coord(g, qz, 2);
  // only the first kk slots are used; the others stay at the smallest key
  // and never become the worst
  unsigned long long best[KK];
#pragma unroll
  for (int i = 0; i < KK; ++i) best[i] = i < kk ? ~0ull : 0ull;
  unsigned long long worst = ~0ull;
  int wi = 0;
  const int rmax = max(g.dims[0], max(g.dims[1], g.dims[2]));
  for (int r = 0; r <= rmax; ++r) {
    for (int dz = -r; dz <= r; ++dz) {
      const int z = cz + dz;
      if (z < 0 || z >= g.dims[2]) continue;
      for (int dy = -r; dy <= r; ++dy) {
        const int y = cy + dy;
        if (y < 0 || y >= g.dims[1]) continue;
        const bool face = dz == -r || dz == r || dy == -r || dy == r;
        for (int dx = -r; dx <= r; dx += (face || r == 0) ? 1 : 2 * r) {
          const int x = cx + dx;
          if (x < 0 || x >= g.dims[0]) continue;
          const int c = (z * g.dims[1] + y) * g.dims[0] + x;
          const int e = cs[c + 1];
          for (int s = cs[c]; s < e; ++s) {
            const float4 p = P[s];
            const int k = __float_as_int(p.w);
            const uint32_t bits = __float_as_uint(sqdist_rn(qx, qy, qz, p.x, p.y, p.z));
            if (k == j || bits > (uint32_t)(worst >> 32)) continue;
            const unsigned long long key = ((unsigned long long)bits << 32) | (uint32_t)k;
            if (key >= worst) continue;
#pragma unroll
            for (int i = 0; i < KK; ++i) best[i] = i == wi ? key : best[i];
            worst = 0ull;
#pragma unroll
            for (int i = 0; i < KK; ++i)
              if (best[i] > worst) {
                worst = best[i];
                wi = i;
              }
          }
        }
      }
    }
    if (worst != ~0ull) {  // the list is full: is anything closer still possible?
      const float reach = ((float)r - 1.0f / 1024.0f) * g.h;
      if (reach > 0.0f && __uint_as_float((uint32_t)(worst >> 32)) < reach * reach) break;
    }
  }
  // sort the kk keys ascending (the unused slots hold 0 and sort first)
#pragma unroll
  for (int i = 1; i < KK; ++i)
#pragma unroll
    for (int t = KK - 1; t >= i; --t)
      if (best[t] < best[t - 1]) {
        const unsigned long long x = best[t];
        best[t] = best[t - 1];
        best[t - 1] = x;
      }
  int32_t* out = nbr + ((size_t)b * N + j) * kk;
#pragma unroll
  for (int i = 0; i < KK; ++i)
    if (i >= KK - kk) out[i - (KK - kk)] = (int32_t)(best[i] & 0xFFFFFFFFull);
}

// More neighbours (8 < kk <= kKnnGridMax): the same shell search, one thread
// per query (queries in cell order), with the kk best keys in a max-heap in
// shared memory (slot i of thread t at [i][t]: the threads of a warp touch
// distinct banks); the root is the worst kept key.  A heapsort leaves them
// ascending at the end.
__global__ void __launch_bounds__(128) k_knn_grid_heap(const float* __restrict__ pos, int N, int kk,
                                                       int gmax, const GridInfo* __restrict__ info,
                                                       const int32_t* __restrict__ cell_start,
                                                       const float4* __restrict__ sorted,
                                                       int32_t* __restrict__ nbr) {
  extern __shared__ unsigned long long s_heap[];  // [kk][blockDim.x]
  const int jj = blockIdx.x * blockDim.x + threadIdx.x;  // the jj-th token in cell order
  const int b = blockIdx.y;
  if (jj >= N) return;
  const int T = blockDim.x;
  unsigned long long* H = s_heap + threadIdx.x;  // H[i * T] is slot i
  const GridInfo g = info[b];
  const int32_t* cs = cell_start + (size_t)b * (gmax + 1);
  const float4* P = sorted + (size_t)b * N;
  const float4 qp = P[jj];
  const int j = __float_as_int(qp.w);
  const float qx = qp.x, qy = qp.y, qz = qp.z;
  const int cx = grid_coord(g, qx, 0), cy = grid_coord(g, qy, 1), cz = grid_coord(g, qz, 2);
  int cnt = 0;
  unsigned long long worst = ~0ull;  // the root once the heap is full
  // the root replaced by key (smaller than it), sifted down within n slots
  auto sift_down = [&](unsigned long long key, int n) {
    int i = 0;
    for (;;) {
      const int l = 2 * i + 1;
      if (l >= n) break;
      const int r = l + 1;
      unsigned long long ck = H[(size_t)l * T];
      int c = l;
      if (r < n) {
        const unsigned long long rk = H[(size_t)r * T];
        if (rk > ck) {
          ck = rk;
          c = r;
        }
      }
      if (ck <= key) break;
      H[(size_t)i * T] = ck;
      i = c;
    }
    H[(size_t)i * T] = key;
  };
  const int rmax = max(g.dims[0], max(g.dims[1], g.dims[2]));
  for (int r = 0; r <= rmax; ++r) {
    for (int dz = -r; dz <= r; ++dz) {
      const int z = cz + dz;
      if (z < 0 || z >= g.dims[2]) continue;
      for (int dy = -r; dy <= r; ++dy) {
        const int y = cy + dy;
        if (y < 0 || y >= g.dims[1]) continue;
        const bool face = dz == -r || dz == r || dy == -r || dy == r;
        for (int dx = -r; dx <= r; dx += (face || r == 0) ? 1 : 2 * r) {
          const int x = cx + dx;
          if (x < 0 || x >= g.dims[0]) continue;
          const int c = (z * g.dims[1] + y) * g.dims[0] + x;
          const int e = cs[c + 1];
          for (int s = cs[c]; s < e; ++s) {
            const float4 p = P[s];
            const int k = __float_as_int(p.w);
            const uint32_t bits = __float_as_uint(sqdist_rn(qx, qy, qz, p.x, p.y, p.z));
            if (k == j || bits > (uint32_t)(worst >> 32)) continue;
            const unsigned long long key = ((unsigned long long)bits << 32) | (uint32_t)k;
            if (key >= worst) continue;
            if (cnt < kk) {  // filling: sift the new key up
              int i = cnt++;
              while (i > 0) {
                const int pi = (i - 1) >> 1;
                const unsigned long long pk = H[(size_t)pi * T];
                if (pk >= key) break;
                H[(size_t)i * T] = pk;
                i = pi;
              }
              H[(size_t)i * T] = key;
              if (cnt == kk) worst = H[0];
            } else {
              sift_down(key, kk);
              worst = H[0];
            }
          }
        }
      }
    }
    if (cnt == kk) {  // the heap is full: is anything closer still possible?
      const float reach = ((float)r - 1.0f / 1024.0f) * g.h;
      if (reach > 0.0f && __uint_as_float((uint32_t)(worst >> 32)) < reach * reach) break;
    }
  }
  // heapsort: the largest to the end, repeatedly
  for (int n = kk; n > 1; --n) {
    const unsigned long long top = H[0];
    const unsigned long long last = H[(size_t)(n - 1) * T];
    H[(size_t)(n - 1) * T] = top;
    sift_down(last, n - 1);
  }
  int32_t* out = nbr + ((size_t)b * N + j) * kk;
  for (int i = 0; i < kk; ++i) out[i] = (int32_t)(H[(size_t)i * T] & 0xFFFFFFFFull);
}

// The largest pinned-fp32 squared distance over pairs, into stats.d2_max_bits,
// from the neighbour grid (points sorted by cell).  A lower bound L is the
// largest d^2 among the extreme points of 13 directions (an actual pair).
// For two cells whose coordinates differ by (dx, dy, dz) cells, any two of
// their points are at most (|d| + 1) h + delta apart along each axis (delta
// covers the rounding of the cell assignment), so the pair of cells can hold
// a pair above L only if sum ((|d| + 1) h + delta)^2, inflated for fp32
// rounding, reaches L.  Cells that reach L with no cell of the grid's corners
// are dropped; the pairs of the remaining cells that pass the test are
// evaluated with the same arithmetic as every other kernel, so the result is
// exactly the largest d^2.  Blocks (part, scene); part p takes every P-th
// row of candidate-cell pairs.
constexpr int DIA_THREADS = 512, DIA_PARTS = 4, DIA_DIRS = 13;

__device__ __forceinline__ uint32_t warp_max_u32(uint32_t v) {
  for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

__device__ __forceinline__ float dia_dir_dot(int d, float x, float y, float z) {
  switch (d) {
    case 0: return x;
    case 1: return y;
    case 2: return z;
    case 3: return x + y;
    case 4: return x - y;
    case 5: return x + z;
    case 6: return x - z;
    case 7: return y + z;
    case 8: return y - z;
    case 9: return x + y + z;
    case 10: return x + y - z;
    case 11: return x - y + z;
    default: return -x + y + z;
  }
}

__global__ void __launch_bounds__(DIA_THREADS) k_diameter_grid(
    int N, int gmax, const GridInfo* __restrict__ info, const int32_t* __restrict__ cell_start,
    const float4* __restrict__ sorted, SceneStats* stats) {
  extern __shared__ int s_cand[];  // candidate cells, [gmax]
  __shared__ unsigned long long s_ext[2 * DIA_DIRS];
  __shared__ int s_ncand, s_wcnt[DIA_THREADS / 32];
  __shared__ uint32_t s_m[DIA_THREADS / 32];
  const int b = blockIdx.y;
  const GridInfo g = info[b];
  const int32_t* cs = cell_start + (size_t)b * (gmax + 1);
  const float4* P = sorted + (size_t)b * N;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (threadIdx.x < 2 * DIA_DIRS) s_ext[threadIdx.x] = 0ull;
  if (threadIdx.x == 0) s_ncand = 0;
  __syncthreads();

  // extreme points of 13 directions (max of +u and of -u), as (key, slot)
  for (int d = 0; d < DIA_DIRS; ++d) {
    unsigned long long hi = 0ull, lo = 0ull;
    for (int i = threadIdx.x; i < N; i += DIA_THREADS) {
      const float4 p = P[i];
      const float v = dia_dir_dot(d, p.x, p.y, p.z);
      const unsigned long long kh = ((unsigned long long)f2key(v) << 32) | (uint32_t)i;
      const unsigned long long kl = ((unsigned long long)f2key(-v) << 32) | (uint32_t)i;
      hi = kh > hi ? kh : hi;
      lo = kl > lo ? kl : lo;
    }
    hi = warp_max_u64(hi);
    lo = warp_max_u64(lo);
    if (lane == 0) {
      atomicMax(&s_ext[2 * d], hi);
      atomicMax(&s_ext[2 * d + 1], lo);
    }
  }
  __syncthreads();
  uint32_t m = 0u;  // the largest d^2 bits this thread has seen
  for (int e = threadIdx.x; e < 2 * DIA_DIRS * 2 * DIA_DIRS; e += DIA_THREADS) {
    const int u = e / (2 * DIA_DIRS), v = e % (2 * DIA_DIRS);
    const float4 a = P[(uint32_t)(s_ext[u] & 0xFFFFFFFFull)];
    const float4 c = P[(uint32_t)(s_ext[v] & 0xFFFFFFFFull)];
    m = max(m, __float_as_uint(sqdist_rn(a.x, a.y, a.z, c.x, c.y, c.z)));
  }
  m = warp_max_u32(m);
  if (lane == 0) s_m[w] = m;
  __syncthreads();
  uint32_t Lb = s_m[0];
  for (int i = 1; i < DIA_THREADS / 32; ++i) Lb = max(Lb, s_m[i]);
  const float L = __uint_as_float(Lb);

  // bound of two cells' d^2 from their coordinate differences
  float span = 0.0f;
  for (int a = 0; a < 3; ++a) span = fmaxf(span, fabsf(g.lo[a]) + (float)g.dims[a] * g.h);
  const float delta = 1e-3f * g.h + 1e-5f * span;
  auto bound = [&](int ax, int ay, int az, int bx, int by, int bz) -> float {
    const float ex = (float)(abs(ax - bx) + 1) * g.h + delta;
    const float ey = (float)(abs(ay - by) + 1) * g.h + delta;
    const float ez = (float)(abs(az - bz) + 1) * g.h + delta;
    return (ex * ex + ey * ey + ez * ez) * 1.000244140625f;  // 1 + 2^-12
  };
  // the candidate cells in ascending order (every block of the scene lists
  // them alike, so the parts split the pairs without gaps or overlaps)
  const int d0 = g.dims[0], d1 = g.dims[1], d2 = g.dims[2];
  for (int base = 0; base < g.ncells; base += DIA_THREADS) {
    const int c = base + threadIdx.x;
    bool cand = false;
    if (c < g.ncells && cs[c + 1] > cs[c]) {
      const int cx = c % d0, cy = (c / d0) % d1, cz = c / (d0 * d1);
      float far = 0.0f;
      for (int k = 0; k < 8; ++k)
        far = fmaxf(far, bound(cx, cy, cz, (k & 1) ? d0 - 1 : 0, (k & 2) ? d1 - 1 : 0,
                               (k & 4) ? d2 - 1 : 0));
      cand = far >= L;
    }
    const uint32_t bal = __ballot_sync(0xFFFFFFFFu, cand);
    if (lane == 0) s_wcnt[w] = __popc(bal);
    __syncthreads();
    int off = s_ncand;
    for (int i = 0; i < w; ++i) off += s_wcnt[i];
    if (cand) s_cand[off + __popc(bal & ((1u << lane) - 1u))] = c;
    __syncthreads();  // every thread has read s_ncand and s_wcnt
    if (threadIdx.x == 0) {
      int tot = 0;
      for (int i = 0; i < DIA_THREADS / 32; ++i) tot += s_wcnt[i];
      s_ncand += tot;
    }
    __syncthreads();
  }
  const int M = s_ncand;

  // rows of candidate-cell pairs: warp (part, w) takes rows r = part + P*w, ...
  const int nw = DIA_THREADS / 32;
  for (int r = blockIdx.x + DIA_PARTS * w; r < M; r += DIA_PARTS * nw) {
    const int A = s_cand[r];
    const int ax = A % d0, ay = (A / d0) % d1, az = A / (d0 * d1);
    const int a0 = cs[A], a1 = cs[A + 1];
    for (int t = r + lane; t < M; t += 32) {
      const int Bc = s_cand[t];
      const int bx = Bc % d0, by = (Bc / d0) % d1, bz = Bc / (d0 * d1);
      if (bound(ax, ay, az, bx, by, bz) < L) continue;
      const int b0 = cs[Bc], b1 = cs[Bc + 1];
      for (int i = a0; i < a1; ++i) {
        const float4 p = P[i];
        for (int j = b0; j < b1; ++j) {
          const float4 q = P[j];
          m = max(m, __float_as_uint(sqdist_rn(p.x, p.y, p.z, q.x, q.y, q.z)));
        }
      }
    }
  }
  m = warp_max_u32(m);
  __syncthreads();  // every warp has read s_m above
  if (lane == 0) s_m[w] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t mm = s_m[0];
    for (int i = 1; i < nw; ++i) mm = max(mm, s_m[i]);
    atomicMax(&stats[b].d2_max_bits, mm);
  }
}

int grid_cells_max(int64_t N) {
  int64_t G = 1;
  while (4 * G * G * G < N) ++G;
  return (int)(G * G * G);
}

int launch_knn_grid(const float* pos, int64_t B, int64_t N, int kk, int32_t* nbr,
                    SceneStats* stats, GridInfo* info, int32_t* cell_start, float4* sorted,
                    cudaStream_t s) {
  const int gmax = grid_cells_max(N);
  if (kk > kKnnGridMax) return CP_EINVAL;
  const size_t smem = sizeof(int) * (size_t)(gmax + 1);
  if (smem > 48 * 1024 &&
      (cuda_status(cudaFuncSetAttribute(k_grid_build, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        (int)smem),
                   "launch_knn_grid: smem attribute") != CP_OK ||
       cuda_status(cudaFuncSetAttribute(k_diameter_grid,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                   "launch_knn_grid: smem attribute") != CP_OK))
    return CP_ECUDA;
  k_grid_build<<<(unsigned)B, 1024, smem, s>>>(pos, (int)N, gmax, info, cell_start, sorted);
  CP_TRY_STATUS(last_launch_status());
  k_diameter_grid<<<dim3(DIA_PARTS, (unsigned)B), DIA_THREADS, smem, s>>>((int)N, gmax, info,
                                                                          cell_start, sorted,
                                                                          stats);
  CP_TRY_STATUS(last_launch_status());
  if (kk <= 0) return CP_OK;
  if (kk <= 8) {
    dim3 grid((unsigned)((N + 127) / 128), (unsigned)B);
    k_knn_grid<8><<<grid, 128, 0, s>>>(pos, (int)N, kk, gmax, info, cell_start, sorted, nbr);
    return last_launch_status();
  }
  const int T = kk <= 64 ? 128 : 64;  // heaps of T x kk keys: at most 64 KB
  const size_t hsmem = sizeof(unsigned long long) * (size_t)T * (size_t)kk;
  if (hsmem > 48 * 1024 &&
      cuda_status(cudaFuncSetAttribute(k_knn_grid_heap, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)hsmem),
                  "launch_knn_grid: heap smem attribute") != CP_OK)
    return CP_ECUDA;
  dim3 grid((unsigned)((N + T - 1) / T), (unsigned)B);
  k_knn_grid_heap<<<grid, T, hsmem, s>>>(pos, (int)N, kk, gmax, info, cell_start, sorted, nbr);
  return last_launch_status();
}

__global__ void k_diameter(const SceneStats* stats, int B, float* out) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < B) out[b] = sqrtf(__uint_as_float(stats[b].d2_max_bits));
}

int launch_diameter(const SceneStats* stats, int64_t B, float* out, cudaStream_t s) {
  k_diameter<<<(unsigned)((B + 127) / 128), 128, 0, s>>>(stats, (int)B, out);
  return last_launch_status();
}

// ---------------------------------------------------------------------------
// Normalisers from the reduced statistics.
// ---------------------------------------------------------------------------
__global__ void k_finalize_norms(const SceneStats* stats, int B, int norm_mode,
                                 SceneNorms* norms, float* norms_out) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const SceneStats st = stats[b];
  SceneNorms nm;
  const float cmax = key2f(st.cos_max_key), cmin = key2f(st.cos_min_key);
  // min-max over all pairs (the Gram's extremes), or the bounds of
  // d_f = 1 - cos itself, [0, 2]
  nm.f_lo = norm_mode == 1 ? 0.0f : 1.0f - cmax;
  nm.f_hi = norm_mode == 1 ? 2.0f : 1.0f - cmin;
  nm.x_lo = 0.0f;  // diagonal pairs: d_x(j, j) = 0
  nm.x_hi = sqrtf(__uint_as_float(st.d2_max_bits));
  nm.t_lo = 0.0f;  // d_tau(j, j) = 0 and d_tau >= 0
  nm.t_hi = (float)(st.tau_max - st.tau_min);
  const float rf = nm.f_hi - nm.f_lo, rx = nm.x_hi - nm.x_lo, rt = nm.t_hi - nm.t_lo;
  nm.f_rinv = rf > (float)kRangeEps ? 1.0f / rf : 0.0f;
  nm.x_rinv = rx > (float)kRangeEps ? 1.0f / rx : 0.0f;
  nm.t_rinv = rt > (float)kRangeEps ? 1.0f / rt : 0.0f;
  for (int i = 0; i < 7; ++i) nm.pad[i] = 0.0f;
  norms[b] = nm;
  if (norms_out) {
    float* o = norms_out + 6 * (size_t)b;
    o[0] = nm.f_lo; o[1] = nm.f_hi; o[2] = nm.x_lo; o[3] = nm.x_hi; o[4] = nm.t_lo; o[5] = nm.t_hi;
  }
}

int launch_finalize_norms(const SceneStats* stats, int64_t B, int norm_mode, SceneNorms* norms,
                          float* norms_out, cudaStream_t s) {
  k_finalize_norms<<<(unsigned)((B + 127) / 128), 128, 0, s>>>(stats, (int)B, norm_mode, norms,
                                                               norms_out);
  return last_launch_status();
}

}  // namespace cp
