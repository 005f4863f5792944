// K5 as Sec. 3.5 prints it (sgs_mode 2): Eqs. srpot_sinkhorn, greedy_flow,
// sgs_select and sgs_update read word for word.
//
// At greedy step l the selected tokens s_0 .. s_{l-1} are the sources of an
// entropic semi-relaxed OT (Eq. srpot_sinkhorn), each with mass 1/K, and
// every token is a target with capacity v_j.  Its plan has the Gibbs form
// P_ij = exp((f_i + g_j - C(s_i, j)) / eps) with g <= 0, and block
// coordinate ascent on the dual alternates
//   rows:    f_i = eps log(1/K) - eps LSE_j((g_j - C(s_i, j)) / eps)   (P 1 = u)
//   columns: g_j = min(0, eps log v_j - eps LSE_i((f_i - C(s_i, j)) / eps))
//            (the capacity cap P^T 1 <= v; a column below it keeps g_j = 0)
// for sot_iters iterations, the column potentials carried over from step
// l-1 (zeros at l = 1).  The residual capacity (Eq. greedy_flow) is
//   r_j = max(v_j - sum_i P_ij, 0)     (r = v at l = 0),
// and the next token minimises the residual-weighted local cost (Eq.
// sgs_select)  score(t) = sum_{j in M_g(t)} r_j C(t, j)  over the
// unselected tokens, lowest index on equal scores.
//
// The path is HBM-bound: each iteration reads the l selected rows of the
// dense cost twice (rows, then columns), the score reads every candidate's
// row once.  One launch per phase covers all B scenes: columns a thread per
// target column (the l source indices and potentials staged in shared
// memory, the cost read coalesced along the row; a block spreads 32 columns
// over 16 groups of source rows), rows a block per source row, scores a warp
// per candidate; every thread keeps eight loads in flight.  Each step's winner is the smallest
// (score bits, index) key, reduced with one 64-bit atomicMin per block into
// that step's slot (initialised to all ones), so no separate argmin pass
// runs; non-negative floats order like their bit patterns, and every score
// is a sum of products of non-negative numbers.  Log-sum-exp is accumulated
// online (the running maximum rescales the running sum only when it grows).
#include "common.cuh"

namespace cp {
namespace {

constexpr int LIT_THREADS = 256;

struct Lse {
  float m, s;  // running maximum and sum of exp(x - m)
};
__device__ __forceinline__ void lse_add(Lse& a, float x) {
  if (x > a.m) {
    a.s = a.s * expf(a.m - x) + 1.0f;  // expf(-inf) = 0 on the first finite term
    a.m = x;
  } else if (x > -INFINITY) {
    a.s += expf(x - a.m);
  }
}
__device__ __forceinline__ Lse lse_merge(Lse a, Lse b) {
  if (a.m < b.m) {
    const Lse t = a;
    a = b;
    b = t;
  }
  if (b.m > -INFINITY) a.s += b.s * expf(b.m - a.m);
  return a;
}
__device__ __forceinline__ float lse_value(const Lse& a) {
  return a.m > -INFINITY ? a.m + logf(a.s) : -INFINITY;
}
__device__ __forceinline__ Lse warp_lse(Lse a) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    Lse b;
    b.m = __shfl_xor_sync(0xFFFFFFFFu, a.m, o);
    b.s = __shfl_xor_sync(0xFFFFFFFFu, a.s, o);
    a = lse_merge(a, b);
  }
  return a;
}
__device__ __forceinline__ int key_index(unsigned long long k) {
  return (int)(uint32_t)(k & 0xFFFFFFFFull);
}

// Row potentials of the l sources: f_i = eps log u - eps LSE_j((g_j - C_ij) / eps).
// One block per source row: thread x takes the columns x, x + 256, ...,
// eight loads in flight before their terms are added in column order; the
// threads' partial log-sum-exps merge in a fixed order (warps by butterfly,
// then the 8 warps in order).
__global__ void __launch_bounds__(LIT_THREADS) k_lit_rows(
    const float* __restrict__ C, int64_t ldc, int N, int K, int l,
    const unsigned long long* __restrict__ keys, const float* __restrict__ gpot, float eps,
    float inv_eps, float log_u, float* __restrict__ fpot) {
  __shared__ float s_m[LIT_THREADS / 32], s_s[LIT_THREADS / 32];
  const int b = blockIdx.y, i = blockIdx.x;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int s = key_index(keys[(size_t)b * K + i]);
  const float* row = C + ((size_t)b * N + s) * ldc;
  const float* g = gpot + (size_t)b * N;
  Lse a{-INFINITY, 0.0f};
  for (int j0 = threadIdx.x; j0 < N; j0 += 8 * LIT_THREADS) {
    float x[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int j = j0 + u * LIT_THREADS;
      x[u] = j < N ? (__ldg(g + j) - __ldg(row + j)) * inv_eps : -INFINITY;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) lse_add(a, x[u]);
  }
  a = warp_lse(a);
  if (lane == 0) {
    s_m[w] = a.m;
    s_s[w] = a.s;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    Lse t{s_m[0], s_s[0]};
    for (int q = 1; q < LIT_THREADS / 32; ++q) t = lse_merge(t, Lse{s_m[q], s_s[q]});
    fpot[(size_t)b * K + i] = eps * (log_u - lse_value(t));
  }
}

// Per target column j, LSE_i((f_i - C(s_i, j)) / eps) over the l sources.
// A block takes 32 columns (threadIdx.x) and splits the sources over 16 row
// groups (threadIdx.y: i = y, y + 16, ...), each warp reading 128
// contiguous bytes of a source row; the 16 partial log-sum-exps of a column
// merge in a fixed order.  RESID = false: the column potential g_j (the
// capacity cap).  RESID = true: the residual r_j = max(v_j - exp(g_j / eps +
// LSE), 0), and block 0 marks the previous step's pick as selected.
constexpr int LC_COLS = 32, LC_GROUPS = 16, LC_CHUNK = 256;
template <bool RESID>
__global__ void __launch_bounds__(LC_COLS * LC_GROUPS) k_lit_cols(
    const float* __restrict__ C, int64_t ldc, int N, int K, int l,
    const unsigned long long* __restrict__ keys, const float* __restrict__ fpot,
    const float* __restrict__ v, float eps, float inv_eps, float* __restrict__ gpot,
    float* __restrict__ resid, uint8_t* __restrict__ chosen) {
  __shared__ int s_idx[LC_CHUNK];
  __shared__ float s_f[LC_CHUNK];
  __shared__ float s_m[LC_GROUPS][LC_COLS], s_s[LC_GROUPS][LC_COLS];
  const int b = blockIdx.y;
  const int tx = threadIdx.x, ty = threadIdx.y;
  const int tid = ty * LC_COLS + tx;
  const int j = blockIdx.x * LC_COLS + tx;
  if (RESID && l > 0 && blockIdx.x == 0 && tid == 0)
    chosen[(size_t)b * N + key_index(keys[(size_t)b * K + l - 1])] = 1;
  const float* Cb = C + (size_t)b * N * ldc;
  Lse a{-INFINITY, 0.0f};
  for (int i0 = 0; i0 < l; i0 += LC_CHUNK) {
    const int n = min(LC_CHUNK, l - i0);
    __syncthreads();  // the previous chunk is consumed
    if (tid < n) {
      s_idx[tid] = key_index(keys[(size_t)b * K + i0 + tid]);
      s_f[tid] = fpot[(size_t)b * K + i0 + tid];
    }
    __syncthreads();
    if (j < N)
      for (int i1 = ty; i1 < n; i1 += 8 * LC_GROUPS) {  // eight loads in flight
        float x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int ii = i1 + u * LC_GROUPS;
          x[u] = ii < n ? (s_f[ii] - __ldg(Cb + (size_t)s_idx[ii] * ldc + j)) * inv_eps
                        : -INFINITY;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) lse_add(a, x[u]);
      }
  }
  s_m[ty][tx] = a.m;
  s_s[ty][tx] = a.s;
  __syncthreads();
  if (ty != 0 || j >= N) return;
  for (int q = 1; q < LC_GROUPS; ++q) a = lse_merge(a, Lse{s_m[q][tx], s_s[q][tx]});
  const float vj = v[(size_t)b * N + j];
  if (!RESID) {
    gpot[(size_t)b * N + j] = vj > 0.0f ? fminf(0.0f, eps * (logf(vj) - lse_value(a))) : -INFINITY;
  } else {
    const float gj = l > 0 ? gpot[(size_t)b * N + j] : 0.0f;
    const float lv = lse_value(a);
    const float col = (lv > -INFINITY && gj > -INFINITY) ? expf(gj * inv_eps + lv) : 0.0f;
    resid[(size_t)b * N + j] = fmaxf(vj - col, 0.0f);
  }
}

// score(t) = sum_{j in M_g(t)} r_j C(t, j) for every unselected t; the
// block's smallest (score, index) key goes to keys[b][l] by atomicMin.
__global__ void __launch_bounds__(LIT_THREADS) k_lit_score(
    const float* __restrict__ C, int64_t ldc, int N, int K, int l, int g, int kk,
    const int32_t* __restrict__ nbr, const float* __restrict__ resid,
    const uint8_t* __restrict__ chosen, unsigned long long* __restrict__ keys) {
  __shared__ unsigned long long s_min[LIT_THREADS / 32];
  const int b = blockIdx.y;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * (LIT_THREADS / 32) + w;
  unsigned long long key = ~0ull;
  if (t < N && !chosen[(size_t)b * N + t]) {
    const float* row = C + ((size_t)b * N + t) * ldc;
    const float* r = resid + (size_t)b * N;
    float s = 0.0f;
    if (g >= N) {
      for (int j = lane; j < N; j += 32) s = fmaf(__ldg(r + j), __ldg(row + j), s);
    } else {
      if (lane == 0) s = r[t] * row[t];
      const int32_t* nb = nbr + ((size_t)b * N + t) * kk;
      for (int q = lane; q < g - 1; q += 32) {
        const int jj = __ldg(nb + q);
        s = fmaf(__ldg(r + jj), __ldg(row + jj), s);
      }
    }
    s = warp_sum(s);
    s = s > 0.0f ? s : 0.0f;  // a -0 sum keys as +0
    key = ((unsigned long long)__float_as_uint(s) << 32) | (uint32_t)t;
  }
  key = warp_min_u64(key);
  if (lane == 0) s_min[w] = key;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long m = s_min[0];
    for (int i = 1; i < LIT_THREADS / 32; ++i) m = s_min[i] < m ? s_min[i] : m;
    if (m != ~0ull) atomicMin(keys + (size_t)b * K + l, m);
  }
}

// The K picks in order, their scores, and the coverage objective of the
// selected set, F(S) = sum_j v_j min(m0, min_{s in S, j in M_g(s)} C(s, j)),
// in double: thread r sums j = r, r + blockDim, ... in order, then a fixed
// tree over the block.  One block (1024 threads) per scene; m in shared
// memory (N floats), lowered with integer atomicMin on the bit patterns of
// the non-negative costs.
__global__ void __launch_bounds__(1024) k_lit_finish(
    const float* __restrict__ C, int64_t ldc, int N, int K, int g, int kk,
    const int32_t* __restrict__ nbr, const float* __restrict__ v,
    const unsigned long long* __restrict__ keys, float m0, int32_t* __restrict__ order32,
    float* __restrict__ gains, double* __restrict__ objective) {
  extern __shared__ float sm_m[];
  __shared__ double s_red[32];
  const int b = blockIdx.x;
  for (int l = threadIdx.x; l < K; l += blockDim.x) {
    const unsigned long long k = keys[(size_t)b * K + l];
    order32[(size_t)b * K + l] = key_index(k);
    if (gains) gains[(size_t)b * K + l] = __uint_as_float((uint32_t)(k >> 32));
  }
  if (!objective) return;
  for (int j = threadIdx.x; j < N; j += blockDim.x) sm_m[j] = m0;
  __syncthreads();
  const float* Cb = C + (size_t)b * N * ldc;
  unsigned int* mbits = reinterpret_cast<unsigned int*>(sm_m);
  for (int l = 0; l < K; ++l) {
    const int s = key_index(keys[(size_t)b * K + l]);
    const float* row = Cb + (size_t)s * ldc;
    if (g >= N) {
      for (int j = threadIdx.x; j < N; j += blockDim.x) {
        const float c = __ldg(row + j);
        atomicMin(mbits + j, __float_as_uint(c > 0.0f ? c : 0.0f));  // -0 as +0
      }
    } else {
      for (int q = threadIdx.x; q < g; q += blockDim.x) {
        const int j = q == 0 ? s : __ldg(nbr + ((size_t)b * N + s) * kk + q - 1);
        const float c = __ldg(row + j);
        atomicMin(mbits + j, __float_as_uint(c > 0.0f ? c : 0.0f));
      }
    }
  }
  __syncthreads();
  double acc = 0.0;
  for (int j = threadIdx.x; j < N; j += blockDim.x)
    acc += (double)v[(size_t)b * N + j] * (double)sm_m[j];
  acc = warp_sum(acc);
  if ((threadIdx.x & 31) == 0) s_red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double F = 0.0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) F += s_red[i];
    objective[b] = F;
  }
}

}  // namespace

size_t sgs_literal_ws_bytes(int64_t B, int64_t N, int64_t K) {
  auto up = [](size_t x) { return (x + 255) & ~(size_t)255; };
  const size_t BN = (size_t)B * (size_t)N, BK = (size_t)B * (size_t)K;
  return up(sizeof(float) * BK) + up(sizeof(float) * BN) + up(sizeof(float) * BN) +
         up(sizeof(unsigned long long) * BK) + up(BN);
}

int launch_sgs_literal(const float* cost, int64_t ldc, const int32_t* nbr, const float* v,
                       const DevParams& P, int64_t B, int64_t N, int64_t K, int32_t* order32,
                       float* gains, double* objective, void* scratch, cudaStream_t s) {
  if (B <= 0 || N <= 0 || K <= 0) return CP_OK;
  auto up = [](size_t x) { return (x + 255) & ~(size_t)255; };
  const size_t BN = (size_t)B * (size_t)N, BK = (size_t)B * (size_t)K;
  unsigned char* base = static_cast<unsigned char*>(scratch);
  float* fpot = reinterpret_cast<float*>(base);
  float* gpot = reinterpret_cast<float*>(base + up(sizeof(float) * BK));
  float* resid = reinterpret_cast<float*>(base + up(sizeof(float) * BK) + up(sizeof(float) * BN));
  unsigned long long* keys = reinterpret_cast<unsigned long long*>(
      base + up(sizeof(float) * BK) + 2 * up(sizeof(float) * BN));
  uint8_t* chosen = base + up(sizeof(float) * BK) + 2 * up(sizeof(float) * BN) +
                    up(sizeof(unsigned long long) * BK);
  CP_TRY_STATUS(cuda_status(cudaMemsetAsync(keys, 0xFF, sizeof(unsigned long long) * BK, s),
                            "launch_sgs_literal: keys"));
  CP_TRY_STATUS(cuda_status(cudaMemsetAsync(gpot, 0, sizeof(float) * BN, s),
                            "launch_sgs_literal: potentials"));
  CP_TRY_STATUS(cuda_status(cudaMemsetAsync(chosen, 0, BN, s), "launch_sgs_literal: chosen"));
  const float eps = P.sot_eps, inv_eps = 1.0f / P.sot_eps;
  const float log_u = (float)(-log((double)K));
  const int n = (int)N, k = (int)K, g = P.g, kk = P.kk;
  const dim3 gcols((unsigned)((N + LC_COLS - 1) / LC_COLS), (unsigned)B);
  const dim3 bcols(LC_COLS, LC_GROUPS);
  const dim3 gscore((unsigned)((N + LIT_THREADS / 32 - 1) / (LIT_THREADS / 32)), (unsigned)B);
  for (int l = 0; l < k; ++l) {
    if (l > 0) {
      const dim3 grows((unsigned)l, (unsigned)B);
      for (int it = 0; it < P.sot_iters; ++it) {
        k_lit_rows<<<grows, LIT_THREADS, 0, s>>>(cost, ldc, n, k, l, keys, gpot, eps, inv_eps,
                                                 log_u, fpot);
        CP_TRY_STATUS(last_launch_status());
        k_lit_cols<false><<<gcols, bcols, 0, s>>>(cost, ldc, n, k, l, keys, fpot, v, eps,
                                                  inv_eps, gpot, resid, chosen);
        CP_TRY_STATUS(last_launch_status());
      }
    }
    k_lit_cols<true><<<gcols, bcols, 0, s>>>(cost, ldc, n, k, l, keys, fpot, v, eps, inv_eps,
                                             gpot, resid, chosen);
    CP_TRY_STATUS(last_launch_status());
    k_lit_score<<<gscore, LIT_THREADS, 0, s>>>(cost, ldc, n, k, l, g, kk, nbr, resid, chosen,
                                               keys);
    CP_TRY_STATUS(last_launch_status());
  }
  const size_t smem = sizeof(float) * (size_t)N;
  if (smem > 48 * 1024 &&
      cuda_status(cudaFuncSetAttribute(k_lit_finish, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem),
                  "launch_sgs_literal: smem attribute") != CP_OK)
    return CP_ECUDA;
  k_lit_finish<<<(unsigned)B, 1024, smem, s>>>(cost, ldc, n, k, g, kk, nbr, v, keys, P.m0,
                                               order32, gains, objective);
  return last_launch_status();
}

}  // namespace cp
