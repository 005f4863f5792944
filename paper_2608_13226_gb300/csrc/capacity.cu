// K4: FST capacity (Sec. 3.4, Eqs. fst_capacity_score, fst_capacity) and the
// cost slab of the local SGS neighbourhoods (Eq. local_neighbor).
#include "common.cuh"
#include "bf16_dot.cuh"

namespace cp {

// r_j = (1/n) sum_{k in N_n(j)} alpha_f d^_f(j,k) + alpha_x d^_x(j,k) + alpha_tau d^_tau(j,k)
// One block per token, one warp per neighbour (warp w takes k = N_n(j)[q]
// for q = w, w + warps, ...): the warps read the token's own row together,
// so L1 serves it once for all of them, and each reads one neighbour row.
// The dot products run over 16-byte feature vectors; the terms are summed in
// neighbour order by one thread.
constexpr int CAP_WARPS = 8;

template <typename T>
__device__ __forceinline__ float row_dot(const T* a, const T* b, int D, int lane) {
  constexpr int V = Vec16<T>::n;
  float dot = 0.0f;
  for (int d = lane * V; d < D; d += 32 * V) {
    float x[V], y[V];
    Vec16<T>::load(a + d, x);
    Vec16<T>::load(b + d, y);
#pragma unroll
    for (int i = 0; i < V; ++i) dot = fmaf(x[i], y[i], dot);
  }
  return dot;
}
template <>
__device__ __forceinline__ float row_dot<__nv_bfloat16>(const __nv_bfloat16* a,
                                                        const __nv_bfloat16* b, int D, int lane) {
  float dot = 0.0f;
  for (int d = lane * 8; d < D; d += 256)
    dot = dot8_bf16(__ldg(reinterpret_cast<const uint4*>(a + d)),
                    __ldg(reinterpret_cast<const uint4*>(b + d)), dot);
  return dot;
}

template <typename T>
__global__ void __launch_bounds__(32 * CAP_WARPS) k_capacity_r(
    const T* __restrict__ F_all, const float* __restrict__ inv_all, const float* __restrict__ pos_all,
    const int32_t* __restrict__ frame_all, const SceneNorms* __restrict__ norms,
    const int32_t* __restrict__ nbr_all, DevParams P, int N, int D, float* __restrict__ r_all) {
  constexpr int CHUNK = 256;
  __shared__ float s_term[CHUNK];  // the terms of neighbours q0 .. q0 + CHUNK - 1
  const int j = blockIdx.x;
  const int b = blockIdx.y;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nw = (int)(blockDim.x >> 5);
  const T* F = F_all + (size_t)b * N * D;
  const float* inv = inv_all + (size_t)b * N;
  const float* X = pos_all + (size_t)b * N * 3;
  const int32_t* TAU = frame_all + (size_t)b * N;
  const int32_t* nb = nbr_all + ((size_t)b * N + j) * P.kk;
  const SceneNorms nm = norms[b];
  const T* fj = F + (size_t)j * D;
  float acc = 0.0f;  // thread 0's running sum, in neighbour order
  for (int q0 = 0; q0 < P.n_cap; q0 += CHUNK) {
    const int qn = min(CHUNK, P.n_cap - q0);
    for (int qq = w; qq < qn; qq += nw) {
      const int k = __ldg(nb + q0 + qq);
      const T* fk = F + (size_t)k * D;
      const float dot = warp_sum(row_dot<T>(fj, fk, D, lane));
      const float cosv = clamp_cos(dot * inv[j] * inv[k]);
      const float tf = ((1.0f - cosv) - nm.f_lo) * nm.f_rinv;
      const float dx = sqrtf(sqdist_rn(X[3 * j], X[3 * j + 1], X[3 * j + 2], X[3 * k],
                                       X[3 * k + 1], X[3 * k + 2]));
      const float tx = (dx - nm.x_lo) * nm.x_rinv;
      const int dt = TAU[j] - TAU[k];
      const float tt = dt > 0 ? (float)dt * nm.t_rinv : 0.0f;
      if (lane == 0) s_term[qq] = P.alpha_f * tf + P.alpha_x * tx + P.alpha_tau * tt;
    }
    __syncthreads();
    if (threadIdx.x == 0)
      for (int qq = 0; qq < qn; ++qq) acc += s_term[qq];
    __syncthreads();
  }
  if (threadIdx.x == 0) r_all[(size_t)b * N + j] = P.n_cap > 0 ? acc / (float)P.n_cap : 0.0f;
}

// The same r_j from stored cosines in place of the dot product, the rest
// identical: the normaliser Gram's output, the upper triangle of
// [B][N][ldc] (cos(j, k) at [min(j, k)][max(j, k)]); or, given pos_of, the
// flagged Morton tiles of the local path (cos(j, k) at [min(pos)][max(pos)]).
// One thread per token; its n gathers fall in one row, near its own index
// (nearest neighbours sit in the same or adjacent frames).
__global__ void __launch_bounds__(256) k_capacity_r_cos(
    const float* __restrict__ cos_all, int64_t ldc, const float* __restrict__ pos_all,
    const int32_t* __restrict__ frame_all, const SceneNorms* __restrict__ norms,
    const int32_t* __restrict__ nbr_all, DevParams P, int N, const int32_t* __restrict__ pos_of,
    float* __restrict__ r_all) {
  const int j = blockIdx.x * 256 + threadIdx.x;
  const int b = blockIdx.y;
  if (j >= N) return;
  const int32_t* po = pos_of ? pos_of + (size_t)b * N : nullptr;
  const float* crow = cos_all + ((size_t)b * N + j) * (size_t)ldc;
  const float* X = pos_all + (size_t)b * N * 3;
  const int32_t* TAU = frame_all + (size_t)b * N;
  const int32_t* nb = nbr_all + ((size_t)b * N + j) * P.kk;
  const SceneNorms nm = norms[b];
  const float xj = X[3 * j], yj = X[3 * j + 1], zj = X[3 * j + 2];
  const int tj = TAU[j];
  float acc = 0.0f;
  for (int q = 0; q < P.n_cap; ++q) {
    const int k = nb[q];
    float cosv;
    if (po) {
      const int a = po[j], c = po[k];
      cosv = cos_all[((size_t)b * N + min(a, c)) * (size_t)ldc + max(a, c)];
    } else {
      cosv = k > j ? crow[k] : cos_all[((size_t)b * N + k) * (size_t)ldc + j];
    }
    const float tf = ((1.0f - cosv) - nm.f_lo) * nm.f_rinv;
    const float dx = sqrtf(sqdist_rn(xj, yj, zj, X[3 * k], X[3 * k + 1], X[3 * k + 2]));
    const float tx = (dx - nm.x_lo) * nm.x_rinv;
    const int dt = tj - TAU[k];
    const float tt = dt > 0 ? (float)dt * nm.t_rinv : 0.0f;
    acc += P.alpha_f * tf + P.alpha_x * tx + P.alpha_tau * tt;
  }
  r_all[(size_t)b * N + j] = P.n_cap > 0 ? acc / (float)P.n_cap : 0.0f;
}

// v_j = r_j / sum_l r_l (phi = identity), uniform when the sum is 0 or the
// uniform-capacity ablation is on.  One block per scene; the sum is taken in
// fp64 in a fixed order.
__global__ void __launch_bounds__(1024) k_capacity_v(const float* __restrict__ r_all, int N,
                                                     int mode, float* __restrict__ v_all,
                                                     float* __restrict__ v_out) {
  const int b = blockIdx.x;
  const float* r = r_all + (size_t)b * N;
  double part = 0.0;
  for (int j = threadIdx.x; j < N; j += blockDim.x) part += (double)r[j];
  part = warp_sum(part);
  __shared__ double s_part[32];
  __shared__ double s_total;
  if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = part;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) t += s_part[i];
    s_total = t;
  }
  __syncthreads();
  const double total = s_total;
  const bool uniform = mode == 1 || !(total > 0.0);
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    const float vj = uniform ? (float)(1.0 / (double)N) : (float)((double)r[j] / total);
    v_all[(size_t)b * N + j] = vj;
    if (v_out) v_out[(size_t)b * N + j] = vj;
  }
}

int launch_capacity(const void* feats, int dtype, const float* inv, const float* pos,
                    const int32_t* frame, const SceneNorms* norms, const int32_t* nbr,
                    const DevParams& P, int64_t B, int64_t N, int64_t D, float* r, float* v,
                    float* v_out, cudaStream_t s, const float* cos, int64_t ldc,
                    const int32_t* pos_of) {
  // one block per token, a warp per neighbour (at most CAP_WARPS)
  const dim3 grid((unsigned)N, (unsigned)B);
  const int warps = P.n_cap < 1 ? 1 : (P.n_cap < CAP_WARPS ? P.n_cap : CAP_WARPS);
  if (cos)
    k_capacity_r_cos<<<dim3((unsigned)((N + 255) / 256), (unsigned)B), 256, 0, s>>>(
        cos, ldc, pos, frame, norms, nbr, P, (int)N, pos_of, r);
  else if (dtype == CP_BF16)
    k_capacity_r<__nv_bfloat16><<<grid, 32 * warps, 0, s>>>(
        (const __nv_bfloat16*)feats, inv, pos, frame, norms, nbr, P, (int)N, (int)D, r);
  else
    k_capacity_r<float><<<grid, 32 * warps, 0, s>>>((const float*)feats, inv, pos, frame, norms,
                                                        nbr, P, (int)N, (int)D, r);
  int st = last_launch_status();
  if (st != CP_OK) return st;
  k_capacity_v<<<(unsigned)B, 1024, 0, s>>>(r, (int)N, P.cap_mode, v, v_out);
  return last_launch_status();
}

// slab[b][t][k] = C(t, M_g(t)[k]) with M_g(t)[0] = t and M_g(t)[k] the k-th
// nearest other token for k >= 1.
__global__ void k_slab(const float* __restrict__ cost, int64_t ldc, const int32_t* __restrict__ nbr,
                       int kk, int g, int N, float* __restrict__ slab) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int b = blockIdx.y;
  if (i >= (int64_t)N * g) return;
  const int t = (int)(i / g), k = (int)(i % g);
  const int j = k == 0 ? t : nbr[((size_t)b * N + t) * kk + (k - 1)];
  slab[(size_t)b * N * g + i] = cost[(size_t)b * N * ldc + (size_t)t * ldc + j];
}

int launch_slab(const float* cost, int64_t ldc, const int32_t* nbr, const DevParams& P, int64_t B,
                int64_t N, float* slab, cudaStream_t s) {
  const int64_t n = N * P.g;
  dim3 grid((unsigned)((n + 255) / 256), (unsigned)B);
  k_slab<<<grid, 256, 0, s>>>(cost, ldc, nbr, P.kk, P.g, (int)N, slab);
  return last_launch_status();
}

}  // namespace cp
