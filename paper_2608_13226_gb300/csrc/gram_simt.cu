// K2/K3 for fp32 features (bf16 features use gram_tc.cu): Gram tiles with fp32 FMA (TF32 tensor cores would
// round the features to 10 mantissa bits, far outside the fp32 tolerance),
// with two epilogues:
//   MINMAX  max and min of cos(f_i, f_j) over the pairs of the tile (the
//           feature normaliser of Sec. 3.3); only tiles touching i <= j run,
//           as cos is symmetric
//   COST    the FST cost of Eq. fst_cost, stored row-major with stride ldc
// 128x128 output tile per 256-thread block, 8x8 outputs per thread, K
// chunks of 16 staged through shared memory.
#include "common.cuh"

namespace cp {

constexpr int ST_BM = 128, ST_BK = 16, ST_THREADS = 256;
enum { EPI_MINMAX = 0, EPI_COST = 1 };

template <typename T>
__device__ __forceinline__ void stage_tile(const T* __restrict__ F, int row0, int N, int D,
                                           int k0, float (*S)[ST_BM + 4]) {
  constexpr int V = Vec16<T>::n;            // elements per 16-byte load
  constexpr int PER_ROW = ST_BK / V;        // loads per row per chunk
  for (int i = threadIdx.x; i < ST_BM * PER_ROW; i += ST_THREADS) {
    const int r = i / PER_ROW, c = (i % PER_ROW) * V;
    float x[V];
    const int gr = row0 + r, gc = k0 + c;
    if (gr < N && gc < D) {
      Vec16<T>::load(F + (size_t)gr * D + gc, x);
    } else {
#pragma unroll
      for (int q = 0; q < V; ++q) x[q] = 0.0f;
    }
#pragma unroll
    for (int q = 0; q < V; ++q) S[c + q][r] = x[q];
  }
}

template <typename T, int EPI>
__global__ void __launch_bounds__(ST_THREADS) k_gram_simt(
    const T* __restrict__ F_all, const float* __restrict__ inv_all, const float* __restrict__ pos_all,
    const int32_t* __restrict__ frame_all, const SceneNorms* __restrict__ norms, DevParams P,
    int N, int D, float* __restrict__ cost, int64_t ldc, SceneStats* stats) {
  const int b = blockIdx.z;
  const int row0 = blockIdx.y * ST_BM, col0 = blockIdx.x * ST_BM;
  if (EPI == EPI_MINMAX && col0 + ST_BM - 1 < row0) return;  // only j < i inside
  const T* F = F_all + (size_t)b * N * D;
  const float* inv = inv_all + (size_t)b * N;

  __shared__ __align__(16) float As[ST_BK][ST_BM + 4];
  __shared__ __align__(16) float Bs[ST_BK][ST_BM + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.0f;

  for (int k0 = 0; k0 < D; k0 += ST_BK) {
    stage_tile<T>(F, row0, N, D, k0, As);
    stage_tile<T>(F, col0, N, D, k0, Bs);
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < ST_BK; ++kk) {
      float a[8], bb[8];
      const float4 a0 = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
      const float4 a1 = *reinterpret_cast<const float4*>(&As[kk][64 + ty * 4]);
      const float4 b0 = *reinterpret_cast<const float4*>(&Bs[kk][tx * 4]);
      const float4 b1 = *reinterpret_cast<const float4*>(&Bs[kk][64 + tx * 4]);
      a[0] = a0.x; a[1] = a0.y; a[2] = a0.z; a[3] = a0.w;
      a[4] = a1.x; a[5] = a1.y; a[6] = a1.z; a[7] = a1.w;
      bb[0] = b0.x; bb[1] = b0.y; bb[2] = b0.z; bb[3] = b0.w;
      bb[4] = b1.x; bb[5] = b1.y; bb[6] = b1.z; bb[7] = b1.w;
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], bb[j], acc[i][j]);
    }
    __syncthreads();
  }

  float cmax = -INFINITY, cmin = INFINITY;
  SceneNorms nm;
  const float* X = pos_all + (size_t)b * N * 3;
  const int32_t* TAU = frame_all + (size_t)b * N;
  float* Cb = nullptr;
  if (EPI == EPI_COST) {
    nm = norms[b];
    Cb = cost + (size_t)b * N * ldc;
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int gi = row0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
    if (gi >= N) continue;
    const float inv_i = inv[gi];
    float xi = 0.f, yi = 0.f, zi = 0.f;
    int ti = 0;
    if (EPI == EPI_COST) {
      xi = X[3 * gi]; yi = X[3 * gi + 1]; zi = X[3 * gi + 2];
      ti = TAU[gi];
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int gj = col0 + (j < 4 ? tx * 4 + j : 64 + tx * 4 + (j - 4));
      if (gj >= N) {
        if (EPI == EPI_COST && gj < ldc) Cb[(size_t)gi * ldc + gj] = 0.0f;
        continue;
      }
      float c = clamp_cos(acc[i][j] * inv_i * inv[gj]);
      if (gi == gj && inv_i > 0.0f) c = 1.0f;  // cos(f, f) = 1 exactly
      if (EPI == EPI_MINMAX) {
        cmax = fmaxf(cmax, c);
        cmin = fminf(cmin, c);
      } else {
        const float d2 = sqdist_rn(xi, yi, zi, X[3 * gj], X[3 * gj + 1], X[3 * gj + 2]);
        Cb[(size_t)gi * ldc + gj] = fst_cost_from(c, d2, ti, TAU[gj], nm, P);
      }
    }
  }
  if (EPI == EPI_MINMAX) {
    for (int o = 16; o > 0; o >>= 1) {
      cmax = fmaxf(cmax, __shfl_xor_sync(0xFFFFFFFFu, cmax, o));
      cmin = fminf(cmin, __shfl_xor_sync(0xFFFFFFFFu, cmin, o));
    }
    if ((threadIdx.x & 31) == 0 && cmax >= cmin) {
      atomicMax(&stats[b].cos_max_key, f2key(cmax));
      atomicMin(&stats[b].cos_min_key, f2key(cmin));
    }
  }
}

int launch_gram_minmax_simt(const void* feats, int dtype, const float* inv, int64_t B, int64_t N,
                            int64_t D, SceneStats* stats, cudaStream_t s) {
  const unsigned nt = (unsigned)((N + ST_BM - 1) / ST_BM);
  dim3 grid(nt, nt, (unsigned)B);
  DevParams P{};
  if (dtype != CP_F32) return CP_EINVAL;  // bf16 features run on the tensor cores
  k_gram_simt<float, EPI_MINMAX><<<grid, ST_THREADS, 0, s>>>(
      (const float*)feats, inv, nullptr, nullptr, nullptr, P, (int)N, (int)D, nullptr, 0, stats);
  return last_launch_status();
}

int launch_cost_simt(const void* feats, int dtype, const float* inv, const float* pos,
                     const int32_t* frame, const SceneNorms* norms, const DevParams& P, int64_t B,
                     int64_t N, int64_t D, float* cost, int64_t ldc, cudaStream_t s) {
  const unsigned nt = (unsigned)((N + ST_BM - 1) / ST_BM);
  dim3 grid(nt, nt, (unsigned)B);
  if (dtype != CP_F32) return CP_EINVAL;  // bf16 features run on the tensor cores
  k_gram_simt<float, EPI_COST><<<grid, ST_THREADS, 0, s>>>(
      (const float*)feats, inv, pos, frame, norms, P, (int)N, (int)D, cost, ldc, nullptr);
  return last_launch_status();
}

}  // namespace cp
