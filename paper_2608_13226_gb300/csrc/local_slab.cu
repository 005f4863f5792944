// The cosines of the local SGS neighbourhoods (Eq. local_neighbor) without
// the all-pairs Gram, for the bounded feature normaliser (d_f / 2, which
// needs no pass over all pairs).
//
// Tokens are laid out in Morton order (Sec. 4.1's curve over 3D cells, the
// order Lite groups in): spatially near tokens sit at nearby positions, so
// the neighbour pairs (t, j in N(t)) fall into a few tiles of the
// position x position Gram around its diagonal.  A pass over the neighbour
// lists flags every 256 x 256 tile of the upper triangle (row positions
// 256 P.., column positions 256 J.., P <= J) that holds a pair, one scan
// lists the flagged tiles of all scenes, and the tensor-core Gram
// (gram_tc.cu) computes exactly those tiles of the Morton-ordered features,
// storing whole tiles at their position coordinates in the cosine buffer.
// The slab and the capacity then read cos(t, j) at [min(pos(t), pos(j))]
// [max(...)], inside a flagged tile.  Everything else of the buffer is
// never written nor read.  On a long-video scene (N = 8192, 63 neighbours)
// 183 of the 528 upper-triangle tiles are flagged.
#include "common.cuh"

namespace cp {
namespace {

constexpr int LS_TILE = 256;  // tile side of the flags (one pair-MMA unit)

// Position of every token, and the features and token records (x, y, z,
// 1/||f||) in Morton order: a warp per position, 16-byte copies.
__global__ void __launch_bounds__(256) k_morton_gather(const uint4* __restrict__ feats,
                                                       const float4* __restrict__ tok,
                                                       const int32_t* __restrict__ perm, int N,
                                                       int D16, uint4* __restrict__ feats_m,
                                                       float4* __restrict__ tok_m,
                                                       int32_t* __restrict__ pos_of) {
  const int b = blockIdx.y;
  const int p = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (p >= N) return;
  const size_t sb = (size_t)b * N;
  const int t = __ldg(perm + sb + p);
  const uint4* src = feats + (sb + t) * (size_t)D16;
  uint4* dst = feats_m + (sb + p) * (size_t)D16;
  for (int i = lane; i < D16; i += 32) dst[i] = __ldg(src + i);
  if (lane == 0) {
    tok_m[sb + p] = __ldg(tok + sb + t);
    pos_of[sb + t] = p;
  }
}

// flags[b][P][J] = 1 (P <= J) when a token at a position of tile P has a
// stored neighbour (any of its kk) at a position of tile J, or the other way
// round: a pair's cosine is read at [min(pos)][max(pos)], the upper
// triangle of the position Gram, so only tiles with P <= J are computed.
__global__ void __launch_bounds__(256) k_tile_flags(const int32_t* __restrict__ perm,
                                                    const int32_t* __restrict__ pos_of,
                                                    const int32_t* __restrict__ nbr, int N, int kk,
                                                    int T, uint8_t* __restrict__ flags) {
  const int b = blockIdx.y;
  const int p = blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= N) return;
  const size_t sb = (size_t)b * N;
  const int t = __ldg(perm + sb + p);
  const int32_t* nb = nbr + (sb + t) * kk;
  uint8_t* f = flags + (size_t)b * T * T;
  const int P = p / LS_TILE;
  for (int k = 0; k < kk; ++k) {
    const int J = __ldg(pos_of + sb + __ldg(nb + k)) / LS_TILE;
    f[(size_t)min(P, J) * T + max(P, J)] = 1;  // every writer stores the same byte
  }
}

// One block: the flagged tiles of every scene, in (scene, P, J) order, as
// units (b << 16) | (P << 8) | J, and their count.
__global__ void __launch_bounds__(1024) k_tile_units(const uint8_t* __restrict__ flags, int total,
                                                     uint32_t* __restrict__ units,
                                                     int* __restrict__ n_units, int T) {
  __shared__ int s_warp[32];
  __shared__ int s_base;
  if (threadIdx.x == 0) s_base = 0;
  __syncthreads();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  for (int c0 = 0; c0 < total; c0 += 1024) {
    const int i = c0 + (int)threadIdx.x;
    const int on = i < total && flags[i] ? 1 : 0;
    const unsigned bal = __ballot_sync(0xFFFFFFFFu, on);
    if (lane == 0) s_warp[w] = __popc(bal);
    __syncthreads();
    if (threadIdx.x == 0) {  // exclusive prefix of the warp counts
      int run = s_base;
      for (int q = 0; q < 32; ++q) {
        const int c = s_warp[q];
        s_warp[q] = run;
        run += c;
      }
      s_base = run;
    }
    __syncthreads();
    if (on) {
      const int at = s_warp[w] + __popc(bal & ((1u << lane) - 1u));
      const int b = i / (T * T), r = i - b * T * T;
      units[at] = ((uint32_t)b << 16) | ((uint32_t)(r / T) << 8) | (uint32_t)(r % T);
    }
    __syncthreads();  // s_warp and s_base are reused
  }
  if (threadIdx.x == 0) *n_units = s_base;
}

}  // namespace

int local_tiles(int64_t N) { return (int)((N + LS_TILE - 1) / LS_TILE); }

int launch_local_blocks(const void* feats, const float4* tok, const int32_t* perm,
                        const int32_t* nbr, int kk, int64_t B, int64_t N, int64_t D,
                        void* feats_m, float4* tok_m, int32_t* pos_of, uint8_t* flags,
                        uint32_t* units, int* n_units, cudaStream_t s) {
  const int T = local_tiles(N);
  if (T > 255 || B > 65535) return CP_EUNSUPPORTED;
  const int D16 = (int)(D * 2 / 16);  // bf16 rows of D % 8 == 0
  k_morton_gather<<<dim3((unsigned)((N + 7) / 8), (unsigned)B), 256, 0, s>>>(
      static_cast<const uint4*>(feats), tok, perm, (int)N, D16, static_cast<uint4*>(feats_m),
      tok_m, pos_of);
  CP_TRY_STATUS(last_launch_status());
  CP_TRY_STATUS(cuda_status(cudaMemsetAsync(flags, 0, (size_t)B * T * T, s), "tile flags"));
  k_tile_flags<<<dim3((unsigned)((N + 255) / 256), (unsigned)B), 256, 0, s>>>(
      perm, pos_of, nbr, (int)N, kk, T, flags);
  CP_TRY_STATUS(last_launch_status());
  k_tile_units<<<1, 1024, 0, s>>>(flags, (int)(B * T * T), units, n_units, T);
  return last_launch_status();
}

}  // namespace cp
