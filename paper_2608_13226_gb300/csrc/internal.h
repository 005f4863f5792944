// Internal declarations of the CoverPrune CUDA library: parameter blocks
// passed to kernels, per-scene normalisers and the host-side launchers of
// every kernel.  Not part of the public ABI (include/coverprune.h is).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "coverprune.h"

namespace cp {

// Method parameters in the form the kernels use them.
struct DevParams {
  float lambda_f, lambda_x, lambda_tau;
  float kappa, inv_log1p_kappa;
  float alpha_f, alpha_x, alpha_tau;
  float voxel, m0;
  int n_cap;   // capacity neighbours, already clamped to N-1
  int g;       // SGS neighbourhood incl. the token itself; == N means all
  int kk;      // neighbours stored per token = max(n_cap, g-1) (g < N) or n_cap
  int cap_mode;
  int sgs_mode;  // 0 = lazy evaluation of gains, 1 = every gain every step, 2 = literal rule
  int norm_mode;  // feature normaliser: 0 = min-max over all pairs, 1 = d_f / 2
  float sot_eps;  // literal rule: entropic weight of the semi-relaxed OT
  int sot_iters;  // literal rule: Sinkhorn iterations per greedy step
  uint64_t timeout_ns;
};

// Per-scene min-max normalisers (Sec. 3.3).  lo/hi are the extremes of each
// discrepancy; *_rinv = 1 / (hi - lo), or 0 when the range is <= 1e-6 (the
// normalised term is then 0).
struct SceneNorms {
  float f_lo, f_hi, x_lo, x_hi, t_lo, t_hi;
  float f_rinv, x_rinv, t_rinv;
  float pad[7];
};
static_assert(sizeof(SceneNorms) == 64, "SceneNorms layout");

// Raw per-scene statistics gathered by atomics before the normalisers are
// finalised: order-preserving keys of max/min cosine and max squared
// distance, frame range and the bounding-box minimum (Morton origin).
struct SceneStats {
  uint32_t cos_max_key, cos_min_key, d2_max_bits;
  int32_t tau_min, tau_max;
  float bbox_min[3];
  uint32_t pad[8];
};
static_assert(sizeof(SceneStats) == 64, "SceneStats layout");

// Uniform grid of one scene for the neighbour search (32 bytes).
struct GridInfo {
  float lo[3];   // bounding-box minimum
  float h;       // cell side
  float inv_h;
  int dims[3];   // cells per axis
  int ncells;
  int pad;
};
static_assert(sizeof(GridInfo) == 40, "GridInfo layout");

// Cell coordinate of x along axis a, clamped to the grid.
__host__ __device__ inline int grid_coord(const GridInfo& g, float x, int a) {
  const int c = (int)floorf((x - g.lo[a]) * g.inv_h);
  return c < 0 ? 0 : (c >= g.dims[a] ? g.dims[a] - 1 : c);
}
__host__ __device__ inline int grid_cell(const GridInfo& g, const float* p) {
  return (grid_coord(g, p[2], 2) * g.dims[1] + grid_coord(g, p[1], 1)) * g.dims[0] +
         grid_coord(g, p[0], 0);
}

constexpr double kRangeEps = 1e-6;

// Layout of the 256-byte status block at the start of every workspace
// (zeroed at the start of every call):
//   int32 [0]      status word (cp_status of the first device-side error)
//   int32 [4..7]   diagnostics of a CP_EDEVICE (step, scene, block, index)
//   uint32 [16]    barrier self-test counter (byte 64)
//   uint64 [16..17] (bytes 128..143) SGS gain evaluations and rounds
constexpr size_t kStatusBytes = 256;
constexpr size_t kCallStatsOffset = 128;

// Device attributes cached per device.
struct DeviceInfo {
  int sm_count;
  int max_smem_optin;
  int cc_major, cc_minor;
};
int device_info(DeviceInfo* out);

// ---------------------------------------------------------------------------
// Launchers (each returns a cp_status; all enqueue on `s`).
// ---------------------------------------------------------------------------

// K0: per-scene frame range and bounding-box minimum; initialises the
// atomically reduced fields of `stats`.
int launch_scene_stats(const float* pos, const int32_t* frame, int64_t B, int64_t N,
                       SceneStats* stats, cudaStream_t s);
// K0: inverse feature norms inv[b*N + j] (0 for a zero feature) and the
// packed per-token record tok[b*N + j] = (x, y, z, inv) the Gram epilogues read.
int launch_inv_norms(const void* feats, int dtype, const float* pos, int64_t B, int64_t N,
                     int64_t D, float* inv, float4* tok, cudaStream_t s);
// K1: per token the kk nearest other tokens by (fp32 d^2, index) into
// nbr[(b*N + j)*kk + q]; also the scene's largest squared distance.
int grid_cells_max(int64_t N);
// Neighbour counts the grid search serves (larger ones take the brute-force kernels).
constexpr int kKnnGridMax = 128;
int launch_knn_grid(const float* pos, int64_t B, int64_t N, int kk, int32_t* nbr,
                    SceneStats* stats, GridInfo* info, int32_t* cell_start, float4* sorted,
                    cudaStream_t s);
int launch_knn(const float* pos, const float4* tok, int64_t B, int64_t N, int kk, int32_t* nbr, SceneStats* stats,
               cudaStream_t s);
// K2 (fp32 SIMT and bf16 tensor-core variants): max and min cosine over all
// pairs into stats.
int launch_gram_minmax(const void* feats, int dtype, const float* inv, const float4* tok,
                       int64_t B, int64_t N, int64_t D, SceneStats* stats, int* status,
                       uint64_t timeout_ns, cudaStream_t s,
                       float* cos_out = nullptr, int64_t ldc = 0);
// Scene diameter sqrt(max d^2) from stats into out[b].
int launch_diameter(const SceneStats* stats, int64_t B, float* out, cudaStream_t s);
// Normalisers from stats (norm_mode 1: the feature range is [0, 2] instead of
// the Gram's extremes).  Optionally also the public [B, 6] float copy.
int launch_finalize_norms(const SceneStats* stats, int64_t B, int norm_mode, SceneNorms* norms,
                          float* norms_out, cudaStream_t s);
// K3 for fp32 features: the FST cost C[b][s][t] into cost + b*N*ldc + s*ldc
// + t for t < N; columns N <= t < ldc are written as 0.  (bf16 features:
// launch_gram_minmax stores the cosines, then launch_fst_apply.)
int launch_cost(const void* feats, int dtype, const float* inv, const float4* tok,
                const float* pos, const int32_t* frame, const SceneNorms* norms,
                const DevParams& P, int64_t B, int64_t N, int64_t D, float* cost, int64_t ldc,
                cudaStream_t s);
// K4: capacity score r and capacity v (Eqs. fst_capacity_score, fst_capacity).
// cos (may be null): every cosine, [B][N][ldc], as the normaliser pass
// stores it; the pairs' cosines are then read from it, not recomputed.
int launch_capacity(const void* feats, int dtype, const float* inv, const float* pos,
                    const int32_t* frame, const SceneNorms* norms, const int32_t* nbr,
                    const DevParams& P, int64_t B, int64_t N, int64_t D, float* r, float* v,
                    float* v_out, cudaStream_t s, const float* cos = nullptr,
                    int64_t ldc = 0, const int32_t* pos_of = nullptr);
// Local SGS, bf16 features: the same slab computed from the stored cosines
// (cos [B][N][ldc], as the normaliser pass writes them), without a dense cost.
// (pos_of given: cos(t, j) at [min(pos)][max(pos)] of the flagged Morton tiles).
int launch_slab_cos(const float* cos, int64_t ldc, const int32_t* nbr, const float4* tok,
                    const int32_t* frame, const SceneNorms* norms, const DevParams& P, int64_t B,
                    int64_t N, float* slab, cudaStream_t s, const int32_t* pos_of = nullptr);
// Local SGS with the bounded normaliser, bf16 features: Morton-ordered
// features and token records, each token's position, and the list of
// 256 x 256 position tiles holding a neighbour pair (units (b << 16) |
// (P << 8) | J, count in *n_units; at most B * T * T units, T = local_tiles(N)).
int local_tiles(int64_t N);
int launch_local_blocks(const void* feats, const float4* tok, const int32_t* perm,
                        const int32_t* nbr, int kk, int64_t B, int64_t N, int64_t D,
                        void* feats_m, float4* tok_m, int32_t* pos_of, uint8_t* flags,
                        uint32_t* units, int* n_units, cudaStream_t s);
// The listed tiles of the Gram of the Morton-ordered bf16 features, whole,
// stored at their position coordinates in cos_out [B][N][ldc].
int launch_gram_tiles(const void* feats_m, const float4* tok_m, int64_t B, int64_t N, int64_t D,
                      const uint32_t* units, const int* n_units, int64_t max_units, int* status,
                      uint64_t timeout_ns, cudaStream_t s, float* cos_out, int64_t ldc);
// Local SGS: slab[b][t][k] = C(t, M_g(t)[k]) gathered from the dense cost.
int launch_slab(const float* cost, int64_t ldc, const int32_t* nbr, const DevParams& P,
                int64_t B, int64_t N, float* slab, cudaStream_t s);
// Column tiles of the elementwise cost pass: the number of partial row sums
// it writes per row into g0, [B][fst_apply_slots(ldc)][N].
int fst_apply_slots(int64_t ldc);
// K5: K greedy steps; order32[b*K + l] = token added at step l.  Local
// lazy SGS (g < N) also needs rev_off [B][N+1] and rev [B][N*g] (scratch for
// the reverse neighbourhoods).
int launch_sgs(const float* cost, int64_t ldc, const float* slab, const int32_t* nbr,
               const float* v, const DevParams& P, int64_t B, int64_t N, int64_t K,
               int32_t* order32, float* gains, double* objective, uint64_t* partials,
               uint32_t* counters, int* status, cudaStream_t s, const float* g0 = nullptr,
               int32_t* rev_off = nullptr, int32_t* rev = nullptr);
// K5 as Sec. 3.5 prints it (sgs_mode 2): entropic semi-relaxed OT residual
// and the residual-weighted local cost; needs the dense cost [B][N][ldc]
// and sgs_literal_ws_bytes(B, N, K) bytes of scratch (256-byte aligned).
size_t sgs_literal_ws_bytes(int64_t B, int64_t N, int64_t K);
int launch_sgs_literal(const float* cost, int64_t ldc, const int32_t* nbr, const float* v,
                       const DevParams& P, int64_t B, int64_t N, int64_t K, int32_t* order32,
                       float* gains, double* objective, void* scratch, cudaStream_t s);
// Sort the B rows of K int32 indices ascending into int64 (and copy the
// unsorted order out as int64 if order64 != NULL).
int launch_sort_kept(const int32_t* idx32, int64_t B, int64_t K, int64_t* kept,
                     int64_t* order64, cudaStream_t s);
// K6: Morton order perm[b*N + p].
int launch_morton(const float* pos, const SceneStats* stats, const DevParams& P, int64_t B,
                  int64_t N, int32_t* perm, cudaStream_t s);
// K7: capacity-guided group starts gs[b*(K+1) + q] (int32).
int launch_groups(const float* v, const int32_t* perm, int64_t B, int64_t N, int64_t K,
                  uint64_t* prefix, int32_t* gs, cudaStream_t s);
// K8: per-group prototype and its score; objective = sum of scores.
int launch_lite_proto(const void* feats, int dtype, const float* inv, const float* pos,
                      const int32_t* frame, const SceneNorms* norms, const float* v,
                      const int32_t* perm, const int32_t* gs, const DevParams& P, int64_t B,
                      int64_t N, int64_t D, int64_t K, int32_t* proto, double* score,
                      double* objective, cudaStream_t s);
// K9: row gather of the kept tokens.
int launch_gather(const void* feats, int dtype, const float* pos, const int32_t* frame,
                  int64_t B, int64_t N, int64_t D, const int64_t* kept, int64_t K,
                  void* feats_out, float* pos_out, int32_t* frame_out, int32_t* status,
                  cudaStream_t s);
// Barrier self-test (see coverprune_barrier_selftest).
int launch_barrier_selftest(int n_blocks, int expected, uint64_t timeout_ns, uint32_t* ctr,
                            int* status, cudaStream_t s);

// Largest N the selection kernels keep in shared memory.
constexpr int64_t kMaxSelectN = 16384;
// Largest N whose neighbour keys fit one block's shared memory.
constexpr int64_t kMaxKnnN = 49152;

// Counts one kernel launch under the calling thread's current stage.
void note_launch();
// Records "where: CUDA error name" as the calling thread's last error.
void note_cuda_error(const char* where, cudaError_t e);
inline int cuda_status(cudaError_t e, const char* where = "cuda call") {
  if (e == cudaSuccess) return CP_OK;
  note_cuda_error(where, e);
  (void)cudaGetLastError();  // do not let a failed call resurface at the next launch
  return CP_ECUDA;
}
// After every <<<>>> launch: count it and report launch errors.
inline int launch_status(const char* where) {
  note_launch();
  return cuda_status(cudaGetLastError(), where);
}
#define last_launch_status() launch_status(__func__)
// Records a plain message as the calling thread's last error.
void note_message(const char* msg);

#define CP_TRY_STATUS(x)          \
  do {                            \
    int _st = (x);                \
    if (_st != CP_OK) return _st; \
  } while (0)

}  // namespace cp
