// Host side of the C ABI declared in include/coverprune.h: argument
// validation (nothing is launched on bad input), workspace planning and the
// launch sequence of each entry point.
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <vector>

#include "internal.h"

namespace cp {

// Tensor-core (bf16) and SIMT (fp32) variants of the Gram kernels.
int launch_gram_minmax_simt(const void* feats, int dtype, const float* inv, int64_t B, int64_t N,
                            int64_t D, SceneStats* stats, cudaStream_t s);
int launch_cost_simt(const void* feats, int dtype, const float* inv, const float* pos,
                     const int32_t* frame, const SceneNorms* norms, const DevParams& P, int64_t B,
                     int64_t N, int64_t D, float* cost, int64_t ldc, cudaStream_t s);
int64_t sgs_partials_count(int64_t B, int64_t N);
int launch_gram_minmax_tc(const void* feats, const float4* tok, int64_t B, int64_t N, int64_t D,
                          SceneStats* stats, int* status, uint64_t timeout_ns, cudaStream_t s,
                          float* cos_out, int64_t ldc);
int launch_fst_apply(float* cost, int64_t ldc, int64_t B, int64_t N, const float4* tok,
                     const int32_t* frame, const SceneNorms* norms, const DevParams& P,
                     const float* v, float* g0, cudaStream_t s);

// ---------------------------------------------------------------------------
// Stage timing and launch counting.
// ---------------------------------------------------------------------------
static std::atomic<int64_t> g_launches[CP_STAGE_COUNT];
static std::atomic<int> g_prof_on{0};
static std::mutex g_prof_mu;
struct StageEvents {
  int stage;
  cudaEvent_t start, stop;
};
static std::vector<StageEvents> g_prof_events;
static thread_local int t_stage = CP_STAGE_PREP;

void note_launch() { g_launches[t_stage].fetch_add(1, std::memory_order_relaxed); }

static thread_local char t_last_error[256] = "";

void note_message(const char* msg) { snprintf(t_last_error, sizeof(t_last_error), "%s", msg); }

void note_cuda_error(const char* where, cudaError_t e) {
  snprintf(t_last_error, sizeof(t_last_error), "%s: %s (%s)", where, cudaGetErrorName(e),
           cudaGetErrorString(e));
}

// Marks the kernels launched while it lives as belonging to `stage`; with
// profiling on, brackets them with CUDA events on the call's stream.
class Stage {
 public:
  Stage(int stage, cudaStream_t s) : prev_(t_stage), s_(s) {
    t_stage = stage;
    ev_.stage = stage;
    if (g_prof_on.load(std::memory_order_relaxed) &&
        cudaEventCreate(&ev_.start) == cudaSuccess) {
      if (cudaEventCreate(&ev_.stop) == cudaSuccess) {
        cudaEventRecord(ev_.start, s_);
        active_ = true;
      } else {
        cudaEventDestroy(ev_.start);
      }
    }
  }
  ~Stage() {
    if (active_) {
      cudaEventRecord(ev_.stop, s_);
      std::lock_guard<std::mutex> lk(g_prof_mu);
      g_prof_events.push_back(ev_);
    }
    t_stage = prev_;
  }

 private:
  int prev_;
  cudaStream_t s_;
  StageEvents ev_{};
  bool active_ = false;
};

// ---------------------------------------------------------------------------
// Device attribute cache.
// ---------------------------------------------------------------------------
static std::mutex g_dev_mu;
static DeviceInfo g_dev[64];
static bool g_dev_ok[64];

int device_info(DeviceInfo* out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return CP_ECUDA;
  std::lock_guard<std::mutex> lk(g_dev_mu);
  if (!g_dev_ok[dev]) {
    DeviceInfo di{};
    if (cudaDeviceGetAttribute(&di.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&di.max_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess ||
        cudaDeviceGetAttribute(&di.cc_major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&di.cc_minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
      return CP_ECUDA;
    g_dev[dev] = di;
    g_dev_ok[dev] = true;
  }
  *out = g_dev[dev];
  return CP_OK;
}

// bf16 features: tcgen05 tensor cores; fp32 features: fp32 FMA tiles (TF32
// would round the features to 10 mantissa bits).  cos_out (bf16 only; may
// be null): every cosine stored [B][N][ldc] for the elementwise cost pass.
int launch_gram_minmax(const void* feats, int dtype, const float* inv, const float4* tok,
                       int64_t B, int64_t N, int64_t D, SceneStats* stats, int* status,
                       uint64_t timeout_ns, cudaStream_t s, float* cos_out, int64_t ldc) {
  if (dtype == CP_BF16)
    return launch_gram_minmax_tc(feats, tok, B, N, D, stats, status, timeout_ns, s, cos_out, ldc);
  return launch_gram_minmax_simt(feats, dtype, inv, B, N, D, stats, s);
}

// fp32 features: the FST cost on the SIMT cores (bf16 features take the
// stored cosines and launch_fst_apply instead).
int launch_cost(const void* feats, int dtype, const float* inv, const float4* tok,
                const float* pos, const int32_t* frame, const SceneNorms* norms,
                const DevParams& P, int64_t B, int64_t N, int64_t D, float* cost, int64_t ldc,
                cudaStream_t s) {
  if (dtype == CP_BF16) {
    note_message("launch_cost: bf16 features take the stored-cosine cost pass");
    return CP_EUNSUPPORTED;
  }
  return launch_cost_simt(feats, dtype, inv, pos, frame, norms, P, B, N, D, cost, ldc, s);
}

// ---------------------------------------------------------------------------
// Validation
// ---------------------------------------------------------------------------
static bool finite_nonneg(float x) { return isfinite(x) && x >= 0.0f; }
static bool aligned(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

static int check_params(const cp_params* p) {
  if (!p || p->struct_size != sizeof(cp_params)) return CP_EINVAL;
  if (!finite_nonneg(p->lambda_f) || !finite_nonneg(p->lambda_x) || !finite_nonneg(p->lambda_tau))
    return CP_EINVAL;
  if (!finite_nonneg(p->alpha_f) || !finite_nonneg(p->alpha_x) || !finite_nonneg(p->alpha_tau))
    return CP_EINVAL;
  if (!(isfinite(p->kappa) && p->kappa > 0.0f)) return CP_EINVAL;
  if (!(isfinite(p->voxel_m) && p->voxel_m > 0.0f)) return CP_EINVAL;
  if (!isfinite(p->m0)) return CP_EINVAL;
  if (!(isfinite(p->timeout_ms) && p->timeout_ms > 0.0f)) return CP_EINVAL;
  if (p->n_cap < 0 || p->g < 0) return CP_EINVAL;
  if (p->capacity_mode != 0 && p->capacity_mode != 1) return CP_EINVAL;
  if (p->sgs_mode < 0 || p->sgs_mode > 2) return CP_EINVAL;
  if (!(isfinite(p->sot_eps) && p->sot_eps > 0.0f)) return CP_EINVAL;
  if (p->sot_iters < 1 || p->sot_iters > 10000) return CP_EINVAL;
  if (p->norm_mode != 0 && p->norm_mode != 1) return CP_EINVAL;
  return CP_OK;
}

static int check_shapes(int dtype, int64_t B, int64_t N, int64_t D, int64_t K) {
  if (dtype != CP_F32 && dtype != CP_BF16) return CP_EINVAL;
  if (B < 0 || N < 0 || K < 0 || K > N || D < 1) return CP_EINVAL;
  if (B > 65535 || N > 0x7FFFFFFF) return CP_EINVAL;
  if (dtype == CP_BF16 && D % 8 != 0) return CP_EINVAL;
  if (dtype == CP_F32 && D % 4 != 0) return CP_EINVAL;
  return CP_OK;
}

static DevParams dev_params(const cp_params* p, int64_t N) {
  DevParams d{};
  d.lambda_f = p->lambda_f;
  d.lambda_x = p->lambda_x;
  d.lambda_tau = p->lambda_tau;
  d.kappa = p->kappa;
  d.inv_log1p_kappa = (float)(1.0 / log1p((double)p->kappa));
  d.alpha_f = p->alpha_f;
  d.alpha_x = p->alpha_x;
  d.alpha_tau = p->alpha_tau;
  d.voxel = p->voxel_m;
  d.m0 = p->m0 > 0.0f ? p->m0 : p->lambda_f + p->lambda_x + p->lambda_tau;
  const int64_t nmax = N > 0 ? N - 1 : 0;
  d.n_cap = (int)(p->n_cap < nmax ? p->n_cap : nmax);
  d.g = (p->g == 0 || p->g >= N) ? (int)N : p->g;
  d.kk = d.g < N ? (d.n_cap > d.g - 1 ? d.n_cap : d.g - 1) : d.n_cap;
  d.cap_mode = p->capacity_mode;
  d.sgs_mode = p->sgs_mode;
  d.norm_mode = p->norm_mode;
  d.sot_eps = p->sot_eps;
  d.sot_iters = p->sot_iters;
  d.timeout_ns = (uint64_t)((double)p->timeout_ms * 1.0e6);
  return d;
}

// ---------------------------------------------------------------------------
// Workspace plan.  Every region starts on a 256-byte boundary.
// ---------------------------------------------------------------------------
struct Plan {
  size_t hdr, counters, stats, norms, inv, tok, nbr, r, v;
  size_t grid_info, grid_start, grid_pts;         // neighbour grid (kk <= kKnnGridMax)
  size_t cost, slab, partials, order32, g0;       // select
  size_t lit;                                     // literal SGS (sgs_mode 2) scratch
  size_t lfeats, ltok, lperm, lpos, lflags, lunits, lnunits;  // local Morton tiles
  size_t rev_off, rev;                            // local SGS reverse neighbourhoods
  size_t perm, prefix, gs, proto, score;          // lite
  size_t total;
  int64_t ldc;
};

static size_t align_up(size_t x) { return (x + 255) & ~(size_t)255; }


// Workspace of coverprune_knn: status block, scene statistics, the grid.
static size_t knn_ws_bytes(int64_t B, int64_t N) {
  return align_up(256) + align_up(sizeof(SceneStats) * (size_t)B) +
         align_up(sizeof(GridInfo) * (size_t)B) +
         align_up(sizeof(int32_t) * (size_t)B * (size_t)(grid_cells_max(N) + 1)) +
         align_up(sizeof(float4) * (size_t)B * (size_t)N);
}

// Local SGS with the bounded feature normaliser on bf16 features computes
// only the Morton tiles that hold a neighbour pair (local_slab.cu), not the
// all-pairs Gram.
static bool local_tiles_path(int op, int dtype, int64_t N, const DevParams& d) {
  return op == CP_OP_SELECT && dtype == CP_BF16 && d.g < N && d.norm_mode == 1 &&
         d.sgs_mode != 2;
}

static void plan_ws(int op, int64_t B, int64_t N, int64_t D, int64_t K, int dtype,
                    const DevParams& d, Plan* pl) {
  memset(pl, 0, sizeof(*pl));
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t at = off;
    off = align_up(off + (bytes > 0 ? bytes : 1));
    return at;
  };
  const size_t BN = (size_t)B * (size_t)N;
  pl->ldc = (N + 3) & ~(int64_t)3;
  pl->hdr = take(256);  // [0] status word, [64] self-test counter
  pl->counters = take(sizeof(uint32_t) * (size_t)B);
  pl->stats = take(sizeof(SceneStats) * (size_t)B);
  pl->norms = take(sizeof(SceneNorms) * (size_t)B);
  pl->inv = take(sizeof(float) * BN);
  pl->tok = take(sizeof(float4) * BN);
  pl->nbr = take(sizeof(int32_t) * BN * (size_t)d.kk);
  if (d.kk <= kKnnGridMax) {
    pl->grid_info = take(sizeof(GridInfo) * (size_t)B);
    pl->grid_start = take(sizeof(int32_t) * (size_t)B * (size_t)(grid_cells_max(N) + 1));
    pl->grid_pts = take(sizeof(float4) * BN);
  }
  pl->r = take(sizeof(float) * BN);
  pl->v = take(sizeof(float) * BN);
  if (op == CP_OP_SELECT) {
    pl->cost = take(sizeof(float) * BN * (size_t)pl->ldc);
    if (d.sgs_mode == 2) pl->lit = take(sgs_literal_ws_bytes(B, N, K));
    if (d.g < N && d.sgs_mode != 2) {
      pl->slab = take(sizeof(float) * BN * (size_t)d.g);
      pl->rev_off = take(sizeof(int32_t) * (BN + (size_t)B));
      pl->rev = take(sizeof(int32_t) * BN * (size_t)d.g);
    }
    if (local_tiles_path(op, dtype, N, d)) {
      const size_t T = (size_t)local_tiles(N);
      pl->lfeats = take(2 * BN * (size_t)D);
      pl->ltok = take(sizeof(float4) * BN);
      pl->lperm = take(sizeof(int32_t) * BN);
      pl->lpos = take(sizeof(int32_t) * BN);
      pl->lflags = take((size_t)B * T * T);
      pl->lunits = take(sizeof(uint32_t) * (size_t)B * T * T);
      pl->lnunits = take(sizeof(int));
    }
    pl->partials = take(sizeof(uint64_t) * (size_t)sgs_partials_count(B, N));
    pl->order32 = take(sizeof(int32_t) * (size_t)B * (size_t)K);
    pl->g0 = take(sizeof(float) * BN * (size_t)fst_apply_slots(pl->ldc));
  } else if (op == CP_OP_LITE) {
    pl->perm = take(sizeof(int32_t) * BN);
    pl->prefix = take(sizeof(uint64_t) * BN);
    pl->gs = take(sizeof(int32_t) * (size_t)B * (size_t)(K + 1));
    pl->proto = take(sizeof(int32_t) * (size_t)B * (size_t)K);
    pl->score = take(sizeof(double) * (size_t)B * (size_t)K);
  }
  pl->total = off;
}

static int check_limits(int op, int64_t N, const DevParams& d) {
  if (op == CP_OP_COST) {
    if (N > kMaxKnnN) return CP_EUNSUPPORTED;
  } else if (N > kMaxSelectN) {
    return CP_EUNSUPPORTED;
  }
  // neighbour list + keys of one kNN block must fit shared memory
  int64_t L = 2;
  while (L < d.kk) L <<= 1;
  if (8 * L + 4 * N > 200 * 1024) return CP_EUNSUPPORTED;
  return CP_OK;
}

template <typename T>
static T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<unsigned char*>(ws) + off);
}

#define CP_TRY(x)                  \
  do {                             \
    int _st = (x);                 \
    if (_st != CP_OK) return _st;  \
  } while (0)

// Stats, inverse norms, neighbours and normalisers: the shared front of
// every entry point.
// cos_out (bf16 features only, may be null): the normaliser pass also stores
// every cosine there, [B][N][ldc], for launch_fst_apply.
static int run_front(const void* feats, int dtype, const float* pos, const int32_t* frame,
                     int64_t B, int64_t N, int64_t D, const DevParams& d, const Plan& pl, void* ws,
                     float* norms_out, cudaStream_t s, float* cos_out = nullptr,
                     int64_t ldc = 0) {
  int* status = at<int>(ws, pl.hdr);
  SceneStats* stats = at<SceneStats>(ws, pl.stats);
  {
    Stage st(CP_STAGE_PREP, s);
    CP_TRY(cuda_status(cudaMemsetAsync(status, 0, kStatusBytes, s), "status block"));
    CP_TRY(launch_scene_stats(pos, frame, B, N, stats, s));
    CP_TRY(launch_inv_norms(feats, dtype, pos, B, N, D, at<float>(ws, pl.inv),
                            at<float4>(ws, pl.tok), s));
    if (d.kk <= kKnnGridMax)
      CP_TRY(launch_knn_grid(pos, B, N, d.kk, at<int32_t>(ws, pl.nbr), stats,
                             at<GridInfo>(ws, pl.grid_info), at<int32_t>(ws, pl.grid_start),
                             at<float4>(ws, pl.grid_pts), s));
    else
      CP_TRY(launch_knn(pos, at<float4>(ws, pl.tok), B, N, d.kk, at<int32_t>(ws, pl.nbr), stats,
                        s));
  }
  // the Gram gives the min-max feature normaliser and, for bf16 inputs, the
  // stored cosines; with the bounded normaliser and no cosines to store
  // (Lite, or fp32 inputs) it does not run
  cos_out = dtype == CP_BF16 ? cos_out : nullptr;
  if (d.norm_mode == 0 || cos_out) {
    Stage st(CP_STAGE_GRAM, s);
    CP_TRY(launch_gram_minmax(feats, dtype, at<float>(ws, pl.inv), at<float4>(ws, pl.tok), B, N,
                              D, stats, status, d.timeout_ns, s, cos_out, ldc));
  }
  Stage st(CP_STAGE_PREP, s);
  CP_TRY(launch_finalize_norms(stats, B, d.norm_mode, at<SceneNorms>(ws, pl.norms), norms_out,
                               s));
  return CP_OK;
}

static int check_inputs(const void* feats, const float* pos, const int32_t* frame) {
  if (!feats || !pos || !frame) return CP_EINVAL;
  if (!aligned(feats, 16) || !aligned(pos, 4) || !aligned(frame, 4)) return CP_EINVAL;
  return CP_OK;
}

static int check_ws(int op, int64_t B, int64_t N, int64_t D, int64_t K, int dtype,
                    const DevParams& d, void* ws, size_t ws_bytes, Plan* pl) {
  plan_ws(op, B, N, D, K, dtype, d, pl);
  if (!ws || !aligned(ws, 256) || ws_bytes < pl->total) return CP_EWORKSPACE;
  return CP_OK;
}

// Records the caller's inputs_done event (cp_params) on the call's stream.
static int record_inputs_done(const cp_params* p, cudaStream_t s) {
  if (!p->inputs_done) return CP_OK;
  return cuda_status(cudaEventRecord(static_cast<cudaEvent_t>(p->inputs_done), s),
                     "inputs_done event");
}

}  // namespace cp

using namespace cp;

extern "C" {

void cp_default_params(cp_params* p) {
  if (!p) return;
  memset(p, 0, sizeof(*p));
  p->struct_size = sizeof(cp_params);
  p->lambda_f = p->lambda_x = p->lambda_tau = 1.0f;
  p->kappa = 10.0f;
  p->alpha_f = p->alpha_x = p->alpha_tau = 1.0f;
  p->n_cap = 8;
  p->g = 0;
  p->capacity_mode = 0;
  p->voxel_m = 0.2f;
  p->m0 = 0.0f;
  p->timeout_ms = 2000.0f;
  p->sgs_mode = 0;
  p->norm_mode = 0;
  p->sot_eps = 0.05f;
  p->sot_iters = 20;
  p->inputs_done = nullptr;
}

int64_t coverprune_budget(double R, int64_t N) {
  if (!(R > 0.0 && R <= 1.0) || N < 1) return -1;
  double k = ceil(R * (double)N - 1e-9);
  if (k < 1.0) k = 1.0;
  if (k > (double)N) k = (double)N;
  return (int64_t)k;
}

const char* coverprune_status_string(int status) {
  switch (status) {
    case CP_OK: return "ok";
    case CP_EINVAL: return "invalid argument";
    case CP_EWORKSPACE: return "workspace missing, misaligned or too small";
    case CP_ECUDA: return "CUDA error";
    case CP_ETIMEOUT: return "device-side wait timed out";
    case CP_EUNSUPPORTED: return "unsupported size or configuration";
    case CP_EDEVICE: return "device-side consistency check failed";
    default: return "unknown status";
  }
}

int coverprune_version(void) { return 100; }

const char* coverprune_last_error(void) { return t_last_error; }

int coverprune_workspace_size(int op, int64_t B, int64_t N, int64_t D, int64_t K, int dtype,
                              const cp_params* p, size_t* bytes) {
  if (!bytes) return CP_EINVAL;
  CP_TRY(check_params(p));
  if (op != CP_OP_COST && op != CP_OP_SELECT && op != CP_OP_LITE && op != CP_OP_KNN)
    return CP_EINVAL;
  if (op == CP_OP_KNN) {
    if (B < 0 || N < 0 || B > 65535 || N > kMaxKnnN) return CP_EINVAL;
    *bytes = knn_ws_bytes(B > 0 ? B : 1, N);
    return CP_OK;
  }
  CP_TRY(check_shapes(dtype, B, N, D, op == CP_OP_COST ? 0 : K));
  DevParams d = dev_params(p, N);
  CP_TRY(check_limits(op, N, d));
  Plan pl;
  plan_ws(op, B, N, D, op == CP_OP_COST ? 0 : K, dtype, d, &pl);
  *bytes = pl.total;
  return CP_OK;
}

int coverprune_check(const void* ws, cp_stream_t stream) {
  if (!ws) return CP_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  CP_TRY(cuda_status(cudaStreamSynchronize(s), "coverprune_check: stream"));
  int st = 0;
  CP_TRY(cuda_status(cudaMemcpy(&st, ws, sizeof(int), cudaMemcpyDeviceToHost),
                     "coverprune_check: status copy"));
  return st;
}

int coverprune_call_stats(const void* ws, cp_stream_t stream, cp_call_stats* out) {
  if (!ws || !out) return CP_EINVAL;
  CP_TRY(cuda_status(cudaStreamSynchronize((cudaStream_t)stream), "coverprune_call_stats: stream"));
  unsigned long long v[3] = {0, 0, 0};
  CP_TRY(cuda_status(cudaMemcpy(v, static_cast<const unsigned char*>(ws) + kCallStatsOffset,
                                sizeof(v), cudaMemcpyDeviceToHost),
                     "coverprune_call_stats: copy"));
  out->gain_evaluations = v[0];
  out->rounds = v[1];
  out->cost_bytes_read = v[2];
  return CP_OK;
}

int coverprune_cost(const void* feats, int dtype, const float* pos, const int32_t* frame,
                    int64_t B, int64_t N, int64_t D, const cp_params* p, float* cost,
                    float* capacity, float* norms, void* ws, size_t ws_bytes, cp_stream_t stream) {
  CP_TRY(check_params(p));
  CP_TRY(check_shapes(dtype, B, N, D, 0));
  if (B == 0 || N == 0) return CP_OK;
  CP_TRY(check_inputs(feats, pos, frame));
  if ((cost && !aligned(cost, 4)) || (capacity && !aligned(capacity, 4)) ||
      (norms && !aligned(norms, 4)))
    return CP_EINVAL;
  DevParams d = dev_params(p, N);
  CP_TRY(check_limits(CP_OP_COST, N, d));
  Plan pl;
  CP_TRY(check_ws(CP_OP_COST, B, N, D, 0, dtype, d, ws, ws_bytes, &pl));
  cudaStream_t s = (cudaStream_t)stream;
  // bf16: the normaliser pass stores the cosines into the output (the
  // capacity reads its pairs there), then one elementwise pass turns them
  // into the cost
  CP_TRY(run_front(feats, dtype, pos, frame, B, N, D, d, pl, ws, norms, s, cost, N));
  const SceneNorms* nm = at<SceneNorms>(ws, pl.norms);
  const float* cosines = dtype == CP_BF16 ? cost : nullptr;
  if (capacity) {
    Stage st(CP_STAGE_CAPACITY, s);
    CP_TRY(launch_capacity(feats, dtype, at<float>(ws, pl.inv), pos, frame, nm,
                           at<int32_t>(ws, pl.nbr), d, B, N, D, at<float>(ws, pl.r),
                           at<float>(ws, pl.v), capacity, s, cosines, N));
  }
  if (cost) {
    Stage st(CP_STAGE_COST, s);
    if (dtype == CP_BF16)
      CP_TRY(launch_fst_apply(cost, N, B, N, at<float4>(ws, pl.tok), frame, nm, d, nullptr,
                              nullptr, s));
    else
      CP_TRY(launch_cost(feats, dtype, at<float>(ws, pl.inv), at<float4>(ws, pl.tok), pos, frame,
                         nm, d, B, N, D, cost, N, s));
  }
  return record_inputs_done(p, s);
}

int coverprune_select(const void* feats, int dtype, const float* pos, const int32_t* frame,
                      int64_t B, int64_t N, int64_t D, int64_t K, const cp_params* p,
                      int64_t* kept, int64_t* order, float* gains, double* objective, void* ws,
                      size_t ws_bytes, cp_stream_t stream) {
  CP_TRY(check_params(p));
  CP_TRY(check_shapes(dtype, B, N, D, K));
  if (B == 0 || N == 0 || K == 0) return CP_OK;
  CP_TRY(check_inputs(feats, pos, frame));
  if (!kept || !aligned(kept, 8) || (order && !aligned(order, 8)) ||
      (gains && !aligned(gains, 4)) || (objective && !aligned(objective, 8)))
    return CP_EINVAL;
  DevParams d = dev_params(p, N);
  CP_TRY(check_limits(CP_OP_SELECT, N, d));
  Plan pl;
  CP_TRY(check_ws(CP_OP_SELECT, B, N, D, K, dtype, d, ws, ws_bytes, &pl));
  cudaStream_t s = (cudaStream_t)stream;
  int* status = at<int>(ws, pl.hdr);
  float* C = at<float>(ws, pl.cost);
  // the all-pairs Gram stores every cosine into C for the cost pass; the
  // local path with the bounded normaliser stores only the Morton tiles it
  // needs (below), so the front runs no Gram for it
  const bool tiles = local_tiles_path(CP_OP_SELECT, dtype, N, d);
  CP_TRY(run_front(feats, dtype, pos, frame, B, N, D, d, pl, ws, nullptr, s, tiles ? nullptr : C,
                   pl.ldc));
  const SceneNorms* nm = at<SceneNorms>(ws, pl.norms);
  const float* inv = at<float>(ws, pl.inv);
  const int32_t* nbr = at<int32_t>(ws, pl.nbr);
  float* v = at<float>(ws, pl.v);
  const int32_t* pos_of = nullptr;  // tiles: cos(t, j) at [min(pos)][max(pos)] of C
  if (tiles) {
    Stage st(CP_STAGE_SLAB, s);
    int32_t* perm = at<int32_t>(ws, pl.lperm);
    const int64_t T = local_tiles(N);
    CP_TRY(launch_morton(pos, at<SceneStats>(ws, pl.stats), d, B, N, perm, s));
    CP_TRY(launch_local_blocks(feats, at<float4>(ws, pl.tok), perm, nbr, d.kk, B, N, D,
                               at<void>(ws, pl.lfeats), at<float4>(ws, pl.ltok),
                               at<int32_t>(ws, pl.lpos), at<uint8_t>(ws, pl.lflags),
                               at<uint32_t>(ws, pl.lunits), at<int>(ws, pl.lnunits), s));
    CP_TRY(launch_gram_tiles(at<void>(ws, pl.lfeats), at<float4>(ws, pl.ltok), B, N, D,
                             at<uint32_t>(ws, pl.lunits), at<int>(ws, pl.lnunits), B * T * T,
                             status, d.timeout_ns, s, C, pl.ldc));
    pos_of = at<int32_t>(ws, pl.lpos);
  }
  {
    Stage st(CP_STAGE_CAPACITY, s);
    CP_TRY(launch_capacity(feats, dtype, inv, pos, frame, nm, nbr, d, B, N, D, at<float>(ws, pl.r),
                           v, nullptr, s, dtype == CP_BF16 ? C : nullptr, pl.ldc, pos_of));
  }
  // the dense lazy selection starts from bounds the cost pass sums
  float* g0 = (dtype == CP_BF16 && d.g >= N && d.sgs_mode == 0) ? at<float>(ws, pl.g0) : nullptr;
  // local SGS reads only the N x g slab: for bf16 it comes straight from
  // the stored cosines, and the dense cost is never formed (the literal rule
  // transports from the selected tokens to every token, so it takes the
  // dense cost whatever g is)
  float* slab = (d.g < N && d.sgs_mode != 2) ? at<float>(ws, pl.slab) : nullptr;
  {
    Stage st(CP_STAGE_COST, s);
    if (dtype == CP_BF16 && slab)
      CP_TRY(launch_slab_cos(C, pl.ldc, nbr, at<float4>(ws, pl.tok), frame, nm, d, B, N, slab,
                             s, pos_of));
    else if (dtype == CP_BF16)
      CP_TRY(launch_fst_apply(C, pl.ldc, B, N, at<float4>(ws, pl.tok), frame, nm, d, v, g0, s));
    else
      CP_TRY(launch_cost(feats, dtype, inv, at<float4>(ws, pl.tok), pos, frame, nm, d, B, N, D, C,
                         pl.ldc, s));
  }
  // the greedy selection reads none of feats, pos, frame
  CP_TRY(record_inputs_done(p, s));
  int32_t* order32 = at<int32_t>(ws, pl.order32);
  {
    Stage st(CP_STAGE_SGS, s);
    if (slab && dtype != CP_BF16) CP_TRY(launch_slab(C, pl.ldc, nbr, d, B, N, slab, s));
    if (d.sgs_mode == 2)
      CP_TRY(launch_sgs_literal(C, pl.ldc, nbr, v, d, B, N, K, order32, gains, objective,
                                at<void>(ws, pl.lit), s));
    else
      CP_TRY(launch_sgs(C, pl.ldc, slab, nbr, v, d, B, N, K, order32, gains, objective,
                        at<uint64_t>(ws, pl.partials), at<uint32_t>(ws, pl.counters), status, s,
                        g0, slab ? at<int32_t>(ws, pl.rev_off) : nullptr,
                        slab ? at<int32_t>(ws, pl.rev) : nullptr));
  }
  Stage st(CP_STAGE_OUTPUT, s);
  CP_TRY(launch_sort_kept(order32, B, K, kept, order, s));
  return CP_OK;
}

int coverprune_lite_select(const void* feats, int dtype, const float* pos, const int32_t* frame,
                           int64_t B, int64_t N, int64_t D, int64_t K, const cp_params* p,
                           int64_t* kept, int32_t* group_start, double* objective, void* ws,
                           size_t ws_bytes, cp_stream_t stream) {
  CP_TRY(check_params(p));
  CP_TRY(check_shapes(dtype, B, N, D, K));
  if (B == 0 || N == 0 || K == 0) return CP_OK;
  CP_TRY(check_inputs(feats, pos, frame));
  if (!kept || !aligned(kept, 8) || (group_start && !aligned(group_start, 4)) ||
      (objective && !aligned(objective, 8)))
    return CP_EINVAL;
  DevParams d = dev_params(p, N);
  d.g = (int)N;  // Lite uses the capacity neighbours only
  d.kk = d.n_cap;
  CP_TRY(check_limits(CP_OP_LITE, N, d));
  Plan pl;
  CP_TRY(check_ws(CP_OP_LITE, B, N, D, K, dtype, d, ws, ws_bytes, &pl));
  cudaStream_t s = (cudaStream_t)stream;
  CP_TRY(run_front(feats, dtype, pos, frame, B, N, D, d, pl, ws, nullptr, s));
  const SceneNorms* nm = at<SceneNorms>(ws, pl.norms);
  const float* inv = at<float>(ws, pl.inv);
  float* v = at<float>(ws, pl.v);
  {
    Stage st(CP_STAGE_CAPACITY, s);
    CP_TRY(launch_capacity(feats, dtype, inv, pos, frame, nm, at<int32_t>(ws, pl.nbr), d, B, N,
                           D, at<float>(ws, pl.r), v, nullptr, s));
  }
  int32_t* perm = at<int32_t>(ws, pl.perm);
  int32_t* gs = group_start ? group_start : at<int32_t>(ws, pl.gs);
  {
    Stage st(CP_STAGE_LITE_ORDER, s);
    CP_TRY(launch_morton(pos, at<SceneStats>(ws, pl.stats), d, B, N, perm, s));
    CP_TRY(launch_groups(v, perm, B, N, K, at<uint64_t>(ws, pl.prefix), gs, s));
  }
  int32_t* proto = at<int32_t>(ws, pl.proto);
  {
    Stage st(CP_STAGE_LITE_PROTO, s);
    CP_TRY(launch_lite_proto(feats, dtype, inv, pos, frame, nm, v, perm, gs, d, B, N, D, K, proto,
                             at<double>(ws, pl.score), objective, s));
  }
  CP_TRY(record_inputs_done(p, s));
  Stage st(CP_STAGE_OUTPUT, s);
  CP_TRY(launch_sort_kept(proto, B, K, kept, nullptr, s));
  return CP_OK;
}

int coverprune_knn(const float* pos, int64_t B, int64_t N, int64_t k, int32_t* nbr,
                   float* diameter, void* ws, size_t ws_bytes, cp_stream_t stream) {
  if (B < 0 || N < 0 || B > 65535 || k < 0 || (N > 0 && k > N - 1)) return CP_EINVAL;
  if (B == 0 || N == 0) return CP_OK;
  if (N > kMaxKnnN) return CP_EUNSUPPORTED;
  if (!pos || !aligned(pos, 4) || (k > 0 && (!nbr || !aligned(nbr, 4))) ||
      (diameter && !aligned(diameter, 4)))
    return CP_EINVAL;
  int64_t L = 2;
  while (L < k) L <<= 1;
  if (8 * L + 4 * N > 200 * 1024) return CP_EUNSUPPORTED;
  if (!ws || !aligned(ws, 256) || ws_bytes < knn_ws_bytes(B, N)) return CP_EWORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  const size_t st_off = align_up(256);
  const size_t gi_off = st_off + align_up(sizeof(SceneStats) * (size_t)B);
  const size_t gs_off = gi_off + align_up(sizeof(GridInfo) * (size_t)B);
  const size_t gp_off = gs_off + align_up(sizeof(int32_t) * (size_t)B * (grid_cells_max(N) + 1));
  SceneStats* stats = at<SceneStats>(ws, st_off);
  CP_TRY(cuda_status(cudaMemsetAsync(ws, 0, sizeof(int), s)));
  CP_TRY(launch_scene_stats(pos, nullptr, B, N, stats, s));  // frames are not needed
  if (k <= kKnnGridMax)
    CP_TRY(launch_knn_grid(pos, B, N, (int)k, k > 0 ? nbr : nullptr, stats,
                           at<GridInfo>(ws, gi_off), at<int32_t>(ws, gs_off),
                           at<float4>(ws, gp_off), s));
  else
    CP_TRY(launch_knn(pos, nullptr, B, N, (int)k, nbr, stats, s));
  if (diameter) CP_TRY(launch_diameter(stats, B, diameter, s));
  return CP_OK;
}

int coverprune_gather(const void* feats, int dtype, const float* pos, const int32_t* frame,
                      int64_t B, int64_t N, int64_t D, const int64_t* kept, int64_t K,
                      void* feats_out, float* pos_out, int32_t* frame_out, int32_t* status,
                      cp_stream_t stream) {
  CP_TRY(check_shapes(dtype, B, N, D, K));
  if (B == 0 || K == 0) return CP_OK;
  if (!feats || !kept || !feats_out || !aligned(feats, 16) || !aligned(feats_out, 16) ||
      !aligned(kept, 8))
    return CP_EINVAL;
  if ((pos_out && (!pos || !aligned(pos, 4) || !aligned(pos_out, 4))) ||
      (frame_out && (!frame || !aligned(frame, 4) || !aligned(frame_out, 4))) ||
      (status && !aligned(status, 4)))
    return CP_EINVAL;
  Stage st(CP_STAGE_OUTPUT, (cudaStream_t)stream);
  return launch_gather(feats, dtype, pos, frame, B, N, D, kept, K, feats_out, pos_out, frame_out,
                       status, (cudaStream_t)stream);
}

int coverprune_profile_enable(int on) {
  g_prof_on.store(on ? 1 : 0);
  return CP_OK;
}

int coverprune_profile_read(double* ms, int64_t* launches, int n) {
  if (n < 0) return CP_EINVAL;
  std::vector<StageEvents> evs;
  {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    evs.swap(g_prof_events);
  }
  std::vector<double> acc(CP_STAGE_COUNT, 0.0);
  int rc = CP_OK;
  for (const StageEvents& e : evs) {
    float t = 0.0f;
    if (cudaEventSynchronize(e.stop) != cudaSuccess ||
        cudaEventElapsedTime(&t, e.start, e.stop) != cudaSuccess)
      rc = CP_ECUDA;
    acc[e.stage] += t;
    cudaEventDestroy(e.start);
    cudaEventDestroy(e.stop);
  }
  for (int i = 0; i < CP_STAGE_COUNT; ++i) {
    const int64_t c = g_launches[i].exchange(0);
    if (i < n) {
      if (ms) ms[i] = acc[i];
      if (launches) launches[i] = c;
    }
  }
  return rc;
}

int coverprune_barrier_selftest(int32_t n_blocks, int32_t expected, float timeout_ms, void* ws,
                                size_t ws_bytes, cp_stream_t stream) {
  if (!ws || !aligned(ws, 256) || ws_bytes < 256) return CP_EWORKSPACE;
  if (!(isfinite(timeout_ms) && timeout_ms > 0.0f) || n_blocks < 1 || expected < 0)
    return CP_EINVAL;
  int* status = static_cast<int*>(ws);
  uint32_t* ctr = reinterpret_cast<uint32_t*>(static_cast<unsigned char*>(ws) + 64);
  return launch_barrier_selftest(n_blocks, expected, (uint64_t)((double)timeout_ms * 1.0e6), ctr,
                                 status, (cudaStream_t)stream);
}

}  // extern "C"
