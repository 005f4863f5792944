/*
 * coverprune.h -- C ABI of the GB300 (sm_103a) CoverPrune hot path.
 *
 * CoverPrune ("Coverage-Driven Token Pruning for 3D VLMs via Optimal
 * Transport") keeps K of the N visual tokens of a 3D scene so that the kept
 * set covers the whole scene in the optimal-transport sense (Sec. 3.2,
 * Eqs. pruning_problem, 3dto_ot, 3dto_select).  This library computes, on one
 * GPU:
 *   - the Feature-Spatial-Temporal transport cost C      (Sec. 3.3, Eqs. fst_metrics, fst_cost)
 *   - the FST target capacity v                          (Sec. 3.4, Eqs. fst_capacity_score, fst_capacity)
 *   - Spatial-Guided Greedy Selection of K tokens         (Sec. 3.5, Eqs. srpot, local_neighbor,
 *                                                          greedy_flow, sgs_select, sgs_update)
 *   - the CoverPrune-Lite selection                      (Sec. 4, Eqs. lite_group, lite_select)
 *   - the compaction of the kept tokens                  (Sec. 3.2 / Sec. 5.1: the kept tokens
 *                                                          are the LLM's visual input)
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Pointers are DEVICE pointers owned by the caller unless a comment says
 *    otherwise.  The library never allocates device memory and never frees
 *    what it is given.  Scratch memory is the caller's workspace `ws` of at
 *    least coverprune_workspace_size() bytes, 256-byte aligned; it must not
 *    be used by anything else until the stream has passed the call.
 *  - Work is enqueued on `stream` (0 = legacy default stream) and the call
 *    returns without synchronising.  Outputs are valid once the stream has
 *    reached the call.
 *  - A batch of B independent scenes of N tokens each is laid out scene-major
 *    and contiguous:
 *        feats [B, N, D]  row-major, element type `dtype`, base 16-B aligned;
 *                         D % 8 == 0 for CP_BF16, D % 4 == 0 for CP_F32
 *        pos   [B, N, 3]  float32 metres (3D global coordinate x_j)
 *        frame [B, N]     int32 frame index (timestamp tau_j)
 *    Token order is the index space: indices in outputs are int64 in [0, N)
 *    within their scene.
 *  - Errors detectable on the host (bad sizes, NULL or misaligned pointers,
 *    non-finite or out-of-range parameters, too small a workspace) return a
 *    non-zero cp_status before anything is launched.  A CUDA launch error
 *    returns CP_ECUDA.  A condition that only the device can see (a grid
 *    barrier that gave up waiting) is recorded in a status word at the start
 *    of the workspace and is read by coverprune_check().
 *  - Sizes: 0 <= B; 0 <= K <= N.  B == 0, N == 0 or K == 0 are valid no-ops
 *    that write nothing.  The selection entry points need N <= 16384
 *    (their per-scene state lives in on-chip shared memory); larger N returns
 *    CP_EUNSUPPORTED.
 *  - Thread safety: calls on different streams with different workspaces
 *    may run concurrently.  The library's only global state is a per-device
 *    cache of device attributes and kernel attributes, filled on first use.
 */
#ifndef COVERPRUNE_H_
#define COVERPRUNE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* cudaStream_t without pulling in the CUDA headers. */
typedef struct CUstream_st* cp_stream_t;

typedef enum {
  CP_OK = 0,
  CP_EINVAL = 1,       /* bad argument (size, pointer, alignment, parameter) */
  CP_EWORKSPACE = 2,   /* ws NULL / misaligned or ws_bytes too small */
  CP_ECUDA = 3,        /* a CUDA runtime call or launch failed */
  CP_ETIMEOUT = 4,     /* a device-side wait gave up (see coverprune_check) */
  CP_EUNSUPPORTED = 5, /* valid request outside what this build supports */
  CP_EDEVICE = 6       /* a device-side consistency check failed (see coverprune_check) */
} cp_status;

typedef enum { CP_F32 = 0, CP_BF16 = 1 } cp_dtype;

/* Which entry point a workspace is sized for. */
typedef enum {
  CP_OP_COST = 0,
  CP_OP_SELECT = 1,
  CP_OP_LITE = 2,
  CP_OP_KNN = 3
} cp_op;

/*
 * Method parameters.  Fill with cp_default_params() and override fields.
 *   lambda_f, lambda_x, lambda_tau  weights of Eq. fst_cost (>= 0, finite;
 *                                   default 1, 1, 1 as in Sec. 5.1)
 *   kappa                           phi_kappa(x) = log(1+kappa x)/log(1+kappa)
 *                                   of Eq. fst_cost (> 0; default 10 -- the
 *                                   paper gives no value)
 *   alpha_f, alpha_x, alpha_tau     weights of Eq. fst_capacity_score (>= 0;
 *                                   default 1, 1, 1 as in Sec. 5.1)
 *   n_cap                           |N_n(t_j)|, 3D neighbours of the capacity
 *                                   score (>= 0, clamped to N-1; default 8)
 *   g                               |M_g(t)| of Eq. local_neighbor, the
 *                                   token itself plus its g-1 nearest others;
 *                                   0 or >= N means every token (default 0)
 *   capacity_mode                   0 = FST capacity (Sec. 3.4); 1 = uniform
 *                                   v = 1/N (the "w/o FST capacity" ablation)
 *   voxel_m                         Morton cell edge in metres for Lite
 *                                   (> 0; default 0.2)
 *   m0                              coverage cost of a token nobody covers
 *                                   yet; <= 0 means lambda_f+lambda_x+lambda_tau,
 *                                   the largest value C can take (default 0)
 *   timeout_ms                      limit of every device-side wait, after
 *                                   which the kernel records CP_ETIMEOUT and
 *                                   returns (> 0; default 2000)
 *   sgs_mode                        how SGS finds each step's winner: 0 =
 *                                   lazy (a gain computed at an earlier step
 *                                   bounds the current one, so only
 *                                   candidates whose bound could still win
 *                                   are re-evaluated; default), 1 = every
 *                                   gain every step (the same picks); 2 =
 *                                   the rule as Sec. 3.5 prints it: at step
 *                                   l the entropic semi-relaxed OT of Eq.
 *                                   srpot_sinkhorn from the l selected
 *                                   tokens (mass 1/K each) to the target
 *                                   capacity v gives the residual
 *                                   r = [v - P^T 1]_+ (Eq. greedy_flow) and
 *                                   the next token minimises
 *                                   sum_{j in M_g(t)} r_j C(t, j) (Eq.
 *                                   sgs_select; lowest index on ties); a
 *                                   different selection, which scores a
 *                                   candidate whose neighbourhood is already
 *                                   served as 0 and so picks beside the
 *                                   selected tokens (the default reading
 *                                   maximises the coverage gain instead)
 *   sot_eps                         entropic weight eps of Eq. srpot_sinkhorn
 *                                   for sgs_mode 2 (> 0, finite; default
 *                                   0.05 -- the paper gives no value)
 *   sot_iters                       Sinkhorn iterations per greedy step for
 *                                   sgs_mode 2 (1..10000; default 20; the
 *                                   target potentials carry over from the
 *                                   previous step -- the paper gives no
 *                                   iteration count)
 *   norm_mode                       feature normaliser of Eq. fst_cost: 0 =
 *                                   min-max of d_f over all ordered pairs of
 *                                   the scene (Sec. 3.3; default); 1 =
 *                                   bounded, d_f / 2 (d_f = 1 - cos lies in
 *                                   [0, 2]), which needs no all-pairs pass, so
 *                                   Lite runs without the N^2 D Gram (the
 *                                   complexity Sec. 4 states).  The spatial
 *                                   and temporal normalisers are the same in
 *                                   both.  The two agree whenever the scene
 *                                   holds a pair with cos = -1.
 *   inputs_done                     not a method parameter: a cudaEvent_t
 *                                   (passed as void*) or NULL.  When given,
 *                                   the call records it on its stream once it
 *                                   has read the last of feats, pos and frame;
 *                                   work ordered after that event may
 *                                   overwrite them (a serving loop's next
 *                                   upload, say).  coverprune_select records
 *                                   it before its greedy selection, the other
 *                                   calls on return.  The caller owns the
 *                                   event (default NULL).
 */
typedef struct {
  uint32_t struct_size; /* = sizeof(cp_params); set by cp_default_params */
  float lambda_f, lambda_x, lambda_tau;
  float kappa;
  float alpha_f, alpha_x, alpha_tau;
  int32_t n_cap;
  int32_t g;
  int32_t capacity_mode;
  float voxel_m;
  float m0;
  float timeout_ms;
  int32_t sgs_mode;
  int32_t norm_mode;
  float sot_eps;
  int32_t sot_iters;
  void* inputs_done;
} cp_params;

/* Fills *p with the defaults listed above.  Host only; p must not be NULL. */
void cp_default_params(cp_params* p);

/* K = ceil(R * N) of Sec. 3.2 (pruning budget for retention ratio R in
 * (0, 1]), clamped to [1, N].  Returns -1 if R is not in (0, 1] or N < 1. */
int64_t coverprune_budget(double R, int64_t N);

/* Bytes of workspace that entry point `op` needs for these sizes; written to
 * *bytes.  Returns CP_OK or CP_EINVAL/CP_EUNSUPPORTED for sizes the entry
 * point would reject.  Host only; touches no device. */
int coverprune_workspace_size(int op, int64_t B, int64_t N, int64_t D, int64_t K,
                              int dtype, const cp_params* p, size_t* bytes);

/* Static string for a cp_status value ("unknown status" otherwise). */
const char* coverprune_status_string(int status);

/* Synchronises `stream`, then reads the device status word that the last
 * call using workspace `ws` left there: CP_OK, or CP_ETIMEOUT if a grid
 * barrier or pipeline wait gave up.  Returns CP_ECUDA if the stream itself
 * reports an error. */
int coverprune_check(const void* ws, cp_stream_t stream);

/*
 * coverprune_cost -- the FST cost and capacity of each scene.
 *   Sec. 3.3 Eqs. fst_metrics, fst_cost; Sec. 3.4 Eqs. fst_capacity_score,
 *   fst_capacity.
 *
 *   cost      [B, N, N] float32 or NULL.  cost[b, s, t] = C(s, t): row s is
 *             the retained (source) token, column t the original token it
 *             covers:
 *               C = lambda_f d^_f + lambda_x phi_kappa(d^_x) + lambda_tau d^_tau
 *             with d_f = 1 - cos(f_s, f_t), d_x = ||x_s - x_t||,
 *             d_tau = max(tau_s - tau_t, 0), each min-max normalised over
 *             all N*N ordered pairs of the scene (diagonal included, so
 *             every minimum of d_x and d_tau is 0); a range <= 1e-6 makes
 *             that term 0; cos := 0 if a feature has zero norm.
 *   capacity  [B, N] float32 or NULL.  v of Eq. fst_capacity with phi = the
 *             identity: r_j = mean over the n_cap nearest other tokens k (3D
 *             distance, ties to the lower index) of
 *             alpha_f d^_f(j,k) + alpha_x d^_x(j,k) + alpha_tau d^_tau(j,k),
 *             v_j = r_j / sum_l r_l (uniform if the sum is 0 or
 *             capacity_mode == 1).  sum_j v_j = 1.
 *   norms     [B, 6] float32 or NULL: (f_lo, f_hi, x_lo, x_hi, tau_lo, tau_hi),
 *             the min and max of d_f, d_x, d_tau over the scene.
 *   bf16 features use the tensor cores (tcgen05, fp32 accumulation); fp32
 *   features use fp32 FMA arithmetic.
 */
int coverprune_cost(const void* feats, int dtype, const float* pos, const int32_t* frame,
                    int64_t B, int64_t N, int64_t D, const cp_params* p,
                    float* cost, float* capacity, float* norms,
                    void* ws, size_t ws_bytes, cp_stream_t stream);

/*
 * coverprune_select -- full CoverPrune: FST cost, FST capacity and
 * Spatial-Guided Greedy Selection of K tokens per scene.
 *   Sec. 3.5, Eqs. srpot, local_neighbor, greedy_flow, sgs_select, sgs_update.
 *
 *   The semi-relaxed OT of Eq. srpot with the source support and its
 *   capacity as decision variables is solved in closed form: every target t_j
 *   sends its mass v_j to its cheapest selected source among those whose
 *   neighbourhood M_g contains it, so the state is the coverage cost
 *   m_j = min(m0, min_{s in S, j in M_g(s)} C(s, j)) and the objective is
 *   F(S) = sum_j v_j m_j.  Each of the K steps adds the unselected token t
 *   with the largest local decrease
 *       gain(t) = sum_{j in M_g(t)} v_j max(m_j - C(t, j), 0)
 *   (the lowest index among equal gains).  Gains are evaluated in float32
 *   with a fixed summation order, so repeated calls return identical results.
 *
 *   kept       [B, K] int64, the selected indices in ascending order
 *   order      [B, K] int64 or NULL, the indices in selection order
 *   gains      [B, K] float32 or NULL, gain of the token added at each step
 *   objective  [B] float64 or NULL, F(S) after the K steps
 */
int coverprune_select(const void* feats, int dtype, const float* pos, const int32_t* frame,
                      int64_t B, int64_t N, int64_t D, int64_t K, const cp_params* p,
                      int64_t* kept, int64_t* order, float* gains, double* objective,
                      void* ws, size_t ws_bytes, cp_stream_t stream);

/*
 * coverprune_lite_select -- CoverPrune-Lite.
 *   Sec. 4.1 Eqs. lite_group, lite_select; Sec. 4.2 Eqs. blk_plan, blk_ot.
 *
 *   Tokens are ordered along a 3D Morton curve (cell q = floor((x - min)/voxel_m)
 *   per axis, clamped to [0, 1023], x in bit 3i, y in bit 3i+1, z in bit 3i+2;
 *   ties by index) and cut into K contiguous groups of capacity ~1/K, computed
 *   exactly in integers: Q_j = rint(v_j 2^40); group q >= 1 starts one past the
 *   first position whose running mass reaches q/K of the total, then starts
 *   are forced strictly increasing with room for the remaining groups.  Each
 *   group keeps s_q = argmin_{t in G_q} sum_{j in G_q} v_j C(t, j) (lowest
 *   index on ties), with C and v exactly as in coverprune_cost.
 *
 *   kept         [B, K] int64, the prototypes in ascending order
 *   group_start  [B, K+1] int32 or NULL, b_0 = 0 < b_1 < ... < b_K = N:
 *                group q is Morton positions [b_q, b_{q+1})
 *   objective    [B] float64 or NULL, sum_q sum_{j in G_q} v_j C(s_q, j)
 */
int coverprune_lite_select(const void* feats, int dtype, const float* pos,
                           const int32_t* frame, int64_t B, int64_t N, int64_t D,
                           int64_t K, const cp_params* p, int64_t* kept,
                           int32_t* group_start, double* objective,
                           void* ws, size_t ws_bytes, cp_stream_t stream);

/*
 * coverprune_knn -- the 3D neighbour sets the method is built on: the
 * capacity neighbours N_n(t_j) of Eq. fst_capacity_score and the SGS
 * neighbourhood M_g(t) of Eq. local_neighbor (M_g(t) = {t} plus the first g-1
 * entries of t's row).
 *   nbr       [B, N, k] int32: for every token j its k nearest OTHER tokens,
 *             ordered by squared distance computed in float32 with one
 *             rounding per operation ((dx*dx + dy*dy) + dz*dz, no fused
 *             multiply-add), ties broken by the lower index.  0 <= k <= N-1.
 *   diameter  [B] float32 or NULL: the largest pairwise distance of each
 *             scene (the spatial normaliser of Sec. 3.3).
 *   ws        at least coverprune_workspace_size(CP_OP_KNN, B, N, 8, 0, ...).
 */
int coverprune_knn(const float* pos, int64_t B, int64_t N, int64_t k, int32_t* nbr,
                   float* diameter, void* ws, size_t ws_bytes, cp_stream_t stream);

/*
 * coverprune_knn_noalloc -- coverprune_knn for callers that cannot allocate
 * device memory.  The paper has no counterpart: this is a deployment
 * variant of the neighbour step above, for hosts that own every device
 * buffer themselves (a fixed, sealed memory pool; a plugin without access
 * to an allocator) and can pass inputs and outputs but no workspace.
 *   Same arguments, results and ordering as coverprune_knn, without ws.
 *   Its scratch is a fixed array inside the library (65,792 bytes on every
 *   GPU that loads the library, kept until the process exits): at most
 *   1024 scenes per call; more returns CP_EUNSUPPORTED (see
 *   coverprune_last_error).  It calls no allocating routine.
 *   The first call on each device looks up the array's device address once
 *   (a runtime query made with that device current); make that first call
 *   before any stream capture.
 *   All calls share the array and each call rewrites the part it reads, so
 *   consecutive calls are independent; calls that overlap on the GPU
 *   (concurrent streams or host threads on one device) race on it.
 */
int coverprune_knn_noalloc(const float* pos, int64_t B, int64_t N, int64_t k, int32_t* nbr,
                           float* diameter, cp_stream_t stream);

/*
 * coverprune_gather -- compaction of the kept tokens (the pruned visual
 * input of Sec. 3.2).
 *   feats_out [B, K, D] = feats[b, kept[b, k], :] (byte copy, same dtype)
 *   pos_out   [B, K, 3] or NULL,  frame_out [B, K] or NULL likewise.
 *   kept      [B, K] int64 indices in [0, N).  An index out of range is
 *             skipped (its output row is left untouched) and recorded as
 *             CP_EINVAL in *status if status is not NULL.
 *   status    device int32 or NULL; written only on a bad index.
 *   Needs no workspace.
 */
int coverprune_gather(const void* feats, int dtype, const float* pos, const int32_t* frame,
                      int64_t B, int64_t N, int64_t D, const int64_t* kept, int64_t K,
                      void* feats_out, float* pos_out, int32_t* frame_out,
                      int32_t* status, cp_stream_t stream);

/*
 * coverprune_barrier_selftest -- exercises the device-side wait limit
 * without any fault: launches `n_blocks` co-resident blocks that wait for
 * `expected` arrivals on a grid barrier in ws (only n_blocks arrive).  With
 * expected > n_blocks the wait runs out after timeout_ms and the kernel
 * records CP_ETIMEOUT in the workspace status word (read it with
 * coverprune_check); with expected <= n_blocks it passes and records CP_OK.
 * ws needs 256 bytes.
 */
int coverprune_barrier_selftest(int32_t n_blocks, int32_t expected, float timeout_ms,
                                void* ws, size_t ws_bytes, cp_stream_t stream);

/*
 * Stage timing and launch counting (for benchmarks; no device memory).
 * Every kernel the library launches is counted under the stage it belongs
 * to.  With profiling enabled, each entry point also records a pair of CUDA
 * events around each stage on the call's own stream.  coverprune_profile_read
 * waits for the recorded events, writes per-stage milliseconds (0 when
 * profiling was off) and launch counts accumulated since the previous read
 * into ms[0..n) and launches[0..n) (either may be NULL), then clears them.
 * Stages: CP_STAGE_PREP (frame range, norms, neighbours, normalisers),
 * CP_STAGE_GRAM (feature normaliser GEMM), CP_STAGE_COST (cost GEMM),
 * CP_STAGE_CAPACITY, CP_STAGE_SGS (greedy selection incl. local slab),
 * CP_STAGE_LITE_ORDER (Morton order and groups), CP_STAGE_LITE_PROTO
 * (prototypes), CP_STAGE_OUTPUT (sort of kept indices, gather),
 * CP_STAGE_SLAB (local SGS with the bounded feature normaliser: the Morton
 * tile pairs that hold a neighbour pair and their cosines, in place of the
 * all-pairs Gram).
 * Host only; thread-safe.  Returns CP_OK or CP_ECUDA.
 */
typedef enum {
  CP_STAGE_PREP = 0,
  CP_STAGE_GRAM = 1,
  CP_STAGE_COST = 2,
  CP_STAGE_CAPACITY = 3,
  CP_STAGE_SGS = 4,
  CP_STAGE_LITE_ORDER = 5,
  CP_STAGE_LITE_PROTO = 6,
  CP_STAGE_OUTPUT = 7,
  CP_STAGE_SLAB = 8,
  CP_STAGE_COUNT = 9
} cp_stage;
int coverprune_profile_enable(int on);
int coverprune_profile_read(double* ms, int64_t* launches, int n);

/*
 * Counters of the last coverprune_select that used workspace `ws`
 * (synchronises `stream` first):
 *   gain_evaluations  candidate gains computed, over all scenes and steps;
 *                     each reads one row of the cost (N floats) or of the
 *                     local slab (g floats)
 *   rounds            decision rounds over all scenes and steps (lazy mode:
 *                     a step needs one or more; full sweep: one per step)
 *   cost_bytes_read   bytes of cost rows (or slab rows and their neighbour
 *                     indices) the selection reads: every gain evaluation,
 *                     and once per scene and step the winner's row for the
 *                     coverage update; the dense lazy kernel skips row
 *                     blocks whose terms are known to be zero, so this can
 *                     be well below gain_evaluations * 4N
 * Returns CP_OK, CP_EINVAL or CP_ECUDA.
 */
typedef struct {
  uint64_t gain_evaluations;
  uint64_t rounds;
  uint64_t cost_bytes_read;
} cp_call_stats;
int coverprune_call_stats(const void* ws, cp_stream_t stream, cp_call_stats* out);

/* Description of the last CP_ECUDA returned on the calling thread: which
 * step failed and the CUDA error name ("" if none).  Host only. */
const char* coverprune_last_error(void);

/* Library version: major * 10000 + minor * 100 + patch. */
int coverprune_version(void);

#ifdef __cplusplus
}
#endif

#endif /* COVERPRUNE_H_ */
