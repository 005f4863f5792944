/*
 * CoverPrune CPU oracle -- TEST INFRASTRUCTURE, not part of the product.
 *
 * A plain, slow, scalar restatement in double precision of what the
 * CoverPrune hot path computes ("CoverPrune: Coverage-Driven Token Pruning
 * for 3D VLMs via Optimal Transport"):
 *   - FST discrepancies and cost            (Sec. 3.3, Eqs. fst_metrics, fst_cost)
 *   - FST target capacity                   (Sec. 3.4, Eqs. fst_capacity_score, fst_capacity)
 *   - Spatial-Guided Greedy Selection (SGS) (Sec. 3.5, Eqs. srpot, local_neighbor,
 *                                            greedy_flow, sgs_select, sgs_update)
 *   - CoverPrune-Lite                       (Sec. 4.1-4.2, Eqs. lite_group, lite_select,
 *                                            blk_plan, blk_ot)
 * Only the test suite, the smoke check and the benchmark's CPU-baseline leg
 * may load this file.  It shares no code, header or table with the CUDA
 * library and includes nothing from it.
 *
 * Precision: every quantity is double, except where a floating-point result
 * decides an integer (nearest-neighbour order, Morton voxel), which is done in
 * IEEE single precision with every operation rounded separately (no
 * contraction into fused multiply-adds).  The build passes -ffp-contract=off
 * and the static assertion below rejects compilers that evaluate float
 * expressions in a wider format.
 *
 * Readings of points the paper leaves open (each documented in the design
 * notes of the repository):
 *   R1 min-max normalisation runs over all N*N ordered pairs (i, j) including
 *      i == j; a range at or below 1e-6 (below single-precision resolution of
 *      a cosine) makes that normalised term 0.
 *   R2 cos := 0 when either feature has zero norm; cos is clamped to [-1, 1].
 *   R3 phi_kappa(x) = log(1 + kappa x) / log(1 + kappa).
 *   R4 capacity neighbours N_n(j): the n nearest *other* tokens in 3D, ordered
 *      by (squared distance in single precision, index); n is clamped to N-1.
 *      The capacity map phi is the identity; if sum r == 0 the capacity is
 *      uniform.
 *   R5 SGS: the semi-relaxed OT with source support and source capacity as
 *      decision variables has the closed-form plan "each target sends its
 *      mass to its cheapest selected source"; the state is the current
 *      coverage cost m_j, the objective F(S) = sum_j v_j m_j, and the selected
 *      token maximises the local marginal decrease
 *      gain(t) = sum_{j in M_g(t)} v_j max(m_j - C(t,j), 0), lowest index on
 *      exact ties.  m starts at M0.
 *   R6 M_g(t) = {t} plus the g-1 nearest other tokens (same order as R4);
 *      g == N means every token.
 *   R7 Morton: per axis q = floor((x - min) / voxel) in single precision,
 *      clamped to [0, 1023]; x fills bit 3i, y bit 3i+1, z bit 3i+2; order by
 *      (code, index).
 *   R8 Lite grouping in exact integers: Q_j = rint(v_j * 2^40) with v_j in
 *      single precision; group q >= 1 starts one past the first position
 *      where the running sum reaches q/K of the total; starts are then forced
 *      strictly increasing with room for the remaining groups.
 *   R9 Lite prototype: lowest original index on exact ties.
 */
#include <float.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#if !defined(FLT_EVAL_METHOD) || FLT_EVAL_METHOD != 0
#error "the oracle needs float expressions evaluated in float (FLT_EVAL_METHOD == 0)"
#endif

#define ORC_OK 0
#define ORC_EINVAL 1
#define ORC_ENOMEM 2

/* Thread count of the OpenMP loops (rows of independent work only; the
 * results do not depend on it). */
void orc_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}

int orc_get_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* Threshold under which a min-max range counts as empty (reading R1). */
#define ORC_RANGE_EPS 1e-6

/* Weights of Eqs. fst_cost and fst_capacity_score. */
typedef struct {
  double lambda_f, lambda_x, lambda_tau; /* Eq. fst_cost */
  double kappa;                          /* phi_kappa of Eq. fst_cost */
  double alpha_f, alpha_x, alpha_tau;    /* Eq. fst_capacity_score */
} orc_weights;

/* Per-scene min-max normalisers (Sec. 3.3: "min-max normalized within the
 * current sample").  d_hat = (d - lo) / (hi - lo), or 0 when hi - lo <= eps. */
typedef struct {
  double f_lo, f_hi;     /* range of d_f = 1 - cos over all ordered pairs */
  double x_lo, x_hi;     /* range of d_x = ||x_s - x_t|| */
  double tau_lo, tau_hi; /* range of d_tau = ReLU(tau_s - tau_t) */
} orc_norms;

/* ------------------------------------------------------------------ */
/* Discrepancies of Eq. fst_metrics                                    */
/* ------------------------------------------------------------------ */

static double feat_norm(const double* f, int64_t D) {
  double s = 0.0;
  for (int64_t d = 0; d < D; ++d) s += f[d] * f[d];
  return sqrt(s);
}

/* ||f_j|| for every token, computed once per call. */
static double* all_norms(const double* F, int64_t N, int64_t D) {
  double* nrm = (double*)malloc(sizeof(double) * (size_t)N);
  if (!nrm) return NULL;
  for (int64_t j = 0; j < N; ++j) nrm[j] = feat_norm(F + j * D, D);
  return nrm;
}

/* d_f(s,t) = 1 - cos(f_s, f_t), with reading R2 (nrm = feature norms). */
static double disc_f(const double* F, const double* nrm, int64_t D, int64_t s,
                     int64_t t) {
  if (nrm[s] == 0.0 || nrm[t] == 0.0) return 1.0; /* cos := 0 */
  double dot = 0.0;
  for (int64_t d = 0; d < D; ++d) dot += F[s * D + d] * F[t * D + d];
  double c = dot / (nrm[s] * nrm[t]);
  if (c > 1.0) c = 1.0;
  if (c < -1.0) c = -1.0;
  return 1.0 - c;
}

/* d_x(s,t) = ||x_s - x_t||_2 */
static double disc_x(const float* X, int64_t s, int64_t t) {
  double dx = (double)X[3 * s + 0] - (double)X[3 * t + 0];
  double dy = (double)X[3 * s + 1] - (double)X[3 * t + 1];
  double dz = (double)X[3 * s + 2] - (double)X[3 * t + 2];
  return sqrt(dx * dx + dy * dy + dz * dz);
}

/* d_tau(s,t) = ReLU(tau_s - tau_t) */
static double disc_tau(const int32_t* tau, int64_t s, int64_t t) {
  double z = (double)tau[s] - (double)tau[t];
  return z > 0.0 ? z : 0.0;
}

static double normalise(double d, double lo, double hi) {
  double range = hi - lo;
  if (range <= ORC_RANGE_EPS) return 0.0;
  return (d - lo) / range;
}

/* phi_kappa(x) = log(1 + kappa x) / log(1 + kappa)   (Eq. fst_cost) */
static double phi_kappa(double x, double kappa) {
  return log1p(kappa * x) / log1p(kappa);
}

/* C(s,t) of Eq. fst_cost: row s is the retained (source) token, t the
 * original (target) token it covers. */
static double fst_cost(const double* F, const double* nrm, int64_t D,
                       const float* X, const int32_t* tau, const orc_weights* w,
                       const orc_norms* nm, int64_t s, int64_t t) {
  double df = normalise(disc_f(F, nrm, D, s, t), nm->f_lo, nm->f_hi);
  double dx = normalise(disc_x(X, s, t), nm->x_lo, nm->x_hi);
  double dt = normalise(disc_tau(tau, s, t), nm->tau_lo, nm->tau_hi);
  return w->lambda_f * df + w->lambda_x * phi_kappa(dx, w->kappa) +
         w->lambda_tau * dt;
}

/* ------------------------------------------------------------------ */
/* Normalisers: min and max of each discrepancy over all ordered pairs */
/* ------------------------------------------------------------------ */

/* feat_mode 0: the range of d_f over all ordered pairs, as for d_x and
 * d_tau (Sec. 3.3).  feat_mode 1, the bounded feature normaliser: d_f =
 * 1 - cos always lies in [0, 2] (cos is clamped to [-1, 1]), so that range
 * stands in for the measured one and d_f is not visited; d_x and d_tau keep
 * their measured ranges. */
int orc_normalisers_mode(int64_t N, int64_t D, const double* F, const float* X,
                         const int32_t* tau, int feat_mode, orc_norms* out) {
  if (N < 1 || D < 1 || !F || !X || !tau || !out) return ORC_EINVAL;
  if (feat_mode != 0 && feat_mode != 1) return ORC_EINVAL;
  double* nrm = all_norms(F, N, D);
  if (!nrm) return ORC_ENOMEM;
  double f_lo = INFINITY, f_hi = -INFINITY;
  double x_lo = INFINITY, x_hi = -INFINITY;
  double t_lo = INFINITY, t_hi = -INFINITY;
  /* All N*N ordered pairs, diagonal included (reading R1).  d_f and d_x are
   * symmetric in (s, t), so the pairs t >= s already give their extremes. */
#pragma omp parallel for schedule(dynamic, 8) \
    reduction(min : f_lo, x_lo, t_lo) reduction(max : f_hi, x_hi, t_hi)
  for (int64_t s = 0; s < N; ++s) {
    for (int64_t t = 0; t < N; ++t) {
      if (t >= s) {
        if (feat_mode == 0) {
          double df = disc_f(F, nrm, D, s, t);
          if (df < f_lo) f_lo = df;
          if (df > f_hi) f_hi = df;
        }
        double dx = disc_x(X, s, t);
        if (dx < x_lo) x_lo = dx;
        if (dx > x_hi) x_hi = dx;
      }
      double dt = disc_tau(tau, s, t);
      if (dt < t_lo) t_lo = dt;
      if (dt > t_hi) t_hi = dt;
    }
  }
  free(nrm);
  if (feat_mode == 1) {
    f_lo = 0.0;
    f_hi = 2.0;
  }
  out->f_lo = f_lo; out->f_hi = f_hi;
  out->x_lo = x_lo; out->x_hi = x_hi;
  out->tau_lo = t_lo; out->tau_hi = t_hi;
  return ORC_OK;
}

int orc_normalisers(int64_t N, int64_t D, const double* F, const float* X,
                    const int32_t* tau, orc_norms* out) {
  return orc_normalisers_mode(N, D, F, X, tau, 0, out);
}

/* ------------------------------------------------------------------ */
/* FST cost (Eq. fst_cost)                                             */
/* ------------------------------------------------------------------ */

/* Rows [s0, s1) of C, each of length N, written to out[(s - s0) * N + t]. */
int orc_cost_rows(int64_t N, int64_t D, const double* F, const float* X,
                  const int32_t* tau, const orc_weights* w, const orc_norms* nm,
                  int64_t s0, int64_t s1, double* out) {
  if (N < 1 || D < 1 || s0 < 0 || s1 > N || s0 > s1 || !out) return ORC_EINVAL;
  double* nrm = all_norms(F, N, D);
  if (!nrm) return ORC_ENOMEM;
#pragma omp parallel for schedule(dynamic, 4)
  for (int64_t s = s0; s < s1; ++s)
    for (int64_t t = 0; t < N; ++t)
      out[(s - s0) * N + t] = fst_cost(F, nrm, D, X, tau, w, nm, s, t);
  free(nrm);
  return ORC_OK;
}

/* C(S[p], T[p]) for a list of P sampled pairs. */
int orc_cost_pairs(int64_t N, int64_t D, const double* F, const float* X,
                   const int32_t* tau, const orc_weights* w, const orc_norms* nm,
                   int64_t P, const int64_t* S, const int64_t* T, double* out) {
  if (N < 1 || D < 1 || P < 0 || !out) return ORC_EINVAL;
  for (int64_t p = 0; p < P; ++p)
    if (S[p] < 0 || S[p] >= N || T[p] < 0 || T[p] >= N) return ORC_EINVAL;
  double* nrm = all_norms(F, N, D);
  if (!nrm) return ORC_ENOMEM;
#pragma omp parallel for schedule(static)
  for (int64_t p = 0; p < P; ++p)
    out[p] = fst_cost(F, nrm, D, X, tau, w, nm, S[p], T[p]);
  free(nrm);
  return ORC_OK;
}

/* ------------------------------------------------------------------ */
/* 3D nearest neighbours (capacity set N_n, SGS neighbourhood M_g)     */
/* ------------------------------------------------------------------ */

/* Squared distance in single precision, one rounding per operation. */
static float sqdist_f32(const float* X, int64_t a, int64_t b) {
  float dx = X[3 * a + 0] - X[3 * b + 0];
  float dy = X[3 * a + 1] - X[3 * b + 1];
  float dz = X[3 * a + 2] - X[3 * b + 2];
  float xx = dx * dx;
  float yy = dy * dy;
  float zz = dz * dz;
  float s = xx + yy;
  return s + zz;
}

/* For every token j: the k nearest other tokens, ordered by (d^2, index).
 * out is [N, k]. */
int orc_knn_others(int64_t N, const float* X, int64_t k, int32_t* out) {
  if (N < 1 || k < 0 || k > N - 1 || !X || (k > 0 && !out)) return ORC_EINVAL;
  if (k == 0) return ORC_OK;
  int failed = 0;
#pragma omp parallel
  {
    float* bd = (float*)malloc(sizeof(float) * (size_t)k);
    int64_t* bi = (int64_t*)malloc(sizeof(int64_t) * (size_t)k);
    if (!bd || !bi) {
#pragma omp atomic write
      failed = 1;
    }
#pragma omp for schedule(dynamic, 16)
    for (int64_t j = 0; j < N; ++j) {
      if (!bd || !bi) continue;
      int64_t cnt = 0; /* sorted list of the best cnt candidates so far */
      for (int64_t c = 0; c < N; ++c) {
        if (c == j) continue;
        float d = sqdist_f32(X, j, c);
        /* candidates arrive in increasing index, so on equal d the one
         * already in the list has the lower index and stays in front */
        if (cnt == k && !(d < bd[k - 1])) continue;
        int64_t pos = cnt < k ? cnt : k - 1;
        while (pos > 0 && d < bd[pos - 1]) {
          bd[pos] = bd[pos - 1];
          bi[pos] = bi[pos - 1];
          --pos;
        }
        bd[pos] = d;
        bi[pos] = c;
        if (cnt < k) ++cnt;
      }
      for (int64_t q = 0; q < k; ++q) out[j * k + q] = (int32_t)bi[q];
    }
    free(bd);
    free(bi);
  }
  return failed ? ORC_ENOMEM : ORC_OK;
}

/* ------------------------------------------------------------------ */
/* FST capacity (Eqs. fst_capacity_score, fst_capacity)                */
/* ------------------------------------------------------------------ */

/* nbr is [N, n]: the capacity neighbours N_n(j).  mode 0 = FST capacity,
 * mode 1 = uniform capacity (the "w/o FST capacity" ablation).  r_out may be
 * NULL. */
int orc_capacity(int64_t N, int64_t D, const double* F, const float* X,
                 const int32_t* tau, const orc_weights* w, const orc_norms* nm,
                 int64_t n, const int32_t* nbr, int mode, double* r_out,
                 double* v_out) {
  if (N < 1 || D < 1 || n < 0 || n > N - 1 || !v_out) return ORC_EINVAL;
  double* r = (double*)malloc(sizeof(double) * (size_t)N);
  double* nrm = all_norms(F, N, D);
  if (!r || !nrm) {
    free(r); free(nrm);
    return ORC_ENOMEM;
  }
  /* r_j: mean FST discrepancy (without phi_kappa) to the n neighbours;
   * the first argument of each discrepancy is t_j. */
#pragma omp parallel for schedule(static)
  for (int64_t j = 0; j < N; ++j) {
    double acc = 0.0;
    for (int64_t q = 0; q < n; ++q) {
      int64_t k = nbr[j * n + q];
      acc += w->alpha_f * normalise(disc_f(F, nrm, D, j, k), nm->f_lo, nm->f_hi) +
             w->alpha_x * normalise(disc_x(X, j, k), nm->x_lo, nm->x_hi) +
             w->alpha_tau * normalise(disc_tau(tau, j, k), nm->tau_lo, nm->tau_hi);
    }
    r[j] = n > 0 ? acc / (double)n : 0.0;
  }
  /* v_j = phi(r_j) / sum_l phi(r_l), phi = identity (reading R4) */
  double total = 0.0;
  for (int64_t j = 0; j < N; ++j) total += r[j];
  for (int64_t j = 0; j < N; ++j) {
    if (r_out) r_out[j] = r[j];
    v_out[j] = (mode == 1 || total <= 0.0) ? 1.0 / (double)N : r[j] / total;
  }
  free(r);
  free(nrm);
  return ORC_OK;
}

/* ------------------------------------------------------------------ */
/* Spatial-Guided Greedy Selection (Sec. 3.5, reading R5/R6)           */
/* ------------------------------------------------------------------ */

/* Is target j in M_g(t)?  nbr_g is [N, g-1] (the g-1 nearest others of t),
 * or NULL for g == N. */
static int in_neighbourhood(int64_t t, int64_t j, int64_t g, int64_t N,
                            const int32_t* nbr_g) {
  if (g >= N) return 1;
  if (j == t) return 1;
  for (int64_t q = 0; q < g - 1; ++q)
    if (nbr_g[t * (g - 1) + q] == j) return 1;
  return 0;
}

/* gain(t) = sum_{j in M_g(t)} v_j max(m_j - C(t,j), 0) */
static double sgs_gain(int64_t t, int64_t N, const double* C, const double* v,
                       const double* m, int64_t g, const int32_t* nbr_g) {
  double acc = 0.0;
  if (g >= N) {
    for (int64_t j = 0; j < N; ++j) {
      double d = m[j] - C[t * N + j];
      if (d > 0.0) acc += v[j] * d;
    }
  } else {
    double d = m[t] - C[t * N + t];
    if (d > 0.0) acc += v[t] * d;
    for (int64_t q = 0; q < g - 1; ++q) {
      int64_t j = nbr_g[t * (g - 1) + q];
      d = m[j] - C[t * N + j];
      if (d > 0.0) acc += v[j] * d;
    }
  }
  return acc;
}

/* F(S) = sum_j v_j m_j with m_j = min(M0, min_{s in S, j in M_g(s)} C(s,j)).
 * For g == N and M0 >= max C this is the semi-relaxed OT value of Eq. srpot
 * with the source capacity free (reading R5). */
int orc_objective(int64_t N, const double* C, const double* v, int64_t g,
                  const int32_t* nbr_g, double M0, int64_t nS, const int64_t* S,
                  double* out) {
  if (N < 1 || nS < 0 || !C || !v || !out) return ORC_EINVAL;
  if (g <= 0) g = N;
  if (g > 1 && g < N && !nbr_g) return ORC_EINVAL;  /* M_g(t) needs t's g-1 neighbours */
  double F = 0.0;
  for (int64_t j = 0; j < N; ++j) {
    double m = M0;
    for (int64_t p = 0; p < nS; ++p) {
      int64_t s = S[p];
      if (s < 0 || s >= N) return ORC_EINVAL;
      if (in_neighbourhood(s, j, g, N, nbr_g) && C[s * N + j] < m) m = C[s * N + j];
    }
    F += v[j] * m;
  }
  *out = F;
  return ORC_OK;
}

/* K greedy steps on a given cost matrix C [N, N] (row = source) and target
 * capacity v.  g <= 0 or g >= N means M_g = all tokens.
 *
 * forced (may be NULL): if given, step l adds forced[l] to S instead of the
 * oracle's own argmax (teacher forcing), while the outputs still report the
 * oracle's own argmax and gains at that step.
 *
 * Outputs per step l (any may be NULL):
 *   best_idx[l]   the argmax over t not in S (lowest index on exact ties)
 *   best_gain[l]  its gain
 *   second[l]     the largest gain among the other candidates (-1 if none)
 *   picked_gain[l] gain of the token actually added (== best_gain unless forced)
 *   F_after[l]    objective after the step
 * order[l] is the token added at step l. */
int orc_sgs(int64_t N, const double* C, const double* v, int64_t g,
            const int32_t* nbr_g, int64_t K, double M0, const int64_t* forced,
            int64_t* order, int64_t* best_idx, double* best_gain, double* second,
            double* picked_gain, double* F_after) {
  if (N < 1 || K < 0 || K > N || !C || !v) return ORC_EINVAL;
  if (g <= 0 || g > N) g = N;
  if (g > 1 && g < N && !nbr_g) return ORC_EINVAL;
  double* m = (double*)malloc(sizeof(double) * (size_t)N);
  double* gain = (double*)malloc(sizeof(double) * (size_t)N);
  char* chosen = (char*)calloc((size_t)N, 1);
  if (!m || !gain || !chosen) {
    free(m); free(gain); free(chosen);
    return ORC_ENOMEM;
  }
  for (int64_t j = 0; j < N; ++j) m[j] = M0;
  int rc = ORC_OK;
  for (int64_t l = 0; l < K; ++l) {
#pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < N; ++t)
      gain[t] = chosen[t] ? -1.0 : sgs_gain(t, N, C, v, m, g, nbr_g);
    /* argmax, lowest index among exact equals (strict > keeps the first) */
    int64_t b = -1;
    for (int64_t t = 0; t < N; ++t)
      if (!chosen[t] && (b < 0 || gain[t] > gain[b])) b = t;
    double sec = -1.0;
    for (int64_t t = 0; t < N; ++t)
      if (!chosen[t] && t != b && gain[t] > sec) sec = gain[t];
    int64_t pick = b;
    if (forced) {
      pick = forced[l];
      if (pick < 0 || pick >= N || chosen[pick]) { rc = ORC_EINVAL; break; }
    }
    if (best_idx) best_idx[l] = b;
    if (best_gain) best_gain[l] = gain[b];
    if (second) second[l] = sec;
    if (picked_gain) picked_gain[l] = gain[pick];
    if (order) order[l] = pick;
    /* S <- S u {t*} (Eq. sgs_update); the served targets' coverage cost
     * drops to what t* offers them */
    chosen[pick] = 1;
    for (int64_t j = 0; j < N; ++j)
      if (in_neighbourhood(pick, j, g, N, nbr_g) && C[pick * N + j] < m[j])
        m[j] = C[pick * N + j];
    if (F_after) {
      double F = 0.0;
      for (int64_t j = 0; j < N; ++j) F += v[j] * m[j];
      F_after[l] = F;
    }
  }
  free(m); free(gain); free(chosen);
  return rc;
}

/* ------------------------------------------------------------------ */
/* CoverPrune-Lite (Sec. 4)                                            */
/* ------------------------------------------------------------------ */

/* Spread the low 10 bits of q so that bit i lands on bit 3i. */
static uint32_t spread3(uint32_t q) {
  uint32_t out = 0;
  for (int i = 0; i < 10; ++i) out |= ((q >> i) & 1u) << (3 * i);
  return out;
}

typedef struct {
  uint32_t code;
  int64_t idx;
} code_idx;

static int cmp_code_idx(const void* a, const void* b) {
  const code_idx* x = (const code_idx*)a;
  const code_idx* y = (const code_idx*)b;
  if (x->code != y->code) return x->code < y->code ? -1 : 1;
  if (x->idx != y->idx) return x->idx < y->idx ? -1 : 1;
  return 0;
}

/* Morton code of every token (reading R7) and the permutation that orders
 * tokens by (code, index).  code_out and/or perm_out may be NULL. */
int orc_morton(int64_t N, const float* X, float voxel, uint32_t* code_out,
               int64_t* perm_out) {
  if (N < 1 || !X || !(voxel > 0.0f)) return ORC_EINVAL;
  float lo[3];
  for (int a = 0; a < 3; ++a) {
    lo[a] = X[a];
    for (int64_t j = 1; j < N; ++j)
      if (X[3 * j + a] < lo[a]) lo[a] = X[3 * j + a];
  }
  code_idx* ci = (code_idx*)malloc(sizeof(code_idx) * (size_t)N);
  if (!ci) return ORC_ENOMEM;
  for (int64_t j = 0; j < N; ++j) {
    uint32_t q[3];
    for (int a = 0; a < 3; ++a) {
      float rel = X[3 * j + a] - lo[a];
      float cell = floorf(rel / voxel);
      if (cell < 0.0f) cell = 0.0f;
      if (cell > 1023.0f) cell = 1023.0f;
      q[a] = (uint32_t)cell;
    }
    uint32_t code = spread3(q[0]) | (spread3(q[1]) << 1) | (spread3(q[2]) << 2);
    ci[j].code = code;
    ci[j].idx = j;
    if (code_out) code_out[j] = code;
  }
  qsort(ci, (size_t)N, sizeof(code_idx), cmp_code_idx);
  if (perm_out)
    for (int64_t p = 0; p < N; ++p) perm_out[p] = ci[p].idx;
  free(ci);
  return ORC_OK;
}

/* Capacity-guided grouping of Eq. lite_group in exact integers (reading
 * R8).  v is the single-precision capacity, perm the Morton order.  Writes
 * the K+1 group starts b[0] = 0 < b[1] < ... < b[K] = N (positions in the
 * Morton order).  Also returns the fixed-point masses Q (may be NULL). */
int orc_lite_groups(int64_t N, int64_t K, const float* v, const int64_t* perm,
                    int64_t* b, uint64_t* Q_out) {
  if (N < 1 || K < 1 || K > N || !v || !perm || !b) return ORC_EINVAL;
  uint64_t* P = (uint64_t*)malloc(sizeof(uint64_t) * (size_t)N);
  if (!P) return ORC_ENOMEM;
  uint64_t run = 0;
  for (int64_t p = 0; p < N; ++p) {
    double vj = (double)v[perm[p]];
    if (!(vj >= 0.0)) vj = 0.0;
    uint64_t q = (uint64_t)rint(vj * 1099511627776.0); /* 2^40 */
    if (Q_out) Q_out[perm[p]] = q;
    run += q;
    P[p] = run; /* inclusive running mass */
  }
  uint64_t total = P[N - 1];
  b[0] = 0;
  b[K] = N;
  int64_t best = INT64_MIN; /* running max of (ideal start - q) */
  int64_t p = 0;
  for (int64_t q = 1; q < K; ++q) {
    /* first position whose running mass reaches q/K of the total:
     * P(p) * K >= q * total, compared exactly in 128 bits */
    while (p < N && (unsigned __int128)P[p] * (unsigned __int128)K <
                        (unsigned __int128)q * (unsigned __int128)total)
      ++p;
    int64_t ideal = (p < N ? p : N - 1) + 1; /* close the group with p inside */
    if (ideal - q > best) best = ideal - q;
    int64_t lift = best < (N - K) ? best : (N - K);
    b[q] = q + lift;
  }
  free(P);
  return ORC_OK;
}

/* Per-group prototype of Eq. lite_select with the FST cost of Eq. fst_cost
 * (global normalisers) and capacity v (double).  perm and b come from
 * orc_morton / orc_lite_groups.  proto[q] is the chosen token of group q,
 * score[q] its capacity-weighted cost; *objective = sum_q score[q], the value
 * of Eq. blk_ot for the chosen prototypes when group masses are exactly 1/K.
 * Any output may be NULL. */
int orc_lite_select(int64_t N, int64_t D, const double* F, const float* X,
                    const int32_t* tau, const orc_weights* w, const orc_norms* nm,
                    const double* v, const int64_t* perm, const int64_t* b,
                    int64_t K, int64_t* proto, double* score, double* objective) {
  if (N < 1 || D < 1 || K < 1 || K > N || !v || !perm || !b) return ORC_EINVAL;
  double total = 0.0;
  int bad = 0;
  for (int64_t q = 0; q < K; ++q)
    if (b[q] < 0 || b[q + 1] > N || b[q] >= b[q + 1]) bad = 1;
  if (bad) return ORC_EINVAL;
  double* nrm = all_norms(F, N, D);
  if (!nrm) return ORC_ENOMEM;
#pragma omp parallel for schedule(dynamic, 1) reduction(+ : total)
  for (int64_t q = 0; q < K; ++q) {
    int64_t best_t = -1;
    double best_s = 0.0;
    for (int64_t a = b[q]; a < b[q + 1]; ++a) {
      int64_t t = perm[a];
      double s = 0.0;
      for (int64_t c = b[q]; c < b[q + 1]; ++c) {
        int64_t j = perm[c];
        s += v[j] * fst_cost(F, nrm, D, X, tau, w, nm, t, j);
      }
      if (best_t < 0 || s < best_s || (s == best_s && t < best_t)) {
        best_t = t;
        best_s = s;
      }
    }
    if (proto) proto[q] = best_t;
    if (score) score[q] = best_s;
    total += best_s;
  }
  free(nrm);
  if (objective) *objective = total;
  return ORC_OK;
}

/* ------------------------------------------------------------------ */
/* Literal SGS with an entropic semi-relaxed OT (Sec. 3.5 read word for */
/* word: Eqs. srpot_sinkhorn, greedy_flow, sgs_select, sgs_update)      */
/* ------------------------------------------------------------------ */

/* log(sum_k exp(x_k)) by shifting with the largest term; -inf when every
 * term is -inf (or n == 0). */
static double log_sum_exp(const double* x, int64_t n) {
  double mx = -INFINITY;
  for (int64_t k = 0; k < n; ++k)
    if (x[k] > mx) mx = x[k];
  if (mx == -INFINITY) return -INFINITY;
  double s = 0.0;
  for (int64_t k = 0; k < n; ++k) s += exp(x[k] - mx);
  return mx + log(s);
}

/* Entropic semi-relaxed OT of Eq. srpot_sinkhorn,
 *   min_P <C, P> - eps H(P)  s.t.  P 1 = u,  P^T 1 <= v,
 * between m sources (row i of C holds C(source i, target j), j < N) and N
 * targets, by block coordinate ascent on its dual.  The plan is
 * P_ij = exp((f_i + g_j - C_ij) / eps) with g <= 0; each iteration first
 * maximises the dual over f (rows: P 1 = u),
 *   f_i = eps log u_i - eps log sum_j exp((g_j - C_ij) / eps),
 * then over g <= 0 (columns: the capacity cap; a column below its capacity
 * keeps g_j = 0),
 *   g_j = min(0, eps log v_j - eps log sum_i exp((f_i - C_ij) / eps))
 * (g_j = -inf when v_j = 0).  g holds the starting point on entry (zeros
 * for a cold start) and the result on exit; f gets the row potentials.
 * colsum (may be NULL) gets P^T 1 of the final potentials; P (may be NULL)
 * the plan, [m, N].  The loops are plain; no tolerance stops them early. */
int orc_sot_sinkhorn(int64_t m, int64_t N, const double* C, const double* u, const double* v,
                     double eps, int64_t iters, double* f, double* g, double* colsum,
                     double* P) {
  if (m < 0 || N < 1 || iters < 0 || !(eps > 0.0) || (m > 0 && (!C || !u || !f)) || !v || !g)
    return ORC_EINVAL;
  int64_t w = m > N ? m : N;
  double* x = (double*)malloc(sizeof(double) * (size_t)(w > 0 ? w : 1));
  if (!x) return ORC_ENOMEM;
  for (int64_t it = 0; it < iters && m > 0; ++it) {
    for (int64_t i = 0; i < m; ++i) {
      for (int64_t j = 0; j < N; ++j) x[j] = (g[j] - C[i * N + j]) / eps;
      f[i] = eps * log(u[i]) - eps * log_sum_exp(x, N);
    }
    for (int64_t j = 0; j < N; ++j) {
      if (!(v[j] > 0.0)) {
        g[j] = -INFINITY;
        continue;
      }
      for (int64_t i = 0; i < m; ++i) x[i] = (f[i] - C[i * N + j]) / eps;
      double gj = eps * log(v[j]) - eps * log_sum_exp(x, m);
      g[j] = gj < 0.0 ? gj : 0.0;
    }
  }
  for (int64_t j = 0; j < N; ++j) {
    double s = 0.0;
    for (int64_t i = 0; i < m; ++i) {
      double p = exp((f[i] + g[j] - C[i * N + j]) / eps);
      if (P) P[i * N + j] = p;
      s += p;
    }
    if (colsum) colsum[j] = s;
  }
  free(x);
  return ORC_OK;
}

/* K steps of SGS as Eqs. greedy_flow and sgs_select print it (reading A10
 * of the design notes; the default hot path uses the coverage-gain reading
 * R5 instead).  At step l the sources are the l selected tokens, each with
 * mass 1/K; the plan P_l of the entropic semi-relaxed OT against the target
 * capacity v (orc_sot_sinkhorn, `iters` iterations, the target potentials
 * warm-started from step l-1, zeros at l = 1) gives the residual capacity
 *   r_j = max(v_j - (P_l^T 1)_j, 0)      (r = v at l = 0),
 * and the next token minimises the residual-weighted local cost
 *   score(t) = sum_{j in M_g(t)} r_j C(t, j)
 * over the unselected tokens (lowest index among exact equals).  C [N, N]
 * row = source; g <= 0 or g >= N means M_g = all tokens, else nbr_g [N,
 * g-1] lists t's nearest others.
 *
 * forced (may be NULL): step l adds forced[l] instead of the argmin while
 * the outputs still report the oracle's own argmin.  Outputs per step
 * (any may be NULL): order (token added), best_idx / best_score (the
 * argmin and its score), second (the smallest score among the other
 * candidates, +inf if none), picked_score (score of the token added). */
int orc_sgs_literal(int64_t N, const double* C, const double* v, int64_t g,
                    const int32_t* nbr_g, int64_t K, double eps, int64_t iters,
                    const int64_t* forced, int64_t* order, int64_t* best_idx,
                    double* best_score, double* second, double* picked_score) {
  if (N < 1 || K < 0 || K > N || !C || !v || !(eps > 0.0) || iters < 0) return ORC_EINVAL;
  if (g <= 0 || g > N) g = N;
  if (g > 1 && g < N && !nbr_g) return ORC_EINVAL;
  int64_t* sel = (int64_t*)malloc(sizeof(int64_t) * (size_t)(K > 0 ? K : 1));
  double* rows = (double*)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1) * (size_t)N);
  double* u = (double*)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1));
  double* fpot = (double*)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1));
  double* gpot = (double*)calloc((size_t)N, sizeof(double));
  double* col = (double*)malloc(sizeof(double) * (size_t)N);
  double* r = (double*)malloc(sizeof(double) * (size_t)N);
  double* score = (double*)malloc(sizeof(double) * (size_t)N);
  char* chosen = (char*)calloc((size_t)N, 1);
  int rc = ORC_OK;
  if (!sel || !rows || !u || !fpot || !gpot || !col || !r || !score || !chosen) {
    rc = ORC_ENOMEM;
    goto done;
  }
  for (int64_t l = 0; l < K; ++l) {
    /* Eq. greedy_flow: residual target capacity after the step-l plan */
    if (l == 0) {
      for (int64_t j = 0; j < N; ++j) r[j] = v[j];
    } else {
      for (int64_t i = 0; i < l; ++i) u[i] = 1.0 / (double)K;
      rc = orc_sot_sinkhorn(l, N, rows, u, v, eps, iters, fpot, gpot, col, NULL);
      if (rc != ORC_OK) break;
      for (int64_t j = 0; j < N; ++j) {
        double d = v[j] - col[j];
        r[j] = d > 0.0 ? d : 0.0;
      }
    }
    /* Eq. sgs_select */
#pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < N; ++t) {
      if (chosen[t]) {
        score[t] = INFINITY;
        continue;
      }
      double s = 0.0;
      if (g >= N) {
        for (int64_t j = 0; j < N; ++j) s += r[j] * C[t * N + j];
      } else {
        s += r[t] * C[t * N + t];
        for (int64_t q = 0; q < g - 1; ++q) {
          int64_t j = nbr_g[t * (g - 1) + q];
          s += r[j] * C[t * N + j];
        }
      }
      score[t] = s;
    }
    int64_t b = -1;
    for (int64_t t = 0; t < N; ++t)
      if (!chosen[t] && (b < 0 || score[t] < score[b])) b = t;
    double sec = INFINITY;
    for (int64_t t = 0; t < N; ++t)
      if (!chosen[t] && t != b && score[t] < sec) sec = score[t];
    int64_t pick = b;
    if (forced) {
      pick = forced[l];
      if (pick < 0 || pick >= N || chosen[pick]) {
        rc = ORC_EINVAL;
        break;
      }
    }
    if (best_idx) best_idx[l] = b;
    if (best_score) best_score[l] = score[b];
    if (second) second[l] = sec;
    if (picked_score) picked_score[l] = score[pick];
    if (order) order[l] = pick;
    /* Eq. sgs_update */
    chosen[pick] = 1;
    sel[l] = pick;
    memcpy(rows + l * N, C + pick * N, sizeof(double) * (size_t)N);
  }
done:
  free(sel); free(rows); free(u); free(fpot); free(gpot); free(col); free(r); free(score);
  free(chosen);
  return rc;
}
