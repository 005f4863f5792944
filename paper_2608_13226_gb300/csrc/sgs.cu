// K5: Spatial-Guided Greedy Selection (Sec. 3.5, Eqs. srpot, local_neighbor,
// greedy_flow, sgs_select, sgs_update).
//
// The semi-relaxed OT of Eq. srpot, with the source support and its capacity
// as decision variables, has a closed-form plan: every target t_j sends its
// mass v_j to its cheapest selected source among those whose neighbourhood
// M_g contains it.  Its value is F(S) = sum_j v_j m_j with the coverage cost
// m_j = min(m0, min_{s in S, j in M_g(s)} C(s, j)), and the residual-weighted
// marginal cost of adding t is -gain(t) with
//     gain(t) = sum_{j in M_g(t)} v_j max(m_j - C(t, j), 0).
// Each step adds the unselected token with the largest gain (lowest index
// among equal gains) and lowers m on its neighbourhood.
//
// One persistent cooperative grid: each scene owns `cps` co-resident blocks.
// Every block keeps the whole (m_j, v_j) state of its scene in shared memory;
// per step the blocks sweep disjoint candidate rows (one warp per row,
// float4 streaming loads of C), publish their best (gain, index) key, meet at
// a scene-local grid barrier (bounded wait), all reduce the same partials to
// the same winner and apply the same update to their copy of m.
#include "common.cuh"

namespace cp {

constexpr int SGS_THREADS = 512;
constexpr int SGS_WARPS = SGS_THREADS / 32;

__device__ __forceinline__ float4 ld_stream_f4(const float4* p) {
  float4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(r.x), "=f"(r.y), "=f"(r.z), "=f"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ unsigned long long gain_key(float gain, int t) {
  // gain >= 0, so its bits order like its value; lower index wins ties
  return ((unsigned long long)__float_as_uint(gain) << 32) | (0xFFFFFFFFu - (uint32_t)t);
}

// One term of gain(t) = sum_j v_j max(m_j - C(t, j), 0), each operation
// rounded once: the computed gain can only decrease when m decreases, which
// makes a gain computed at an earlier step an upper bound of the current one.
__device__ __forceinline__ float gain_term(float acc, float v, float m, float c) {
  return __fmaf_rn(v, fmaxf(__fsub_rn(m, c), 0.0f), acc);
}

// Partial gain over quarter q of a dense padded row (ncols % 4 == 0, pad
// v = 0): the row's float4 chunks are cut into four contiguous quarters;
// lane l sums chunks l, l+32, ... of the quarter in ascending order, then a
// butterfly (identical result in every lane).
__device__ __forceinline__ float quarter_gain(const float* __restrict__ crow, const float* sm_m,
                                              const float* sm_v, int ncols, int q, int lane) {
  const float4* row = reinterpret_cast<const float4*>(crow);
  const float4* m4 = reinterpret_cast<const float4*>(sm_m);
  const float4* v4 = reinterpret_cast<const float4*>(sm_v);
  const int nq = ncols >> 2;
  const int Q4 = (nq + 3) >> 2;
  const int q_end = min(nq, (q + 1) * Q4);
  float acc = 0.0f;
  int i = q * Q4 + lane;
  for (; i + 224 < q_end; i += 256) {
    float4 cs[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) cs[u] = ld_stream_f4(row + i + 32 * u);
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const float4 mm = m4[i + 32 * u], vv = v4[i + 32 * u];
      acc = gain_term(acc, vv.x, mm.x, cs[u].x);
      acc = gain_term(acc, vv.y, mm.y, cs[u].y);
      acc = gain_term(acc, vv.z, mm.z, cs[u].z);
      acc = gain_term(acc, vv.w, mm.w, cs[u].w);
    }
  }
  for (; i < q_end; i += 32) {
    const float4 c0 = ld_stream_f4(row + i);
    const float4 mm = m4[i], vv = v4[i];
    acc = gain_term(acc, vv.x, mm.x, c0.x);
    acc = gain_term(acc, vv.y, mm.y, c0.y);
    acc = gain_term(acc, vv.z, mm.z, c0.z);
    acc = gain_term(acc, vv.w, mm.w, c0.w);
  }
  return warp_sum(acc);
}

// The four quarter sums combined in one fixed order.
__device__ __forceinline__ float combine_quarters(float s0, float s1, float s2, float s3) {
  return __fadd_rn(__fadd_rn(__fadd_rn(s0, s1), s2), s3);
}

// gain(t) over a dense padded row, by one warp: the same quarters and the
// same combination as the four-warp evaluation of the lazy kernel, so every
// kernel computes bit-identical gains.
__device__ __forceinline__ float dense_row_gain(const float* __restrict__ crow,
                                                const float* sm_m, const float* sm_v, int ncols,
                                                int lane) {
  const float s0 = quarter_gain(crow, sm_m, sm_v, ncols, 0, lane);
  const float s1 = quarter_gain(crow, sm_m, sm_v, ncols, 1, lane);
  const float s2 = quarter_gain(crow, sm_m, sm_v, ncols, 2, lane);
  const float s3 = quarter_gain(crow, sm_m, sm_v, ncols, 3, lane);
  return combine_quarters(s0, s1, s2, s3);
}

// gain(t) over the local neighbourhood M_g(t): slab row of g costs, member
// k = 0 is t itself, members k >= 1 are t's nearest others.
__device__ __forceinline__ float local_row_gain(const float* __restrict__ srow,
                                                const int32_t* __restrict__ nb, int t, int g,
                                                const float* sm_m, const float* sm_v, int lane) {
  float acc = 0.0f;
  for (int k = lane; k < g; k += 32) {
    const int j = k == 0 ? t : nb[k - 1];
    acc = gain_term(acc, sm_v[j], sm_m[j], srow[k]);
  }
  return warp_sum(acc);
}

// F(S) = sum_j v_j m_j in fp64, in one fixed order whatever the block size
// (>= 512 threads): thread r < 512 sums j = r, r+512, ...; then 16 warp
// butterflies; then the 16 warp sums in order.  Every thread of the block
// must call it; the result is valid in thread 0.
__device__ __forceinline__ double objective_sum(const float* sm_m, const float* sm_v, int N) {
  __shared__ double s_part[16];
  double part = 0.0;
  if (threadIdx.x < 512)
    for (int j = threadIdx.x; j < N; j += 512) part += (double)sm_v[j] * (double)sm_m[j];
  if (threadIdx.x < 512) part = warp_sum(part);
  if (threadIdx.x < 512 && (threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = part;
  __syncthreads();
  double t = 0.0;
  if (threadIdx.x == 0)
    for (int i = 0; i < 16; ++i) t += s_part[i];
  return t;
}

template <bool LOCAL>
__global__ void __launch_bounds__(SGS_THREADS) k_sgs(
    const float* __restrict__ cost, int64_t ldc, const float* __restrict__ slab,
    const int32_t* __restrict__ nbr, const float* __restrict__ v_all, DevParams P, int N, int K,
    int cps, int scene0, int32_t* __restrict__ order32, float* __restrict__ gains,
    double* __restrict__ objective, unsigned long long* partials, uint32_t* counters,
    int* status) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int ncols = LOCAL ? N : (int)ldc;  // dense rows are padded to ldc (C = 0, v = 0)
  float* sm_m = reinterpret_cast<float*>(smem);                  // [ncols] coverage cost m_j
  float* sm_v = sm_m + ncols;                                    // [ncols] capacity v_j
  uint32_t* chosen = reinterpret_cast<uint32_t*>(sm_v + ncols);  // [ceil(N/32)] bitset
  __shared__ unsigned long long s_best[SGS_WARPS];
  __shared__ int s_pick, s_bad;
  __shared__ float s_gain;

  const int b = scene0 + blockIdx.x / cps;
  const int c = blockIdx.x % cps;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* v = v_all + (size_t)b * N;
  const float* Cb = LOCAL ? nullptr : cost + (size_t)b * N * ldc;
  const float* Sb = LOCAL ? slab + (size_t)b * N * P.g : nullptr;
  const int32_t* NB = nbr + (size_t)b * N * P.kk;
  unsigned long long* part = partials;  // [2][B][cps]
  const int nchosen = (N + 31) >> 5;

  for (int j = threadIdx.x; j < ncols; j += SGS_THREADS) {
    sm_m[j] = j < N ? P.m0 : 0.0f;
    sm_v[j] = j < N ? v[j] : 0.0f;
  }
  for (int i = threadIdx.x; i < nchosen; i += SGS_THREADS) chosen[i] = 0u;
  __syncthreads();

  const int gw = c * SGS_WARPS + w, nw = cps * SGS_WARPS;
  const size_t nscenes = gridDim.x / cps;
  bool alive = true;
  unsigned long long my_evals = 0ull;  // rows this warp evaluated (lane 0 counts)
  for (int step = 0; step < K && alive; ++step) {
    unsigned long long best = 0ull;
    for (int t = gw; t < N; t += nw) {
      if (chosen[t >> 5] & (1u << (t & 31))) continue;
      const float acc =
          LOCAL ? local_row_gain(Sb + (size_t)t * P.g, NB + (size_t)t * P.kk, t, P.g, sm_m, sm_v,
                                 lane)
                : dense_row_gain(Cb + (size_t)t * ldc, sm_m, sm_v, ncols, lane);
      ++my_evals;
      const unsigned long long key = gain_key(acc, t);
      best = key > best ? key : best;
    }
    if (lane == 0) s_best[w] = best;
    __syncthreads();
    const int par = step & 1;
    if (threadIdx.x == 0) {
      unsigned long long m = s_best[0];
      for (int i = 1; i < SGS_WARPS; ++i) m = s_best[i] > m ? s_best[i] : m;
      part[((size_t)par * nscenes + (b - scene0)) * cps + c] = m;
    }
    if (!grid_barrier(counters + b, (uint32_t)(step + 1) * (uint32_t)cps, status, P.timeout_ns)) {
      alive = false;
      break;
    }
    if (w == 0) {
      unsigned long long m = 0ull;
      const unsigned long long* pp = part + ((size_t)par * nscenes + (b - scene0)) * cps;
      for (int i = lane; i < cps; i += 32) {
        // each reading lane acquires: a weak load may be served a stale copy
        const unsigned long long x = ld_acquire_u64(pp + i);
        m = x > m ? x : m;
      }
      m = warp_max_u64(m);
      if (lane == 0) {
        const int pk = (int)(0xFFFFFFFFu - (uint32_t)(m & 0xFFFFFFFFull));
        s_pick = pk;
        s_gain = __uint_as_float((uint32_t)(m >> 32));
        // decided once, before anyone updates the state: a winner must be an
        // unselected token (never expected to fail)
        s_bad = pk < 0 || pk >= N || (chosen[pk >> 5] & (1u << (pk & 31))) != 0u;
      }
    }
    __syncthreads();
    const int pick = s_pick;
    if (s_bad) {
      if (threadIdx.x == 0 && atomicCAS(status, 0, CP_EDEVICE) == 0) {
        status[4] = step;  // where it happened, for diagnosis
        status[5] = b;
        status[6] = c;
        status[7] = pick;
      }
      alive = false;
      break;
    }
    if (threadIdx.x == 0) {
      chosen[pick >> 5] |= 1u << (pick & 31);
      if (c == 0) {
        order32[(size_t)b * K + step] = pick;
        if (gains) gains[(size_t)b * K + step] = s_gain;
      }
    }
    // S <- S u {t*} (Eq. sgs_update): lower the coverage cost of its targets
    if (!LOCAL) {
      const float* row = Cb + (size_t)pick * ldc;
      for (int j = threadIdx.x; j < N; j += SGS_THREADS) sm_m[j] = fminf(sm_m[j], __ldg(row + j));
    } else {
      const float* srow = Sb + (size_t)pick * P.g;
      const int32_t* nb = NB + (size_t)pick * P.kk;
      for (int k = threadIdx.x; k < P.g; k += SGS_THREADS) {
        const int j = k == 0 ? pick : nb[k - 1];
        sm_m[j] = fminf(sm_m[j], srow[k]);
      }
    }
    __syncthreads();
  }

  unsigned long long* cstats = reinterpret_cast<unsigned long long*>(
      reinterpret_cast<unsigned char*>(status) + kCallStatsOffset);
  if (lane == 0 && my_evals) atomicAdd(&cstats[0], my_evals);
  if (c == 0 && threadIdx.x == 0) atomicAdd(&cstats[1], (unsigned long long)K);
  if (c == 0 && alive && objective) {
    const double F = objective_sum(sm_m, sm_v, N);
    if (threadIdx.x == 0) objective[b] = F;
  }
}

template <bool LOCAL>
static int sgs_launch_impl(const float* cost, int64_t ldc, const float* slab, const int32_t* nbr,
                           const float* v, const DevParams& P, int64_t B, int64_t N, int64_t K,
                           int32_t* order32, float* gains, double* objective,
                           unsigned long long* partials, uint32_t* counters, int* status,
                           cudaStream_t s) {
  DeviceInfo di;
  if (device_info(&di) != CP_OK) return CP_ECUDA;
  const int64_t ncols = LOCAL ? N : ldc;
  const size_t smem = 2 * sizeof(float) * (size_t)ncols + sizeof(uint32_t) * (size_t)((N + 31) / 32);
  auto fn = k_sgs<LOCAL>;
  if (smem > 48 * 1024 &&
      cuda_status(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                  "launch_sgs: smem attribute") != CP_OK)
    return CP_ECUDA;
  int per_sm = 0;
  if (cuda_status(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, SGS_THREADS, smem),
                  "launch_sgs: occupancy") != CP_OK)
    return CP_ECUDA;
  if (per_sm < 1) return CP_EUNSUPPORTED;
  const int64_t slots = (int64_t)per_sm * di.sm_count;
  const int64_t per_launch = B < slots ? B : slots;  // scenes resident together
  int cps = (int)(slots / per_launch);
  // a scene never needs more blocks than it has candidate rows per warp
  const int64_t max_cps = (N + SGS_WARPS - 1) / SGS_WARPS;
  if (cps > max_cps) cps = (int)max_cps;
  if (cps < 1) cps = 1;
  if (cuda_status(cudaMemsetAsync(counters, 0, sizeof(uint32_t) * (size_t)B, s),
                  "launch_sgs: counters") != CP_OK)
    return CP_ECUDA;
  if (cuda_status(cudaMemsetAsync(partials, 0,
                                  sizeof(unsigned long long) * 2 * (size_t)per_launch * cps, s),
                  "launch_sgs: partials") != CP_OK)
    return CP_ECUDA;
  for (int64_t b0 = 0; b0 < B; b0 += per_launch) {
    const int64_t nb = (B - b0) < per_launch ? (B - b0) : per_launch;
    int Ni = (int)N, Ki = (int)K, scene0 = (int)b0;
    DevParams Pc = P;
    void* args[] = {(void*)&cost, (void*)&ldc, (void*)&slab, (void*)&nbr, (void*)&v, (void*)&Pc,
                    (void*)&Ni, (void*)&Ki, (void*)&cps, (void*)&scene0, (void*)&order32,
                    (void*)&gains, (void*)&objective, (void*)&partials, (void*)&counters,
                    (void*)&status};
    cudaError_t e = cudaLaunchCooperativeKernel((const void*)fn, dim3((unsigned)(nb * cps)),
                                                dim3(SGS_THREADS), args, smem, s);
    note_launch();
    if (cuda_status(e, "launch_sgs: cooperative launch") != CP_OK) return CP_ECUDA;
  }
  return CP_OK;
}


// ---------------------------------------------------------------------------
// Lazy evaluation of the same greedy (exact, bit-identical picks).
//
// A gain computed at an earlier step is an upper bound of the current one
// (gain_term is monotone in m and m only decreases), so the step's winner --
// the largest (gain, -index) key -- is found without evaluating every
// candidate: keep the last computed gain ub[t] of every token; a candidate
// whose bound is exact this step ("fresh") and larger than every other bound
// is the winner.  One block of 32 warps per scene; warp w owns the
// candidates [w*S, (w+1)*S).  Each round every warp reports the largest
// bound of its slice; if the overall largest is fresh the step is decided,
// otherwise each warp whose slice-best is stale and could still beat the
// best fresh key recomputes that row.  Step 0 evaluates every candidate.
// No inter-block synchronisation: blocks are independent scenes.
// ---------------------------------------------------------------------------
constexpr int LZ_THREADS = 1024;
constexpr int LZ_WARPS = LZ_THREADS / 32;

template <bool LOCAL>
__global__ void __launch_bounds__(LZ_THREADS, 1) k_sgs_lazy(
    const float* __restrict__ cost, int64_t ldc, const float* __restrict__ slab,
    const int32_t* __restrict__ nbr, const float* __restrict__ v_all, DevParams P, int N, int K,
    int32_t* __restrict__ order32, float* __restrict__ gains, double* __restrict__ objective,
    int* status) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int ncols = LOCAL ? N : (int)ldc;
  const int nwords = (N + 31) >> 5;
  float* sm_m = reinterpret_cast<float*>(smem);                 // [ncols] coverage cost
  float* sm_v = sm_m + ncols;                                   // [ncols] capacity
  float* ub = sm_v + ncols;                                     // [N] last computed gain
  uint32_t* chosen = reinterpret_cast<uint32_t*>(ub + N);       // [nwords]
  uint32_t* fresh = chosen + nwords;                            // [nwords]
  __shared__ unsigned long long s_wkey[LZ_WARPS];
  __shared__ int s_wfresh[LZ_WARPS];
  unsigned long long my_evals = 0ull, my_rounds = 0ull;  // lane 0 / thread 0 count

  const int b = blockIdx.x;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* v = v_all + (size_t)b * N;
  const float* Cb = LOCAL ? nullptr : cost + (size_t)b * N * ldc;
  const float* Sb = LOCAL ? slab + (size_t)b * N * P.g : nullptr;
  const int32_t* NB = nbr + (size_t)b * N * P.kk;

  for (int j = threadIdx.x; j < ncols; j += LZ_THREADS) {
    sm_m[j] = j < N ? P.m0 : 0.0f;
    sm_v[j] = j < N ? v[j] : 0.0f;
  }
  for (int i = threadIdx.x; i < nwords; i += LZ_THREADS) chosen[i] = 0u;
  __syncthreads();

  auto gain_of = [&](int t) -> float {
    return LOCAL ? local_row_gain(Sb + (size_t)t * P.g, NB + (size_t)t * P.kk, t, P.g, sm_m, sm_v,
                                  lane)
                 : dense_row_gain(Cb + (size_t)t * ldc, sm_m, sm_v, ncols, lane);
  };
  // step 0: every gain exactly
  for (int t = w; t < N; t += LZ_WARPS) {
    const float g0 = gain_of(t);
    if (lane == 0) ub[t] = g0;
    ++my_evals;
  }
  const int S = (N + LZ_WARPS - 1) / LZ_WARPS;
  const int t_lo = w * S, t_hi = min(N, t_lo + S);

  for (int step = 0; step < K; ++step) {
    for (int i = threadIdx.x; i < nwords; i += LZ_THREADS) fresh[i] = step == 0 ? ~0u : 0u;
    __syncthreads();
    int pick = -1;
    for (int round = 0; round <= N; ++round) {
      ++my_rounds;
      unsigned long long best = 0ull;
      for (int t = t_lo + lane; t < t_hi; t += 32)
        if (!(chosen[t >> 5] & (1u << (t & 31)))) {
          const unsigned long long key = gain_key(ub[t], t);
          best = key > best ? key : best;
        }
      best = warp_max_u64(best);
      if (lane == 0) {
        const int bt = (int)(0xFFFFFFFFu - (uint32_t)(best & 0xFFFFFFFFull));
        s_wkey[w] = best;
        s_wfresh[w] = best != 0ull && ((fresh[bt >> 5] >> (bt & 31)) & 1u);
      }
      __syncthreads();
      unsigned long long G = 0ull, BF = 0ull;
      for (int i = 0; i < LZ_WARPS; ++i) {
        const unsigned long long k = s_wkey[i];
        G = k > G ? k : G;
        if (s_wfresh[i]) BF = k > BF ? k : BF;
      }
      const unsigned long long mine = s_wkey[w];
      const bool mine_fresh = s_wfresh[w] != 0;
      __syncthreads();  // s_wkey / s_wfresh are rewritten next round
      if (G != 0ull && G == BF) {  // the largest bound is exact: the winner
        pick = (int)(0xFFFFFFFFu - (uint32_t)(G & 0xFFFFFFFFull));
        break;
      }
      if (G == 0ull) break;  // no candidate left (never for K <= N)
      if (!mine_fresh && mine > BF) {  // this slice's best might still win
        const int t = (int)(0xFFFFFFFFu - (uint32_t)(mine & 0xFFFFFFFFull));
        const float g = gain_of(t);
        ++my_evals;
        if (lane == 0) {
          ub[t] = g;
          atomicOr(&fresh[t >> 5], 1u << (t & 31));
        }
      }
      __syncthreads();
    }
    // every thread checks the winner before anyone updates the state
    const bool bad = pick < 0 || pick >= N || (chosen[pick >> 5] & (1u << (pick & 31))) != 0u;
    __syncthreads();
    if (bad) {  // never expected; block-uniform (every thread has the same pick)
      if (threadIdx.x == 0 && atomicCAS(status, 0, CP_EDEVICE) == 0) {
        status[4] = step;
        status[5] = b;
        status[6] = 0;
        status[7] = pick;
      }
      return;
    }
    if (threadIdx.x == 0) {
      chosen[pick >> 5] |= 1u << (pick & 31);
      order32[(size_t)b * K + step] = pick;
      if (gains) gains[(size_t)b * K + step] = ub[pick];
    }
    // S <- S u {t*} (Eq. sgs_update)
    if (!LOCAL) {
      const float* row = Cb + (size_t)pick * ldc;
      for (int j = threadIdx.x; j < N; j += LZ_THREADS) sm_m[j] = fminf(sm_m[j], __ldg(row + j));
    } else {
      const float* srow = Sb + (size_t)pick * P.g;
      const int32_t* nb = NB + (size_t)pick * P.kk;
      for (int k = threadIdx.x; k < P.g; k += LZ_THREADS) {
        const int j = k == 0 ? pick : nb[k - 1];
        sm_m[j] = fminf(sm_m[j], srow[k]);
      }
    }
    __syncthreads();
  }

  unsigned long long* cstats = reinterpret_cast<unsigned long long*>(
      reinterpret_cast<unsigned char*>(status) + kCallStatsOffset);
  if (lane == 0 && my_evals) atomicAdd(&cstats[0], my_evals);
  if (threadIdx.x == 0) atomicAdd(&cstats[1], my_rounds);
  if (objective) {
    const double F = objective_sum(sm_m, sm_v, N);
    if (threadIdx.x == 0) objective[b] = F;
  }
}


// ---------------------------------------------------------------------------
// Dense lazy SGS on a thread-block cluster.  The C blocks of a cluster share
// one scene: block c owns the candidates [c*NC, (c+1)*NC) and keeps its own
// copy of the scene's (m, v); its 32 warps form 8 quads, each owning a slice
// of the block's candidates.  A round: every quad scans its slice for the
// best bound; the C*8 quad bests are exchanged through distributed shared
// memory after a cluster barrier; if the largest is exact (fresh) it is the
// step's winner, otherwise every quad whose stale best could still win
// re-evaluates it, one quarter of the row per warp (quarters combined in the
// fixed order of dense_row_gain, so the gains are bit-identical to the full
// sweep's).  The winner's row then lowers every block's copy of m.
//
// The round barrier is a monotone arrival counter in block 0's shared
// memory (release add, acquire spin bounded by the call's time limit; no
// phase can alias).  The quad bests are double-buffered by round parity, so
// one barrier per round suffices.  Errors never return early: every block
// reaches the final hardware cluster barrier, after which no block touches
// another's shared memory.
// ---------------------------------------------------------------------------
constexpr int QD_QUADS = LZ_WARPS / 4;

__device__ __forceinline__ void quad_sync(int k) {
  asm volatile("bar.sync %0, 128;" ::"r"(1 + k) : "memory");
}
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ uint32_t map_rank(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ unsigned long long ld_dsmem_u64(uint32_t a) {
  unsigned long long v;
  asm volatile("ld.shared::cluster.u64 %0, [%1];" : "=l"(v) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ uint32_t ld_dsmem_u32(uint32_t a) {
  uint32_t v;
  asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ uint32_t ld_acquire_dsmem_u32(uint32_t a) {
  uint32_t v;
  asm volatile("ld.acquire.cluster.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ void red_release_dsmem_add(uint32_t a, uint32_t v) {
  asm volatile("red.release.cluster.shared::cluster.add.u32 [%0], %1;" ::"r"(a), "r"(v)
               : "memory");
}
__device__ __forceinline__ void hw_cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}

__global__ void __launch_bounds__(LZ_THREADS, 1) k_sgs_lazy_cl(
    const float* __restrict__ cost, int64_t ldc, const float* __restrict__ v_all, DevParams P,
    int N, int K, int C, int32_t* __restrict__ order32, float* __restrict__ gains,
    double* __restrict__ objective, int* status) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int ncols = (int)ldc;
  const int NC = (N + C - 1) / C;                 // candidates per block
  const int nwords = (NC + 31) >> 5;
  float* sm_m = reinterpret_cast<float*>(smem);   // [ncols] coverage cost (full copy)
  float* sm_v = sm_m + ncols;                     // [ncols] capacity
  float* ub = sm_v + ncols;                       // [NC] last computed gain, own candidates
  uint32_t* chosen = reinterpret_cast<uint32_t*>(ub + NC);  // [nwords] own candidates
  uint32_t* fresh = chosen + nwords;                        // [nwords]
  __shared__ unsigned long long s_wq[LZ_WARPS];
  __shared__ unsigned long long s_key[2][QD_QUADS];  // by round parity, read by the cluster
  __shared__ uint32_t s_fresh[2][QD_QUADS];
  __shared__ float s_part[QD_QUADS][4];
  __shared__ unsigned long long s_G, s_BF;
  __shared__ uint32_t s_ctr;                      // round barrier counter (used in block 0)
  __shared__ int s_ok;

  const uint32_t crank = cluster_ctarank();
  const int b = blockIdx.x / C;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k = w >> 2, q = w & 3, tq = threadIdx.x & 127;
  const int c0 = (int)crank * NC;                 // first candidate of this block
  const int nown = max(0, min(N, c0 + NC) - c0);  // own candidates
  const float* v = v_all + (size_t)b * N;
  const float* Cb = cost + (size_t)b * N * ldc;
  unsigned long long my_evals = 0ull, my_rounds = 0ull;
  const uint32_t ctr0 = map_rank(smem_addr(&s_ctr), 0);

  for (int j = threadIdx.x; j < ncols; j += LZ_THREADS) {
    sm_m[j] = j < N ? P.m0 : 0.0f;
    sm_v[j] = j < N ? v[j] : 0.0f;
  }
  for (int i = threadIdx.x; i < nwords; i += LZ_THREADS) chosen[i] = 0u;
  if (threadIdx.x == 0) s_ctr = 0u;
  hw_cluster_sync();  // every block initialised before anyone arrives on block 0

  // step 0: every own candidate's gain exactly, one warp per row
  for (int t = w; t < nown; t += LZ_WARPS) {
    const float g0 = dense_row_gain(Cb + (size_t)(c0 + t) * ldc, sm_m, sm_v, ncols, lane);
    if (lane == 0) ub[t] = g0;
    ++my_evals;
  }
  const int S = (nown + QD_QUADS - 1) / QD_QUADS;
  const int t_lo = k * S, t_hi = min(nown, t_lo + S);  // quad slice, own indices
  uint32_t gr = 0;  // rounds so far (all blocks count alike)
  bool ok = true;

  for (int step = 0; step < K && ok; ++step) {
    for (int i = threadIdx.x; i < nwords; i += LZ_THREADS) fresh[i] = step == 0 ? ~0u : 0u;
    __syncthreads();
    int pick = -1;
    for (int round = 0; round <= N && ok; ++round, ++gr) {
      ++my_rounds;
      const int par = gr & 1;
      unsigned long long best = 0ull;
      for (int t = t_lo + tq; t < t_hi; t += 128)
        if (!(chosen[t >> 5] & (1u << (t & 31)))) {
          const unsigned long long key = gain_key(ub[t], c0 + t);
          best = key > best ? key : best;
        }
      best = warp_max_u64(best);
      if (lane == 0) s_wq[w] = best;
      quad_sync(k);
      if (q == 0 && lane == 0) {
        unsigned long long kb = s_wq[4 * k];
        for (int i = 1; i < 4; ++i) kb = s_wq[4 * k + i] > kb ? s_wq[4 * k + i] : kb;
        const int bt = (int)(0xFFFFFFFFu - (uint32_t)(kb & 0xFFFFFFFFull)) - c0;
        s_key[par][k] = kb;
        s_fresh[par][k] = kb != 0ull && ((fresh[bt >> 5] >> (bt & 31)) & 1u);
      }
      // cluster round barrier: arrive on block 0's counter, wait for C * (gr+1)
      __syncthreads();
      if (threadIdx.x == 0) {
        int good = 1;
        red_release_dsmem_add(ctr0, 1u);
        const uint32_t target = (gr + 1u) * (uint32_t)C;
        const uint64_t t0 = globaltimer_ns();
        uint32_t spins = 0;
        while (ld_acquire_dsmem_u32(ctr0) < target) {
          if ((++spins & 63u) == 0) {
            if (ld_volatile_i32(status) != 0) { good = 0; break; }
            if (globaltimer_ns() - t0 > P.timeout_ns) {
              set_status(status, CP_ETIMEOUT);
              good = 0;
              break;
            }
          }
        }
        s_ok = good;
      }
      __syncthreads();
      if (!s_ok) {
        ok = false;
        break;
      }
      if (w == 0) {  // gather the cluster's quad bests
        unsigned long long G = 0ull, BF = 0ull;
        (void)ld_acquire_dsmem_u32(ctr0);  // this lane's own acquire of the round
        for (int e = lane; e < C * QD_QUADS; e += 32) {
          const uint32_t r = (uint32_t)(e / QD_QUADS), kk = (uint32_t)(e % QD_QUADS);
          const unsigned long long key = ld_dsmem_u64(map_rank(smem_addr(&s_key[par][kk]), r));
          const uint32_t fr = ld_dsmem_u32(map_rank(smem_addr(&s_fresh[par][kk]), r));
          G = key > G ? key : G;
          if (fr) BF = key > BF ? key : BF;
        }
        G = warp_max_u64(G);
        BF = warp_max_u64(BF);
        if (lane == 0) {
          s_G = G;
          s_BF = BF;
        }
      }
      __syncthreads();
      const unsigned long long G = s_G, BF = s_BF;
      if (G != 0ull && G == BF) {  // the largest bound is exact: the winner
        pick = (int)(0xFFFFFFFFu - (uint32_t)(G & 0xFFFFFFFFull));
        ++gr;
        break;
      }
      if (G == 0ull) {  // no candidate left (never for K <= N)
        ++gr;
        break;
      }
      const unsigned long long mine = s_key[par][k];
      if (!s_fresh[par][k] && mine > BF) {  // this quad's best might still win
        const int t = (int)(0xFFFFFFFFu - (uint32_t)(mine & 0xFFFFFFFFull));
        const float part = quarter_gain(Cb + (size_t)t * ldc, sm_m, sm_v, ncols, q, lane);
        if (lane == 0) s_part[k][q] = part;
        quad_sync(k);
        if (q == 0 && lane == 0) {
          const int tl = t - c0;
          ub[tl] = combine_quarters(s_part[k][0], s_part[k][1], s_part[k][2], s_part[k][3]);
          atomicOr(&fresh[tl >> 5], 1u << (tl & 31));  // quads may share a word
          ++my_evals;
        }
      }
      __syncthreads();
    }
    if (!ok) break;
    const bool bad = pick < 0 || pick >= N ||
                     (pick >= c0 && pick < c0 + nown &&
                      (chosen[(pick - c0) >> 5] & (1u << ((pick - c0) & 31))) != 0u);
    __syncthreads();
    if (bad) {  // never expected; cluster-uniform
      if (threadIdx.x == 0 && crank == 0 && atomicCAS(status, 0, CP_EDEVICE) == 0) {
        status[4] = step;
        status[5] = b;
        status[6] = (int)crank;
        status[7] = pick;
      }
      ok = false;
      break;
    }
    if (threadIdx.x == 0) {
      if (pick >= c0 && pick < c0 + nown) chosen[(pick - c0) >> 5] |= 1u << ((pick - c0) & 31);
      if (crank == 0) {
        order32[(size_t)b * K + step] = pick;
        if (gains) gains[(size_t)b * K + step] = __uint_as_float((uint32_t)(s_G >> 32));
      }
    }
    // S <- S u {t*} (Eq. sgs_update), on this block's copy of m
    const float* row = Cb + (size_t)pick * ldc;
    for (int j = threadIdx.x; j < N; j += LZ_THREADS) sm_m[j] = fminf(sm_m[j], __ldg(row + j));
    __syncthreads();
  }

  unsigned long long* cstats = reinterpret_cast<unsigned long long*>(
      reinterpret_cast<unsigned char*>(status) + kCallStatsOffset);
  if (lane == 0 && my_evals) atomicAdd(&cstats[0], my_evals);
  if (threadIdx.x == 0 && crank == 0) atomicAdd(&cstats[1], my_rounds);
  if (ok && crank == 0 && objective) {
    const double F = objective_sum(sm_m, sm_v, N);
    if (threadIdx.x == 0) objective[b] = F;
  }
  hw_cluster_sync();  // nobody leaves while a peer may still read its shared memory
}

// Blocks per scene for the cluster kernel: the largest power of two <= 8
// such that every scene's cluster can be resident at once.
static int cluster_size_for(int64_t B, int sm_count) {
  int C = 8;
  while (C > 1 && (int64_t)C * B > sm_count) C >>= 1;
  return C;
}

static int sgs_lazy_cluster_launch(const float* cost, int64_t ldc, const float* v,
                                   const DevParams& P, int64_t B, int64_t N, int64_t K,
                                   int32_t* order32, float* gains, double* objective, int* status,
                                   cudaStream_t s) {
  DeviceInfo di;
  if (device_info(&di) != CP_OK) return CP_ECUDA;
  auto fn = k_sgs_lazy_cl;
  for (int C = cluster_size_for(B, di.sm_count); C >= 1; C >>= 1) {
    const int64_t NC = (N + C - 1) / C;
    const size_t smem = sizeof(float) * (size_t)(2 * ldc + NC) +
                        2 * sizeof(uint32_t) * (size_t)((NC + 31) / 32);
    if (cuda_status(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem),
                    "launch_sgs_lazy_cluster: smem attribute") != CP_OK)
      return CP_ECUDA;
    if (C > 8 &&
        cuda_status(cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1),
                    "launch_sgs_lazy_cluster: cluster attribute") != CP_OK)
      return CP_ECUDA;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(B * C));
    cfg.blockDim = dim3(LZ_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, (const void*)fn, &cfg) != cudaSuccess ||
        clusters < 1) {
      (void)cudaGetLastError();
      continue;  // this cluster shape cannot be resident: try a smaller one
    }
    int Ni = (int)N, Ki = (int)K;
    cudaError_t e = cudaLaunchKernelEx(&cfg, fn, cost, ldc, v, P, Ni, Ki, C, order32, gains,
                                       objective, status);
    note_launch();
    return cuda_status(e, "launch_sgs_lazy_cluster");
  }
  note_message("launch_sgs_lazy_cluster: no resident cluster shape");
  return CP_EUNSUPPORTED;
}

template <bool LOCAL>
static int sgs_lazy_launch(const float* cost, int64_t ldc, const float* slab, const int32_t* nbr,
                           const float* v, const DevParams& P, int64_t B, int64_t N, int64_t K,
                           int32_t* order32, float* gains, double* objective, int* status,
                           cudaStream_t s) {
  const int64_t ncols = LOCAL ? N : ldc;
  const size_t smem = sizeof(float) * (size_t)(2 * ncols + N) +
                      2 * sizeof(uint32_t) * (size_t)((N + 31) / 32);
  if (!LOCAL)
    return sgs_lazy_cluster_launch(cost, ldc, v, P, B, N, K, order32, gains, objective, status, s);
  auto fn = k_sgs_lazy<true>;
  if (smem > 48 * 1024 &&
      cuda_status(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                  "launch_sgs_lazy: smem attribute") != CP_OK)
    return CP_ECUDA;
  fn<<<(unsigned)B, LZ_THREADS, smem, s>>>(cost, ldc, slab, nbr, v, P, (int)N, (int)K, order32,
                                          gains, objective, status);
  return last_launch_status();
}

int launch_sgs(const float* cost, int64_t ldc, const float* slab, const int32_t* nbr,
               const float* v, const DevParams& P, int64_t B, int64_t N, int64_t K,
               int32_t* order32, float* gains, double* objective, uint64_t* partials,
               uint32_t* counters, int* status, cudaStream_t s) {
  auto* part = reinterpret_cast<unsigned long long*>(partials);
  if (P.sgs_mode == 0) {
    if (P.g < N)
      return sgs_lazy_launch<true>(cost, ldc, slab, nbr, v, P, B, N, K, order32, gains, objective,
                                   status, s);
    return sgs_lazy_launch<false>(cost, ldc, slab, nbr, v, P, B, N, K, order32, gains, objective,
                                  status, s);
  }
  if (P.g < N)
    return sgs_launch_impl<true>(cost, ldc, slab, nbr, v, P, B, N, K, order32, gains, objective,
                                 part, counters, status, s);
  return sgs_launch_impl<false>(cost, ldc, slab, nbr, v, P, B, N, K, order32, gains, objective,
                                part, counters, status, s);
}

// Upper bound of the partial slots the launcher may use: 2 * B * cps with
// cps <= ceil(N / SGS_WARPS).
int64_t sgs_partials_count(int64_t B, int64_t N) {
  return 2 * B * ((N + SGS_WARPS - 1) / SGS_WARPS);
}

// ---------------------------------------------------------------------------
// Barrier self-test: n_blocks co-resident blocks wait for `expected`
// arrivals; with expected > n_blocks the bounded wait must run out.
// ---------------------------------------------------------------------------
__global__ void k_barrier_selftest(uint32_t* ctr, uint32_t expected, int* status,
                                   uint64_t timeout_ns) {
  grid_barrier(ctr, expected, status, timeout_ns);
}

int launch_barrier_selftest(int n_blocks, int expected, uint64_t timeout_ns, uint32_t* ctr,
                            int* status, cudaStream_t s) {
  DeviceInfo di;
  if (device_info(&di) != CP_OK) return CP_ECUDA;
  if (n_blocks < 1 || n_blocks > di.sm_count || expected < 0) return CP_EINVAL;
  if (cudaMemsetAsync(ctr, 0, sizeof(uint32_t), s) != cudaSuccess) return CP_ECUDA;
  if (cudaMemsetAsync(status, 0, sizeof(int), s) != cudaSuccess) return CP_ECUDA;
  uint32_t exp_u = (uint32_t)expected;
  void* args[] = {(void*)&ctr, (void*)&exp_u, (void*)&status, (void*)&timeout_ns};
  cudaError_t e = cudaLaunchCooperativeKernel((const void*)k_barrier_selftest, dim3(n_blocks),
                                              dim3(64), args, 0, s);
  note_launch();
  return cuda_status(e);
}

// ---------------------------------------------------------------------------
// Ascending sort of K indices per scene (bitonic, shared memory).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) k_sort_kept(const int32_t* __restrict__ idx32, int K, int L,
                                                    int64_t* __restrict__ kept,
                                                    int64_t* __restrict__ order64) {
  extern __shared__ int32_t sk[];
  const int b = blockIdx.x;
  const int32_t* in = idx32 + (size_t)b * K;
  for (int i = threadIdx.x; i < L; i += blockDim.x) sk[i] = i < K ? in[i] : INT32_MAX;
  if (order64)
    for (int i = threadIdx.x; i < K; i += blockDim.x) order64[(size_t)b * K + i] = in[i];
  __syncthreads();
  for (int size = 2; size <= L; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < (L >> 1); i += blockDim.x) {
        const int a = 2 * i - (i & (stride - 1));
        const int c = a + stride;
        const bool up = (a & size) == 0;
        const int32_t x = sk[a], y = sk[c];
        if ((x > y) == up) { sk[a] = y; sk[c] = x; }
      }
      __syncthreads();
    }
  }
  for (int i = threadIdx.x; i < K; i += blockDim.x) kept[(size_t)b * K + i] = sk[i];
}

int launch_sort_kept(const int32_t* idx32, int64_t B, int64_t K, int64_t* kept, int64_t* order64,
                     cudaStream_t s) {
  int L = 2;
  while (L < K) L <<= 1;
  const size_t smem = sizeof(int32_t) * (size_t)L;
  if (smem > 48 * 1024 &&
      cuda_status(cudaFuncSetAttribute(k_sort_kept, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem),
                  "launch_sort_kept: smem attribute") != CP_OK)
    return CP_ECUDA;
  k_sort_kept<<<(unsigned)B, 1024, smem, s>>>(idx32, (int)K, L, kept, order64);
  return last_launch_status();
}

}  // namespace cp
