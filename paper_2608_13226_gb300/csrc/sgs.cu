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
// v = 0).  The row's float4 chunks are taken in iterations of 32 (iteration
// it: chunks 32 it .. 32 it + 31, 512 contiguous bytes) and quarter q owns
// the iterations q, q + 4, q + 8, ...: a row's positive terms cluster by
// token index (nearby tokens), and interleaving spreads them evenly over the
// four quarters.  Lane l sums chunk 32 it + l of each owned iteration in
// ascending order, then a butterfly (identical result in every lane).
__device__ __forceinline__ float quarter_gain(const float* __restrict__ crow, const float* sm_m,
                                              const float* sm_v, int ncols, int q, int lane) {
  const float4* row = reinterpret_cast<const float4*>(crow);
  const float4* m4 = reinterpret_cast<const float4*>(sm_m);
  const float4* v4 = reinterpret_cast<const float4*>(sm_v);
  const int nq = ncols >> 2;
  float acc = 0.0f;
  int i = 32 * q + lane;
  for (; i + 7 * 128 < nq; i += 8 * 128) {
    float4 cs[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) cs[u] = ld_stream_f4(row + i + 128 * u);
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const float4 mm = m4[i + 128 * u], vv = v4[i + 128 * u];
      acc = gain_term(acc, vv.x, mm.x, cs[u].x);
      acc = gain_term(acc, vv.y, mm.y, cs[u].y);
      acc = gain_term(acc, vv.z, mm.z, cs[u].z);
      acc = gain_term(acc, vv.w, mm.w, cs[u].w);
    }
  }
  for (; i < nq; i += 128) {
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

// quarter_gain over the blocks a mask names.  Quarter q's u-th iteration
// holds chunks 32 (4u + q) + lane; bit u >> bit_shift of m16 says whether iteration u may hold a positive term.  An
// iteration whose terms are all zero leaves every lane's sum unchanged (each
// term is v * max(m - C, 0) = +0 and acc + 0 = acc), so skipping it returns
// exactly quarter_gain's value.  A term stays zero once m <= C, because m
// only decreases; out16 gets the bits of the iterations that still have
// some m > C.  Up to 8 needed iterations are loaded before any is summed.
__device__ __forceinline__ float quarter_gain_masked(const float* __restrict__ crow,
                                                     const float* sm_m, const float* sm_v,
                                                     int ncols, int q, int lane, uint32_t m16,
                                                     int bit_shift, uint32_t& out16, int& nread) {
  const float4* row = reinterpret_cast<const float4*>(crow);
  const float4* m4 = reinterpret_cast<const float4*>(sm_m);
  const float4* v4 = reinterpret_cast<const float4*>(sm_v);
  const int nq = ncols >> 2;
  const int NI = (nq + 31) >> 5;                    // iterations of the whole row
  const int nit = NI > q ? (NI - q + 3) >> 2 : 0;   // ... owned by quarter q
  uint32_t todo = m16 & 0xFFFFu;
  if (bit_shift) {  // each bit covers two iterations: spread bit i to bits 2i, 2i+1
    todo = (todo | (todo << 8)) & 0x00FF00FFu;
    todo = (todo | (todo << 4)) & 0x0F0F0F0Fu;
    todo = (todo | (todo << 2)) & 0x33333333u;
    todo = (todo | (todo << 1)) & 0x55555555u;
    todo |= todo << 1;
  }
  if (nit < 32) todo &= (1u << nit) - 1u;
  nread = __popc(todo);
  float acc = 0.0f;
  uint32_t nzb = 0u;
  while (todo) {
    int us[8];
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      us[s] = todo ? __ffs(todo) - 1 : -1;
      todo &= todo - 1u;
    }
    float4 cs[8];
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      const int i = 128 * us[s] + 32 * q + lane;
      cs[s] = (us[s] >= 0 && i < nq) ? ld_stream_f4(row + i) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if (us[s] < 0) break;  // warp-uniform
      const int i = 128 * us[s] + 32 * q + lane;
      bool nz = false;
      if (i < nq) {
        const float4 mm = m4[i], vv = v4[i];
        // d = max(m - C, 0) is +0 or positive, so the OR of the bit
        // patterns is zero iff all four terms are zero
        const float d0 = fmaxf(__fsub_rn(mm.x, cs[s].x), 0.0f);
        const float d1 = fmaxf(__fsub_rn(mm.y, cs[s].y), 0.0f);
        const float d2 = fmaxf(__fsub_rn(mm.z, cs[s].z), 0.0f);
        const float d3 = fmaxf(__fsub_rn(mm.w, cs[s].w), 0.0f);
        acc = __fmaf_rn(vv.x, d0, acc);
        acc = __fmaf_rn(vv.y, d1, acc);
        acc = __fmaf_rn(vv.z, d2, acc);
        acc = __fmaf_rn(vv.w, d3, acc);
        nz = (__float_as_uint(d0) | __float_as_uint(d1) | __float_as_uint(d2) |
              __float_as_uint(d3)) != 0u;
      }
      if (__any_sync(0xFFFFFFFFu, nz)) nzb |= 1u << (us[s] >> bit_shift);
    }
  }
  out16 = nzb;
  return warp_sum(acc);
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
  unsigned long long my_update_bytes = 0ull;  // coverage-update reads (thread 0 of block 0)
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
        my_update_bytes += LOCAL ? 8ull * (unsigned long long)P.g : 4ull * (unsigned long long)N;
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
  if (lane == 0 && my_evals)
    atomicAdd(&cstats[2], my_evals * (unsigned long long)(LOCAL ? 8 * P.g : 4 * ldc));
  if (my_update_bytes) atomicAdd(&cstats[2], my_update_bytes);
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
// whose bound is exact ("fresh") and larger than every other bound is the
// winner.
// ---------------------------------------------------------------------------
constexpr int LZ_THREADS = 1024;
constexpr int LZ_WARPS = LZ_THREADS / 32;

// Reverse neighbourhoods of the local SGS, per scene in CSR form:
// rev[rev_off[j] .. rev_off[j+1]) = the t with j in M_g(t) (M_g(t)[0] = t,
// M_g(t)[k] = nbr[t][k-1]), in no particular order.  One block per scene;
// counts and cursors in shared memory [N].
__global__ void __launch_bounds__(1024) k_rev_build(const int32_t* __restrict__ nbr_all, int N,
                                                    int g, int kk, int32_t* __restrict__ off_all,
                                                    int32_t* __restrict__ rev_all) {
  extern __shared__ int s_c[];  // [N]
  __shared__ int s_sum[1024];
  const int b = blockIdx.x;
  const int32_t* NB = nbr_all + (size_t)b * N * kk;
  int32_t* off = off_all + (size_t)b * (N + 1);
  int32_t* rev = rev_all + (size_t)b * N * g;
  const int64_t ng = (int64_t)N * g;
  for (int j = threadIdx.x; j < N; j += blockDim.x) s_c[j] = 0;
  __syncthreads();
  for (int64_t i = threadIdx.x; i < ng; i += blockDim.x) {
    const int t = (int)(i / g), k = (int)(i % g);
    atomicAdd(&s_c[k == 0 ? t : NB[(size_t)t * kk + (k - 1)]], 1);
  }
  __syncthreads();
  // exclusive prefix of the counts: each thread a contiguous chunk, then a
  // scan of the 1024 chunk sums
  const int chunk = (N + blockDim.x - 1) / blockDim.x;
  const int c0 = min(N, (int)threadIdx.x * chunk), c1 = min(N, c0 + chunk);
  int part = 0;
  for (int j = c0; j < c1; ++j) part += s_c[j];
  s_sum[threadIdx.x] = part;
  __syncthreads();
  for (int d = 1; d < (int)blockDim.x; d <<= 1) {
    const int x = threadIdx.x >= (unsigned)d ? s_sum[threadIdx.x - d] : 0;
    __syncthreads();
    s_sum[threadIdx.x] += x;
    __syncthreads();
  }
  int run = s_sum[threadIdx.x] - part;  // the exclusive prefix of this chunk
  for (int j = c0; j < c1; ++j) {
    const int n = s_c[j];
    off[j] = run;
    s_c[j] = run;  // from here on: the next free slot of j
    run += n;
  }
  if (threadIdx.x == 0) off[N] = (int)ng;
  __syncthreads();
  for (int64_t i = threadIdx.x; i < ng; i += blockDim.x) {
    const int t = (int)(i / g), k = (int)(i % g);
    const int j = k == 0 ? t : NB[(size_t)t * kk + (k - 1)];
    rev[atomicAdd(&s_c[j], 1)] = t;
  }
}

// Local SGS (g < N, Eq. local_neighbor), lazy, one block of 32 warps per
// scene; warp w owns the candidates t = w (mod 32), so the tokens near a pick
// (nearby indices), whose bounds go stale together, are re-evaluated by
// different warps in the same round.  The update of a pick w
// lowers m only on M_g(w), so gain(t) changes only if M_g(t) holds a target
// whose m dropped: exactly the t on that target's reverse list.  Those lose
// their exact mark ("dirty set"); every other bound stays exact -- its terms,
// and so its rounded sum, are unchanged.  A round reads every warp's best key
// and whether it is exact: if the block's largest is exact it is the winner,
// otherwise each warp whose best is stale and above the largest exact one
// re-evaluates it (one warp a row, local_row_gain), and its second best too
// when that one is stale and above it as well, then rescans its slice.
// Step 0 evaluates every candidate; no inter-block synchronisation.
__global__ void __launch_bounds__(LZ_THREADS, 1) k_sgs_local(
    const float* __restrict__ slab, const int32_t* __restrict__ nbr,
    const float* __restrict__ v_all, const int32_t* __restrict__ rev_off_all,
    const int32_t* __restrict__ rev_all, DevParams P, int N, int K,
    int32_t* __restrict__ order32, float* __restrict__ gains, double* __restrict__ objective,
    int* status) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int nwords = (N + 31) >> 5;
  float* sm_m = reinterpret_cast<float*>(smem);            // [N] coverage cost
  float* sm_v = sm_m + N;                                  // [N] capacity
  float* ub = sm_v + N;                                    // [N] last computed gain
  uint32_t* chosen = reinterpret_cast<uint32_t*>(ub + N);  // [nwords]
  uint32_t* fresh = chosen + nwords;                       // [nwords]
  __shared__ unsigned long long s_wkey[LZ_WARPS];          // each warp's best key
  __shared__ unsigned long long s_wkey2[LZ_WARPS];         // ... and its second best
  __shared__ int s_wfr[LZ_WARPS];                          // ... and whether it is exact
  __shared__ int s_pick, s_bad;
  unsigned long long my_evals = 0ull, my_rounds = 0ull, my_bytes = 0ull;

  const int b = blockIdx.x;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = P.g, kk = P.kk;
  const float* v = v_all + (size_t)b * N;
  const float* Sb = slab + (size_t)b * N * g;
  const int32_t* NB = nbr + (size_t)b * N * kk;
  const int32_t* roff = rev_off_all + (size_t)b * (N + 1);
  const int32_t* rev = rev_all + (size_t)b * N * g;

  for (int j = threadIdx.x; j < N; j += LZ_THREADS) {
    sm_m[j] = P.m0;
    sm_v[j] = v[j];
  }
  for (int i = threadIdx.x; i < nwords; i += LZ_THREADS) {
    chosen[i] = 0u;
    fresh[i] = ~0u;
  }
  __syncthreads();
  auto gain_of = [&](int t) -> float {
    return local_row_gain(Sb + (size_t)t * g, NB + (size_t)t * kk, t, g, sm_m, sm_v, lane);
  };
  for (int t = w; t < N; t += LZ_WARPS) {  // step 0: every gain exactly
    const float g0 = gain_of(t);
    if (lane == 0) ub[t] = g0;
    ++my_evals;
  }
  __syncthreads();
  auto is_fresh = [&](unsigned long long key) -> int {
    const int t = (int)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
    return key != 0ull && ((fresh[t >> 5] >> (t & 31)) & 1u);
  };
  auto rescan = [&]() {  // the warp's best and second-best keys
    unsigned long long best = 0ull, second = 0ull;
    for (int t = w + LZ_WARPS * lane; t < N; t += LZ_WARPS * 32)
      if (!(chosen[t >> 5] & (1u << (t & 31)))) {
        const unsigned long long key = gain_key(ub[t], t);
        if (key > best) {
          second = best;
          best = key;
        } else if (key > second) {
          second = key;
        }
      }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {  // merge the lanes' top two
      const unsigned long long ob = __shfl_xor_sync(0xFFFFFFFFu, best, o);
      const unsigned long long os = __shfl_xor_sync(0xFFFFFFFFu, second, o);
      const unsigned long long lo = best < ob ? best : ob;
      best = best > ob ? best : ob;
      const unsigned long long s2 = second > os ? second : os;
      second = lo > s2 ? lo : s2;
    }
    if (lane == 0) {
      s_wkey[w] = best;
      s_wkey2[w] = second;
      s_wfr[w] = is_fresh(best);
    }
  };
  rescan();
  __syncthreads();

  for (int step = 0; step < K; ++step) {
    int pick = -1;
    for (int round = 0; round <= N; ++round) {
      ++my_rounds;
      // lane i reads warp i's entry; two warp maxima give G and BF
      const unsigned long long ki = s_wkey[lane];
      const int fi = s_wfr[lane];
      const unsigned long long G = warp_max_u64(ki);
      const unsigned long long BF = warp_max_u64(fi ? ki : 0ull);
      const unsigned long long mine = __shfl_sync(0xFFFFFFFFu, ki, w);
      const bool mine_fresh = __shfl_sync(0xFFFFFFFFu, fi, w) != 0;
      __syncthreads();  // every warp has read s_wkey / s_wfr before any rescan
      if (G != 0ull && G == BF) {  // the largest bound is exact: the winner
        pick = (int)(0xFFFFFFFFu - (uint32_t)(G & 0xFFFFFFFFull));
        break;
      }
      if (G == 0ull) break;  // no candidate left (never for K <= N)
      if (!mine_fresh && mine > BF) {  // this slice's best might still win
        const int t = (int)(0xFFFFFFFFu - (uint32_t)(mine & 0xFFFFFFFFull));
        // so may its second best when stale and above the largest exact
        // key: evaluated in the same round (any stale candidate may be)
        const unsigned long long k2 = s_wkey2[w];
        const int t2 = (k2 > BF && !is_fresh(k2)) ? (int)(0xFFFFFFFFu - (uint32_t)(k2 & 0xFFFFFFFFull))
                                                  : -1;
        const float gt = gain_of(t);
        const float gt2 = t2 >= 0 ? gain_of(t2) : 0.0f;
        ++my_evals;
        if (lane == 0) {
          ub[t] = gt;
          atomicOr(&fresh[t >> 5], 1u << (t & 31));
          if (t2 >= 0) {
            ub[t2] = gt2;
            atomicOr(&fresh[t2 >> 5], 1u << (t2 & 31));
          }
        }
        if (t2 >= 0) ++my_evals;
        __syncwarp();
        rescan();
      }
      __syncthreads();
    }
    if (threadIdx.x == 0) {  // decided once, before anyone updates the state
      s_pick = pick;
      s_bad = pick < 0 || pick >= N || (chosen[pick >> 5] & (1u << (pick & 31))) != 0u;
    }
    __syncthreads();
    pick = s_pick;
    if (s_bad) {  // never expected; block-uniform
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
      my_bytes += 8ull * (unsigned long long)g;
    }
    // S <- S u {t*} (Eq. sgs_update) on M_g(t*), one warp a member: a target
    // whose m drops makes every candidate on its reverse list stale
    for (int k = w; k < g; k += LZ_WARPS) {
      const int j = k == 0 ? pick : NB[(size_t)pick * kk + (k - 1)];
      const float c = Sb[(size_t)pick * g + k];
      const float mj = sm_m[j];
      if (c < mj) {  // warp-uniform
        __syncwarp();
        if (lane == 0) sm_m[j] = c;
        for (int e = roff[j] + lane; e < roff[j + 1]; e += 32) {
          const int t = rev[e];
          atomicAnd(&fresh[t >> 5], ~(1u << (t & 31)));
        }
      }
    }
    __syncthreads();
    // the warp that held the pick rescans; the others re-read whether their
    // best is still exact (their bounds did not change)
    if (w == (pick & (LZ_WARPS - 1))) {
      rescan();
    } else if (lane == 0) {
      s_wfr[w] = is_fresh(s_wkey[w]);
    }
    __syncthreads();
  }

  unsigned long long* cstats = reinterpret_cast<unsigned long long*>(
      reinterpret_cast<unsigned char*>(status) + kCallStatsOffset);
  if (lane == 0 && my_evals) atomicAdd(&cstats[0], my_evals);
  if (threadIdx.x == 0) atomicAdd(&cstats[1], my_rounds);
  if (lane == 0 && my_evals) atomicAdd(&cstats[2], my_evals * 8ull * (unsigned long long)g);
  if (my_bytes) atomicAdd(&cstats[2], my_bytes);
  if (objective) {
    const double F = objective_sum(sm_m, sm_v, N);
    if (threadIdx.x == 0) objective[b] = F;
  }
}


// ---------------------------------------------------------------------------
// Dense lazy SGS on a thread-block cluster.  The C blocks of a cluster share
// one scene: block c owns the candidates t = c (mod C) and keeps its own
// copy of the scene's (m, v); its 32 warps form 8 quads, quad k owning the
// block's candidates of own index k (mod 8).  Interleaving spreads tokens
// with nearby indices -- in a scene they are nearby in space, so one pick
// lowers their gains together -- over all quads of the cluster, which then
// re-evaluate them in the same round.  A step has two phases.
//
//  1. Local certification, with block barriers only.  Each round every quad
//     finds the best key of its slice.  If the block's largest key is exact
//     ("fresh") it is the block's result r_c; if it is below the cluster's
//     hint h (the largest exact key any block has computed this step) the
//     block cannot hold the winner and r_c is its best fresh key; otherwise
//     every quad whose stale best could still win re-evaluates it, one
//     quarter of the row per warp (quarters combined in the fixed order of
//     dense_row_gain, so gains are bit-identical to the full sweep's).  A
//     new exact key is pushed into every block's hint: a max over keys
//     tagged with the step, so a late push from an earlier step never wins.
//     Each own candidate keeps a 64-bit mask of the row blocks that held a
//     positive term at its last evaluation (when the masks fit in shared
//     memory); an evaluation reads only those blocks (quarter_gain_masked).
//  2. Exchange.  Block c stores r_c into its slot in every block and adds to
//     that block's arrival counter (release); every block waits on its own
//     counter (acquire, bounded) and takes the largest result.
//
// The largest result is the step's winner: every key of block c is at most
// r_c or below a hint, and the block that computed a hint reports a result
// at least as large; so max_c r_c bounds every candidate's key and is itself
// an exact key.  Slots and counters are double-buffered by step parity (a
// block can be at most one step ahead of a peer's exchange).  Errors never
// return early: every block reaches the final hardware cluster barrier,
// after which no block touches another's shared memory.
// ---------------------------------------------------------------------------
constexpr int CL_MAX = 16;  // blocks per cluster (16: the non-portable maximum)

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
__device__ __forceinline__ void st_dsmem_u64(uint32_t a, unsigned long long v) {
  asm volatile("st.shared::cluster.u64 [%0], %1;" ::"r"(a), "l"(v) : "memory");
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
__device__ __forceinline__ void red_dsmem_max_u64(uint32_t a, unsigned long long v) {
  asm volatile("red.relaxed.cluster.shared::cluster.max.u64 [%0], %1;" ::"r"(a), "l"(v)
               : "memory");
}
__device__ __forceinline__ unsigned long long ld_volatile_u64(const unsigned long long* p) {
  return *reinterpret_cast<const volatile unsigned long long*>(p);
}
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
__device__ __forceinline__ void hw_cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}

// Hint format: step in bits 45.., gain bits in 14..44, 16383 - index in
// 0..13 (N <= 16384 and K <= N): a later step's hint is always larger.
__device__ __forceinline__ unsigned long long tag_key(unsigned long long key, int step) {
  const uint32_t t = 0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull);
  return ((unsigned long long)step << 45) | ((key >> 32) << 14) | (16383u - t);
}
__device__ __forceinline__ unsigned long long untag_key(unsigned long long h, int step) {
  if ((int)(h >> 45) != step || h == 0ull) return 0ull;
  const uint32_t t = 16383u - (uint32_t)(h & 0x3FFFull);
  return (((h >> 14) & 0x7FFFFFFFull) << 32) | (0xFFFFFFFFu - t);
}

// Launch arguments of k_sgs_lazy_cl, precomputed on the host and read from
// the parameter space (the kernel runs at 64 registers a thread).
struct LzClArgs {
  const float* cost;   // [B][N][ldc]
  const float* v;      // [B][N]
  const float* g0;     // [B][g0_slots][N] first-gain partial sums from the cost pass, or null
  int g0_slots;
  int32_t* order32;    // [B][K]
  float* gains;        // [B][K] or null
  double* objective;   // [B] or null
  int* status;
  int64_t ldc;
  uint64_t timeout_ns;
  float m0;
  int N, K;
  int C, lgC;          // blocks per cluster, a power of two, and its log2
  int NC;              // candidates per block, ceil(N / C)
  int nwords;          // words of a candidate bitmap, ceil(NC / 32)
  int use_mask;        // block masks kept in shared memory
  int bit_shift;       // log2 of the quarter iterations per mask bit (0 or 1)
  uint32_t off_v, off_ub, off_chosen, off_fresh, off_nzm;  // dynamic smem offsets
};

// Every own unselected candidate's gain at the current m, warp w taking
// own rows w, w + nwarps, ...: the quarter sums of its block mask folded as
// combine_quarters does, so exactly a decision round's value; its mask is
// renewed.  Kept out of line (called once a launch) so that the step loop
// keeps its registers.
__device__ __noinline__ void sweep_rows(const LzClArgs& a, const float* Cb, const float* sm_m,
                                        const float* sm_v, float* ub, const uint32_t* chosen,
                                        uint16_t* nzm, unsigned long long* s_stats, int nown,
                                        uint32_t crank, int w, int nwarps, int lane) {
  const int ncols = (int)a.ldc;
  for (int tl = w; tl < nown; tl += nwarps) {
    if (chosen[tl >> 5] & (1u << (tl & 31))) continue;
    const float* crow = Cb + (size_t)((tl << a.lgC) | (int)crank) * a.ldc;
    float g1 = 0.0f;
    int nr_all = 0;
#pragma unroll 1
    for (int qq = 0; qq < 4; ++qq) {
      uint32_t o;
      int nr;
      const float sq = quarter_gain_masked(crow, sm_m, sm_v, ncols, qq, lane, nzm[4 * tl + qq],
                                           a.bit_shift, o, nr);
      g1 = qq == 0 ? sq : __fadd_rn(g1, sq);
      if (lane == 0) nzm[4 * tl + qq] = (uint16_t)o;
      nr_all += nr;
    }
    if (lane == 0) {
      ub[tl] = g1;
      atomicAdd(&s_stats[0], 1ull);
      atomicAdd(&s_stats[2], 512ull * (unsigned long long)nr_all);
    }
  }
}

// WARPS warps a block (32: one block an SM; 16: two blocks an SM, of
// different clusters, so one block runs while the other waits), in quads
// of 4 warps.
template <int WARPS>
__global__ void __launch_bounds__(32 * WARPS, 1024 / (32 * WARPS))
    k_sgs_lazy_cl(const __grid_constant__ LzClArgs a) {
  constexpr int kThreads = 32 * WARPS, kQuads = WARPS / 4;
  constexpr int kLQ = kQuads == 8 ? 3 : 2;  // log2(kQuads)
  static_assert(kQuads == 8 || kQuads == 4, "4 or 8 quads");
  extern __shared__ __align__(16) unsigned char smem[];
  float* sm_m = reinterpret_cast<float*>(smem);                    // [ldc] coverage cost
  float* sm_v = reinterpret_cast<float*>(smem + a.off_v);          // [ldc] capacity
  float* ub = reinterpret_cast<float*>(smem + a.off_ub);           // [NC] last computed gain
  uint32_t* chosen = reinterpret_cast<uint32_t*>(smem + a.off_chosen);  // [nwords]
  uint32_t* fresh = reinterpret_cast<uint32_t*>(smem + a.off_fresh);    // [nwords]
  uint16_t* nzm = reinterpret_cast<uint16_t*>(smem + a.off_nzm);   // [NC][4] if use_mask
  __shared__ unsigned long long s_wq[WARPS];    // best key of each warp's candidates
  __shared__ unsigned long long s_qkey[kQuads];  // best key of each quad
  __shared__ uint32_t s_qfresh[kQuads];          // ... and whether it is exact
  __shared__ float s_part[kQuads][4];
  __shared__ unsigned long long s_G[3], s_BF[3];   // block's largest key / largest exact
                                                   // key, one slot per round (mod 3)
  __shared__ unsigned long long s_hint;            // tagged; pushed by every block
  __shared__ unsigned long long s_H[3];            // the hint for each decision slot
  __shared__ unsigned long long s_res[2][CL_MAX];  // exchange: results, by step parity
  __shared__ unsigned long long s_resm[2][CL_MAX];  // exchange: their block masks
  __shared__ uint32_t s_cnt[2];                    // exchange arrivals, by step parity
  __shared__ unsigned long long s_W, s_WM;
  __shared__ unsigned long long s_stats[3];        // evaluations, rounds, cost bytes read
  __shared__ int s_ok;                             // 1 ok, 0 stop, 2 inconsistent winner

  const int ncols = (int)a.ldc;
  const int lgC = a.lgC;
  const uint32_t crank = cluster_ctarank();
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k = w >> 2, q = w & 3;
  // own index tl <-> candidate t = (tl << lgC) | crank; quad k scans the own
  // indices k + kQuads * (threadIdx.x & 127) + 128 kQuads i, so warp
  // 4 * (tl & (kQuads - 1)) + ((tl >> (kLQ + 5)) & 3) holds tl
  const int nown = a.N > (int)crank ? (a.N - (int)crank + a.C - 1) >> lgC : 0;
  const float* Cb = a.cost + (size_t)(blockIdx.x >> lgC) * a.N * a.ldc;

  {
    const float* v = a.v + (size_t)(blockIdx.x >> lgC) * a.N;
    for (int j = threadIdx.x; j < ncols; j += kThreads) {
      sm_m[j] = j < a.N ? a.m0 : 0.0f;
      sm_v[j] = j < a.N ? v[j] : 0.0f;
    }
  }
  for (int i = threadIdx.x; i < a.nwords; i += kThreads) {
    chosen[i] = 0u;
    fresh[i] = a.g0 ? 0u : ~0u;  // step 0: exact gains from the sweep below, or bounds
  }
  if (threadIdx.x < 3) {
    s_stats[threadIdx.x] = 0ull;
    s_G[threadIdx.x] = 0ull;
    s_BF[threadIdx.x] = 0ull;
  }
  if (threadIdx.x == 0) {
    s_hint = 0ull;
    s_cnt[0] = s_cnt[1] = 0u;
  }
  hw_cluster_sync();  // every block initialised before any peer writes to it

  if (a.g0) {
    // step 0 from the cost pass's partial row sums: the same terms as
    // the gain (exact products v d, each fused into a rounded sum), summed
    // in another order, so like the gain within gamma_(n-1) =
    // (n-1)u / (1 - (n-1)u) of the exact sum (u = 2^-24, n <= 16384 terms:
    // the two differ by a factor below 1 + 2^-9); scaled by 1 + 2^-8 and
    // rounded up they bound the gain, and are marked stale
    const float* g0 = a.g0 + (size_t)(blockIdx.x >> lgC) * a.g0_slots * a.N;
    for (int tl = threadIdx.x; tl < nown; tl += kThreads) {
      const int t = (tl << lgC) | (int)crank;
      float sum = 0.0f;  // the slots in order; their loads issued together
#pragma unroll 16
      for (int sl = 0; sl < a.g0_slots; ++sl) sum = __fadd_rn(sum, __ldg(g0 + (size_t)sl * a.N + t));
      ub[tl] = __fmaf_ru(fmaxf(sum, 0.0f), 1.00390625f, 1.0e-30f);
      if (a.use_mask)
        for (int qq = 0; qq < 4; ++qq) nzm[4 * tl + qq] = (uint16_t)0xFFFFu;
    }
  }
  // step 0 otherwise: every own candidate's gain exactly, one warp per row
  for (int tl = a.g0 ? nown : w; tl < nown; tl += WARPS) {
    const float* crow = Cb + (size_t)((tl << lgC) | (int)crank) * a.ldc;
    float g0;
    if (a.use_mask) {
      // combine_quarters is the left fold ((s0 + s1) + s2) + s3
      int nr_all = 0;
      g0 = 0.0f;
#pragma unroll 1
      for (int qq = 0; qq < 4; ++qq) {
        uint32_t o;
        int nr;
        const float sq =
            quarter_gain_masked(crow, sm_m, sm_v, ncols, qq, lane, 0xFFFFu, a.bit_shift, o, nr);
        g0 = qq == 0 ? sq : __fadd_rn(g0, sq);
        if (lane == 0) nzm[4 * tl + qq] = (uint16_t)o;
        nr_all += nr;
      }
      if (lane == 0) atomicAdd(&s_stats[2], 512ull * (unsigned long long)nr_all);
    } else {
      g0 = dense_row_gain(crow, sm_m, sm_v, ncols, lane);
      if (lane == 0) atomicAdd(&s_stats[2], 4ull * (unsigned long long)ncols);
    }
    if (lane == 0) {
      ub[tl] = g0;
      atomicAdd(&s_stats[0], 1ull);
    }
  }
  __syncthreads();

  // the best key of this warp's remaining candidates, into s_wq[w]
  auto warp_rescan = [&]() {
    unsigned long long best = 0ull;
    for (int tl = k + kQuads * (threadIdx.x & 127); tl < nown; tl += kQuads * 128)
      if (!(chosen[tl >> 5] & (1u << (tl & 31)))) {
        const unsigned long long key = gain_key(ub[tl], (tl << lgC) | (int)crank);
        best = key > best ? key : best;
      }
    best = warp_max_u64(best);
    if (lane == 0) s_wq[w] = best;
  };
  // quad leader: the quad's best key and whether it is exact
  auto quad_best = [&]() -> unsigned long long {
    unsigned long long kb = s_wq[4 * k];
    for (int i = 1; i < 4; ++i) kb = s_wq[4 * k + i] > kb ? s_wq[4 * k + i] : kb;
    const int bt = (int)(0xFFFFFFFFu - (uint32_t)(kb & 0xFFFFFFFFull)) >> lgC;
    s_qkey[k] = kb;
    s_qfresh[k] = kb != 0ull && ((fresh[bt >> 5] >> (bt & 31)) & 1u);
    return kb;
  };

  bool ok = true;
  int slot = 0;  // decision slot of the next round
  warp_rescan();  // step 0 starts from every warp's best

  for (int step = 0; step < a.K && ok; ++step) {
    if (step == 1 && a.use_mask) {
      // ---- step 1 as one sweep.  The first pick lowers m across the whole
      // scene, so every bound left by step 0 is far above every gain of
      // step 1 and the lazy rounds would evaluate all candidates anyway,
      // one per quad and round.  Here each warp streams through its share
      // of the block's rows instead, with no decision between rows: the
      // same quarter sums in the same fold as a round's evaluation, so the
      // same gains and masks.  Every bound is then exact.
      __syncthreads();  // step 0's update of m and its chosen bit are done
      sweep_rows(a, Cb, sm_m, sm_v, ub, chosen, nzm, s_stats, nown, crank, w, WARPS, lane);
      for (int i = threadIdx.x; i < a.nwords; i += kThreads) fresh[i] = ~0u;
      __syncthreads();
      warp_rescan();
    }
    // ---- step start: the quad bests into the first decision slot (the
    // warp that held the last pick has rescanned; m is updated, and the
    // bounds the pick may have changed are stale)
    quad_sync(k);  // this quad's fresh bits and warp bests of the last step's end are settled
    if (q == 0) {
      unsigned long long kb = 0ull;
      uint32_t fr = 0u;
      if (lane == 0) {
        kb = quad_best();
        fr = s_qfresh[k];
        atomicMax(&s_G[slot], kb);
        if (fr) atomicMax(&s_BF[slot], kb);
      }
      kb = __shfl_sync(0xFFFFFFFFu, kb, 0);
      fr = __shfl_sync(0xFFFFFFFFu, fr, 0);
      if (fr && lane < a.C)  // an exact best from the start: lane r tells block r
        red_dsmem_max_u64(map_rank(smem_addr(&s_hint), (uint32_t)lane), tag_key(kb, step));
    }
    if (threadIdx.x == 0) s_H[slot] = untag_key(ld_volatile_u64(&s_hint), step);
    __syncthreads();

    // ---- phase 1: this block's result.  A round reads its slot, clears
    // the slot two rounds ahead (read two rounds ago) and fills the next;
    // nothing a round reads is written before the block barrier that ends
    // it, so every thread takes the same decisions.
    unsigned long long R = 0ull;
    for (int round = 0; round <= a.NC; ++round) {
      const unsigned long long G = s_G[slot], BF = s_BF[slot], H = s_H[slot];
      const unsigned long long mine = s_qkey[k];
      const uint32_t mine_fresh = s_qfresh[k];
      const int nslot = slot == 2 ? 0 : slot + 1;
      const int cslot = nslot == 2 ? 0 : nslot + 1;
      if (threadIdx.x == 0) {
        s_G[cslot] = 0ull;
        s_BF[cslot] = 0ull;
        ++s_stats[1];
      }
      slot = nslot;
      if (G == 0ull) break;  // no candidate left in this block
      if (G == BF) {         // the block's largest bound is exact
        R = G;
        break;
      }
      if (G < H) {  // nothing here can beat an exact key of another block
        R = BF;
        break;
      }
      const unsigned long long floor_key = BF > H ? BF : H;
      if (!mine_fresh && mine > floor_key) {  // this quad's best might still win
        const int t = (int)(0xFFFFFFFFu - (uint32_t)(mine & 0xFFFFFFFFull));
        const int tl = t >> lgC;
        float part;
        if (a.use_mask) {
          uint32_t o;
          int nr;
          part = quarter_gain_masked(Cb + (size_t)t * a.ldc, sm_m, sm_v, ncols, q, lane,
                                     nzm[4 * tl + q], a.bit_shift, o, nr);
          if (lane == 0) {
            nzm[4 * tl + q] = (uint16_t)o;
            atomicAdd(&s_stats[2], 512ull * (unsigned long long)nr);
          }
        } else {
          part = quarter_gain(Cb + (size_t)t * a.ldc, sm_m, sm_v, ncols, q, lane);
          if (lane == 0) atomicAdd(&s_stats[2], (unsigned long long)ncols);  // a quarter row
        }
        if (lane == 0) s_part[k][q] = part;
        quad_sync(k);
        if (q == 0) {  // the quad's first warp records the gain
          const float g = combine_quarters(s_part[k][0], s_part[k][1], s_part[k][2], s_part[k][3]);
          if (lane == 0) {
            ub[tl] = g;
            atomicOr(&fresh[tl >> 5], 1u << (tl & 31));  // quads may share a word
            atomicAdd(&s_stats[0], 1ull);
          }
          const unsigned long long nk = gain_key(g, t);
          if (nk > floor_key && lane < a.C)  // a new best exact key: lane r tells block r
            red_dsmem_max_u64(map_rank(smem_addr(&s_hint), (uint32_t)lane), tag_key(nk, step));
        }
        quad_sync(k);
        if (w == 4 * k + ((tl >> (kLQ + 5)) & 3)) warp_rescan();  // the warp holding t
        quad_sync(k);
        if (q == 0 && lane == 0) (void)quad_best();
      }
      if (q == 0 && lane == 0) {  // every quad into the next decision
        atomicMax(&s_G[slot], s_qkey[k]);
        if (s_qfresh[k]) atomicMax(&s_BF[slot], s_qkey[k]);
      }
      if (threadIdx.x == 0) s_H[slot] = untag_key(ld_volatile_u64(&s_hint), step);
      __syncthreads();
    }

    // ---- phase 2: exchange the C results with their block masks.  Meanwhile
    // warp 1 of each quad prefetches into L2 the blocks of the quad's best
    // candidate, which the next step's first round will most likely
    // re-evaluate (most bounds go stale with the pick)
    const int par = step & 1;
    if (q == 1 && a.use_mask) {
      const unsigned long long kb = s_qkey[k];
      if (kb != 0ull && kb != R) {
        const int t = (int)(0xFFFFFFFFu - (uint32_t)(kb & 0xFFFFFFFFull));
        const int tl = t >> lgC;
        const int nq = ncols >> 2;
        const float4* row = reinterpret_cast<const float4*>(Cb + (size_t)t * a.ldc);
        for (int bb = lane; bb < 64; bb += 32) {
          if (!((nzm[4 * tl + (bb >> 4)] >> (bb & 15)) & 1u)) continue;
          const int u0 = (bb & 15) << a.bit_shift, u1 = ((bb & 15) + 1) << a.bit_shift;
          for (int u = u0; u < u1; ++u) {
            const int i0 = 128 * u + 32 * (bb >> 4);  // iteration 4u + quarter
            if (i0 < nq) prefetch_l2(row + i0, (uint32_t)(16 * min(32, nq - i0)));
          }
        }
      }
    }
    if (w == 0) {
      if (lane < a.C) {
        unsigned long long RM = R == 0ull ? 0ull : ~0ull;
        if (R != 0ull && a.use_mask) {
          const int tl = (int)(0xFFFFFFFFu - (uint32_t)(R & 0xFFFFFFFFull)) >> lgC;
          RM = (unsigned long long)nzm[4 * tl] | ((unsigned long long)nzm[4 * tl + 1] << 16) |
               ((unsigned long long)nzm[4 * tl + 2] << 32) |
               ((unsigned long long)nzm[4 * tl + 3] << 48);
        }
        st_dsmem_u64(map_rank(smem_addr(&s_res[par][crank]), lane), R);
        st_dsmem_u64(map_rank(smem_addr(&s_resm[par][crank]), lane), RM);
        red_release_dsmem_add(map_rank(smem_addr(&s_cnt[par]), lane), 1u);
      }
      if (lane == 0) {
        int good = 1;
        const uint32_t own_cnt = map_rank(smem_addr(&s_cnt[par]), crank);
        const uint32_t target = (uint32_t)a.C * (uint32_t)((step >> 1) + 1);
        uint64_t t0 = 0;  // read the clock only once the wait is not short
        uint32_t spins = 0;
        while (ld_acquire_dsmem_u32(own_cnt) < target) {
          if ((++spins & 63u) == 0) {
            if (ld_volatile_i32(a.status) != 0) { good = 0; break; }
            if (t0 == 0) {
              t0 = globaltimer_ns();
            } else if (globaltimer_ns() - t0 > a.timeout_ns) {
              set_status(a.status, CP_ETIMEOUT);
              good = 0;
              break;
            }
          }
        }
        unsigned long long W = 0ull, WM = 0ull;
        if (good) {
          for (int r = 0; r < a.C; ++r) {
            const unsigned long long x = ld_volatile_u64(&s_res[par][r]);
            if (x > W) {
              W = x;
              WM = ld_volatile_u64(&s_resm[par][r]);
            }
          }
          // the winner must be a valid candidate that this block, if it owns
          // it, has not picked before (never expected otherwise)
          const int pick = W == 0ull ? -1 : (int)(0xFFFFFFFFu - (uint32_t)(W & 0xFFFFFFFFull));
          const int ptl = pick >> lgC;
          if (pick < 0 || pick >= a.N ||
              ((pick & (a.C - 1)) == (int)crank && (chosen[ptl >> 5] & (1u << (ptl & 31))))) {
            good = 2;
            if (atomicCAS(a.status, 0, CP_EDEVICE) == 0) {
              a.status[4] = step;
              a.status[5] = (int)(blockIdx.x >> lgC);
              a.status[6] = (int)crank;
              a.status[7] = pick;
            }
          }
        }
        s_W = W;
        s_WM = WM;
        s_ok = good;
      }
    }
    __syncthreads();
    if (s_ok != 1) {
      ok = false;
      break;
    }
    const unsigned long long W = s_W, WM = s_WM;
    const int pick = (int)(0xFFFFFFFFu - (uint32_t)(W & 0xFFFFFFFFull));
    const int ptl = pick >> lgC;
    const bool own = (pick & (a.C - 1)) == (int)crank;
    if (threadIdx.x == 0 && crank == 0) {
      const size_t o = (size_t)(blockIdx.x >> lgC) * a.K + step;
      s_stats[2] += (unsigned long long)__popcll(WM) * (512ull << a.bit_shift);  // update reads
      a.order32[o] = pick;
      if (a.gains) a.gains[o] = __uint_as_float((uint32_t)(W >> 32));
    }
    // S <- S u {t*} (Eq. sgs_update), on this block's copy of m.  Only the
    // row blocks of the winner's mask can lower m: the winner was evaluated
    // at the current m, and a block outside its mask has m <= C throughout.
    // Pad columns hold C = 0 and m = 0, so whole float4 chunks are safe.
    {
      const float4* row = reinterpret_cast<const float4*>(Cb + (size_t)pick * a.ldc);
      float4* m4 = reinterpret_cast<float4*>(sm_m);
      const int nq = ncols >> 2;
      for (int bb = w; bb < 64; bb += WARPS) {
        if (!((WM >> bb) & 1ull)) continue;
        const int u0 = (bb & 15) << a.bit_shift, u1 = ((bb & 15) + 1) << a.bit_shift;
        for (int u = u0; u < u1; ++u) {
          const int i = 128 * u + 32 * (bb >> 4) + lane;  // iteration 4u + quarter
          if (i < nq) {
            const float4 c = __ldg(row + i);
            float4 mm = m4[i];
            mm.x = fminf(mm.x, c.x);
            mm.y = fminf(mm.y, c.y);
            mm.z = fminf(mm.z, c.z);
            mm.w = fminf(mm.w, c.w);
            m4[i] = mm;
          }
        }
      }
    }
    // A bound stays exact when its candidate had no positive term in any
    // row block the pick lowers m on (the winner's mask WM): its terms, and
    // so their rounded sum, are unchanged.  Its mask stays exact too (m is
    // unchanged inside it).  Every other bound goes stale (all of them
    // without masks); the warp that held the pick drops it.
    // Each quad clears the bits of its own candidates (the ones its warps
    // rescan), so a quad barrier orders them before the quad's next read.
    if (a.use_mask) {
      for (int tl = k + kQuads * (threadIdx.x & 127); tl < nown; tl += kQuads * 128) {
        const uint32_t bit = 1u << (tl & 31);
        if (fresh[tl >> 5] & bit) {  // only this thread changes this bit
          const unsigned long long mk =
              (unsigned long long)nzm[4 * tl] | ((unsigned long long)nzm[4 * tl + 1] << 16) |
              ((unsigned long long)nzm[4 * tl + 2] << 32) |
              ((unsigned long long)nzm[4 * tl + 3] << 48);
          if (mk & WM) atomicAnd(&fresh[tl >> 5], ~bit);
        }
      }
    } else {
      for (int tl = k + kQuads * (threadIdx.x & 127); tl < nown; tl += kQuads * 128)
        atomicAnd(&fresh[tl >> 5], ~(1u << (tl & 31)));
    }
    if (own && w == 4 * (ptl & (kQuads - 1)) + ((ptl >> (kLQ + 5)) & 3)) {
      if (lane == 0) chosen[ptl >> 5] |= 1u << (ptl & 31);
      __syncwarp();
      warp_rescan();
    }
  }

  unsigned long long* cstats = reinterpret_cast<unsigned long long*>(
      reinterpret_cast<unsigned char*>(a.status) + kCallStatsOffset);
  __syncthreads();
  if (threadIdx.x == 0) {
    atomicAdd(&cstats[0], s_stats[0]);
    if (crank == 0) atomicAdd(&cstats[1], s_stats[1]);
    atomicAdd(&cstats[2], s_stats[2]);
  }
  if (ok && crank == 0 && a.objective) {
    const double F = objective_sum(sm_m, sm_v, a.N);
    if (threadIdx.x == 0) a.objective[blockIdx.x >> lgC] = F;
  }
  hw_cluster_sync();  // nobody leaves while a peer may still write to its shared memory
}

// Blocks per scene for the cluster kernel: the largest power of two <= 16
// such that every scene's cluster can be resident at once (16 only where
// the device runs that many clusters of 16 at a time; checked at launch).
static int cluster_size_for(int64_t B, int sm_count) {
  int C = CL_MAX;
  while (C > 1 && (int64_t)C * B > sm_count) C >>= 1;
  return C;
}

// One launch of the lazy kernel with WARPS warps a block on clusters of C
// blocks.  Returns 1 (nothing launched) when that shape cannot be resident
// -- every scene's cluster at once when all_resident -- else a status.
template <int WARPS>
static int lazy_launch_shape(LzClArgs a, int C, bool all_resident, int64_t B, int64_t N,
                             int64_t ldc, const DeviceInfo& di, cudaStream_t s) {
  auto fn = k_sgs_lazy_cl<WARPS>;
  a.C = C;
  a.lgC = C >= 16 ? 4 : C >= 8 ? 3 : C >= 4 ? 2 : C >= 2 ? 1 : 0;
  a.NC = (int)((N + C - 1) / C);
  a.nwords = (a.NC + 31) / 32;
  const int nit_max = (int)(((ldc / 4 + 31) / 32 + 3) / 4);  // iterations per quarter
  a.bit_shift = nit_max <= 16 ? 0 : 1;
  a.off_v = (uint32_t)(sizeof(float) * ldc);
  a.off_ub = (uint32_t)(sizeof(float) * 2 * ldc);
  a.off_chosen = a.off_ub + (uint32_t)(sizeof(float) * a.NC);
  a.off_fresh = a.off_chosen + (uint32_t)(sizeof(uint32_t) * a.nwords);
  a.off_nzm = a.off_fresh + (uint32_t)(sizeof(uint32_t) * a.nwords);
  const size_t smem_plain = a.off_nzm;
  const size_t smem_mask = smem_plain + 4 * sizeof(uint16_t) * (size_t)a.NC;
  // the block masks live in shared memory when they fit beside (m, v)
  a.use_mask = smem_mask + 2048 <= (size_t)di.max_smem_optin ? 1 : 0;
  const size_t smem = a.use_mask ? smem_mask : smem_plain;
  if (cuda_status(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem),
                  "launch_sgs_lazy_cluster: smem attribute") != CP_OK)
    return CP_ECUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(B * C));
  cfg.blockDim = dim3(32 * WARPS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (C > 8 && cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
                   cudaSuccess) {
    (void)cudaGetLastError();
    return 1;
  }
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, (const void*)fn, &cfg) != cudaSuccess ||
      clusters < 1 || (all_resident && clusters < B)) {
    (void)cudaGetLastError();
    return 1;  // this cluster shape cannot be resident
  }
  cudaError_t e = cudaLaunchKernelEx(&cfg, fn, a);
  note_launch();
  return cuda_status(e, "launch_sgs_lazy_cluster");
}

// The cluster shape: C blocks of 32 warps, C the largest power of two <= 16
// with every scene resident at once; where that C is below 16, clusters of
// 2C blocks of 16 warps instead, two blocks an SM (from different
// clusters), when every scene's cluster can be resident.
static int sgs_lazy_cluster_launch(const float* cost, int64_t ldc, const float* v,
                                   const DevParams& P, int64_t B, int64_t N, int64_t K,
                                   int32_t* order32, float* gains, double* objective, int* status,
                                   cudaStream_t s, const float* g0) {
  DeviceInfo di;
  if (device_info(&di) != CP_OK) return CP_ECUDA;
  LzClArgs a{};
  a.cost = cost;
  a.v = v;
  a.g0 = g0;
  a.g0_slots = fst_apply_slots(ldc);  // per column tile of the elementwise cost pass
  a.order32 = order32;
  a.gains = gains;
  a.objective = objective;
  a.status = status;
  a.ldc = ldc;
  a.timeout_ns = P.timeout_ns;
  a.m0 = P.m0;
  a.N = (int)N;
  a.K = (int)K;
  const int C32 = cluster_size_for(B, di.sm_count);
  if (C32 < CL_MAX) {
    const int st = lazy_launch_shape<16>(a, 2 * C32, true, B, N, ldc, di, s);
    if (st != 1) return st;
  }
  for (int C = C32; C >= 1; C >>= 1) {
    const int st = lazy_launch_shape<32>(a, C, C > 8, B, N, ldc, di, s);
    if (st != 1) return st;
  }
  note_message("launch_sgs_lazy_cluster: no resident cluster shape");
  return CP_EUNSUPPORTED;
}

static int sgs_local_launch(const float* slab, const int32_t* nbr, const float* v,
                            const DevParams& P, int64_t B, int64_t N, int64_t K, int32_t* order32,
                            float* gains, double* objective, int* status, int32_t* rev_off,
                            int32_t* rev, cudaStream_t s) {
  const size_t rsmem = sizeof(int) * (size_t)N;
  if (rsmem > 48 * 1024 &&
      cuda_status(cudaFuncSetAttribute(k_rev_build, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)rsmem),
                  "launch_sgs_local: reverse-list smem attribute") != CP_OK)
    return CP_ECUDA;
  k_rev_build<<<(unsigned)B, 1024, rsmem, s>>>(nbr, (int)N, P.g, P.kk, rev_off, rev);
  CP_TRY_STATUS(last_launch_status());
  const size_t smem = sizeof(float) * 3 * (size_t)N + 2 * sizeof(uint32_t) * (size_t)((N + 31) / 32);
  if (smem > 48 * 1024 &&
      cuda_status(cudaFuncSetAttribute(k_sgs_local, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem),
                  "launch_sgs_local: smem attribute") != CP_OK)
    return CP_ECUDA;
  k_sgs_local<<<(unsigned)B, LZ_THREADS, smem, s>>>(slab, nbr, v, rev_off, rev, P, (int)N, (int)K,
                                                    order32, gains, objective, status);
  return last_launch_status();
}

int launch_sgs(const float* cost, int64_t ldc, const float* slab, const int32_t* nbr,
               const float* v, const DevParams& P, int64_t B, int64_t N, int64_t K,
               int32_t* order32, float* gains, double* objective, uint64_t* partials,
               uint32_t* counters, int* status, cudaStream_t s, const float* g0,
               int32_t* rev_off, int32_t* rev) {
  auto* part = reinterpret_cast<unsigned long long*>(partials);
  if (P.sgs_mode == 0) {
    if (P.g < N)
      return sgs_local_launch(slab, nbr, v, P, B, N, K, order32, gains, objective, status,
                              rev_off, rev, s);
    return sgs_lazy_cluster_launch(cost, ldc, v, P, B, N, K, order32, gains, objective, status, s,
                                   g0);
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
