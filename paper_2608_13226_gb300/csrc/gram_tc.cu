// K2/K3 for bf16 features on the 5th-generation tensor cores (tcgen05 + TMEM).
//
// The feature Gram G = F F^T of one scene is the method's only dense
// contraction (the cosine of Eq. fst_metrics).  k_gram_tc computes it for
// the pairs i <= j only (the tiles on or above the diagonal) and keeps the
// max and min cosine (the feature normaliser of Sec. 3.3); with an output
// buffer it also stores every cosine of a pair i <= j at [i][j] (the upper
// triangle).  The FST cost of Eq. fst_cost needs the normalisers of the
// whole scene, so it follows as one pass over the stored cosines
// (k_fst_pair, HBM-bound: each cosine read once, C(i, j) and C(j, i)
// written), which also sums the greedy's first gains.
//
// Persistent CTA pairs (clusters of two CTAs, one CTA per SM) issuing the
// pair MMA tcgen05.mma.cta_group::2 (M = 256, N = 256, K = 16): a unit is
// the 256 x 256 tile of row tiles 2p, 2p+1 and one 256-column tile.  Each
// CTA loads only its own operands into its own shared memory: its 128 rows
// of A (row tile 2p + rank) and its 128-row half of B, so a CTA fetches
// 32 KB from L2 per 64-deep step instead of the 48 KB a single-CTA M = 128,
// N = 256 tile needs; the pair instruction reads both CTAs' halves.  Row
// tile 2p + rank's accumulator lands in that CTA's own TMEM.  Each CTA has
// 10 warps:
//   warp 0      TMA producer: 128x64 bf16 boxes, 128-byte swizzle, into a
//               6-stage shared-memory ring (32 KB a stage); both CTAs'
//               copies signal the leader CTA's (rank 0) "full" barrier
//               (.cta_group::2 form), which expects both CTAs' bytes
//   warp 1      allocates 512 TMEM columns (both CTAs, collectively); in the
//               leader lane 0 issues the pair MMA into one of two 128x256
//               fp32 accumulators per CTA (double buffer) and commits to
//               the barriers of both CTAs
//   warps 2..9  epilogue: warps w and w+4 share TMEM lane quadrant w%4 and
//               split the 256 columns; tcgen05.ld 32 lanes x 32 columns at a
//               time, cosines and their min/max in registers; the 32
//               columns' inverse norms are staged per warp in shared memory.
//               Chunks above the diagonal leave through a per-warp 32 x 32
//               shared-memory transpose (the same 4 KB), so that each store
//               instruction writes 4 rows x 128 contiguous bytes: whole L2
//               lines, which L2 takes without reading DRAM first; chunks
//               crossing the diagonal store their pairs j >= i element by
//               element, chunks below it store nothing.  One lane a warp
//               tells the leader that its accumulator is drained.
// Stage hand-offs use mbarriers (a stage's "empty" barrier in each CTA gets
// the leader's MMA commit); the accumulator hand-off uses tcgen05.commit ->
// mbarrier and back.  Every wait is bounded by the call's time limit: on
// expiry the kernel records CP_ETIMEOUT, stops issuing work, waits (bounded)
// for the copies and MMAs it already issued, frees its TMEM and returns.
#include <cuda.h>

#include "common.cuh"

namespace cp {
namespace {

constexpr int TC_BM = 128, TC_BN = 256, TC_BK = 64, TC_STAGES = 6;
constexpr int TC_EPI_WARPS = 8;                     // two per TMEM lane quadrant
constexpr int TC_THREADS = 64 + 32 * TC_EPI_WARPS;  // producer, MMA, epilogue
constexpr uint32_t TC_A_BYTES = TC_BM * TC_BK * 2;  // 16 KB: this CTA's 128 rows of A
constexpr uint32_t TC_BH_BYTES = (TC_BN / 2) * TC_BK * 2;  // 16 KB: this CTA's half of B
constexpr uint32_t TC_STAGE_BYTES = TC_A_BYTES + TC_BH_BYTES;
constexpr uint32_t TC_PAIR_STAGE_BYTES = 2 * TC_STAGE_BYTES;  // what the leader's barrier expects
constexpr uint32_t TC_TMEM_COLS = 512;              // 2 accumulators x 256 fp32 columns
constexpr uint32_t TC_STG_FLOATS = 32 * 32;         // epilogue staging per warp (4 KB)
constexpr uint32_t TC_EMPTY_ARRIVALS = 2 * TC_EPI_WARPS;  // one lane per epilogue warp, both CTAs
constexpr size_t TC_SMEM = (size_t)TC_STAGES * TC_STAGE_BYTES +
                           (size_t)TC_EPI_WARPS * TC_STG_FLOATS * sizeof(float) +
                           1024;  // + alignment slack

// Instruction descriptor of tcgen05.mma kind::f16: D fp32, A and B bf16,
// both K-major, M = 256 (the CTA pair: 128 rows in each), N = 256.
constexpr uint32_t kIdesc = (1u << 4)              // D format: f32
                            | (1u << 7)            // A format: bf16
                            | (1u << 10)           // B format: bf16
                            | ((uint32_t)(TC_BN >> 3) << 17)        // N >> 3
                            | ((uint32_t)((2 * TC_BM) >> 4) << 24);  // M >> 4

struct TcArgs {
  const float4* tok;      // [B*N] (x, y, z, 1/||f||)
  float* cos_out;         // [B][N][ldc] every cosine, or null
  int64_t ldc;
  int vec_ok;             // cos_out rows take 16-byte stores (ldc % 4 == 0, 16-byte base)
  SceneStats* stats;
  int* status;
  int N, B, TI, TJ, num_kb;
  int pairs_per_scene, total_pairs;  // (row-tile pair, column tile) units
  uint64_t timeout_ns;
  // tile-list mode (local SGS with the bounded normaliser): units[u] =
  // (b << 16) | (P << 8) | J for u < *n_units, whole tiles stored, no min/max
  const uint32_t* units;
  const int* n_units;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

// ---- mbarrier ---------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return done != 0;
}
// Waits for the phase of parity `parity` to complete.  Gives up when the
// block has aborted or this wait exceeds timeout_ns (then aborts the block).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          uint64_t timeout_ns, int* status) {
  if (mbar_test(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  uint32_t spins = 0;
  while (!mbar_test(bar, parity)) {
    if ((++spins & 15u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer_ns() - t0 > timeout_ns) {
        set_status(status, CP_ETIMEOUT);
        *abort_flag = 1;
        return false;
      }
    }
  }
  return true;
}

// ---- TMA ---------------------------------------------------------------------
// L2 policies: the feature operands are re-read by every tile of a scene and
// should stay in L2 (evict last); each cost line is written once (evict
// first), so the output stream does not push the features out.
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// Cluster address of the same shared-memory object in the pair's CTA `rank`.
__device__ __forceinline__ uint32_t cluster_addr(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(p)), "r"(rank));
  return r;
}
// A box into this CTA's shared memory at dst; the bytes are counted on the
// mbarrier at cluster address bar_cl, which may lie in the peer CTA of the
// pair (the .cta_group::2 form).
__device__ __forceinline__ void tma_load_3d_pair(const CUtensorMap* map, uint32_t bar_cl,
                                                 uint32_t dst, int x, int y, int z,
                                                 uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".cta_group::2.L2::cache_hint [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar_cl), "l"(policy)
      : "memory");
}
// Arrive (release at cluster scope) on the mbarrier at cluster address bar_cl.
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar_cl) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cl)
               : "memory");
}
__device__ __forceinline__ void st_f4_policy(float* p, const float4& v, uint64_t policy) {
  asm volatile("st.global.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "f"(v.x),
               "f"(v.y), "f"(v.z), "f"(v.w), "l"(policy)
               : "memory");
}
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ---- tcgen05 -------------------------------------------------------------------
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row
// groups 1024 bytes apart (the layout a 128-byte-wide TMA box with
// SWIZZLE_128B writes).  Leading-byte offset unused for this layout.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4)       // start address >> 4
         | ((uint64_t)1 << 16)                     // leading byte offset (unused) = 16 B
         | ((uint64_t)(1024 >> 4) << 32)           // stride byte offset = 1024 B
         | ((uint64_t)1 << 46)                     // descriptor version (fixed 0b001)
         | ((uint64_t)2 << 61);                    // swizzle mode: 128 B
}
// The pair MMA: D[256 x 256] (+)= A B^T, A's rows 0..127 from the leader's
// shared memory and 128..255 from the peer's, B's columns 0..127 from the
// leader's and 128..255 from the peer's (both at the same offsets); each
// CTA's TMEM at tmem_d receives its own 128 rows.  Issued by one thread of
// the leader CTA.
__device__ __forceinline__ void umma_bf16_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                               uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
      : "memory");
}
// Arrive on the mbarrier at bar's offset in both CTAs of the pair once the
// pair MMAs issued so far have completed (an mbarrier signal, not a copy).
__device__ __forceinline__ void umma_commit_pair(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"((uint16_t)0x3)
      : "memory");
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Warp-reduce a scene's running max / min cosine and merge it into stats.
__device__ __forceinline__ void flush_minmax(SceneStats* st, float cmax, float cmin) {
  for (int o = 16; o > 0; o >>= 1) {
    cmax = fmaxf(cmax, __shfl_xor_sync(0xFFFFFFFFu, cmax, o));
    cmin = fminf(cmin, __shfl_xor_sync(0xFFFFFFFFu, cmin, o));
  }
  if ((threadIdx.x & 31) == 0 && cmax >= cmin) {
    atomicMax(&st->cos_max_key, f2key(cmax));
    atomicMin(&st->cos_min_key, f2key(cmin));
  }
}

// Unit p of the schedule -> (scene b, row tile I, column tile J): a unit is
// a pair of row tiles (2P, 2P+1) and the cluster's CTA of rank c computes
// I = 2P + c.  Only the tiles holding a pair i <= j are visited (row tile
// I needs J >= I/2, so a pair needs J >= P).  A scene's units go in bands
// of TC_BAND row-tile pairs, each band column by column (J ascending, then
// P ascending), so the units in flight at once share a few A and B tiles
// in L2 instead of sweeping every column tile of the scene.
constexpr int TC_BAND = 8;
__device__ __forceinline__ void unit_coords(const TcArgs& a, int p, int cr, int& b, int& I,
                                            int& J) {
  if (a.units) {
    const uint32_t u = __ldg(a.units + p);
    b = (int)(u >> 16);
    I = 2 * (int)((u >> 8) & 0xFFu) + cr;
    J = (int)(u & 0xFFu);
    return;
  }
  b = p / a.pairs_per_scene;
  int r = p - b * a.pairs_per_scene;
  const int TP = (a.TI + 1) >> 1;  // == TJ
  int P0 = 0, P1 = min(TC_BAND, TP) - 1;
  for (;;) {  // the band holding unit r: columns J >= P0, min(J, P1) - P0 + 1 units each
    const int hg = P1 - P0 + 1;
    const int cnt = hg * (hg + 1) / 2 + (a.TJ - 1 - P1) * hg;
    if (r < cnt || P1 >= TP - 1) break;
    r -= cnt;
    P0 += TC_BAND;
    P1 = min(P0 + TC_BAND, TP) - 1;
  }
  int Jc = P0;
  for (;;) {
    const int h = min(Jc, P1) - P0 + 1;
    if (r < h || Jc >= a.TJ - 1) break;
    r -= h;
    ++Jc;
  }
  J = Jc;
  I = 2 * (P0 + r) + cr;  // past the last row tile (odd TI): rows read as 0
}

__global__ void __launch_bounds__(TC_THREADS, 1)
    k_gram_tc(const __grid_constant__ CUtensorMap mapA, const TcArgs a) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[TC_STAGES], empty_bar[TC_STAGES];
  __shared__ __align__(8) uint64_t tfull_bar[2], tempty_bar[2];
  __shared__ uint32_t s_tmem_base;
  __shared__ volatile int s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t smem_base = (smem_u32(smem_raw) + 1023u) & ~1023u;  // 1024-B aligned ring
  const int cr = (int)cluster_rank();  // 0: the leader (issues the MMAs); 1: its peer
  const int cid = (int)(blockIdx.x >> 1), ncl = (int)(gridDim.x >> 1);

  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int s = 0; s < TC_STAGES; ++s) {
      mbar_init(&full_bar[s], 1);   // leader only: its producer's arrive + both CTAs' bytes
      mbar_init(&empty_bar[s], 1);  // the leader's MMA commit
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull_bar[i], 1);                   // the leader's MMA commit
      mbar_init(&tempty_bar[i], TC_EMPTY_ARRIVALS);  // leader only: every epilogue warp
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    tma_prefetch_desc(&mapA);
  }
  if (warp == 1) {  // one warp of each CTA, collectively for the pair
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&s_tmem_base)),
                 "r"(TC_TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  cluster_sync_all();  // both CTAs' barriers exist before either signals the other
  const uint32_t tmem_base = s_tmem_base;
  const int total = a.units ? *a.n_units : a.total_pairs;  // units of the whole grid

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t keep = l2_policy_evict_last();
      int stage = 0;
      uint32_t phase = 0;
      uint32_t pending = 0;        // (leader) stages holding a load not yet seen consumed
      uint32_t pend_parity = 0;    // parity of that load's full phase, per stage bit
      for (int p = cid; p < total && !s_abort; p += ncl) {
        int b, I, J;
        unit_coords(a, p, cr, b, I, J);
        for (int kb = 0; kb < a.num_kb; ++kb) {
          if (!mbar_wait(&empty_bar[stage], phase ^ 1u, &s_abort, a.timeout_ns, a.status)) break;
          pending &= ~(1u << stage);
          const uint32_t sa = smem_base + (uint32_t)stage * TC_STAGE_BYTES;
          const uint32_t fb = cluster_addr(&full_bar[stage], 0);  // the leader's barrier
          if (cr == 0) mbar_arrive_expect_tx(&full_bar[stage], TC_PAIR_STAGE_BYTES);
          // this CTA's 128 rows of A, and its 128-row half of the 256-row B tile
          tma_load_3d_pair(&mapA, fb, sa, kb * TC_BK, I * TC_BM, b, keep);
          tma_load_3d_pair(&mapA, fb, sa + TC_A_BYTES, kb * TC_BK, J * TC_BN + cr * TC_BM, b,
                           keep);
          pending |= 1u << stage;
          pend_parity = (pend_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == TC_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (s_abort) {
        // let the copies already issued land before the block exits: the
        // leader sees them on its own barrier (a phase completes once both
        // CTAs' bytes are in); the peer's copies signal the leader, so the
        // peer waits a fixed bounded time instead
        const uint64_t drain = globaltimer_ns() + (cr == 0 ? 50000000ull : 2000000ull);
        if (cr == 0) {
          for (int s = 0; s < TC_STAGES; ++s)
            if (pending & (1u << s))
              while (!mbar_test(&full_bar[s], (pend_parity >> s) & 1u) &&
                     globaltimer_ns() < drain) {
              }
        } else if (pending) {
          while (globaltimer_ns() < drain) {
          }
        }
      } else {
        // every stage released by the leader's MMAs: its last commits to
        // this CTA's barriers have landed before the final cluster barrier
        for (int i = 0; i < TC_STAGES; ++i) {
          if (!mbar_wait(&empty_bar[stage], phase ^ 1u, &s_abort, a.timeout_ns, a.status)) break;
          if (++stage == TC_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (leader)
    if (lane == 0 && cr == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      uint64_t* last_commit = nullptr;
      uint32_t last_parity = 0;
      for (int p = cid; p < total && !s_abort; p += ncl) {
        if (!mbar_wait(&tempty_bar[acc], acc_phase ^ 1u, &s_abort, a.timeout_ns, a.status)) break;
        tc_fence_after();
        const uint32_t tmem_d = tmem_base + (uint32_t)(acc * TC_BN);
        bool ok = true;
        for (int kb = 0; kb < a.num_kb; ++kb) {
          if (!mbar_wait(&full_bar[stage], phase, &s_abort, a.timeout_ns, a.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_base + (uint32_t)stage * TC_STAGE_BYTES;
          const uint64_t adesc = sw128_desc(sa), bdesc = sw128_desc(sa + TC_A_BYTES);
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k)  // 32 bytes further along K per step
            umma_bf16_pair(tmem_d, adesc + (uint64_t)(2 * k), bdesc + (uint64_t)(2 * k),
                           (kb > 0 || k > 0) ? 1u : 0u);
          umma_commit_pair(&empty_bar[stage]);  // frees the stage in both CTAs
          last_commit = &empty_bar[stage];
          last_parity = phase;
          if (++stage == TC_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit_pair(&tfull_bar[acc]);  // both CTAs' accumulators ready for their epilogues
        last_commit = &tfull_bar[acc];
        last_parity = acc_phase;
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
      if (s_abort && last_commit) {
        // the MMAs already issued must finish before TMEM is freed
        const uint64_t drain = globaltimer_ns() + 50000000ull;
        while (!mbar_test(last_commit, last_parity) && globaltimer_ns() < drain) {
        }
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;                        // TMEM lane quadrant of this warp
    const int half = (warp - 2) / 4;               // which 128 of the 256 columns
    const int ew = warp - 2;                       // epilogue warp index (staging slot)
    const int r = q * 32 + lane;                   // row of the tile
    float* stg = reinterpret_cast<float*>(smem_raw + (smem_base - smem_u32(smem_raw)) +
                                          TC_STAGES * TC_STAGE_BYTES) +
                 ew * TC_STG_FLOATS;               // this warp's 32 x 32 staging tile
    float* s_rn = stg;  // the chunk columns' 1/||f||
    const uint64_t stream_out = l2_policy_evict_first();
    const uint32_t tempty_cl0 = cluster_addr(&tempty_bar[0], 0);  // the leader's barriers
    const uint32_t tempty_cl1 = cluster_addr(&tempty_bar[1], 0);
    int acc = 0;
    uint32_t acc_phase = 0;
    float cmax = -INFINITY, cmin = INFINITY;
    int cur_b = -1;
    for (int p = cid; p < total; p += ncl) {
      // lane 0 waits, the warp follows it (keeps the warp converged for the
      // .sync.aligned TMEM loads below)
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&tfull_bar[acc], acc_phase, &s_abort, a.timeout_ns, a.status);
      ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      int b, I, J;
      unit_coords(a, p, cr, b, I, J);
      if (b != cur_b) {
        if (cur_b >= 0 && !a.units) flush_minmax(a.stats + cur_b, cmax, cmin);
        cur_b = b;
        cmax = -INFINITY;
        cmin = INFINITY;
      }
      const int gi = I * TC_BM + r;
      const bool row_ok = gi < a.N;
      const size_t sb = (size_t)b * a.N;
      const float rni = row_ok ? __ldg(a.tok + sb + gi).w : 0.0f;
      const int r0 = I * TC_BM + q * 32;  // first row of this warp
      const uint32_t row_taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * TC_BN);
#pragma unroll 1
      for (int c = half * 4; c < half * 4 + 4; ++c) {
        const int j0 = J * TC_BN + c * 32;
        // stage the 32 columns' inverse norms (one column per lane, coalesced)
        {
          const int jl = j0 + lane;
          const float rnj = jl < a.N ? __ldg(a.tok + sb + jl).w : 0.0f;
          __syncwarp();  // the previous chunk's staging reads are done
          s_rn[lane] = rnj;
          __syncwarp();
        }
        uint32_t v[32];
        tmem_ld32(row_taddr + (uint32_t)(c * 32), v);
        if (row_ok) {
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const int j = j0 + e;
            float cv = 0.0f;  // pad columns N <= j < ldc hold 0
            if (j < a.N) {
              cv = clamp_cos(__uint_as_float(v[e]) * rni * s_rn[e]);
              if (j == gi && rni > 0.0f) cv = 1.0f;  // cos(f, f) = 1 exactly
              cmax = fmaxf(cmax, cv);
              cmin = fminf(cmin, cv);
            }
            v[e] = __float_as_uint(cv);
          }
        }
        if (a.cos_out == nullptr) continue;
        // only the upper triangle (j >= i) is stored: a chunk wholly above
        // the diagonal leaves through the transpose below, one crossing it
        // row by row; chunks below it store nothing
        const int where = a.units ? 1 : (j0 >= r0 + 31 ? 1 : (j0 + 31 < r0 ? -1 : 0));
        if (where == 0 && row_ok) {
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const int j = j0 + e;
            if (j >= gi && j < a.ldc)
              a.cos_out[(sb + (size_t)gi) * (size_t)a.ldc + j] = __uint_as_float(v[e]);
          }
        }
        if (where == 1) {
          // lane l writes row l's eight float4 chunks (chunk c at c ^ (l & 7),
          // so a phase of 8 lanes hits 8 distinct bank groups); store i (of
          // 8) then moves rows 4i + l/8, chunk l % 8: 4 rows x 128 bytes
          __syncwarp();  // every lane is done with the staged norms
#pragma unroll
          for (int c = 0; c < 8; ++c)
            *reinterpret_cast<float4*>(stg + lane * 32 + 4 * (c ^ (lane & 7))) =
                make_float4(__uint_as_float(v[4 * c]), __uint_as_float(v[4 * c + 1]),
                            __uint_as_float(v[4 * c + 2]), __uint_as_float(v[4 * c + 3]));
          __syncwarp();
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int rr = 4 * i + (lane >> 3), c = lane & 7;  // rr < 32
            const float4 val = *reinterpret_cast<const float4*>(stg + rr * 32 + 4 * (c ^ (rr & 7)));
            const int grow = r0 + rr;
            const int col = j0 + 4 * c;
            if (grow < a.N && col < a.ldc) {
              float* dst = a.cos_out + (sb + (size_t)grow) * (size_t)a.ldc + col;
              if (a.vec_ok) {  // col % 4 == 0 and ldc % 4 == 0: the chunk fits
                st_f4_policy(dst, val, stream_out);
              } else {
                dst[0] = val.x;
                if (col + 1 < a.ldc) dst[1] = val.y;
                if (col + 2 < a.ldc) dst[2] = val.z;
                if (col + 3 < a.ldc) dst[3] = val.w;
              }
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();  // every lane's TMEM loads of this accumulator are done
      if (lane == 0) mbar_arrive_cluster(acc ? tempty_cl1 : tempty_cl0);  // free for the leader's MMAs
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
    if (cur_b >= 0 && !a.units) flush_minmax(a.stats + cur_b, cmax, cmin);
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // the leader's MMAs and both CTAs' TMEM reads are over
  if (warp == 1) {     // one warp of each CTA, collectively for the pair
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(TC_TMEM_COLS)
                 : "memory");
  }
  cluster_sync_all();  // neither CTA leaves while the other may still signal it
}

}  // namespace
}  // namespace cp

#include <limits.h>

#include <mutex>

namespace cp {
namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static std::once_flag once;
  static EncodeTiledFn fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
    else
      (void)cudaGetLastError();
  });
  return fn;
}

// 3D view [B][N][D] of the bf16 features; box = 64 features x box_rows tokens
// x 1 scene, 128-byte swizzle; rows past N (and features past D) read as 0.
int make_feature_map(CUtensorMap* map, const void* feats, int64_t B, int64_t N, int64_t D,
                     uint32_t box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) {
    note_message("launch_gram_tc: cuTensorMapEncodeTiled unavailable");
    return CP_ECUDA;
  }
  const cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)N, (cuuint64_t)B};
  const cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)N * (cuuint64_t)D * 2};
  const cuuint32_t box[3] = {(cuuint32_t)TC_BK, box_rows, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(feats), dims,
                         strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                         CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    note_message("launch_gram_tc: cuTensorMapEncodeTiled rejected the feature layout");
    return CP_ECUDA;
  }
  return CP_OK;
}

}  // namespace

int launch_gram_minmax_tc(const void* feats, const float4* tok, int64_t B, int64_t N, int64_t D,
                          SceneStats* stats, int* status, uint64_t timeout_ns, cudaStream_t s,
                          float* cos_out, int64_t ldc) {
  DeviceInfo di;
  if (device_info(&di) != CP_OK) return CP_ECUDA;
  alignas(64) CUtensorMap mapA;  // 64 x 128 boxes: A tiles and the halves of B tiles
  CP_TRY_STATUS(make_feature_map(&mapA, feats, B, N, D, TC_BM));
  TcArgs a{};
  a.tok = tok;
  a.cos_out = cos_out;
  a.ldc = ldc;
  a.vec_ok = (ldc % 4 == 0) && (reinterpret_cast<uintptr_t>(cos_out) % 16 == 0);
  a.stats = stats;
  a.status = status;
  a.N = (int)N;
  a.B = (int)B;
  a.TI = (int)((N + TC_BM - 1) / TC_BM);
  a.TJ = (int)((N + TC_BN - 1) / TC_BN);
  a.num_kb = (int)((D + TC_BK - 1) / TC_BK);
  const int TP = (a.TI + 1) / 2;  // row-tile pairs (TP == TJ)
  int64_t ups = 0;                // units per scene
  for (int P2 = 0; P2 < TP; ++P2) ups += a.TJ - P2;
  const int64_t total = ups * B;
  if (total > INT_MAX) return CP_EUNSUPPORTED;
  a.pairs_per_scene = (int)ups;
  a.total_pairs = (int)total;
  a.timeout_ns = timeout_ns;
  auto fn = k_gram_tc;
  if (cuda_status(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)TC_SMEM),
                  "launch_gram_tc: smem attribute") != CP_OK)
    return CP_ECUDA;
  const int64_t clusters = total < di.sm_count / 2 ? total : di.sm_count / 2;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(2 * clusters));
  cfg.blockDim = dim3(TC_THREADS);
  cfg.dynamicSmemBytes = TC_SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, fn, mapA, a);
  note_launch();
  return cuda_status(e, "launch_gram_tc");
}

// The flagged tiles of the Morton-ordered features (local SGS with the
// bounded normaliser): every unit of units[0 .. *n_units) in whole, stored at
// its position coordinates in cos_out; at most max_units units.
int launch_gram_tiles(const void* feats_m, const float4* tok_m, int64_t B, int64_t N, int64_t D,
                      const uint32_t* units, const int* n_units, int64_t max_units, int* status,
                      uint64_t timeout_ns, cudaStream_t s, float* cos_out, int64_t ldc) {
  DeviceInfo di;
  if (device_info(&di) != CP_OK) return CP_ECUDA;
  alignas(64) CUtensorMap mapA;
  CP_TRY_STATUS(make_feature_map(&mapA, feats_m, B, N, D, TC_BM));
  TcArgs a{};
  a.tok = tok_m;
  a.cos_out = cos_out;
  a.ldc = ldc;
  a.vec_ok = (ldc % 4 == 0) && (reinterpret_cast<uintptr_t>(cos_out) % 16 == 0);
  a.stats = nullptr;
  a.status = status;
  a.N = (int)N;
  a.B = (int)B;
  a.TI = (int)((N + TC_BM - 1) / TC_BM);
  a.TJ = (int)((N + TC_BN - 1) / TC_BN);
  a.num_kb = (int)((D + TC_BK - 1) / TC_BK);
  a.pairs_per_scene = 0;
  a.total_pairs = 0;
  a.timeout_ns = timeout_ns;
  a.units = units;
  a.n_units = n_units;
  if (max_units > INT_MAX) return CP_EUNSUPPORTED;
  auto fn = k_gram_tc;
  if (cuda_status(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)TC_SMEM),
                  "launch_gram_tiles: smem attribute") != CP_OK)
    return CP_ECUDA;
  const int64_t clusters = max_units < di.sm_count / 2 ? max_units : di.sm_count / 2;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(2 * (clusters > 0 ? clusters : 1)));
  cfg.blockDim = dim3(TC_THREADS);
  cfg.dynamicSmemBytes = TC_SMEM;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, fn, mapA, a);
  note_launch();
  return cuda_status(e, "launch_gram_tiles");
}

// ---------------------------------------------------------------------------
// The FST cost from the stored upper triangle of cosines, in place (one pass,
// HBM-bound; each cosine read once, both costs of its pair written), and the
// greedy's first-gain partial sums per 64-column tile.
// ---------------------------------------------------------------------------
namespace {

// FST cost of one pair (Eq. fst_cost) with the weights and normalisers
// folded into per-scene constants:
//   C = kB - kA cos + kL log2(1 + kK d) + kT max(tau_s - tau_t, 0)
// (kA = lambda_f / M_f, kB = kA (1 - min d_f), kK = kappa / M_x,
// kL = lambda_x / log2(1 + kappa), kT = lambda_tau / M_tau); the distance
// d = d2 rsqrt(d2) with d2 kept above 1e-30 (d = 0 gives log2(1) = 0), and
// log2 from the hardware approximation: within ~1e-6 of the plain formula,
// far inside the bf16 parity bar, and C(t, t) = 0 exactly.  Both inputs are
// normal floats (d2 >= 1e-30, 1 + kK d >= 1), where the flush-to-zero forms
// of the two instructions return what the plain ones do, without their
// subnormal-input handling.
__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float rsqrt_approx(float x) {
  float y;
  asm("rsqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
struct FstConst {
  float kA, kB, kK, kL, kT;
};
__device__ __forceinline__ FstConst fst_const(const SceneNorms& nm, const DevParams& P) {
  FstConst k;
  k.kA = P.lambda_f * nm.f_rinv;
  k.kB = k.kA * (1.0f - nm.f_lo);
  k.kK = P.kappa * nm.x_rinv;
  k.kL = P.lambda_x * (0.69314718055994531f * P.inv_log1p_kappa);  // log(1+x) = ln2 log2(1+x)
  k.kT = P.lambda_tau * nm.t_rinv;
  return k;
}
__device__ __forceinline__ float fst_cost_fold(const FstConst& k, float cosv, float dx, float dy,
                                               float dz, float tau_s, float tau_t) {
  const float d2 = fmaxf(fmaf(dz, dz, fmaf(dy, dy, dx * dx)), 1.0e-30f);
  const float lg = lg2_approx(fmaf(k.kK, d2 * rsqrt_approx(d2), 1.0f));
  return fmaf(k.kL, lg, fmaf(k.kT, fmaxf(tau_s - tau_t, 0.0f), fmaf(-k.kA, cosv, k.kB)));
}

constexpr int FP_T = 64;         // tile side
constexpr int FP_THREADS = 256;  // 16 threads a row of a tile, 16 rows a pass

// The FST cost from the stored upper triangle of cosines, in place.  Block
// (J, I, b) with I <= J takes the cosine tile of rows 64I.., columns 64J..:
// it writes C(i, j) there and C(j, i) into the transposed tile (rows 64J..,
// columns 64I..), both from the one cosine (the temporal term is the only
// asymmetric part); a diagonal tile (I == J) takes its lower half from the
// transposed upper half.  Pad columns (N <= j < ldc) get 0.  When g0 is given
// every row's terms v_j max(m0 - C(i, j), 0) over the tile's 64 columns go to
// g0[b][column tile][i] (each slot written by one block).  Per-scene
// constants are folded once (fst_const).
__global__ void __launch_bounds__(FP_THREADS, 4) k_fst_pair(
    float* __restrict__ cost, int64_t ldc, int N, const float4* __restrict__ tok,
    const int32_t* __restrict__ frame, const SceneNorms* __restrict__ norms, DevParams P,
    const float* __restrict__ v, float* __restrict__ g0) {
  const int J = blockIdx.x, I = blockIdx.y, b = blockIdx.z;
  if (J < I) return;
  __shared__ float sL[FP_T][FP_T + 1];  // C(j, i): rows of tile J, columns of tile I
  __shared__ float sU[FP_T][FP_T + 1];  // diagonal tile only: the whole C tile
  __shared__ float4 s_ti[FP_T];
  __shared__ float s_fi[FP_T], s_vi[FP_T];
  const size_t sb = (size_t)b * N;
  const int i0 = I * FP_T, jb = J * FP_T;
  const bool diag = I == J;
  const int tid = threadIdx.x;
  const int T = gridDim.x;
  if (tid < FP_T) {
    const int i = i0 + tid;
    s_ti[tid] = i < N ? __ldg(tok + sb + i) : make_float4(0.f, 0.f, 0.f, 0.f);
    s_fi[tid] = i < N ? (float)__ldg(frame + sb + i) : 0.0f;
    s_vi[tid] = i < N && v ? __ldg(v + sb + i) : 0.0f;
  }
  const FstConst kf = fst_const(norms[b], P);
  const int rl = tid >> 4, c4 = (tid & 15) * 4;  // row in the pass, first column
  // this thread's four columns stay the same in every pass
  float4 tj[4];
  float fj[4], vj[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int j = jb + c4 + u;
    tj[u] = j < N ? __ldg(tok + sb + j) : make_float4(0.f, 0.f, 0.f, 0.f);
    fj[u] = j < N ? (float)__ldg(frame + sb + j) : 0.0f;
    vj[u] = j < N && v ? __ldg(v + sb + j) : 0.0f;
  }
  __syncthreads();
  if (!diag && (ldc & 3) == 0 && (reinterpret_cast<uintptr_t>(cost) & 15) == 0) {
    // an off-diagonal pair with 16-byte rows (the common case): every row of
    // tile I is a token (I < J), every column of tile I lies inside the
    // rows, and this thread's four columns of tile J are all inside or all
    // past the row (ldc % 4 == 0)
    const bool cols_ld = jb + c4 < ldc;
    const bool cols_in = jb + c4 + 3 < N;
    const size_t step16 = (size_t)16 * (size_t)ldc;
    float* up = cost + (sb + (size_t)(i0 + rl)) * (size_t)ldc + (jb + c4);
    // every pass's cosines are loaded before the first store, so the four
    // loads are in flight together (a store of pass p could otherwise alias
    // the load of pass p + 1, which would wait for it)
    float4 xs[FP_T / 16];
#pragma unroll
    for (int pass = 0; pass < FP_T / 16; ++pass)
      xs[pass] = cols_ld ? __ldcs(reinterpret_cast<const float4*>(up + pass * step16))
                         : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int pass = 0; pass < FP_T / 16; ++pass, up += step16) {
      const int r = pass * 16 + rl;
      const float c[4] = {xs[pass].x, xs[pass].y, xs[pass].z, xs[pass].w};
      const float4 ti = s_ti[r];
      const float fi = s_fi[r];
      float o[4];
      float part = 0.0f;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        o[u] = 0.0f;  // pad column
        if (!cols_in && jb + c4 + u >= N) continue;
        // fst_cost_fold for (i, j) and (j, i), sharing all but the temporal term
        const float dx = ti.x - tj[u].x, dy = ti.y - tj[u].y, dz = ti.z - tj[u].z;
        const float d2 = fmaxf(fmaf(dz, dz, fmaf(dy, dy, dx * dx)), 1.0e-30f);
        const float lg = lg2_approx(fmaf(kf.kK, d2 * rsqrt_approx(d2), 1.0f));
        const float base = fmaf(-kf.kA, c[u], kf.kB);
        o[u] = fmaf(kf.kL, lg, fmaf(kf.kT, fmaxf(fi - fj[u], 0.0f), base));
        sL[c4 + u][r] = fmaf(kf.kL, lg, fmaf(kf.kT, fmaxf(fj[u] - fi, 0.0f), base));
        part = __fmaf_rn(vj[u], fmaxf(__fsub_rn(P.m0, o[u]), 0.0f), part);
      }
      if (cols_ld) __stcs(reinterpret_cast<float4*>(up), make_float4(o[0], o[1], o[2], o[3]));
      if (g0) {  // the row's 16 threads (a half warp), in a fixed order
#pragma unroll
        for (int o2 = 8; o2 > 0; o2 >>= 1) part += __shfl_xor_sync(0xFFFFFFFFu, part, o2);
        if ((tid & 15) == 0) g0[((size_t)b * T + J) * (size_t)N + i0 + r] = part;
      }
    }
    __syncthreads();
    float* lo = cost + (sb + (size_t)(jb + rl)) * (size_t)ldc + (i0 + c4);
#pragma unroll
    for (int pass = 0; pass < FP_T / 16; ++pass, lo += step16) {
      const int r = pass * 16 + rl;
      const bool row_ok = jb + r < N;
      float o[4];
      float part = 0.0f;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        o[u] = sL[r][c4 + u];
        part = __fmaf_rn(s_vi[c4 + u], fmaxf(__fsub_rn(P.m0, o[u]), 0.0f), part);
      }
      if (row_ok) __stcs(reinterpret_cast<float4*>(lo), make_float4(o[0], o[1], o[2], o[3]));
      if (g0) {
#pragma unroll
        for (int o2 = 8; o2 > 0; o2 >>= 1) part += __shfl_xor_sync(0xFFFFFFFFu, part, o2);
        if ((tid & 15) == 0 && row_ok) g0[((size_t)b * T + I) * (size_t)N + jb + r] = part;
      }
    }
    return;
  }
  // the general case (a diagonal tile, or rows that are not 16-byte aligned):
  // rows i0 + r (r = pass * 16 + rl), columns jb + c4 .. + 3
#pragma unroll
  for (int pass = 0; pass < FP_T / 16; ++pass) {
    const int r = pass * 16 + rl, i = i0 + r;
    const bool row_ok = i < N;
    float* row = cost + (sb + (size_t)(row_ok ? i : 0)) * (size_t)ldc;
    const bool vec = jb + c4 + 3 < ldc && ((reinterpret_cast<uintptr_t>(row + jb + c4) & 15) == 0);
    float c[4] = {0.f, 0.f, 0.f, 0.f};
    if (row_ok) {
      if (vec) {
        const float4 x = __ldcs(reinterpret_cast<const float4*>(row + jb + c4));
        c[0] = x.x, c[1] = x.y, c[2] = x.z, c[3] = x.w;  // below the diagonal: unused
      } else {
#pragma unroll
        for (int u = 0; u < 4; ++u) c[u] = jb + c4 + u < ldc ? row[jb + c4 + u] : 0.0f;
      }
    }
    const float4 ti = s_ti[r];
    const float fi = s_fi[r];
    float o[4];
    float part = 0.0f;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int cl = c4 + u, j = jb + cl;
      o[u] = 0.0f;  // pad column (or, in a diagonal tile, below the diagonal)
      if (!row_ok || j >= N || (diag && cl < r)) continue;
      // fst_cost_fold for (i, j) and for (j, i): the distance term and the
      // feature term are the same (dx only changes sign), the temporal
      // term is the one difference; the same operations, so the same bits
      const float dx = ti.x - tj[u].x, dy = ti.y - tj[u].y, dz = ti.z - tj[u].z;
      const float d2 = fmaxf(fmaf(dz, dz, fmaf(dy, dy, dx * dx)), 1.0e-30f);
      const float lg = lg2_approx(fmaf(kf.kK, d2 * rsqrt_approx(d2), 1.0f));
      const float base = fmaf(-kf.kA, c[u], kf.kB);
      o[u] = fmaf(kf.kL, lg, fmaf(kf.kT, fmaxf(fi - fj[u], 0.0f), base));
      if (!diag || cl > r)  // C(j, i) from the same cosine
        sL[cl][r] = fmaf(kf.kL, lg, fmaf(kf.kT, fmaxf(fj[u] - fi, 0.0f), base));
      part = __fmaf_rn(vj[u], fmaxf(__fsub_rn(P.m0, o[u]), 0.0f), part);
    }
    if (diag) {  // finished below, once the lower half is known
#pragma unroll
      for (int u = 0; u < 4; ++u) sU[r][c4 + u] = o[u];
      continue;
    }
    if (row_ok) {
      if (vec) {
        __stcs(reinterpret_cast<float4*>(row + jb + c4), make_float4(o[0], o[1], o[2], o[3]));
      } else {
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (jb + c4 + u < ldc) row[jb + c4 + u] = o[u];
      }
    }
    if (g0) {  // the row's 16 threads (a half warp), in a fixed order
#pragma unroll
      for (int o2 = 8; o2 > 0; o2 >>= 1) part += __shfl_xor_sync(0xFFFFFFFFu, part, o2);
      if ((tid & 15) == 0 && row_ok) g0[((size_t)b * T + J) * (size_t)N + i] = part;
    }
  }
  __syncthreads();
  if (diag) {  // the lower half: C(i, j) for j < i is sL[i][j]
    for (int e = tid; e < FP_T * FP_T; e += FP_THREADS) {
      const int r = e / FP_T, cl = e % FP_T;
      if (cl < r) sU[r][cl] = sL[r][cl];
    }
    __syncthreads();
  }
  // the rows of the transposed tile (I < J), or of the whole diagonal tile,
  // from shared memory: stores and their first-gain terms (slot I)
  float(*src)[FP_T + 1] = diag ? sU : sL;
  const int rbase = diag ? i0 : jb;  // first row of that tile
#pragma unroll
  for (int pass = 0; pass < FP_T / 16; ++pass) {
    const int r = pass * 16 + rl, jr = rbase + r;
    const bool row_ok = jr < N;
    float o[4];
    float part = 0.0f;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      o[u] = src[r][c4 + u];
      part = __fmaf_rn(s_vi[c4 + u], fmaxf(__fsub_rn(P.m0, o[u]), 0.0f), part);
    }
    if (row_ok) {
      float* row = cost + (sb + (size_t)jr) * (size_t)ldc;
      if (i0 + c4 + 3 < ldc && ((reinterpret_cast<uintptr_t>(row + i0 + c4) & 15) == 0)) {
        __stcs(reinterpret_cast<float4*>(row + i0 + c4), make_float4(o[0], o[1], o[2], o[3]));
      } else {
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (i0 + c4 + u < ldc) row[i0 + c4 + u] = o[u];
      }
    }
    if (g0) {  // the row's 16 threads (a half warp), in a fixed order
#pragma unroll
      for (int o2 = 8; o2 > 0; o2 >>= 1) part += __shfl_xor_sync(0xFFFFFFFFu, part, o2);
      if ((tid & 15) == 0 && row_ok) g0[((size_t)b * T + I) * (size_t)N + jr] = part;
    }
  }
}

// The local neighbourhoods' costs straight from the stored cosines (the
// upper triangle, cos(t, j) at [min][max]):
// slab[b][t][k] = C(t, M_g(t)[k]) with M_g(t)[0] = t and M_g(t)[k] the k-th
// nearest other token, by the same arithmetic as k_fst_pair (the slab holds
// exactly the entries the dense cost would).  One thread per (t, k).
__global__ void __launch_bounds__(256) k_slab_cos(const float* __restrict__ cos, int64_t ldc, int N,
                                                  int g, int kk, const int32_t* __restrict__ nbr,
                                                  const float4* __restrict__ tok,
                                                  const int32_t* __restrict__ frame,
                                                  const SceneNorms* __restrict__ norms,
                                                  DevParams P, const int32_t* __restrict__ pos_of,
                                                  float* __restrict__ slab) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int b = blockIdx.y;
  if (i >= (int64_t)N * g) return;
  const int t = (int)(i / g), k = (int)(i % g);
  const size_t sb = (size_t)b * N;
  const int j = k == 0 ? t : __ldg(nbr + (sb + t) * kk + (k - 1));
  const FstConst kf = fst_const(norms[b], P);
  const float4 ti = __ldg(tok + sb + t), tj = __ldg(tok + sb + j);
  float c;
  if (pos_of == nullptr)  // the upper triangle of the all-pairs Gram
    c = __ldg(cos + (sb + min(t, j)) * (size_t)ldc + max(t, j));
  else if (k == 0)        // cos(f, f) = 1 exactly, as the Gram's diagonal
    c = ti.w > 0.0f ? 1.0f : 0.0f;
  else {                  // the upper triangle of the flagged Morton tiles
    const int pt = __ldg(pos_of + sb + t), pj = __ldg(pos_of + sb + j);
    c = __ldg(cos + (sb + min(pt, pj)) * (size_t)ldc + max(pt, pj));
  }
  slab[sb * g + i] = fst_cost_fold(kf, c, ti.x - tj.x, ti.y - tj.y, ti.z - tj.z,
                                   (float)__ldg(frame + sb + t), (float)__ldg(frame + sb + j));
}

}  // namespace

int launch_slab_cos(const float* cos, int64_t ldc, const int32_t* nbr, const float4* tok,
                    const int32_t* frame, const SceneNorms* norms, const DevParams& P, int64_t B,
                    int64_t N, float* slab, cudaStream_t s, const int32_t* pos_of) {
  const int64_t n = N * P.g;
  dim3 grid((unsigned)((n + 255) / 256), (unsigned)B);
  k_slab_cos<<<grid, 256, 0, s>>>(cos, ldc, (int)N, P.g, P.kk, nbr, tok, frame, norms, P, pos_of,
                                  slab);
  return last_launch_status();
}

int fst_apply_slots(int64_t ldc) { return (int)((ldc + FP_T - 1) / FP_T); }

int launch_fst_apply(float* cost, int64_t ldc, int64_t B, int64_t N, const float4* tok,
                     const int32_t* frame, const SceneNorms* norms, const DevParams& P,
                     const float* v, float* g0, cudaStream_t s) {
  const unsigned T = (unsigned)fst_apply_slots(ldc);
  k_fst_pair<<<dim3(T, T, (unsigned)B), FP_THREADS, 0, s>>>(cost, ldc, (int)N, tok, frame, norms,
                                                           P, v, g0);
  return last_launch_status();
}

}  // namespace cp
