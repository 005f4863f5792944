// Device-side helpers shared by the CoverPrune kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "internal.h"

namespace cp {

// ---------------------------------------------------------------------------
// Element loads: features are bf16 or fp32; every product and sum is fp32.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

// 16 bytes of features as fp32 values: 4 for fp32, 8 for bf16.
template <typename T> struct Vec16;
template <> struct Vec16<float> {
  static constexpr int n = 4;
  __device__ __forceinline__ static void load(const float* p, float* out) {
    float4 v = __ldg(reinterpret_cast<const float4*>(p));
    out[0] = v.x; out[1] = v.y; out[2] = v.z; out[3] = v.w;
  }
};
template <> struct Vec16<__nv_bfloat16> {
  static constexpr int n = 8;
  __device__ __forceinline__ static void load(const __nv_bfloat16* p, float* out) {
    uint4 v = __ldg(reinterpret_cast<const uint4*>(p));
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      out[2 * i + 0] = __uint_as_float(w[i] << 16);
      out[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  }
};

// ---------------------------------------------------------------------------
// Warp-level tensor-core tile (mma.sync m16n8k16, bf16 operands, fp32
// accumulate): d += A B with A 16 x 16 (row-major; this lane holds rows
// lane/4 and lane/4 + 8, columns 2 (lane % 4) + {0, 1} and + 8) and B 16 x 8
// (column-major; this lane holds column lane/4, rows 2 (lane % 4) + {0, 1}
// and + 8); d rows lane/4 and lane/4 + 8, columns 2 (lane % 4) + {0, 1}.
// Each 32-bit operand register packs two consecutive bf16 of one row.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1,
                                               uint32_t a2, uint32_t a3, uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// ---------------------------------------------------------------------------
// Order-preserving float <-> uint32 keys (for atomicMin / atomicMax).
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t f2key(float f) {
  uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float key2f(uint32_t k) {
  uint32_t b = (k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k;
  return __uint_as_float(b);
}

// ---------------------------------------------------------------------------
// Squared distance in single precision, one rounding per operation (no
// contraction): the same value the neighbour order and Morton cells of the
// method are decided on.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float sqdist_rn(float ax, float ay, float az, float bx, float by,
                                           float bz) {
  float dx = __fsub_rn(ax, bx), dy = __fsub_rn(ay, by), dz = __fsub_rn(az, bz);
  return __fadd_rn(__fadd_rn(__fmul_rn(dx, dx), __fmul_rn(dy, dy)), __fmul_rn(dz, dz));
}

// ---------------------------------------------------------------------------
// The FST cost of one pair from its cosine, squared distance and frames
// (Eq. fst_cost).  nm holds the scene's normalisers (see SceneNorms).
// ---------------------------------------------------------------------------
__device__ __forceinline__ float fst_cost_from(float cosv, float d2, int tau_s, int tau_t,
                                               const SceneNorms& nm, const DevParams& P) {
  float df = 1.0f - cosv;
  float tf = (df - nm.f_lo) * nm.f_rinv;  // f_rinv == 0 when the range is empty
  float dx = sqrtf(d2);
  float tx = log1pf(P.kappa * (dx * nm.x_rinv)) * P.inv_log1p_kappa;
  int dt = tau_s - tau_t;
  float tt = dt > 0 ? (float)dt * nm.t_rinv : 0.0f;
  return P.lambda_f * tf + P.lambda_x * tx + P.lambda_tau * tt;
}

__device__ __forceinline__ float clamp_cos(float c) { return fminf(1.0f, fmaxf(-1.0f, c)); }

// ---------------------------------------------------------------------------
// Warp reductions (fixed butterfly order: deterministic).
// ---------------------------------------------------------------------------
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}
__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}
__device__ __forceinline__ unsigned long long warp_max_u64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    unsigned long long w = __shfl_xor_sync(0xFFFFFFFFu, v, o);
    v = w > v ? w : v;
  }
  return v;
}
__device__ __forceinline__ unsigned long long warp_min_u64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    unsigned long long w = __shfl_xor_sync(0xFFFFFFFFu, v, o);
    v = w < v ? w : v;
  }
  return v;
}

// ---------------------------------------------------------------------------
// Time and bounded waits.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ int ld_volatile_i32(const int* p) {
  return *reinterpret_cast<const volatile int*>(p);
}
__device__ __forceinline__ void red_release_add(uint32_t* p, uint32_t v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
// Record the first device-side error of a call (later ones are dropped).
__device__ __forceinline__ void set_status(int* status, int code) {
  atomicCAS(status, 0, code);
}

// Grid barrier over `nblocks` blocks sharing counter `ctr` (zeroed before the
// launch; the target grows by nblocks every round).  Gives up after
// timeout_ns or as soon as another block has recorded an error; returns false
// then, with the error in *status.  Every thread of the block must call it.
__device__ __forceinline__ bool grid_barrier(uint32_t* ctr, uint32_t target, int* status,
                                             uint64_t timeout_ns) {
  __shared__ int s_ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    __threadfence();
    red_release_add(ctr, 1u);
    uint64_t t0 = globaltimer_ns();
    uint32_t spins = 0;
    while (ld_acquire_u32(ctr) < target) {
      if ((++spins & 63u) == 0) {
        if (ld_volatile_i32(status) != 0) { ok = 0; break; }
        if (globaltimer_ns() - t0 > timeout_ns) {
          set_status(status, CP_ETIMEOUT);
          ok = 0;
          break;
        }
      }
    }
    __threadfence();
    s_ok = ok;
  }
  __syncthreads();
  return s_ok != 0;
}

}  // namespace cp
