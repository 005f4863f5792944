// bf16 rows: dot products with fp32 accumulation on the mixed-precision FMA
// (fma.rn.f32.bf16: the bf16 operands enter the FMA as they are, with no
// widening instructions), and 16-byte asynchronous copies of row pieces into
// shared memory (cp.async), for loops that keep several pieces in flight
// without holding them in registers.
#pragma once
#include <stdint.h>

namespace cp {

// acc + x . y over the 8 bf16 of each operand, element order lo, hi of each
// 32-bit word in turn: fma.rn.f32.bf16 takes the bf16 operands as they are
// (their product is exact in fp32) and rounds once, so each step equals
// fmaf on the widened values and the sum is the same as widening first.
__device__ __forceinline__ float dot8_bf16(const uint4 x, const uint4 y, float acc) {
  asm("{\n\t.reg .b16 xl, xh, yl, yh;\n\t"
      "mov.b32 {xl, xh}, %1;\n\tmov.b32 {yl, yh}, %5;\n\t"
      "fma.rn.f32.bf16 %0, xl, yl, %0;\n\tfma.rn.f32.bf16 %0, xh, yh, %0;\n\t"
      "mov.b32 {xl, xh}, %2;\n\tmov.b32 {yl, yh}, %6;\n\t"
      "fma.rn.f32.bf16 %0, xl, yl, %0;\n\tfma.rn.f32.bf16 %0, xh, yh, %0;\n\t"
      "mov.b32 {xl, xh}, %3;\n\tmov.b32 {yl, yh}, %7;\n\t"
      "fma.rn.f32.bf16 %0, xl, yl, %0;\n\tfma.rn.f32.bf16 %0, xh, yh, %0;\n\t"
      "mov.b32 {xl, xh}, %4;\n\tmov.b32 {yl, yh}, %8;\n\t"
      "fma.rn.f32.bf16 %0, xl, yl, %0;\n\tfma.rn.f32.bf16 %0, xh, yh, %0;\n\t}"
      : "+f"(acc)
      : "r"(x.x), "r"(x.y), "r"(x.z), "r"(x.w), "r"(y.x), "r"(y.y), "r"(y.z), "r"(y.w));
  return acc;
}
// 16 bytes global -> shared through L2 only; zeros, reading nothing, when
// !ok (src must still be a valid address)
__device__ __forceinline__ void cp_async16_zfill(void* dst, const void* src, bool ok) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(
                   (uint32_t)__cvta_generic_to_shared(dst)),
               "l"(src), "r"(ok ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
// this thread's copies of all but the newest N committed groups have landed
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

}  // namespace cp
