// Two-lane float vectors on Blackwell's packed FP32 instructions
// (add/sub/mul/fma .rn.f32x2): a thread relaxes two groups in lockstep, one per
// half, and every add / sub / mul / fma covers both at once.  Each packed
// instruction rounds like the scalar IEEE operation it pairs, but ptxas fuses a
// packed multiply into a following packed add (an FMA) even with .rn given, and
// decides that per kernel: the scalar instantiation (V = float, explicitly
// rounded intrinsics, never fused) and the paired one (V = F2) agree to within
// fp32 rounding, not bit for bit, and so do two kernels running the same code.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace roi {

struct F2 {
  unsigned long long v;
};

__device__ __forceinline__ F2 f2(float a, float b) {
  F2 r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r.v) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ F2 f2(float a) { return f2(a, a); }
__device__ __forceinline__ float lo(F2 x) {
  float a, b;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(x.v));
  return a;
}
__device__ __forceinline__ float hi(F2 x) {
  float a, b;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(x.v));
  return b;
}
__device__ __forceinline__ F2 operator+(F2 a, F2 b) {
  F2 r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r.v) : "l"(a.v), "l"(b.v));
  return r;
}
__device__ __forceinline__ F2 operator-(F2 a, F2 b) {
  F2 r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r.v) : "l"(a.v), "l"(b.v));
  return r;
}
__device__ __forceinline__ F2 operator*(F2 a, F2 b) {
  F2 r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r.v) : "l"(a.v), "l"(b.v));
  return r;
}
__device__ __forceinline__ F2 vfma(F2 a, F2 b, F2 c) {
  F2 r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r.v) : "l"(a.v), "l"(b.v), "l"(c.v));
  return r;
}

// Scalar counterparts with the same (explicit, uncontracted) rounding.
__device__ __forceinline__ float vadd(float a, float b) { return __fadd_rn(a, b); }
__device__ __forceinline__ float vsub(float a, float b) { return __fsub_rn(a, b); }
__device__ __forceinline__ float vmul(float a, float b) { return __fmul_rn(a, b); }
__device__ __forceinline__ float vfma(float a, float b, float c) { return __fmaf_rn(a, b, c); }
__device__ __forceinline__ F2 vadd(F2 a, F2 b) { return a + b; }
__device__ __forceinline__ F2 vsub(F2 a, F2 b) { return a - b; }
__device__ __forceinline__ F2 vmul(F2 a, F2 b) { return a * b; }

// Broadcast constant.
template <class V>
__device__ __forceinline__ V vconst(float c);
template <>
__device__ __forceinline__ float vconst<float>(float c) { return c; }
template <>
__device__ __forceinline__ F2 vconst<F2>(float c) { return f2(c); }

// Lane-wise helpers without a packed instruction.
template <class Fn>
__device__ __forceinline__ float vmap(float a, Fn fn) { return fn(a); }
template <class Fn>
__device__ __forceinline__ F2 vmap(F2 a, Fn fn) { return f2(fn(lo(a)), fn(hi(a))); }
template <class Fn>
__device__ __forceinline__ float vmap2(float a, float b, Fn fn) { return fn(a, b); }
template <class Fn>
__device__ __forceinline__ F2 vmap2(F2 a, F2 b, Fn fn) { return f2(fn(lo(a), lo(b)), fn(hi(a), hi(b))); }

__device__ __forceinline__ float vmax(float a, float b) { return fmaxf(a, b); }
__device__ __forceinline__ F2 vmax(F2 a, F2 b) { return f2(fmaxf(lo(a), lo(b)), fmaxf(hi(a), hi(b))); }
__device__ __forceinline__ float vmin(float a, float b) { return fminf(a, b); }
__device__ __forceinline__ F2 vmin(F2 a, F2 b) { return f2(fminf(lo(a), lo(b)), fminf(hi(a), hi(b))); }

// Per-lane flag mask: bit h set if lane h satisfies `!(x >= t)` (true for NaN).
__device__ __forceinline__ uint32_t vbelow(float x, float t) { return !(x >= t) ? 1u : 0u; }
__device__ __forceinline__ uint32_t vbelow(F2 x, float t) {
  return (!(lo(x) >= t) ? 1u : 0u) | (!(hi(x) >= t) ? 2u : 0u);
}

template <class V>
__host__ __device__ constexpr int vlanes() {
  return sizeof(V) / sizeof(float);
}

}  // namespace roi
