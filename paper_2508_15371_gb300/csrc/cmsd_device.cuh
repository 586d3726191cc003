// Device primitives for sm_103a: fast base-2 exponential, packed bf16x2
// min/max, packed f32x2 arithmetic, streaming loads and GPU-scope atomics
// with acquire-release semantics.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace cmsd {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
// Masked (-inf) drafter logits are clamped to -2^100.  A power of two times
// the float log2(e) is exact, so when a lane's running maximum is itself a
// clamped entry the exponent z*log2e - m*log2e is exactly 0 (no rounding
// residual of a 1e30-sized product leaks into ex2).
constexpr uint32_t kNegClampBits = 0xF1B00000u;       // -2^100 (exact in bf16 and f32)
constexpr uint32_t kNegClamp2 = 0xF1B0F1B0u;          // the same, two bf16 lanes
constexpr uint32_t kNegInf2 = 0xFF80FF80u;            // -inf, two bf16 lanes
// "No element yet": -2^101, below every clamped logit.  Also a power of two, so
// kNegInit * log2(e) is exact and two empty states cancel to exactly 0.
constexpr float kNegInit = -2535301200456458802993406410752.0f;   // -2^101
constexpr unsigned kFull = 0xFFFFFFFFu;
constexpr int kIntMax = 0x7FFFFFFF;

__device__ __forceinline__ float neg_clamp() { return __uint_as_float(kNegClampBits); }
__device__ __forceinline__ float pos_inf() { return __int_as_float(0x7F800000); }
// m * log2(e), rounded on its own (never fused into a neighbouring add): the
// differences of such products must be exactly 0 for equal maxima.
__device__ __forceinline__ float mlog2e(float m) { return __fmul_rn(m, kLog2e); }

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ---- packed bfloat16 pairs ------------------------------------------------
__device__ __forceinline__ uint32_t bmax2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ uint32_t bmin2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("min.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// ---- packed float pairs -----------------------------------------------------
// Two IEEE fp32 values in one 64-bit register pair, operated on by the sm_100+
// packed f32x2 instructions (two independent correctly rounded operations).
typedef unsigned long long u64;
__device__ __forceinline__ u64 pack2(float lo, float hi) {
  u64 r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ float lo32f(u64 r) { return __uint_as_float((uint32_t)r); }
__device__ __forceinline__ float hi32f(u64 r) { return __uint_as_float((uint32_t)(r >> 32)); }
// the two bfloat16 halves of w as two floats (low half first)
__device__ __forceinline__ u64 bf2_to_f2(uint32_t w) {
  u64 r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(w << 16), "r"(w & 0xFFFF0000u));
  return r;
}
__device__ __forceinline__ u64 fma2(u64 a, u64 b, u64 c) {
  u64 d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ u64 add2(u64 a, u64 b) {
  u64 d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ u64 mul2(u64 a, u64 b) {
  u64 d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ u64 dup2(float x) { return pack2(x, x); }
__device__ __forceinline__ u64 ex2_2(u64 x) { return pack2(ex2(lo32f(x)), ex2(hi32f(x))); }

// ---- global memory ------------------------------------------------------------
// GPU-scope add with acquire-release semantics: the caller's earlier stores
// are visible before the add, and what other threads released before their
// adds is visible after it.
__device__ __forceinline__ int atom_add_acq_rel(int* p, int v) {
  int old;
  asm volatile("atom.add.acq_rel.gpu.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}


__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ unsigned long long atom_add_acq_rel_u64(unsigned long long* p,
                                                                   unsigned long long v) {
  unsigned long long old;
  asm volatile("atom.add.acq_rel.gpu.u64 %0, [%1], %2;" : "=l"(old) : "l"(p), "l"(v) : "memory");
  return old;
}
}  // namespace cmsd
