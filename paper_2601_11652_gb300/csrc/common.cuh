// common.cuh -- device-side helpers shared by the verification kernels.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include "wisp_verify.h"

namespace wisp {

// ---------------------------------------------------------------------------
// Workspace header (first 256 bytes of the caller's workspace)
// ---------------------------------------------------------------------------
struct DeviceStatus {
  int32_t code;        // wisp_device_code of the first error, 0 if none
  int32_t pad;
  int64_t request_id;  // request id of that error
};

// Record the first device-side error; later errors are dropped.
__device__ __forceinline__ void report(DeviceStatus *st, int32_t code, const int64_t *request_ids, int r) {
  if (atomicCAS(&st->code, 0, code) == 0) {
    st->request_id = request_ids && r >= 0 ? request_ids[r] : (int64_t)r;  // r < 0: not one request
  }
}

constexpr int kMaxRowsPerHead = 128;  // (Hq/Hkv) * (k+1) rows per KV head of a request
constexpr int kTcRowsPerItem = 64;    // query rows per work item of the tensor-core attention kernel
constexpr int kMaxDraft = 1024;       // k_r limit of the acceptance kernels

// Hardware 2^x (ex2.approx.ftz.f32).  Over every float x in [-126, 0] its relative error is below
// 2^-22.7 (measured exhaustively on GB300 by tests/test_ex2_bound_gpu.py); the acceptance kernels'
// certified bounds use kEx2RelErr for it.  Below -126 the result flushes to zero.
constexpr float kEx2RelErr = 0x1p-22f;
constexpr float kLog2e = 1.4426950408889634f;  // log2(e) rounded to float
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Per-request flags written by the planner
enum : int32_t { REQ_OK = 0, REQ_BAD = 1 };

// ---------------------------------------------------------------------------
// Element loads
// ---------------------------------------------------------------------------
__device__ __forceinline__ float bf16_bits_to_float(uint32_t bits16) {
  return __uint_as_float(bits16 << 16);
}
__device__ __forceinline__ float load_elem(const float *p, int64_t i) { return __ldg(p + i); }
__device__ __forceinline__ float load_elem(const __nv_bfloat16 *p, int64_t i) {
  return __bfloat162float(p[i]);
}

// ---------------------------------------------------------------------------
// Double-float ("ff") arithmetic: a value is hi + lo with |lo| <= ulp(hi)/2.
// Error-free transformations after Knuth (TwoSum), Dekker (FastTwoSum) and the
// FMA-based TwoProd; about 48 significant bits.  Must be compiled without
// fast-math / reassociation.
// ---------------------------------------------------------------------------
struct ff {
  float hi, lo;
};

__device__ __forceinline__ ff ff_two_sum(float a, float b) {
  float s = __fadd_rn(a, b);
  float bb = __fsub_rn(s, a);
  float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return {s, e};
}
__device__ __forceinline__ ff ff_fast_two_sum(float a, float b) {  // requires |a| >= |b| or a == 0
  float s = __fadd_rn(a, b);
  float e = __fsub_rn(b, __fsub_rn(s, a));
  return {s, e};
}
__device__ __forceinline__ ff ff_two_prod(float a, float b) {
  float p = __fmul_rn(a, b);
  float e = __fmaf_rn(a, b, -p);
  return {p, e};
}
__device__ __forceinline__ ff ff_add(ff a, ff b) {
  ff s = ff_two_sum(a.hi, b.hi);
  ff t = ff_two_sum(a.lo, b.lo);
  s.lo = __fadd_rn(s.lo, t.hi);
  s = ff_fast_two_sum(s.hi, s.lo);
  s.lo = __fadd_rn(s.lo, t.lo);
  return ff_fast_two_sum(s.hi, s.lo);
}
__device__ __forceinline__ ff ff_add_f(ff a, float b) {
  ff s = ff_two_sum(a.hi, b);
  s.lo = __fadd_rn(s.lo, a.lo);
  return ff_fast_two_sum(s.hi, s.lo);
}
__device__ __forceinline__ ff ff_neg(ff a) { return {-a.hi, -a.lo}; }
__device__ __forceinline__ ff ff_mul(ff a, ff b) {
  ff p = ff_two_prod(a.hi, b.hi);
  p.lo = __fmaf_rn(a.hi, b.lo, __fmaf_rn(a.lo, b.hi, p.lo));
  return ff_fast_two_sum(p.hi, p.lo);
}
__device__ __forceinline__ ff ff_mul_f(ff a, float b) {
  ff p = ff_two_prod(a.hi, b);
  p.lo = __fmaf_rn(a.lo, b, p.lo);
  return ff_fast_two_sum(p.hi, p.lo);
}
__device__ __forceinline__ bool ff_gt(ff a, ff b) {  // a > b
  return a.hi > b.hi || (a.hi == b.hi && a.lo > b.lo);
}
__device__ __forceinline__ double ff_to_double(ff a) { return (double)a.hi + (double)a.lo; }
__device__ __forceinline__ ff ff_shfl_xor(ff a, int m) {
  return {__shfl_xor_sync(0xffffffffu, a.hi, m), __shfl_xor_sync(0xffffffffu, a.lo, m)};
}
__device__ __forceinline__ ff ff_shfl_up(ff a, int d) {
  return {__shfl_up_sync(0xffffffffu, a.hi, d), __shfl_up_sync(0xffffffffu, a.lo, d)};
}

// 2^(j/256), j = 0..255, as double-float pairs; filled by the host from exp2 in double.
struct Exp2Table {
  float hi[256];
  float lo[256];
};

// exp(x) for x = xh + xl <= 0 (|xl| <= ulp(xh)/2), to about 1e-13 relative error.
// Tang's table-driven method (ACM TOMS 15(2), 1989): x = N ln2/256 + r, |r| <= ln2/512,
// exp(x) = 2^(N div 256) * 2^((N mod 256)/256) * exp(r), exp(r) by its Taylor series to r^4.
// ln2/256 is split into three floats (8 + 24 + 24 bits) so that N*C_HI is exact and
// x - N*C_HI is exact for |x| < 128.  `tab` lives in shared memory.
__device__ __forceinline__ ff ff_exp_nonpos(float xh, float xl, const float *tab_hi, const float *tab_lo) {
  constexpr float kInvC = 0x1.715476p+8f;   // 256 / ln 2
  constexpr float C_HI = 0x1.62p-9f;        // ln2/256 rounded to 8 significant bits
  constexpr float C_MID = 0x1.c85fep-18f;   // next 24 bits
  constexpr float C_LO = -0x1.718432p-43f;  // next 24 bits
  if (!(xh > -87.0f)) return {0.0f, 0.0f};  // exp(x) < 1.7e-38: below ff resolution of any sum >= 1
  const float Nf = rintf(xh * kInvC);
  const int N = (int)Nf;
  const float r1 = __fmaf_rn(-Nf, C_HI, xh);  // exact
  ff p = ff_two_prod(Nf, C_MID);             // exact
  ff s = ff_two_sum(r1, -p.hi);
  s.lo = __fadd_rn(s.lo, __fsub_rn(__fsub_rn(xl, p.lo), __fmul_rn(Nf, C_LO)));
  s = ff_fast_two_sum(s.hi, s.lo);           // r = s.hi + s.lo, |r| <= 1.36e-3
  const float rh = s.hi, rl = s.lo;
  // exp(r) - 1 - r = r^2/2 + r^3/6 + r^4/24 (+ r*rl cross term of r^2/2)
  float poly = __fmul_rn(__fmul_rn(rh, rh), __fmaf_rn(rh, __fmaf_rn(rh, 1.0f / 24.0f, 1.0f / 6.0f), 0.5f));
  poly = __fmaf_rn(rh, rl, poly);
  ff e = ff_two_sum(1.0f, rh);
  e.lo = __fadd_rn(e.lo, __fadd_rn(rl, poly));
  e = ff_fast_two_sum(e.hi, e.lo);
  const int j = N & 255;          // N = 256*kexp + j, 0 <= j < 256 (two's complement)
  const int kexp = (N - j) >> 8;  // in [-126, 0] since x > -87
  e = ff_mul(e, ff{tab_hi[j], tab_lo[j]});
  const float scale = __int_as_float((127 + kexp) << 23);
  return {__fmul_rn(e.hi, scale), __fmul_rn(e.lo, scale)};
}

}  // namespace wisp
