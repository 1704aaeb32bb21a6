// Double-float arithmetic: a value is the unevaluated sum hi + lo of two
// fp32 numbers with |lo| <= ulp(hi) / 2, about 48 significant bits, built
// from fp32 operations only (FP64 throughput on this part is a small
// fraction of FP32's).  Internal to libadt; used where an fp32 result would
// decide an integer (an accept / reject test, an inverse-CDF draw) and the
// oracle decides in fp64.
//
// Algorithms:
//   two_sum, fast_two_sum, two_prod: the error-free transformations of
//     T. J. Dekker, "A floating-point technique for extending the available
//     precision", Numer. Math. 18 (1971), and D. E. Knuth, TAOCP vol. 2
//     (TwoSum); two_prod uses the fused multiply-add.
//   df_add, df_mul: the "accurate" double-word addition and the
//     double-word times double-word product of M. Joldes, J.-M. Muller,
//     V. Popescu, "Tight and rigorous error bounds for basic building blocks
//     of double-word arithmetic", ACM TOMS 44(2), 2017 (Algorithms 6 and 12).
//   df_exp_diff: Tang's table-driven exponential with a Cody-Waite split
//     reduction (W. J. Cody, W. Waite, "Software Manual for the Elementary
//     Functions", 1980); see the function.
// Every addition and multiplication that must round exactly as written uses
// the explicitly rounded intrinsics, which the compiler never contracts.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace dfl {

struct df {
  float hi, lo;
};

__device__ __forceinline__ df make(float hi, float lo) { return df{hi, lo}; }

// s + e = a + b exactly.
__device__ __forceinline__ df two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return df{s, e};
}

// s + e = a + b exactly, for |a| >= |b| (or a = 0).
__device__ __forceinline__ df fast_two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  return df{s, __fsub_rn(b, __fsub_rn(s, a))};
}

// p + e = a * b exactly (barring underflow).
__device__ __forceinline__ df two_prod(float a, float b) {
  const float p = __fmul_rn(a, b);
  return df{p, __fmaf_rn(a, b, -p)};
}

__device__ __forceinline__ df df_add(df x, df y) {
  const df s = two_sum(x.hi, y.hi);
  const df t = two_sum(x.lo, y.lo);
  const df u = fast_two_sum(s.hi, __fadd_rn(s.lo, t.hi));
  return fast_two_sum(u.hi, __fadd_rn(t.lo, u.lo));
}

__device__ __forceinline__ df df_neg(df x) { return df{-x.hi, -x.lo}; }

__device__ __forceinline__ df df_mul(df x, df y) {
  const df c = two_prod(x.hi, y.hi);
  const float tl = __fmul_rn(x.hi, y.lo);
  const float cl = __fmaf_rn(x.lo, y.hi, tl);
  return fast_two_sum(c.hi, __fadd_rn(c.lo, cl));
}

// x * f for an fp32 f.
__device__ __forceinline__ df df_mul_f(df x, float f) {
  const df c = two_prod(x.hi, f);
  return fast_two_sum(c.hi, __fmaf_rn(x.lo, f, c.lo));
}

__device__ __forceinline__ double to_double(df x) { return static_cast<double>(x.hi) + static_cast<double>(x.lo); }

// 2^(j/64), j = 0 .. 63, as double-floats (hi, lo), evaluated in exact
// decimal arithmetic: the table of the reduction in df_exp_diff.  A kernel
// copies it to shared memory (exp_table_to_smem) and passes that copy.
__device__ const float2 kExp2Sixtyfourths[64] = {
    {0x1.0000000000000p+0f, 0.0f}, {0x1.02c9a40000000p+0f, -0x1.887fa00000000p-28f},
    {0x1.059b0e0000000p+0f, -0x1.9d4f520000000p-25f}, {0x1.0874520000000p+0f, -0x1.e2990e0000000p-26f},
    {0x1.0b55860000000p+0f, 0x1.9f31220000000p-25f}, {0x1.0e3ec40000000p+0f, -0x1.a585cc0000000p-25f},
    {0x1.11301e0000000p+0f, -0x1.fdb4960000000p-25f}, {0x1.1429aa0000000p+0f, 0x1.d525bc0000000p-25f},
    {0x1.172b840000000p+0f, -0x1.c157420000000p-27f}, {0x1.1a35be0000000p+0f, 0x1.6df96e0000000p-25f},
    {0x1.1d48740000000p+0f, -0x1.d2e8ca0000000p-25f}, {0x1.2063b80000000p+0f, 0x1.0c519a0000000p-25f},
    {0x1.2387a60000000p+0f, 0x1.ceac480000000p-25f}, {0x1.26b4560000000p+0f, 0x1.789f380000000p-26f},
    {0x1.29e9e00000000p+0f, -0x1.5c04240000000p-25f}, {0x1.2d285a0000000p+0f, 0x1.b900c20000000p-26f},
    {0x1.306fe00000000p+0f, 0x1.4636e20000000p-25f}, {0x1.33c08c0000000p+0f, -0x1.b37d200000000p-25f},
    {0x1.371a740000000p+0f, -0x1.18aac60000000p-25f}, {0x1.3a7db40000000p+0f, -0x1.634c020000000p-25f},
    {0x1.3dea640000000p+0f, 0x1.8246840000000p-25f}, {0x1.4160a20000000p+0f, 0x1.f72e2a0000000p-28f},
    {0x1.44e0860000000p+0f, 0x1.8624b40000000p-30f}, {0x1.486a2c0000000p+0f, -0x1.47d8660000000p-25f},
    {0x1.4bfdae0000000p+0f, -0x1.593abc0000000p-25f}, {0x1.4f9b280000000p+0f, -0x1.2c5a6c0000000p-25f},
    {0x1.5342b60000000p+0f, -0x1.2c56100000000p-25f}, {0x1.56f4740000000p+0f, -0x1.295b040000000p-25f},
    {0x1.5ab07e0000000p+0f, -0x1.5bd5ec0000000p-27f}, {0x1.5e76f20000000p+0f, -0x1.4a5bd60000000p-25f},
    {0x1.6247ec0000000p+0f, -0x1.f8b5500000000p-25f}, {0x1.6623880000000p+0f, 0x1.2a91120000000p-27f},
    {0x1.6a09e60000000p+0f, 0x1.9fcef40000000p-26f}, {0x1.6dfb240000000p+0f, -0x1.cd72e80000000p-27f},
    {0x1.71f75e0000000p+0f, 0x1.1d8bee0000000p-25f}, {0x1.75feb60000000p+0f, -0x1.37b3060000000p-25f},
    {0x1.7a11480000000p+0f, -0x1.829fd00000000p-25f}, {0x1.7e2f340000000p+0f, -0x1.2616340000000p-25f},
    {0x1.82589a0000000p+0f, -0x1.accc7c0000000p-26f}, {0x1.868d9a0000000p+0f, -0x1.2edb440000000p-26f},
    {0x1.8ace540000000p+0f, 0x1.15506e0000000p-27f}, {0x1.8f1aea0000000p+0f, -0x1.baa2320000000p-26f},
    {0x1.93737c0000000p+0f, -0x1.e647440000000p-25f}, {0x1.97d82a0000000p+0f, -0x1.0d8d840000000p-31f},
    {0x1.9c49180000000p+0f, 0x1.51f8480000000p-27f}, {0x1.a0c6680000000p+0f, -0x1.2886a60000000p-26f},
    {0x1.a5503c0000000p+0f, -0x1.b83b540000000p-25f}, {0x1.a9e6b60000000p+0f, -0x1.50c0480000000p-25f},
    {0x1.ae89fa0000000p+0f, -0x1.a94b140000000p-26f}, {0x1.b33a2c0000000p+0f, -0x1.ec3a820000000p-26f},
    {0x1.b7f7700000000p+0f, -0x1.a094380000000p-25f}, {0x1.bcc1ea0000000p+0f, -0x1.f687c60000000p-25f},
    {0x1.c199be0000000p+0f, -0x1.3d56b20000000p-27f}, {0x1.c67f120000000p+0f, 0x1.cafa2a0000000p-25f},
    {0x1.cb720e0000000p+0f, -0x1.8837cc0000000p-27f}, {0x1.d072d40000000p+0f, 0x1.40f1300000000p-25f},
    {0x1.d5818e0000000p+0f, -0x1.822dbc0000000p-27f}, {0x1.da9e600000000p+0f, 0x1.ed99420000000p-27f},
    {0x1.dfc9740000000p+0f, -0x1.908c940000000p-25f}, {0x1.e502ee0000000p+0f, 0x1.e2cffe0000000p-26f},
    {0x1.ea4afa0000000p+0f, 0x1.52486c0000000p-27f}, {0x1.efa1be0000000p+0f, 0x1.cc2b440000000p-25f},
    {0x1.f507660000000p+0f, -0x1.246eb00000000p-26f}, {0x1.fa7c180000000p+0f, 0x1.9e90d80000000p-28f},
};

// Copies the table to shared memory; call from the first 64 threads of a
// block, then synchronise.
__device__ __forceinline__ void exp_table_to_smem(float2* dst) {
  if (threadIdx.x < 64) dst[threadIdx.x] = kExp2Sixtyfourths[threadIdx.x];
}

// e^(a - b) for fp32 a <= b (the difference is formed exactly); 0 where it
// falls below about 2^-124 (or a is -inf).  Relative error about 3e-12.
// Table-driven (P. T. P. Tang, "Table-driven implementation of the
// exponential function in IEEE floating-point arithmetic", ACM TOMS 15(2),
// 1989): d = (64 m + j) ln2/64 + r with |r| <= ln2/128, e^d = 2^m 2^(j/64) e^r,
// ln2/64 split Cody-Waite style into C1 + C2 + C3 with C1 holding 11 bits so
// that k C1 is exact for |k| < 2^13 (and d - k C1 exact by Sterbenz' lemma);
// e^r = (1 + r) + r^2 (1/2 + r (1/6 + r/24)), the tail (below 1.5e-5) in
// fp32.  `tab` is the shared-memory copy of kExp2Sixtyfourths.
__device__ __forceinline__ df df_exp_diff(float a, float b, const float2* tab) {
  const df d = two_sum(a, -b);
  if (!(d.hi > -86.0f)) return df{0.f, 0.f};
  const float C1 = 0x1.62cp-7f, C2 = 0x1.217f7ep-18f, C3 = -0x1.c610cap-43f;
  const float kf = rintf(__fmul_rn(d.hi, 0x1.715476p+6f));  // in [-7940, 0]
  const int k = static_cast<int>(kf);
  const float a0 = __fsub_rn(d.hi, __fmul_rn(kf, C1));
  df r = two_sum(a0, d.lo);
  r = df_add(r, df_neg(two_prod(kf, C2)));
  const float rh = r.hi;
  const float rl = __fsub_rn(r.lo, __fmul_rn(kf, C3));
  // e^r: 1 + r as a pair, the rest folded into the low word
  const float t = __fmul_rn(__fmul_rn(rh, rh), __fmaf_rn(__fmaf_rn(rh, 0x1.555556p-5f, 0x1.555556p-3f), rh, 0.5f));
  const df one_r = two_sum(1.0f, rh);
  const df er = fast_two_sum(one_r.hi, __fadd_rn(one_r.lo, __fadd_rn(rl, t)));
  const int m = k >> 6, j = k & 63;  // floor division: j in [0, 63]
  const float2 tj = tab[j];
  const df v = df_mul(df{tj.x, tj.y}, er);
  const float scale = __int_as_float((m + 127) << 23);  // m >= -125: a normal number
  return df{__fmul_rn(v.hi, scale), __fmul_rn(v.lo, scale)};
}

// max(0, x) for a normalised double-float (its sign is hi's sign).
__device__ __forceinline__ df df_max0(df x) { return x.hi > 0.f ? x : df{0.f, 0.f}; }

// x < y for normalised double-floats: the sign of their difference.
__device__ __forceinline__ bool df_less(df x, df y) { return df_add(x, df_neg(y)).hi < 0.f; }

// 1 / y for a normalised double-float y != 0: one Newton-Raphson step from
// the correctly rounded fp32 reciprocal t of y.hi, r = t + t (1 - y t), with
// 1 - y t formed from the exact product y.hi t (two_prod) less y.lo t.  The
// residual 1 - y t is about 2^-24, so the step leaves a relative error near
// 2^-46.
__device__ __forceinline__ df df_recip(df y) {
  const float t = __frcp_rn(y.hi);
  const df p = two_prod(y.hi, t);
  const float e = __fsub_rn(__fsub_rn(__fsub_rn(1.f, p.hi), p.lo), __fmul_rn(y.lo, t));
  return fast_two_sum(t, __fmul_rn(t, e));
}

// Running sum of many double-float terms: the leading words summed with
// TwoSum, their errors and the trailing words gathered in a second word
// (a compensated sum; its error stays near n u^2 of the sum for the n
// non-negative terms a thread adds here).
struct Acc {
  float s = 0.f, c = 0.f;
  __device__ __forceinline__ void add(df x) {
    const df t = two_sum(s, x.hi);
    s = t.hi;
    c = __fadd_rn(c, __fadd_rn(t.lo, x.lo));
  }
  __device__ __forceinline__ df value_df() const { return fast_two_sum(s, c); }
};

}  // namespace dfl
