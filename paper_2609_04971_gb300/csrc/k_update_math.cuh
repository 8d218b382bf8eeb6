// Arithmetic shared by the beacon-update kernels (k_update.cu for many queries
// per instance, k_update_small.cu for a few): double-float operations, the
// exact per-column sums of bf16 values, the norm data of a centroid and the
// exact re-decision of a close assignment.  Both kernels take their decisions
// and sums with these same operations.
#pragma once
#include "bkv_device.cuh"

namespace bkv {
namespace {

// A query is re-decided exactly when its best and second-best screened unit-centroid
// dots differ by at most this fraction of |q| (about twice the screening error bound).
constexpr float kMarginRel = 1e-4f;

// Double-float arithmetic (an unevaluated sum hi + lo of two fp32 values,
// about 48 significant bits) for the exact re-decisions: fp64 is slow on
// this part.  TwoSum (Knuth) and the FMA-based exact product.
struct DF {
  float hi, lo;
};

__device__ __forceinline__ DF df_add(DF a, DF b) {
  const float s = __fadd_rn(a.hi, b.hi);
  const float bb = __fadd_rn(s, -a.hi);
  const float err = __fadd_rn(__fadd_rn(a.hi, -__fadd_rn(s, -bb)), __fadd_rn(b.hi, -bb));
  const float lo = __fadd_rn(__fadd_rn(a.lo, b.lo), err);
  const float t = __fadd_rn(s, lo);
  return DF{t, __fadd_rn(lo, -__fadd_rn(t, -s))};
}

__device__ __forceinline__ DF df_two_prod(float a, float b) {
  const float p = __fmul_rn(a, b);
  return DF{p, __fmaf_rn(a, b, -p)};
}

__device__ __forceinline__ DF df_mul(DF a, DF b) {
  const float p = __fmul_rn(a.hi, b.hi);
  float e = __fmaf_rn(a.hi, b.hi, -p);
  e = __fmaf_rn(a.hi, b.lo, e);
  e = __fmaf_rn(a.lo, b.hi, e);
  const float t = __fadd_rn(p, e);
  return DF{t, __fadd_rn(e, -__fadd_rn(t, -p))};
}

__device__ __forceinline__ bool df_gt(DF a, DF b) { return a.hi > b.hi || (a.hi == b.hi && a.lo > b.lo); }

// 1 / sqrt(a) for a double-float a > 0: the fp32 estimate y = rsqrtf(a.hi) (about 2^-22
// relative) refined by one Newton-Raphson step for f(y) = 1 / y^2 - a,
// y' = y + y (1 - a y^2) / 2, with the residual 1 - a y^2 formed in double-float
// arithmetic; the result holds about 44 significant bits.  fp64 is slow on this part.
__device__ __forceinline__ DF df_rsqrt(DF a) {
  const float y = rsqrtf(a.hi);
  const DF ay2 = df_mul(a, df_two_prod(y, y));
  const float r = __fadd_rn(__fadd_rn(1.f, -ay2.hi), -ay2.lo);  // 1 - a y^2, about 2^-22: two roundings suffice
  return df_add(DF{y, 0.f}, df_two_prod(y, 0.5f * r));
}

// Exact sums of bf16 values without a 64-bit conversion per element: x is
// split into xh = x rounded to a multiple of 2^-3, xm = the rest rounded to a
// multiple of 2^-20 and xl = what remains (magic-number rounding, fp32 adds
// only, two columns per paired-fp32 instruction); each part's fp32 running
// sum is exact over up to 128 values with |x| < 2^14 (xl is exact for
// |x| >= 2^-31).  `fixed40` turns the three sums into round(sum * 2^40) with
// 32-bit conversions.
struct Parts {
  float h, m, l;
};

__device__ __forceinline__ long long fixed40(const Parts& p) {
  const long long h = static_cast<long long>(__float2int_rn(p.h * 8.0f)) << 37;
  const long long m = static_cast<long long>(__float2int_rn(p.m * 1048576.0f)) << 20;
  const long long l = static_cast<long long>(__float2int_rn(p.l * 274877906944.0f)) << 2;
  return h + m + l;
}

// Float <-> int conversions run on a slow unit of this part, so the small cases below use the
// magic-number route instead: for an integer-valued float x with |x| <= 2^22, x + 1.5 * 2^23 holds the
// integer in its low mantissa bits (the sum stays in [2^23, 2^24], where every integer is exact),
// and for an integer |i| <= 2^22 the reverse subtraction gives float(i) exactly.
__device__ __forceinline__ int magic_f2i(float x) {  // x integer-valued, |x| <= 2^22
  return __float_as_int(__fadd_rn(x, 12582912.f)) - 0x4B400000;
}
__device__ __forceinline__ float magic_i2f(int i) {  // |i| <= 2^22, exact
  return __fadd_rn(__int_as_float(0x4B400000 + i), -12582912.f);
}

// fixed40 for part sums of at most 32 values (a few queries per beacon, the decode-step kernel): each
// scaled part is an integer of magnitude at most 2^22 (|x| < 2^14 for the high part, 2^-4 for the
// middle one, 2^-21 for the low one), so the magic-number conversions are exact and equal fixed40's.
__device__ __forceinline__ long long fixed40_few(const Parts& p) {
  const long long h = static_cast<long long>(magic_f2i(p.h * 8.0f)) << 37;
  const long long m = static_cast<long long>(magic_f2i(p.m * 1048576.0f)) << 20;
  const long long l = static_cast<long long>(magic_f2i(p.l * 274877906944.0f)) << 2;
  return h + m + l;
}

// fixed40_one below 2^-31 in magnitude (e < 96): x * 2^38 = M / 2^(96 - e) rounded to nearest
// even, times 4 (0 once the shift reaches 9).  Out of line: rare, and kept off the common path.
__device__ __noinline__ long long fixed40_one_tiny(int M, int e) {
  const int sh = 96 - e;
  if (sh >= 9) return 0;
  int q = M >> sh;
  const int rem = M & ((1 << sh) - 1), half = 1 << (sh - 1);
  if (rem > half || (rem == half && (q & 1))) ++q;
  return static_cast<long long>(q) << 2;
}

// round(x * 2^40) of one bf16-exact value x (|x| < 2^14), from integer operations on its bits: what
// fixed40 gives for the part sums of x alone (exact for |x| >= 2^-31; below, x * 2^38 rounded to the
// nearest even integer, times 4, as the low part's conversion does).
__device__ __forceinline__ long long fixed40_one(float x) {
  const uint32_t b = __float_as_uint(x);
  const int e = static_cast<int>((b >> 23) & 0xffu);
  const int M = static_cast<int>(((b >> 16) & 0x7fu) | 0x80u);  // the 8-bit significand
  long long F;
  if (e >= 96) {
    F = static_cast<long long>(M) << (e - 94);  // x * 2^40 = M * 2^(e - 94), exact
  } else {
    F = e == 0 ? 0 : fixed40_one_tiny(M, e);  // zero or a subnormal rounds to 0 on the 2^-38 grid
  }
  return (b >> 31) ? -F : F;
}

// Splits the bf16 value x (exact in fp32) into the three parts and adds them.
__device__ __forceinline__ void parts_add(Parts& p, float x) {
  const float xh = __fadd_rn(__fadd_rn(x, 1572864.f), -1572864.f);  // multiple of 2^-3 (1.5 * 2^20 magic)
  const float r = __fadd_rn(x, -xh);
  const float xm = __fadd_rn(__fadd_rn(r, 12.f), -12.f);  // multiple of 2^-20 (1.5 * 2^3 magic)
  p.h = __fadd_rn(p.h, xh);
  p.m = __fadd_rn(p.m, xm);
  p.l = __fadd_rn(p.l, __fadd_rn(r, -xm));
}

// 1 / |c| of a centroid from its double-float sum of squares n2d (fp32 value n2),
// and whether |c|^2 is far from fp32 over- and underflow (`plain`); outside that
// range the same quantity is taken in fp64.
__device__ __noinline__ DF centroid_inv_norm_wide(DF n2d) {
  const double inv = __drcp_rn(sqrt(static_cast<double>(n2d.hi) + static_cast<double>(n2d.lo)));
  const float inv_hi = __double2float_rn(inv);
  return DF{inv_hi, __double2float_rn(inv - static_cast<double>(inv_hi))};
}

__device__ __forceinline__ DF centroid_inv_norm(DF n2d, float n2, bool& plain) {
  plain = n2 > 1e-30f && n2 < 1e30f;
  return plain ? df_rsqrt(n2d) : centroid_inv_norm_wide(n2d);
}

// The fold of a call's exact sum into the running state.  acc * 2^-40 as a double: one
// round-to-nearest conversion of the int64 (exact below 2^53), the power of two applied to
// the exponent field (|acc| >= 1 keeps the result normal).
__device__ __forceinline__ double fixed40_to_double(long long acc) {
  if (acc == 0) return 0.0;
  return __longlong_as_double(__double_as_longlong(__ll2double_rn(acc)) - (40LL << 52));
}

// The double nearest to t * 2^-40 (ties to even) for 0 < |t| < 2^63, from integer operations
// only: the leading bit fixes the exponent, the bits below the 53-bit significand are rounded.
__device__ __forceinline__ double fixed40_round(long long t) {
  const unsigned long long sign = t < 0 ? (1ull << 63) : 0ull;
  const unsigned long long a = t < 0 ? 0ull - static_cast<unsigned long long>(t) : static_cast<unsigned long long>(t);
  int msb = 63 - __clzll(static_cast<long long>(a));
  unsigned long long mant;
  if (msb <= 52) {
    mant = a << (52 - msb);
  } else {
    const int sh = msb - 52;
    mant = a >> sh;
    const unsigned long long rem = a & ((1ull << sh) - 1ull), half = 1ull << (sh - 1);
    if (rem > half || (rem == half && (mant & 1ull))) ++mant;
    if (mant >> 53) {
      mant >>= 1;
      ++msb;
    }
  }
  const unsigned long long e = static_cast<unsigned long long>(msb - 40 + 1023);
  return __longlong_as_double(static_cast<long long>(sign | (e << 52) | (mant & ((1ull << 52) - 1ull))));
}

// fold_sum's fp64 route, out of line (rare: sums off the 2^-40 grid or at 2^22 and above).
__device__ __noinline__ double fold_sum_wide(double s, long long acc) { return __dadd_rn(s, fixed40_to_double(acc)); }

// s + acc * 2^-40 rounded to the nearest double (ties to even), the running sum after a call
// whose exact sum is acc (fixed point, 40 fractional bits).  fp64 arithmetic is slow on this
// part, so the common case stays in integers: when s is a multiple of 2^-40 below 2^22 in
// magnitude (every sum built from queries of 2^-31 or more is) and |acc| < 2^61, s becomes the
// integer s * 2^40, the two integers are added exactly and the total is rounded once.  This is
// the correctly rounded sum, as an fp64 addition of s and acc * 2^-40 (exact below 2^53) gives.
// Other values take the fp64 route.
__device__ __forceinline__ double fold_sum(double s, long long acc) {
  if (acc == 0) return s;
  const unsigned long long bits = static_cast<unsigned long long>(__double_as_longlong(s));
  const int e = static_cast<int>((bits >> 52) & 0x7ff);
  const long long lim = 1LL << 61;
  if (acc > -lim && acc < lim && e < 1023 + 22) {
    long long f = 0;
    bool ok = true;
    if (e != 0) {
      const unsigned long long m = (bits & ((1ull << 52) - 1ull)) | (1ull << 52);
      const int sh = e - 1035;  // s * 2^40 = m * 2^(e - 1075 + 40)
      if (sh >= 0) {
        f = static_cast<long long>(m << sh);
      } else if (sh > -53 && (m & ((1ull << -sh) - 1ull)) == 0ull) {
        f = static_cast<long long>(m >> -sh);
      } else {
        ok = false;  // not a multiple of 2^-40
      }
      if (bits >> 63) f = -f;
    } else {
      ok = (bits << 1) == 0ull;  // +-0; subnormals take the fp64 route
    }
    if (ok) {
      const long long t = f + acc;
      return t == 0 ? 0.0 : fixed40_round(t);
    }
  }
  return fold_sum_wide(s, acc);
}

// fold_sum for warps that have the fp64 pipe to themselves: below 2^53, acc * 2^-40 is exact in
// fp64 and one fp64 addition rounds the sum once, so the result is fold_sum's, without its integer
// instructions; larger sums take fold_sum (which rounds once where the fp64 route would round twice).
__device__ __forceinline__ double fold_sum_fp64(double s, long long acc) {
  const long long lim = 1LL << 53;
  if (acc > -lim && acc < lim) return acc == 0 ? s : __dadd_rn(s, fixed40_to_double(acc));
  return fold_sum(s, acc);
}

// n > 2^22 as nf + nl: nf = fp32(n), nl = fp32(n - nf).  Out of line: the 64-bit conversions run on
// a slow unit of this part, and inlined they would be executed for every count.
__device__ __noinline__ float2 count_split_large(long long n) {
  const float nf = static_cast<float>(n);
  return make_float2(nf, static_cast<float>(n - static_cast<long long>(nf)));
}

// 1 / n for a count n >= 1 as a double-float: the correctly rounded fp32 reciprocal of n
// refined by one Newton-Raphson step r' = r + r (1 - n r), the residual formed exactly.
__device__ __forceinline__ DF count_reciprocal(long long n) {
  // counts up to 2^22 (all practical ones) are exact floats by the magic-number route (nl = 0)
  float nf, nl = 0.f;
  if (n <= (1LL << 22)) {
    nf = magic_i2f(static_cast<int>(n));
  } else {
    const float2 v = count_split_large(n);
    nf = v.x;
    nl = v.y;
  }
  const float r = __frcp_rn(nf);
  const float p = __fmul_rn(nf, r);
  const float pe = __fmaf_rn(nl, r, __fmaf_rn(nf, r, -p));     // n r - p
  const float e = __fadd_rn(__fadd_rn(1.f, -p), -pe);          // 1 - n r (1 - p is exact: p is near 1)
  const float d = __fmul_rn(r, e);
  const float hi = __fadd_rn(r, d);
  return DF{hi, __fadd_rn(d, -__fadd_rn(hi, -r))};
}

// 2^k as a float, for -126 <= k <= 127.
__device__ __forceinline__ float pow2f(int k) { return __uint_as_float(static_cast<uint32_t>(k + 127) << 23); }

// fp32(s * (1 / n)) from the running sum s (fp64) and rcp = count_reciprocal(n), without fp64
// arithmetic: s is split into hi (its significand rounded to 24 bits) and lo (the remainder,
// rounded to fp32) by integer operations on its bits, multiplied by rcp as double-floats and
// rounded once to fp32; within one fp32 ulp of fp32(s / n).  |s| outside [2^-70, 2^100]
// (and zero) takes the fp64 route.
// centroid_value outside [2^-70, 2^100] (and at zero), in fp64; out of line so that its fp64
// instructions are never executed for the common case.
__device__ __noinline__ float centroid_value_wide(double s, DF rcp) {
  return __double2float_rn(__dmul_rn(s, __dadd_rn(static_cast<double>(rcp.hi), static_cast<double>(rcp.lo))));
}

__device__ __forceinline__ float centroid_value(double s, DF rcp) {
  const unsigned long long bits = static_cast<unsigned long long>(__double_as_longlong(s));
  const int e = static_cast<int>((bits >> 52) & 0x7ff);
  if (e < 1023 - 70 || e > 1023 + 100) return centroid_value_wide(s, rcp);
  const unsigned long long m = (bits & ((1ull << 52) - 1)) | (1ull << 52);  // 53-bit significand
  const unsigned long long m_hi = (m + (1ull << 28) - 1 + ((m >> 29) & 1)) >> 29;  // m / 2^29, nearest even
  const long long rem = static_cast<long long>(m) - static_cast<long long>(m_hi << 29);  // |rem| <= 2^28
  // no conversion instructions (a slow unit on this part): m_hi is in [2^23, 2^24], whose float has the
  // bit pattern m_hi + 0x4A800000; rem (|rem| <= 2^28) is rounded to fp32 as the fp32 sum of its exact
  // high part (rem with its low 6 bits cleared) and its exact low 6 bits: one rounding, as a conversion
  const float mh = __int_as_float(static_cast<int>(m_hi) + 0x4A800000);
  const int rem_i = static_cast<int>(rem);
  const float rem_f = __fadd_rn(__fmul_rn(magic_i2f(rem_i >> 6), 64.f), magic_i2f(rem_i & 63));
  float hi = __fmul_rn(mh, pow2f(e - 1046));  // exact: m_hi <= 2^24
  float lo = __fmul_rn(rem_f, pow2f(e - 1075));
  if (bits >> 63) {
    hi = -hi;
    lo = -lo;
  }
  const float p = __fmul_rn(hi, rcp.hi);
  float err = __fmaf_rn(hi, rcp.hi, -p);
  err = __fmaf_rn(hi, rcp.lo, err);
  err = __fmaf_rn(lo, rcp.hi, err);
  return __fadd_rn(p, err);
}

// Exact assignment of one query (warp-wide; x holds this lane's elements lane + 32 j):
// the valid beacon maximising (q . c_b) * (1 / |c_b|) in double-float arithmetic (exact
// products, TwoSum accumulation, then a butterfly over the lanes), ties to the lower
// beacon; -1 for a zero query or when no beacon is valid.  cent_at(b, col) reads centroid
// b; valid(b) is warp-uniform; cninv[b] is 1 / |c_b| (a pointer, or any type with that operator).
template <int D, typename CentAt, typename Valid, typename CnInv>
__device__ __forceinline__ int exact_decision(const float (&x)[D / 32], int nb, CentAt cent_at, Valid valid,
                                              const CnInv& cninv) {
  const int lane = threadIdx.x & 31;
  int nz = 0;
#pragma unroll
  for (int j = 0; j < D / 32; ++j) nz |= x[j] != 0.f;
  DF b1{-INFINITY, 0.f};
  int best_b = -1;
  if (__any_sync(0xffffffffu, nz))
    for (int b = 0; b < nb; ++b) {
      if (!valid(b)) continue;
      DF dt{0.f, 0.f};
#pragma unroll
      for (int j = 0; j < D / 32; ++j) dt = df_add(dt, df_two_prod(x[j], cent_at(b, lane + 32 * j)));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1)
        dt = df_add(dt, DF{__shfl_xor_sync(0xffffffffu, dt.hi, o), __shfl_xor_sync(0xffffffffu, dt.lo, o)});
      const DF cs = df_mul(dt, cninv[b]);
      if (best_b < 0 || df_gt(cs, b1)) {
        b1 = cs;
        best_b = b;
      }
    }
  return best_b;
}

}  // namespace
}  // namespace bkv
