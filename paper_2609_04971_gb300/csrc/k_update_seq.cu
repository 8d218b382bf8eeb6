// Beacon maintenance for a run of decode steps in one launch (Section 3.2,
// Appendix D: Algorithm 2's decode branch, one pre-RoPE query per query head
// per step).  Step t's queries are assigned against the centroids as steps
// 0 .. t-1 left them and folded into the running state before step t + 1.
// The result is, bit for bit, that of one few-query update per step
// (k_update_small.cu): the same exact re-decisions, exact fixed-point sums,
// fold and centroid arithmetic (k_update_math.cuh).
//
// Nothing reads the beacons between two compresses, so a decode loop can hand
// over the steps since the last compress at once.  One CTA of D / 32 warps
// takes one instance at a time (persistent CTAs walk the instances) and keeps
// its running sums and centroids in shared memory for all the steps: read from
// HBM once, written back once (rows of touched beacons only).  Warp w owns
// columns [32 w, 32 w + 32) of every beacon, so the per-step work splits by
// column:
//   queries: each warp loads its columns of the step's G queries (the next
//     step's are prefetched into registers) as fp32, with partial squared
//     norms;
//   screening: each warp forms, over its own columns, the partial squared norm
//     of every beacon's screening row and its partial dot with every query
//     (R lanes per row, packed fp32 multiply-adds); after a CTA barrier the
//     warp that decides query r adds the partials of the D / 32 warps (lane b:
//     beacon b), scales by rsqrtf of the squared norm and takes the best and
//     second best by warp reductions.  A cosine does not change when its
//     vector is scaled, so a beacon touched in this call screens with its
//     running sum (fp32, within 2^-23 relative per element) instead of its
//     centroid, and untouched beacons with their centroids;
//   decision: the best beacon (the lowest one on ties) unless best and second
//     best differ by at most 1e-4 |q| or a norm is extreme; such a close call
//     is re-decided exactly by that warp among the beacons screened within
//     2e-4 |q| of the best, with the few-query kernel's double-float
//     arithmetic on whole rows of exact centroids (recomputed from the sums
//     for touched beacons).  The screened values are within far less than
//     5e-5 |q| of the exact cosines whatever the rounding of the partial sums
//     and of the screening rows, so this decides as the few-query kernel
//     does: where its margin test passes, the screened best is the exact
//     maximum, and otherwise both take the exact argmax;
//   fold: after a second barrier, each lane folds its own column of every
//     touched beacon.  While a warp's running sums are below 2^18 in
//     magnitude and on the 2^-40 grid (what sums of bf16 queries of 2^-31 or
//     more are), each is held exactly as three fp32 parts h + m + l (h a
//     multiple of 2^-3, |m| <= 2^-4 a multiple of 2^-20, |l| <= 2^-21 a
//     multiple of 2^-40); a query element splits exactly into the same three
//     parts, so a step adds its rows with fp32 additions that are all exact
//     and carries between the parts.  That exact total is fold_sum's result
//     below 2^13; from 2^13 on fold_sum rounds it to its double's grid, and so
//     does the fold (the low part rounded).  The few-query kernel rounds
//     elements below 2^-31 (their sum over a beacon's rows, to a multiple of
//     2^-38); a step with such an element sums each beacon's rows first and
//     rounds likewise.  A warp whose columns leave that range (a sum reaching
//     2^18, or one that never was on the grid) keeps doubles and folds with
//     fold_sum.  Centroids are formed at the end, for the touched beacons,
//     from their final sums and counts (centroid_value's arithmetic, without
//     forming the double).
#include "bkv_device.cuh"
#include "bkv_internal.h"
#include "k_update_math.cuh"

namespace bkv {
namespace {

struct SeqArgs {
  int n_inst, nq, nb, n_steps;
  int lg_rows;               // log2 of the lanes that share one centroid row in the screening
  const __nv_bfloat16* q;    // [n_steps][n_inst * nq][D]
  float* cent;               // [n_inst][nb][D]
  double* sums;              // [n_inst][nb][D]
  long long* counts;         // [n_inst][nb]
  int* assign_out;           // [n_steps][n_inst * nq] or nullptr
};

// Shared memory of one CTA (one instance), byte offsets.
struct SeqLayout {
  size_t s, c, q, dots, norms, nzf, mode, qn2, dec, total;
};

__host__ __device__ inline SeqLayout seq_layout(int D, int NQ, int nb, int R) {
  const int W = D / 32;
  int nbp = 1;
  while (nbp < nb) nbp <<= 1;
  SeqLayout L;
  size_t o = 0;
  L.s = o;  // float [3][nb][D]: the parts h, m, l of each running sum (fp64 form: its bits in h and m)
  o += 12ull * nb * D;
  L.c = o;  // float [nb][D + 4R]: screening rows (centroids; fp32 running sums once touched)
  o += 4ull * nb * (D + 4 * R);
  L.q = o;  // float [NQ][D + 4]: the step's queries
  o += 4ull * NQ * (D + 4);
  L.dots = o;  // float [W][NQ][nbp]: partial dots (nbp: nb rounded up to a power of two)
  o += 4ull * W * NQ * nbp;
  L.norms = o;  // float [W][32]: partial squared norms of the screening rows
  o += 4ull * W * 32;
  L.nzf = o;  // uint32 [W]: bit b set when centroid b has a nonzero element among the warp's columns
  o += 4ull * W;
  L.mode = o;  // int [W]: the warp's columns hold integer sums (1) or fp64 sums (0)
  o += 4ull * W;
  L.qn2 = o;  // float [W][NQ]: partial squared norms of the queries
  o += 4ull * W * NQ;
  L.dec = o;  // int [NQ]: the step's decisions
  o += 4ull * NQ;
  L.total = (o + 15) / 16 * 16;
  return L;
}

__device__ __forceinline__ unsigned long long fma2(unsigned long long a, unsigned long long b, unsigned long long c) {
  unsigned long long d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ float sum2(unsigned long long v) {
  return __uint_as_float(static_cast<uint32_t>(v)) + __uint_as_float(static_cast<uint32_t>(v >> 32));
}

// Order-preserving key of a screened value (larger value, larger key); NaN and invalid lanes map to 0.
__device__ __forceinline__ uint32_t order_key(float v, bool valid) {
  const uint32_t u = __float_as_uint(v);
  const uint32_t k = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return (valid && !isnan(v)) ? k : 0u;
}
__device__ __forceinline__ float key_value(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// s as the integer s * 2^40 when s is +0 or a multiple of 2^-40 with |s| < 2^18 (then |S| < 2^58).
__device__ __forceinline__ bool to_fixed(double s, long long& f) {
  const unsigned long long bits = static_cast<unsigned long long>(__double_as_longlong(s));
  const int e = static_cast<int>((bits >> 52) & 0x7ff);
  f = 0;
  if (bits == 0ull) return true;
  if (e == 0 || e >= 1023 + 18) return false;  // -0, subnormal, or |s| >= 2^18
  const unsigned long long m = (bits & ((1ull << 52) - 1ull)) | (1ull << 52);
  const int sh = e - 1035;  // s * 2^40 = m * 2^(e - 1075 + 40)
  unsigned long long v;
  if (sh >= 0) {
    v = m << sh;
  } else if (sh > -53 && (m & ((1ull << -sh) - 1ull)) == 0ull) {
    v = m >> -sh;
  } else {
    return false;  // not a multiple of 2^-40
  }
  f = (bits >> 63) ? -static_cast<long long>(v) : static_cast<long long>(v);
  return true;
}

// The double S * 2^-40 (+0 for S = 0): fold_sum's result for that total (exact when S has at most 53
// significant bits).
__device__ __forceinline__ double from_fixed(long long S) { return S == 0 ? 0.0 : fixed40_round(S); }

// centroid_value(S * 2^-40, rcp) for an S of at most 53 significant bits (|S| < 2^63), without forming
// the double: for a = |S| with leading bit p, the double's 53-bit significand is a shifted to bit 52
// and its exponent field 983 + p, so centroid_value's split gives hi = m_hi * 2^(p - 63) and
// lo = rem * 2^(p - 92).
__device__ __forceinline__ float centroid_fixed(long long S, DF rcp) {
  const unsigned long long a = static_cast<unsigned long long>(S < 0 ? -S : S) | (S == 0 ? 1ull : 0ull);
  const int p = 63 - __clzll(static_cast<long long>(a));
  const unsigned long long m = p >= 52 ? a >> ((p - 52) & 63) : a << ((52 - p) & 63);
  const unsigned long long m_hi = (m + (1ull << 28) - 1 + ((m >> 29) & 1)) >> 29;
  const int rem_i = static_cast<int>(static_cast<long long>(m) - static_cast<long long>(m_hi << 29));
  const float mh = __int_as_float(static_cast<int>(m_hi) + 0x4A800000);
  const float rem_f = __fadd_rn(__fmul_rn(magic_i2f(rem_i >> 6), 64.f), magic_i2f(rem_i & 63));
  float hi = __fmul_rn(mh, pow2f(p - 63));
  float lo = __fmul_rn(rem_f, pow2f(p - 92));
  if (S < 0) {
    hi = -hi;
    lo = -lo;
  }
  const float pr = __fmul_rn(hi, rcp.hi);
  float err = __fmaf_rn(hi, rcp.hi, -pr);
  err = __fmaf_rn(hi, rcp.lo, err);
  err = __fmaf_rn(lo, rcp.hi, err);
  return S == 0 ? 0.f : __fadd_rn(pr, err);
}

// The exact split of a bf16 value (as parts_add makes it): h = x rounded to a multiple of 2^-3, m =
// the rest rounded to a multiple of 2^-20, l = what remains.
__device__ __forceinline__ void split3(float x, float& h, float& m, float& l) {
  h = __fadd_rn(__fadd_rn(x, 1572864.f), -1572864.f);
  const float r = __fadd_rn(x, -h);
  m = __fadd_rn(__fadd_rn(r, 12.f), -12.f);
  l = __fadd_rn(r, -m);
}

// Carries l's multiple of 2^-20 into m and m's multiple of 2^-3 into h, exactly: afterwards
// |m| <= 2^-4 and |l| <= 2^-21 (for |h| < 2^20, |m| < 2^19, |l| < 2^-16, each on its grid).
__device__ __forceinline__ void carry3(float& h, float& m, float& l) {
  const float lc = __fadd_rn(__fadd_rn(l, 12.f), -12.f);
  m = __fadd_rn(m, lc);
  l = __fadd_rn(l, -lc);
  const float mc = __fadd_rn(__fadd_rn(m, 1572864.f), -1572864.f);
  h = __fadd_rn(h, mc);
  m = __fadd_rn(m, -mc);
}

// (h + m + l) * 2^40 as an integer, for carried parts with |h| <= 2^19 (every conversion exact).
__device__ __forceinline__ long long parts_fixed(float h, float m, float l) {
  return (static_cast<long long>(magic_f2i(h * 8.f)) << 37) +
         (static_cast<long long>(magic_f2i(m * 1048576.f)) << 20) +
         static_cast<long long>(magic_f2i(l * 1099511627776.f));
}

// parts_fixed for |h| up to 2^20 (after a step that leaves the range): h by a conversion instruction.
__device__ __noinline__ long long parts_fixed_wide(float h, float m, float l) {
  return (__float2ll_rn(h * 8.f) << 37) + (static_cast<long long>(magic_f2i(m * 1048576.f)) << 20) +
         static_cast<long long>(magic_f2i(l * 1099511627776.f));
}

// Carried parts of S * 2^-40 for |S| < 2^58.
__device__ __forceinline__ void fixed_parts(long long S, float& h, float& m, float& l) {
  const long long hq = (S + (1ll << 36)) >> 37;
  const long long rem = S - (hq << 37);
  const long long mq = (rem + (1ll << 19)) >> 20;
  const long long lq = rem - (mq << 20);
  h = magic_i2f(static_cast<int>(hq)) * 0.125f;
  m = magic_i2f(static_cast<int>(mq)) * 9.5367431640625e-07f;          // 2^-20
  l = magic_i2f(static_cast<int>(lq)) * 9.094947017729282e-13f;        // 2^-40
}

// floor(log2 |h + m + l|) of carried parts with a nonzero total, from the exact integer.
__device__ __noinline__ int parts_exponent(float h, float m, float l) {
  const long long S = parts_fixed(h, m, l);
  return 23 - __clzll(S < 0 ? -S : S);  // (63 - clz) - 40
}

// From 2^13 on, a double's grid is coarser than 2^-40, and fold_sum rounds each step's exact total to
// it (to nearest, ties to even).  For carried parts of a total s with |s| < 2^18 (sv: s to within
// 2^-22 relative) that is the low part rounded to a multiple of 2^(e - 52), e = floor(log2 |s|): h and
// m are multiples of 2^-20, so they do not change, and the total's last kept bit is l's.  e is read
// from sv unless sv lies within 2^-19 relative of a power of two, where it is taken exactly.  The
// rounding adds and subtracts 1.5 * 2^(e - 29), whose ulp is the grid (|l| <= 2^-21 is far below it;
// the constant's even multiple of the grid keeps ties to even); below 2^13 it adds and subtracts 0.
__device__ __forceinline__ void round_to_double(float h, float m, float& l, float sv) {
  const uint32_t bits = __float_as_uint(sv);
  int e = static_cast<int>((bits >> 23) & 0xffu) - 127;
  const uint32_t man = bits & 0x7fffffu;
  if (e >= 12 && (man < 16u || man > 0x7fffefu)) e = parts_exponent(h, m, l);
  const float c = e >= 13 ? __uint_as_float((static_cast<uint32_t>(e + 98) << 23) | 0x400000u) : 0.f;
  l = __fadd_rn(__fadd_rn(l, c), -c);
}

// Per-beacon double-float values held by the lanes of a warp (lane b: beacon b); [b] reads beacon b's
// (b warp-uniform, every lane calling).
struct LaneDF {
  DF v;
  __device__ __forceinline__ DF operator[](int b) const {
    return DF{__shfl_sync(0xffffffffu, v.hi, b), __shfl_sync(0xffffffffu, v.lo, b)};
  }
};

// Shared-memory views of one CTA's instance.
struct SeqShared {
  float *Ph, *Pm, *Pl;  // parts of the running sums, [nb][D] each (fp64 form: bits in Ph and Pm)
  float* C;             // screening rows [nb][CP]
  float* Q;             // the step's queries [NQ][D + 4]
  int* mode;            // [W]: 1 while the warp's columns hold parts
  int CP;
};

// The exact centroid of (beacon b, column c) as the few-query kernel holds it after the steps so far:
// the loaded centroid until b is touched, then centroid_value of its running sum (rcp: 1 / count).
template <int D>
__device__ __forceinline__ float seq_exact_c(const SeqShared& sh, uint32_t touched_all, const LaneDF& rcp, int b, int c) {
  if (!((touched_all >> b) & 1u)) return sh.C[b * sh.CP + c];
  const int i = b * D + c;
  const DF rb = rcp[b];
  if (sh.mode[c >> 5]) return centroid_fixed(parts_fixed(sh.Ph[i], sh.Pm[i], sh.Pl[i]), rb);
  return centroid_value(__hiloint2double(__float_as_int(sh.Pm[i]), __float_as_int(sh.Ph[i])), rb);
}

// Exact re-decision of query r among the candidate beacons (warp-wide; lane b holds beacon b's count):
// the few-query kernel's double-float arithmetic on whole rows of exact centroids.  Out of line: rare.
template <int D>
__device__ __noinline__ int seq_exact(const SeqShared& sh, int r, uint32_t cand, int nb, uint32_t touched_all,
                                      long long cnt) {
  const int lane = threadIdx.x & 31;
  LaneDF rcp{count_reciprocal(cnt > 0 ? cnt : 1)}, cninv{DF{0.f, 0.f}};  // lane b: beacon b's 1 / count
  for (uint32_t m = cand; m; m &= m - 1) {
    const int b = __ffs(m) - 1;
    float n2b = 0.f;
    DF n2d{0.f, 0.f};
#pragma unroll
    for (int k = 0; k < D / 32; ++k) {
      const float c = seq_exact_c<D>(sh, touched_all, rcp, b, lane + 32 * k);
      n2b = fmaf(c, c, n2b);
      n2d = df_add(n2d, df_two_prod(c, c));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) n2b += __shfl_xor_sync(0xffffffffu, n2b, o);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
      n2d = df_add(n2d, DF{__shfl_xor_sync(0xffffffffu, n2d.hi, o), __shfl_xor_sync(0xffffffffu, n2d.lo, o)});
    bool plain = true;
    const DF inv_df = centroid_inv_norm(n2d, n2b, plain);
    if (lane == b) cninv.v = inv_df;
  }
  float x[D / 32];
#pragma unroll
  for (int j = 0; j < D / 32; ++j) x[j] = sh.Q[r * (D + 4) + lane + 32 * j];
  const int d = exact_decision<D>(
      x, nb, [&](int b, int c) { return seq_exact_c<D>(sh, touched_all, rcp, b, c); },
      [&](int b) { return ((cand >> b) & 1u) != 0; }, cninv);
  return d;
}

// Partial dots of the warp's 32 columns of every screening row with every query, and the rows' partial
// squared norms: R lanes per row, lane (row, part) taking 16-byte chunks part, part + R, ... (packed fp32
// multiply-adds, two columns per instruction); the R lanes' partials added by a butterfly.  Query rows
// past the call's nq are zero.
template <int D, int NQ, int R>
__device__ __forceinline__ void seq_screen(const float* crow, const float* qw, float (&acc)[NQ], float& n2) {
  unsigned long long acc2[NQ];
#pragma unroll
  for (int r = 0; r < NQ; ++r) acc2[r] = 0ull;
  unsigned long long n2p = 0ull;
  const int part = threadIdx.x & (R - 1);
#pragma unroll
  for (int i = 0; i < 8 / R; ++i) {
    const int k = part + R * i;
    const ulonglong2 c = *reinterpret_cast<const ulonglong2*>(crow + 4 * k);
    n2p = fma2(c.x, c.x, n2p);
    n2p = fma2(c.y, c.y, n2p);
#pragma unroll
    for (int r = 0; r < NQ; ++r) {
      const ulonglong2 x = *reinterpret_cast<const ulonglong2*>(qw + r * (D + 4) + 4 * k);
      acc2[r] = fma2(x.x, c.x, acc2[r]);
      acc2[r] = fma2(x.y, c.y, acc2[r]);
    }
  }
#pragma unroll
  for (int r = 0; r < NQ; ++r) acc[r] = sum2(acc2[r]);
  n2 = sum2(n2p);
#pragma unroll
  for (int o = 1; o < R; o <<= 1) {
    n2 += __shfl_xor_sync(0xffffffffu, n2, o);
#pragma unroll
    for (int r = 0; r < NQ; ++r) acc[r] += __shfl_xor_sync(0xffffffffu, acc[r], o);
  }
}

template <int D, int NQ>
__global__ void __launch_bounds__(D, (NQ <= 8 ? 6 : 3) * 128 / D) update_seq_kernel(SeqArgs a) {
  constexpr int W = D / 32;  // warps per CTA; warp w owns columns [32 w, 32 w + 32)
  constexpr int QP = D + 4;  // query row pitch (floats)
  constexpr int QU = NQ / 4; // 8-byte query loads per lane and step: NQ rows x 32 columns per warp
  static_assert(NQ % 4 == 0, "query loads of 4 columns, 8 lanes per row");
  extern __shared__ __align__(16) unsigned char seq_sh[];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nb = a.nb, nq = a.nq;
  const int lg_r = a.lg_rows;
  const int row = lane >> lg_r;
  const bool has_row = row < nb;
  const int CP = D + (4 << lg_r);  // screening row pitch (floats): R lanes' 16-byte reads conflict-free
  const int col = 32 * w + lane;   // this lane's column in the fold
  int nbp = 1;                     // nb rounded up to a power of two: the partial dots' row pitch
  while (nbp < nb) nbp <<= 1;
  const SeqLayout lay = seq_layout(D, NQ, nb, 1 << lg_r);
  SeqShared sh;
  sh.Ph = reinterpret_cast<float*>(seq_sh + lay.s);
  sh.Pm = sh.Ph + nb * D;
  sh.Pl = sh.Pm + nb * D;
  sh.C = reinterpret_cast<float*>(seq_sh + lay.c);
  sh.Q = reinterpret_cast<float*>(seq_sh + lay.q);
  sh.mode = reinterpret_cast<int*>(seq_sh + lay.mode);
  sh.CP = CP;
  float* const Ph = sh.Ph;
  float* const Pm = sh.Pm;
  float* const Pl = sh.Pl;
  float* const C_sh = sh.C;
  float* const Q_sh = sh.Q;
  float* dots = reinterpret_cast<float*>(seq_sh + lay.dots);
  float* norms = reinterpret_cast<float*>(seq_sh + lay.norms);
  uint32_t* nzw = reinterpret_cast<uint32_t*>(seq_sh + lay.nzf);  // [W]: the warps' nonzero masks
  float* qn2p = reinterpret_cast<float*>(seq_sh + lay.qn2);
  int* dec_sh = reinterpret_cast<int*>(seq_sh + lay.dec);
  const size_t step_elems = static_cast<size_t>(a.n_inst) * nq * D;  // one step's query block
  // a running sum in fp64 form: its bits in the h and m slots
  auto get_d = [&](int i) { return __hiloint2double(__float_as_int(Pm[i]), __float_as_int(Ph[i])); };
  auto put_d = [&](int i, double v) {
    Ph[i] = __int_as_float(__double2loint(v));
    Pm[i] = __int_as_float(__double2hiint(v));
  };

  for (int e = blockIdx.x; e < a.n_inst; e += gridDim.x) {
    const size_t cbase = static_cast<size_t>(e) * nb * D;
    // ---- this warp's columns of the instance's state (4 beacons' loads in flight per lane); the sums
    // in parts when every one of them allows it.  nzbits bit b: this lane's element of centroid b is
    // nonzero (so the beacon's centroid is nonzero iff some lane of some warp has the bit)
    bool ok = true;
    uint32_t nzbits = 0;
    for (int b0 = 0; b0 < nb; b0 += 4) {
      double sv[4];
      float cv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const size_t g = cbase + static_cast<size_t>(b0 + i < nb ? b0 + i : b0) * D + col;
        sv[i] = a.sums[g];
        cv[i] = a.cent[g];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int b = b0 + i;
        if (b < nb) {
          C_sh[b * CP + col] = cv[i];
          long long f;
          ok &= to_fixed(sv[i], f);
          put_d(b * D + col, sv[i]);
          nzbits |= (cv[i] != 0.f ? 1u : 0u) << b;
        }
      }
    }
    bool fixed = __all_sync(0xffffffffu, ok);
    if (fixed)
      for (int b = 0; b < nb; ++b) {
        const int i = b * D + col;
        long long f;
        to_fixed(get_d(i), f);
        float h, m, l;
        fixed_parts(f, h, m, l);
        Ph[i] = h;
        Pm[i] = m;
        Pl[i] = l;
      }
    if (lane == 0) sh.mode[w] = fixed;
    // lane b: beacon b's count at call start and what the steps added
    const long long cnt_base = lane < nb ? a.counts[static_cast<size_t>(e) * nb + lane] : 0;
    const bool base_pos = cnt_base > 0;
    int cnt_add = 0;
    auto count_of = [&](int b) { return __shfl_sync(0xffffffffu, cnt_base + cnt_add, b); };
    uint32_t touched_all = 0;  // beacons touched by this call (the same in every warp)
    int* assign = a.assign_out ? a.assign_out + static_cast<size_t>(e) * nq : nullptr;  // step 0's row

    // query loads: unit u = lane + 32 k is row u / 8, columns 32 w + 4 (u % 8) .. + 3
    const __nv_bfloat16* qn = a.q + static_cast<size_t>(e) * nq * D + 32 * w;
    uint2 qv[QU];
#pragma unroll
    for (int k = 0; k < QU; ++k) {
      const int u = lane + 32 * k, r = u >> 3;
      qv[k] = r < nq ? *reinterpret_cast<const uint2*>(qn + r * D + 4 * (u & 7)) : make_uint2(0u, 0u);
    }

    for (int t = 0; t < a.n_steps; ++t) {
      // ---- the step's queries (this warp's columns) to shared memory, partial norms; the next step's loads
#pragma unroll
      for (int k = 0; k < QU; ++k) {
        const int u = lane + 32 * k, r = u >> 3;
        const uint2 v = qv[k];
        const float4 x = make_float4(__uint_as_float(v.x << 16), __uint_as_float(v.x & 0xffff0000u),
                                     __uint_as_float(v.y << 16), __uint_as_float(v.y & 0xffff0000u));
        *reinterpret_cast<float4*>(Q_sh + r * QP + 32 * w + 4 * (u & 7)) = x;
        float p = x.x * x.x;
        p = fmaf(x.y, x.y, p);
        p = fmaf(x.z, x.z, p);
        p = fmaf(x.w, x.w, p);
        p += __shfl_xor_sync(0xffffffffu, p, 1);
        p += __shfl_xor_sync(0xffffffffu, p, 2);
        p += __shfl_xor_sync(0xffffffffu, p, 4);
        if ((u & 7) == 0) qn2p[w * NQ + r] = p;
      }
      if (t + 1 < a.n_steps) {
        qn += step_elems;
#pragma unroll
        for (int k = 0; k < QU; ++k) {
          const int u = lane + 32 * k, r = u >> 3;
          qv[k] = r < nq ? *reinterpret_cast<const uint2*>(qn + r * D + 4 * (u & 7)) : make_uint2(0u, 0u);
        }
      }
      __syncwarp();

      // ---- screening over this warp's columns
      {
        float acc[NQ], n2;
        const float* crow = C_sh + (has_row ? row : 0) * CP + 32 * w;
        const float* qw = Q_sh + 32 * w;
        switch (lg_r) {
          case 0: seq_screen<D, NQ, 1>(crow, qw, acc, n2); break;
          case 1: seq_screen<D, NQ, 2>(crow, qw, acc, n2); break;
          case 2: seq_screen<D, NQ, 4>(crow, qw, acc, n2); break;
          default: seq_screen<D, NQ, 8>(crow, qw, acc, n2); break;
        }
        if ((lane & ((1 << lg_r) - 1)) == 0 && has_row) {
#pragma unroll
          for (int r = 0; r < NQ; ++r) dots[(w * NQ + r) * nbp + row] = acc[r];
          norms[w * 32 + row] = n2;
        }
        const uint32_t nzm = __reduce_or_sync(0xffffffffu, nzbits);
        if (lane == 0) nzw[w] = nzm;
      }
      __syncthreads();  // A: partials, and every warp's columns of the queries and the state

      // ---- decisions: warp w takes queries w, w + W, ...; lane b holds beacon b
      {
        float n2 = 0.f;
        uint32_t nzm = 0;
#pragma unroll
        for (int v = 0; v < W; ++v) {
          n2 += norms[v * 32 + lane];
          nzm |= nzw[v];
        }
        const bool valid = lane < nb && (base_pos || cnt_add > 0) && ((nzm >> lane) & 1u);  // count > 0, nonzero centroid
        const uint32_t vmask = __ballot_sync(0xffffffffu, valid);
        const bool degenerate = __any_sync(0xffffffffu, valid && !(n2 > 1e-30f && n2 < 1e30f));
        const float inv = valid ? rsqrtf(n2) : 0.f;
        for (int r = w; r < nq; r += W) {
          float qn2 = 0.f, dot = 0.f;
#pragma unroll
          for (int v = 0; v < W; ++v) {
            qn2 += qn2p[v * NQ + r];
            dot += lane < nb ? dots[(v * NQ + r) * nbp + lane] : 0.f;
          }
          const float val = valid ? dot * inv : -INFINITY;
          const uint32_t key = order_key(val, valid);
          const uint32_t kmax = __reduce_max_sync(0xffffffffu, key);
          const uint32_t at_max = __ballot_sync(0xffffffffu, key == kmax && kmax != 0u);
          int dec = at_max ? __ffs(at_max) - 1 : -1;  // the lowest beacon on ties
          const uint32_t k2 = __reduce_max_sync(0xffffffffu, lane == dec ? 0u : key);
          const float best = kmax ? key_value(kmax) : -INFINITY;
          const float second = k2 ? key_value(k2) : -INFINITY;
          const bool wild = degenerate || !(qn2 > 1e-30f && qn2 < 1e30f);
          // |q| to within a few ulps (the margin has ample room for it)
          const float margin = kMarginRel * (qn2 * rsqrtf(qn2));
          // with a valid beacon but no screened best (every value NaN: an extreme norm), best - second is NaN
          if (vmask != 0u && (wild || !(best - second > margin))) {  // warp-uniform
            // candidates: a screened value is within kMarginRel |q| / 2 of the exact one, so only beacons
            // screened within 2 kMarginRel |q| of the best can have the largest exact value
            const uint32_t cand = wild ? vmask : __ballot_sync(0xffffffffu, valid && val >= best - 2.f * margin);
            dec = seq_exact<D>(sh, r, cand, nb, touched_all, cnt_base + cnt_add);
          }
          if (lane == 0) {
            dec_sh[r] = dec;
            if (assign) assign[r] = dec;
          }
        }
      }
      __syncthreads();  // B: the decisions; every read of other warps' columns is done
      if (assign) assign += static_cast<size_t>(a.n_inst) * nq;

      // ---- fold: lane `col` of every touched beacon
      {
        const int decr = lane < nq ? dec_sh[lane] : -1;  // lane r: query r's beacon
        const uint32_t touched = __reduce_or_sync(0xffffffffu, decr >= 0 ? (1u << decr) : 0u);
        touched_all |= touched;
        bool out = false;  // a sum reaching 2^18 in parts form
        int tiny = 0;
#pragma unroll
        for (int r = 0; r < NQ; ++r) {
          const float x = Q_sh[r * QP + col];
          tiny |= (x != 0.f && fabsf(x) < 4.656612873077393e-10f);  // 2^-31
        }
        if (fixed && !__any_sync(0xffffffffu, tiny)) {
          // every row added into its beacon's parts in row order and carried (all exact)
#pragma unroll
          for (int r = 0; r < NQ; ++r) {
            const int b = __shfl_sync(0xffffffffu, decr, r);
            if (b >= 0) {  // warp-uniform (rows past nq have b = -1)
              const int i = b * D + col;
              float xh, xm, xl;
              split3(Q_sh[r * QP + col], xh, xm, xl);
              float h = __fadd_rn(Ph[i], xh), mm = __fadd_rn(Pm[i], xm), l = __fadd_rn(Pl[i], xl);
              carry3(h, mm, l);
              const float sv = __fadd_rn(__fadd_rn(h, mm), l);  // the sum within 2^-22 relative; 0 iff it is 0
              // the centroid is 0 iff the sum is; sums from 2^13 on are rounded to their double's grid
              if (__any_sync(0xffffffffu, fabsf(sv) >= 8191.f || sv == 0.f)) {
                round_to_double(h, mm, l, sv);
                out |= fabsf(sv) >= 262143.f;
                nzbits = (nzbits & ~(1u << b)) | ((sv != 0.f ? 1u : 0u) << b);
              } else {
                nzbits |= 1u << b;
              }
              Ph[i] = h;
              Pm[i] = mm;
              Pl[i] = l;
              C_sh[b * CP + col] = sv;
              if (lane == b) ++cnt_add;
            }
          }
        } else {
          for (uint32_t m = touched; m; m &= m - 1) {
            const int b = __ffs(m) - 1;
            const int i = b * D + col;
            const uint32_t rows = __ballot_sync(0xffffffffu, lane < nq && decr == b);
            if (lane == b) cnt_add += __popc(rows);
            // the beacon's rows split and summed part by part in row order, as parts_add sums them (exact,
            // but for elements below 2^-31, whose low-part sum fixed40_few rounds to a multiple of 2^-38)
            float hs = 0.f, ms = 0.f, ls = 0.f;
            for (uint32_t mr = rows; mr; mr &= mr - 1) {
              float xh, xm, xl;
              split3(Q_sh[(__ffs(mr) - 1) * QP + col], xh, xm, xl);
              hs = __fadd_rn(hs, xh);
              ms = __fadd_rn(ms, xm);
              ls = __fadd_rn(ls, xl);
            }
            float c;
            if (fixed) {
              ls = magic_i2f(magic_f2i(ls * 274877906944.f)) * 3.637978807091713e-12f;  // to 2^-38, as fixed40_few
              const float lc = __fadd_rn(__fadd_rn(ls, 12.f), -12.f);  // its multiple of 2^-20 into ms
              ms = __fadd_rn(ms, lc);
              ls = __fadd_rn(ls, -lc);
              float h = __fadd_rn(Ph[i], hs), mm = __fadd_rn(Pm[i], ms), l = __fadd_rn(Pl[i], ls);
              carry3(h, mm, l);
              c = __fadd_rn(__fadd_rn(h, mm), l);
              if (__any_sync(0xffffffffu, fabsf(c) >= 8191.f)) round_to_double(h, mm, l, c);
              Ph[i] = h;
              Pm[i] = mm;
              Pl[i] = l;
              out |= fabsf(c) >= 262143.f;
              C_sh[b * CP + col] = c;
            } else {
              const double s_new = fold_sum(get_d(i), fixed40_few(Parts{hs, ms, ls}));
              put_d(i, s_new);
              C_sh[b * CP + col] = __double2float_rn(s_new);
              c = centroid_value(s_new, count_reciprocal(count_of(b)));
            }
            nzbits = (nzbits & ~(1u << b)) | ((c != 0.f ? 1u : 0u) << b);
          }
        }
        if (fixed && __any_sync(0xffffffffu, out)) {
          // a sum reached 2^18: this warp's columns go to fp64 form for good.  The parts hold the
          // running sums exactly (each on its double's grid)
          for (int b = 0; b < nb; ++b) {
            const int i = b * D + col;
            put_d(i, from_fixed(parts_fixed_wide(Ph[i], Pm[i], Pl[i])));
          }
          fixed = false;
          if (lane == 0) sh.mode[w] = 0;
          for (uint32_t m = touched; m; m &= m - 1) {
            const int b = __ffs(m) - 1;
            const double sv = get_d(b * D + col);
            C_sh[b * CP + col] = __double2float_rn(sv);
            const float c = centroid_value(sv, count_reciprocal(count_of(b)));
            nzbits = (nzbits & ~(1u << b)) | ((c != 0.f ? 1u : 0u) << b);
          }
        }
      }
      // the next step's writes (queries, partials, decisions) come after barrier B of this step, and
      // every read of another warp's columns of the state after barrier A of the next one
    }

    // ---- write back this warp's columns of the touched beacons: sums, and centroids from the final
    // sums and counts; the counts
    for (uint32_t m = touched_all; m; m &= m - 1) {
      const int b = __ffs(m) - 1;
      const DF rb = count_reciprocal(count_of(b));
      const int i = b * D + col;
      const size_t g = cbase + static_cast<size_t>(b) * D + col;
      if (fixed) {
        const long long S = parts_fixed(Ph[i], Pm[i], Pl[i]);
        a.sums[g] = from_fixed(S);
        a.cent[g] = centroid_fixed(S, rb);
      } else {
        const double sv = get_d(i);
        a.sums[g] = sv;
        a.cent[g] = centroid_value(sv, rb);
      }
    }
    if (w == 0 && lane < nb) a.counts[static_cast<size_t>(e) * nb + lane] = cnt_base + cnt_add;
    __syncthreads();  // the next instance's loads overwrite the state that other warps read last
  }
}

template <int D, int NQ>
cudaError_t launch_seq_dq(const SeqArgs& a, int sms, cudaStream_t st) {
  const SeqLayout lay = seq_layout(D, NQ, a.nb, 1 << a.lg_rows);
  if (lay.total > 227 * 1024) return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(update_seq_kernel<D, NQ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(lay.total));
  if (e == cudaSuccess)  // all of the SM's on-chip memory as shared memory: the CTAs per SM are smem-bound
    e = cudaFuncSetAttribute(update_seq_kernel<D, NQ>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, update_seq_kernel<D, NQ>, D, lay.total);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorInvalidValue;
  const long long slots = 1ll * per_sm * sms;
  const int grid = static_cast<int>(a.n_inst < slots ? a.n_inst : slots);
  update_seq_kernel<D, NQ><<<grid, D, lay.total, st>>>(a);
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_seq_d(const SeqArgs& a, int sms, cudaStream_t st) {
  if (a.nq <= 4) return launch_seq_dq<D, 4>(a, sms, st);
  if (a.nq <= 8) return launch_seq_dq<D, 8>(a, sms, st);
  if (a.nq <= 16) return launch_seq_dq<D, 16>(a, sms, st);
  return launch_seq_dq<D, 32>(a, sms, st);
}

}  // namespace

cudaError_t launch_update_seq(const Shape& s, const __nv_bfloat16* q_steps, int n_steps, float* cent, double* sums,
                              long long* counts, int* assign_out, cudaStream_t st) {
  if (s.n_inst == 0 || n_steps == 0 || s.nb == 0) return cudaSuccess;
  if (s.G > kUpdateSmallMaxRows || s.nb > kMaxBeacons) return cudaErrorInvalidValue;
  int lg = 0;
  while ((32 >> (lg + 1)) >= s.nb && lg < 3) ++lg;  // 2^lg lanes per row, 2^lg * nb <= 32
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  SeqArgs a{s.n_inst, s.G, s.nb, n_steps, lg, q_steps, cent, sums, counts, assign_out};
  return s.d == 128 ? launch_seq_d<128>(a, sms, st) : launch_seq_d<64>(a, sms, st);
}

}  // namespace bkv
