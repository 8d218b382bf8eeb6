// Checks the beacon update's integer fold (fold_sum in k_update_math.cuh) against the fp64
// route it replaces, __dadd_rn(s, acc * 2^-40), on deterministic adversarial inputs:
//   grid    s a multiple of 2^-40 of every exponent below 2^22, |acc| < 2^53 (both exact
//           paths): results must be bit-identical;
//   halves  sums that land exactly halfway between two doubles (ties to even);
//   large   2^53 <= |acc| < 2^61 (the fp64 route rounds acc * 2^-40 first, which under
//           cancellation can miss by several ulps): bit-identical to the correctly rounded
//           sum, formed on the host from the exact integer s * 2^40 + acc;
//   off     s off the 2^-40 grid, at or beyond 2^22, subnormal or zero (the fp64 route):
//           bit-identical.
// fold_sum_fp64 (the batched kernel's form) must equal fold_sum bit for bit on every input;
// fixed40_few must equal fixed40 on sums of up to 32 values, fixed40_one on single values of every
// exponent; centroid_value must be within one fp32 ulp of s / n.
// Prints one line per class and exits non-zero on any mismatch.  Test code only.
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <vector>

#include "k_update_math.cuh"

namespace {

__global__ void fold_kernel(const double* s, const long long* acc, double* got, double* want, double* got64, int n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  got[i] = bkv::fold_sum(s[i], acc[i]);
  got64[i] = bkv::fold_sum_fp64(s[i], acc[i]);
  want[i] = acc[i] == 0 ? s[i] : __dadd_rn(s[i], bkv::fixed40_to_double(acc[i]));
}

// fixed40_few (magic-number conversions) against fixed40 (conversion instructions) on the part sums
// of up to 32 bf16-exact values, and centroid_value against the exactly computed quotient.
__global__ void parts_kernel(const float* x, int rows, int n, long long* few, long long* ref) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  bkv::Parts p{0.f, 0.f, 0.f};
  for (int r = 0; r < rows; ++r) bkv::parts_add(p, x[static_cast<size_t>(i) * rows + r]);
  few[i] = bkv::fixed40_few(p);
  ref[i] = bkv::fixed40(p);
}

// fixed40_one (integer operations on the bits) against fixed40 of the parts of one value
__global__ void one_kernel(const float* x, int n, long long* one, long long* ref) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  bkv::Parts p{0.f, 0.f, 0.f};
  bkv::parts_add(p, x[i]);
  one[i] = bkv::fixed40_one(x[i]);
  ref[i] = bkv::fixed40(p);
}

__global__ void centroid_kernel(const double* s, const long long* cnt, float* got, int n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  got[i] = bkv::centroid_value(s[i], bkv::count_reciprocal(cnt[i]));
}

uint64_t rng_state = 0x9e3779b97f4a7c15ull;
uint64_t next() {  // xorshift64*
  rng_state ^= rng_state >> 12;
  rng_state ^= rng_state << 25;
  rng_state ^= rng_state >> 27;
  return rng_state * 2685821657736338717ull;
}

double from_bits(uint64_t b) {
  double d;
  std::memcpy(&d, &b, sizeof d);
  return d;
}
uint64_t to_bits(double d) {
  uint64_t b;
  std::memcpy(&b, &d, sizeof b);
  return b;
}

// a multiple of 2^-40 with its leading bit at 2^k (k in [-40, 21]), random sign
double grid_value(int k) {
  const int bits = k + 40 + 1;  // significant bits available above 2^-40
  const int nb = bits < 53 ? bits : 53;
  uint64_t m = (next() >> (64 - nb)) | (1ull << (nb - 1));
  double v = static_cast<double>(m);
  v = std::ldexp(v, k - (nb - 1));
  return (next() & 1) ? -v : v;
}

}  // namespace

int main() {
  std::vector<double> s;
  std::vector<long long> acc;
  std::vector<int> cls;  // 0 grid, 1 halves, 2 large, 3 off
  for (int i = 0; i < 200000; ++i) {
    const int k = -40 + static_cast<int>(next() % 62);
    s.push_back(grid_value(k));
    const int ka = static_cast<int>(next() % 53);
    long long a = static_cast<long long>(next() >> (64 - ka - 1));
    if (next() & 1) a = -a;
    acc.push_back(a);
    cls.push_back(0);
  }
  for (int i = 0; i < 50000; ++i) {  // s + acc * 2^-40 exactly between two doubles of magnitude ~2^13..2^21
    const int k = 13 + static_cast<int>(next() % 8);
    const double base = std::ldexp(static_cast<double>((next() >> 12) | (1ull << 52)), k - 52);  // ulp 2^(k-52)
    const int ulp_exp = k - 52 + 40;                                                             // in 2^-40 units
    s.push_back((next() & 1) ? -base : base);
    long long half = 1LL << (ulp_exp - 1);
    long long a = half * static_cast<long long>(1 + 2 * (next() % 1000));
    if (next() & 1) a = -a;
    acc.push_back(a);
    cls.push_back(1);
  }
  for (int i = 0; i < 50000; ++i) {
    s.push_back(grid_value(-40 + static_cast<int>(next() % 62)));
    const int ka = 53 + static_cast<int>(next() % 8);
    long long a = static_cast<long long>((next() >> (64 - ka - 1)) | (1ull << ka));
    acc.push_back((next() & 1) ? -a : a);
    cls.push_back(2);
  }
  for (int i = 0; i < 50000; ++i) {
    double v;
    switch (i % 5) {
      case 0: v = std::ldexp(static_cast<double>((next() >> 11) | 1ull), -60); break;  // off the grid
      case 1: v = grid_value(22 + static_cast<int>(next() % 20)); break;                // at or beyond 2^22
      case 2: v = from_bits(next() >> 12); break;                                        // subnormal
      case 3: v = (next() & 1) ? -0.0 : 0.0; break;
      default: v = from_bits(next() & ~(0x7ffull << 52) | (static_cast<uint64_t>(900 + next() % 300) << 52));
    }
    s.push_back(v);
    long long a = static_cast<long long>(next() >> 12);
    acc.push_back((next() & 1) ? -a : a);
    cls.push_back(3);
  }
  const int n = static_cast<int>(s.size());
  double *ds, *dg, *dw, *dg64;
  long long* da;
  cudaMalloc(&dg64, sizeof(double) * n);
  cudaMalloc(&ds, sizeof(double) * n);
  cudaMalloc(&dg, sizeof(double) * n);
  cudaMalloc(&dw, sizeof(double) * n);
  cudaMalloc(&da, sizeof(long long) * n);
  cudaMemcpy(ds, s.data(), sizeof(double) * n, cudaMemcpyHostToDevice);
  cudaMemcpy(da, acc.data(), sizeof(long long) * n, cudaMemcpyHostToDevice);
  fold_kernel<<<(n + 255) / 256, 256>>>(ds, da, dg, dw, dg64, n);
  std::vector<double> got(n), want(n), want_route, got64(n);
  cudaError_t e = cudaMemcpy(got.data(), dg, sizeof(double) * n, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemcpy(want.data(), dw, sizeof(double) * n, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemcpy(got64.data(), dg64, sizeof(double) * n, cudaMemcpyDeviceToHost);
  want_route = want;
  if (e != cudaSuccess) {
    std::printf("CUDA error: %s\n", cudaGetErrorString(e));
    return 2;
  }
  long long count[4] = {}, bad[4] = {};
  for (int i = 0; i < n; ++i) {
    const int c = cls[i];
    ++count[c];
    if (c == 2) {
      // s is a multiple of 2^-40 below 2^22: s * 2^40 is an exact integer; the int64 -> double
      // conversion rounds to nearest even, and the scaling by 2^-40 is exact
      const long long t = static_cast<long long>(s[i] * 1099511627776.0) + acc[i];
      want[i] = std::ldexp(static_cast<double>(t), -40);
    }
    const uint64_t g = to_bits(got[i]), w = to_bits(want[i]);
    if (g == w) continue;
    if (bad[c] < 3)
      std::printf("class %d: s=%.17g acc=%lld got=%.17g want=%.17g\n", c, s[i], acc[i], got[i], want[i]);
    ++bad[c];
  }
  const char* names[4] = {"grid", "halves", "large (against the exact sum)", "off"};
  int fail = 0;
  for (int c = 0; c < 4; ++c) {
    std::printf("%s: %lld cases, %lld mismatches\n", names[c], count[c], bad[c]);
    fail |= bad[c] != 0;
  }
  // how often the fp64 route it replaces misses the exact sum in the large class
  long long route_off = 0;
  for (int i = 0; i < n; ++i) {
    if (cls[i] != 2) continue;
    const long long t = static_cast<long long>(s[i] * 1099511627776.0) + acc[i];
    route_off += to_bits(std::ldexp(static_cast<double>(t), -40)) != to_bits(want_route[i]);
  }
  std::printf("fp64 route (rounds twice) off the exact sum in the large class: %lld of %lld\n", route_off, count[2]);
  long long forms_differ = 0;
  for (int i = 0; i < n; ++i) forms_differ += to_bits(got[i]) != to_bits(got64[i]);
  std::printf("fold_sum_fp64 differs from fold_sum: %lld of %d\n", forms_differ, n);
  fail |= forms_differ != 0;
  // ---- fixed40_few against fixed40: 100000 sets of up to 32 values, |x| < 2^14, bf16-exact
  {
    const int sets = 100000, rows = 32;
    std::vector<float> xs(static_cast<size_t>(sets) * rows);
    for (int i = 0; i < sets; ++i)
      for (int r = 0; r < rows; ++r) {
        const int e = -34 + static_cast<int>(next() % 48);                    // 2^-34 .. 2^13
        const float m = static_cast<float>(128 + (next() % 128)) / 128.f;   // 8 significant bits
        float v = std::ldexp(m, e);
        if (next() & 1) v = -v;
        if (i % 7 == 0) v = (r % 2 ? 1.f : -1.f) * std::ldexp(255.f / 128.f, 13);  // extremes, alternating
        if (i % 11 == 0) v = std::ldexp(255.f / 128.f, 13);                         // all at the maximum
        xs[static_cast<size_t>(i) * rows + r] = v;
      }
    float* dx;
    long long *dfew, *dref;
    cudaMalloc(&dx, sizeof(float) * xs.size());
    cudaMalloc(&dfew, sizeof(long long) * sets);
    cudaMalloc(&dref, sizeof(long long) * sets);
    cudaMemcpy(dx, xs.data(), sizeof(float) * xs.size(), cudaMemcpyHostToDevice);
    parts_kernel<<<(sets + 255) / 256, 256>>>(dx, rows, sets, dfew, dref);
    std::vector<long long> hf(sets), hr(sets);
    cudaMemcpy(hf.data(), dfew, sizeof(long long) * sets, cudaMemcpyDeviceToHost);
    cudaMemcpy(hr.data(), dref, sizeof(long long) * sets, cudaMemcpyDeviceToHost);
    long long diff = 0;
    for (int i = 0; i < sets; ++i) diff += hf[i] != hr[i];
    std::printf("fixed40_few differs from fixed40: %lld of %d sets of %d values\n", diff, sets, rows);
    fail |= diff != 0;
    cudaFree(dx);
    cudaFree(dfew);
    cudaFree(dref);
  }
  // ---- fixed40_one against fixed40 on single bf16-exact values of every exponent (2^-140 .. 2^13)
  {
    std::vector<float> xs;
    for (int e = -140; e <= 13; ++e)
      for (int k = 0; k < 128; ++k) {
        const float v = std::ldexp(static_cast<float>(128 + k) / 128.f, e);
        xs.push_back(v);
        xs.push_back(-v);
      }
    xs.push_back(0.f);
    xs.push_back(-0.f);
    const int n1 = static_cast<int>(xs.size());
    float* dx;
    long long *d1, *dr;
    cudaMalloc(&dx, sizeof(float) * n1);
    cudaMalloc(&d1, sizeof(long long) * n1);
    cudaMalloc(&dr, sizeof(long long) * n1);
    cudaMemcpy(dx, xs.data(), sizeof(float) * n1, cudaMemcpyHostToDevice);
    one_kernel<<<(n1 + 255) / 256, 256>>>(dx, n1, d1, dr);
    std::vector<long long> h1(n1), hr(n1);
    cudaMemcpy(h1.data(), d1, sizeof(long long) * n1, cudaMemcpyDeviceToHost);
    cudaMemcpy(hr.data(), dr, sizeof(long long) * n1, cudaMemcpyDeviceToHost);
    long long diff = 0;
    for (int i = 0; i < n1; ++i) {
      if (h1[i] != hr[i] && diff < 3) std::printf("  x = %g: one %lld, parts %lld\n", xs[i], h1[i], hr[i]);
      diff += h1[i] != hr[i];
    }
    std::printf("fixed40_one differs from fixed40 of one value: %lld of %d\n", diff, n1);
    fail |= diff != 0;
    cudaFree(dx);
    cudaFree(d1);
    cudaFree(dr);
  }
  // ---- centroid_value within one fp32 ulp of s / n (host: the fp64 quotient, then fp32)
  {
    const int m = 200000;
    std::vector<double> cs(m);
    std::vector<long long> cn(m);
    for (int i = 0; i < m; ++i) {
      cs[i] = grid_value(-40 + static_cast<int>(next() % 62));
      cn[i] = 1 + static_cast<long long>(next() % (i % 3 == 0 ? 100 : (i % 3 == 1 ? 100000 : 10000000)));
    }
    double* dcs;
    long long* dcn;
    float* dcg;
    cudaMalloc(&dcs, sizeof(double) * m);
    cudaMalloc(&dcn, sizeof(long long) * m);
    cudaMalloc(&dcg, sizeof(float) * m);
    cudaMemcpy(dcs, cs.data(), sizeof(double) * m, cudaMemcpyHostToDevice);
    cudaMemcpy(dcn, cn.data(), sizeof(long long) * m, cudaMemcpyHostToDevice);
    centroid_kernel<<<(m + 255) / 256, 256>>>(dcs, dcn, dcg, m);
    std::vector<float> cg(m);
    cudaMemcpy(cg.data(), dcg, sizeof(float) * m, cudaMemcpyDeviceToHost);
    long long off = 0, exact = 0;
    for (int i = 0; i < m; ++i) {
      const float ref = static_cast<float>(cs[i] / static_cast<double>(cn[i]));
      uint32_t a, b;
      std::memcpy(&a, &cg[i], 4);
      std::memcpy(&b, &ref, 4);
      const long long d = static_cast<long long>(a) - static_cast<long long>(b);
      exact += d == 0;
      off += d > 1 || d < -1;
    }
    std::printf("centroid_value: %lld of %d equal fp32(s / n), %lld more than one ulp away\n", exact, m, off);
    fail |= off != 0;
    cudaFree(dcs);
    cudaFree(dcn);
    cudaFree(dcg);
  }
  cudaFree(dg64);
  cudaFree(ds);
  cudaFree(dg);
  cudaFree(dw);
  cudaFree(da);
  return fail;
}
