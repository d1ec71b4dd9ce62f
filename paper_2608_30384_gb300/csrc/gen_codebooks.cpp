// gen_codebooks.cpp -- writes codebooks_multid.inc, the 2-D and 4-D K=16
// codebooks of the 2-bit and 1-bit RSLM codecs (Sec. 3.2: k-means with K
// clusters on a large set of synthetic N(0, I) samples; Table "Rslm Codec
// Specifications": b=2 uses a 2-D, b=1 a 4-D codebook with K=16).
//
// Development-time generator, not part of the library.  Build and run:
//   g++ -O2 -std=c++17 gen_codebooks.cpp -o /tmp/gen && /tmp/gen > codebooks_multid.inc
//
// Fixed recipe (every step deterministic):
//  * samples: 2^17 vectors of g Gaussians from Box-Muller on SplitMix64
//    (seed 0x52534C4D + 1000 + g; pair i uses outputs 2i, 2i+1 mapped to
//    ((out >> 11) + 0.5) * 2^-53), rounded to the 2^-20 grid so that cluster
//    sums are exact in double in any order;
//  * 8 restarts, each seeded by k-means++ (uniforms (out >> 11) * 2^-53 of
//    SplitMix64 seed 0x52534C4D + 2000 + 100 g + r: first center at
//    floor(u0 n), next centers where the running sum of squared distances
//    first exceeds u_k * total), refined by Lloyd iterations (nearest center,
//    lowest index on ties; new center = exact member mean; an empty cluster
//    keeps its center) until the assignment repeats or 400 passes;
//  * the restart with the lowest distortion wins; its codewords are sorted
//    lexicographically and rounded to the nearest binary16 value.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <vector>

namespace {

constexpr uint64_t kSeed = 0x52534C4Dull;
constexpr int kSamples = 1 << 17;
constexpr int kRestarts = 8;
constexpr int kMaxIters = 400;
constexpr int kK = 16;

uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Output n (0-based) of SplitMix64 started from `seed`.
uint64_t splitmix_at(uint64_t seed, uint64_t n) {
  return mix64(seed + (n + 1) * 0x9E3779B97F4A7C15ull);
}

double sq_dist(const double* x, const double* c, int g) {
  double d = (x[0] - c[0]) * (x[0] - c[0]);
  for (int j = 1; j < g; ++j) d = d + (x[j] - c[j]) * (x[j] - c[j]);
  return d;
}

std::vector<double> make_samples(int g) {
  const int n = kSamples * g;
  std::vector<double> z(n);
  const double grid = std::ldexp(1.0, -20);
  for (int i = 0; i < n / 2; ++i) {
    double u1 = (double(splitmix_at(kSeed + 1000 + g, 2 * i) >> 11) + 0.5) * std::ldexp(1.0, -53);
    double u2 = (double(splitmix_at(kSeed + 1000 + g, 2 * i + 1) >> 11) + 0.5) * std::ldexp(1.0, -53);
    double r = std::sqrt(-2.0 * std::log(u1));
    double th = 2.0 * M_PI * u2;
    z[2 * i] = std::nearbyint(r * std::cos(th) / grid) * grid;
    z[2 * i + 1] = std::nearbyint(r * std::sin(th) / grid) * grid;
  }
  return z;
}

void assign(const std::vector<double>& X, const std::vector<double>& C, int g,
            std::vector<int>& arg, std::vector<double>& best) {
  const int n = int(X.size()) / g;
  for (int i = 0; i < n; ++i) {
    double b = sq_dist(&X[size_t(i) * g], &C[0], g);
    int a = 0;
    for (int k = 1; k < kK; ++k) {
      double d = sq_dist(&X[size_t(i) * g], &C[size_t(k) * g], g);
      if (d < b) { b = d; a = k; }
    }
    arg[i] = a;
    best[i] = b;
  }
}

std::vector<double> kmeanspp(const std::vector<double>& X, int g, uint64_t seed) {
  const int n = int(X.size()) / g;
  std::vector<double> C(size_t(kK) * g);
  auto uni = [&](int k) { return double(splitmix_at(seed, k) >> 11) * std::ldexp(1.0, -53); };
  int first = int(uni(0) * n);
  for (int j = 0; j < g; ++j) C[j] = X[size_t(first) * g + j];
  std::vector<double> d(n), cum(n);
  for (int i = 0; i < n; ++i) d[i] = sq_dist(&X[size_t(i) * g], &C[0], g);
  for (int k = 1; k < kK; ++k) {
    double run = 0.0;
    for (int i = 0; i < n; ++i) { run += d[i]; cum[i] = run; }
    double target = uni(k) * cum[n - 1];
    int j = int(std::upper_bound(cum.begin(), cum.end(), target) - cum.begin());
    if (j > n - 1) j = n - 1;
    for (int t = 0; t < g; ++t) C[size_t(k) * g + t] = X[size_t(j) * g + t];
    for (int i = 0; i < n; ++i) d[i] = std::min(d[i], sq_dist(&X[size_t(i) * g], &X[size_t(j) * g], g));
  }
  return C;
}

double lloyd(const std::vector<double>& X, int g, std::vector<double>& C, int* iters) {
  const int n = int(X.size()) / g;
  std::vector<int> arg(n), prev(n);
  std::vector<double> best(n);
  bool have_prev = false;
  int it = 0;
  for (it = 0; it < kMaxIters; ++it) {
    assign(X, C, g, arg, best);
    if (have_prev && arg == prev) break;
    prev = arg;
    have_prev = true;
    std::vector<double> sum(size_t(kK) * g, 0.0);
    std::vector<long> cnt(kK, 0);
    for (int i = 0; i < n; ++i) {
      cnt[arg[i]]++;
      for (int j = 0; j < g; ++j) sum[size_t(arg[i]) * g + j] += X[size_t(i) * g + j];
    }
    for (int k = 0; k < kK; ++k)
      if (cnt[k])
        for (int j = 0; j < g; ++j) C[size_t(k) * g + j] = sum[size_t(k) * g + j] / double(cnt[k]);
  }
  assign(X, C, g, arg, best);
  double tot = 0.0;
  for (int i = 0; i < n; ++i) tot += best[i];
  *iters = it;
  return tot / double(X.size());
}

// Nearest binary16 value of v (round half to even), returned as double.
double round_f16(double v) {
  if (v == 0.0 || !std::isfinite(v)) return v;
  double a = std::fabs(v);
  int e;
  std::frexp(a, &e);  // a = f 2^e, f in [0.5, 1): exponent of a is e - 1
  int exp2 = e - 1;
  if (exp2 < -14) exp2 = -14;  // subnormal spacing 2^-24
  double q = std::ldexp(1.0, exp2 - 10);
  double r = std::nearbyint(a / q) * q;
  return std::copysign(r, v);
}

void emit(int g) {
  std::vector<double> X = make_samples(g);
  std::vector<double> bestC;
  double bestm = 0.0;
  int bestr = -1, bestit = 0;
  for (int r = 0; r < kRestarts; ++r) {
    std::vector<double> C = kmeanspp(X, g, kSeed + 2000 + 100 * g + r);
    int it = 0;
    double m = lloyd(X, g, C, &it);
    if (bestr < 0 || m < bestm) { bestm = m; bestC = C; bestr = r; bestit = it; }
  }
  std::vector<std::vector<double>> rows(kK, std::vector<double>(g));
  for (int k = 0; k < kK; ++k)
    for (int j = 0; j < g; ++j) rows[k][j] = bestC[size_t(k) * g + j];
  std::sort(rows.begin(), rows.end());
  std::printf("// g=%d: distortion per coordinate on the samples %.9f (restart %d, %d passes)\n", g,
              bestm, bestr, bestit);
  std::printf("static const double kCodebook%dD[16][%d] = {\n", g, g);
  for (int k = 0; k < kK; ++k) {
    std::printf("  {");
    for (int j = 0; j < g; ++j) std::printf("%s%a", j ? ", " : "", round_f16(rows[k][j]));
    std::printf("},\n");
  }
  std::printf("};\n");
}

}  // namespace

int main() {
  std::printf("// Generated by gen_codebooks.cpp; binary16-exact codeword components.\n");
  emit(2);
  emit(4);
  return 0;
}
