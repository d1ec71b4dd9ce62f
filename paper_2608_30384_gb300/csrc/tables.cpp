// tables.cpp -- static tables of the RSLM codec, computed on the host.
//
// * Sign table S1 and in-block permutation P (Sec. 3.1.2): drawn from
//   SplitMix64 (Steele, Lea, Flood 2014), seed 0x52534C4D ("RSLM"); outputs
//   0..255 give S1 (top bit set -> -1), outputs 256..382 drive a Fisher-Yates
//   shuffle of 0..127 (step t swaps entries 127-t and out mod (128-t)).
//   S2 = S1 offset by 127 entries (Sec. 3.1.3, step 4).
// * 1-D Lloyd-Max levels of N(0,1) (Sec. 3.2) by the Lloyd fixed point on
//   the exact density; 2-D / 4-D k-means codebooks from codebooks_multid.inc
//   (written by gen_codebooks.cpp).  All components rounded to binary16.
// * E_max(D) = integral_0^inf 1 - erf(t/sqrt2)^D dt (Sec. 3.2) by composite
//   Gauss-Legendre quadrature.
#include <cmath>
#include <cstring>
#include <vector>

#include "rslm_internal.h"

namespace rslm {
namespace {

#include "codebooks_multid.inc"

constexpr uint64_t kSeed = 0x52534C4Dull;

uint64_t splitmix_at(uint64_t seed, uint64_t n) {
  uint64_t z = seed + (n + 1) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

double round_f16(double v) {
  if (v == 0.0 || !std::isfinite(v)) return v;
  int e;
  std::frexp(std::fabs(v), &e);
  int exp2 = e - 1;
  if (exp2 < -14) exp2 = -14;
  double q = std::ldexp(1.0, exp2 - 10);
  return std::copysign(std::nearbyint(std::fabs(v) / q) * q, v);
}

// Lloyd fixed point for the K-level quantizer of N(0,1).
std::vector<double> lloyd_max(int K) {
  std::vector<double> lv(K), t(K + 1), nw(K);
  for (int i = 0; i < K; ++i) lv[i] = -2.5 + 5.0 * i / (K - 1);
  const double s2 = std::sqrt(2.0), sp = std::sqrt(2.0 * M_PI);
  for (int it = 0; it < 200000; ++it) {
    t[0] = -INFINITY;
    t[K] = INFINITY;
    for (int i = 1; i < K; ++i) t[i] = 0.5 * (lv[i] + lv[i - 1]);
    double diff = 0.0;
    for (int i = 0; i < K; ++i) {
      double pa = std::isinf(t[i]) ? 0.0 : std::exp(-0.5 * t[i] * t[i]) / sp;
      double pb = std::isinf(t[i + 1]) ? 0.0 : std::exp(-0.5 * t[i + 1] * t[i + 1]) / sp;
      double ca = 0.5 * std::erfc(-t[i] / s2), cb = 0.5 * std::erfc(-t[i + 1] / s2);
      nw[i] = (pa - pb) / (cb - ca);
      diff = std::fmax(diff, std::fabs(nw[i] - lv[i]));
    }
    lv = nw;
    if (diff < 1e-15) break;
  }
  return lv;
}

// Gauss-Legendre nodes / weights on [-1, 1] by Newton on P_n.
void gauss_legendre(int n, std::vector<double>& x, std::vector<double>& w) {
  x.assign(n, 0.0);
  w.assign(n, 0.0);
  for (int i = 0; i < n; ++i) {
    double z = std::cos(M_PI * (i + 0.75) / (n + 0.5)), pp = 0.0;
    for (int it = 0; it < 100; ++it) {
      double p1 = 1.0, p2 = 0.0;
      for (int j = 1; j <= n; ++j) {
        double p3 = p2;
        p2 = p1;
        p1 = ((2.0 * j - 1.0) * z * p2 - (j - 1.0) * p3) / j;
      }
      pp = n * (z * p1 - p2) / (z * z - 1.0);
      double z1 = z;
      z = z1 - p1 / pp;
      if (std::fabs(z - z1) < 1e-16) break;
    }
    x[i] = z;
    w[i] = 2.0 / ((1.0 - z * z) * pp * pp);
  }
}

}  // namespace

void rotation_tables(int8_t s1[256], int32_t perm[128]) {
  for (int i = 0; i < 256; ++i) s1[i] = (splitmix_at(kSeed, i) >> 63) ? -1 : 1;
  for (int i = 0; i < 128; ++i) perm[i] = i;
  for (int t = 0; t < 127; ++t) {
    int i = 127 - t;
    int j = int(splitmix_at(kSeed, 256 + t) % uint64_t(i + 1));
    int tmp = perm[i];
    perm[i] = perm[j];
    perm[j] = tmp;
  }
}

RotSpec make_rot_spec(int D, int bits) {
  RotSpec r;
  std::memset(&r, 0, sizeof(r));
  r.D = D;
  int B = 128;
  if (D < 128) {
    B = 1;
    while (B * 2 <= D) B *= 2;
  }
  r.B = B;
  r.logB = 0;
  while ((1 << r.logB) < B) r.logB++;
  r.M = D / B;
  r.overlap = (D % B) ? D - B : -1;
  r.two_pass = !(bits == 4 && D <= 256);
  r.inv_sqrt_B = 1.0 / std::sqrt(double(B));
  int8_t s1[256];
  int32_t p[128];
  rotation_tables(s1, p);
  for (int i = 0; i < 256; ++i) {
    if (s1[i] < 0) r.s1[i >> 5] |= 1u << (i & 31);
    if (s1[(i + 127) % 256] < 0) r.s2[i >> 5] |= 1u << (i & 31);
  }
  for (int k = 0; k < B; ++k) {
    if (B == 128) {
      r.perm[k] = uint8_t(p[k]);
    } else {
      int rev = 0;
      for (int b = 0; b < r.logB; ++b)
        if (k >> b & 1) rev |= 1 << (r.logB - 1 - b);
      r.perm[k] = uint8_t(rev);
    }
  }
  return r;
}

double e_max(int D) {
  static std::vector<double> gx, gw;
  if (gx.empty()) gauss_legendre(12, gx, gw);
  const double s2 = std::sqrt(2.0);
  auto f = [&](double t) { return -std::expm1(D * std::log1p(-std::erfc(t / s2))); };
  double total = 0.0;
  const double h = 0.025;
  for (int p = 0; p < 1600; ++p) {  // [0, 40]
    double a = p * h, mid = a + 0.5 * h, part = 0.0;
    for (size_t i = 0; i < gx.size(); ++i) part += gw[i] * f(mid + 0.5 * h * gx[i]);
    total += 0.5 * h * part;
  }
  return total;
}

bool make_codec_spec(int bits, int D, bool interleaved, CodecSpec* out) {
  CodecSpec c;
  std::memset(&c, 0, sizeof(c));
  c.bits = bits;
  c.K = 16;
  if (bits == 4 || bits == 3) {
    c.g = 1;
    c.K = bits == 4 ? 16 : 8;
    std::vector<double> lv = lloyd_max(c.K);
    for (int k = 0; k < c.K; ++k) c.cbd[k] = round_f16(lv[k]);
    for (int k = 0; k + 1 < c.K; ++k) c.thr[k] = 0.5 * (c.cbd[k] + c.cbd[k + 1]);
  } else if (bits == 2) {
    c.g = 2;
    for (int k = 0; k < 16; ++k)
      for (int j = 0; j < 2; ++j) c.cbd[k * 2 + j] = kCodebook2D[k][j];
  } else if (bits == 1) {
    c.g = 4;
    for (int k = 0; k < 16; ++k)
      for (int j = 0; j < 4; ++j) c.cbd[k * 4 + j] = kCodebook4D[k][j];
  } else {
    return false;
  }
  for (int i = 0; i < c.K * c.g; ++i) c.cbf[i] = float(c.cbd[i]);
  if (D > 0) {
    c.ngroups = (D + c.g - 1) / c.g;
    c.Dp = c.ngroups * c.g;
    c.code_bytes = (c.ngroups + 1) / 2;
    if (bits == 3) {
      // Rslm3: a 3-bit stream, 8 codes in 3 bytes; the device rows hold whole
      // groups of 32 codes (three 32-bit words), interleaved word by word
      c.code_bytes = (3 * c.ngroups + 7) / 8;
      c.stride = (c.ngroups + 31) / 32 * 12;
      c.chunk = interleaved ? 4 : 0;
      if (!interleaved) c.stride = (c.stride + 15) / 16 * 16;
    } else if (interleaved) {
      c.stride = (c.code_bytes + 3) / 4 * 4;
      c.chunk = c.stride % 16 == 0 ? 16 : (c.stride % 8 == 0 ? 8 : 4);
    } else {
      c.stride = (c.code_bytes + 15) / 16 * 16;
      c.chunk = 0;
    }
    c.emax = e_max(D);
  }
  *out = c;
  return true;
}

uint32_t ue_encode_host(double v, int ebits, int mbits) {
  if (!(v > 0.0)) return 0;
  int k;
  double f = std::frexp(v, &k);
  int e = k - 1;
  double m = std::nearbyint((2.0 * f - 1.0) * double(1 << mbits));
  uint32_t mi = uint32_t(m);
  if (mi == (1u << mbits)) {
    mi = 0;
    e += 1;
  }
  int be = e + (1 << (ebits - 1)) - 1;
  if (be <= 0) return 0;
  if (be > (1 << ebits) - 1) return (((1u << ebits) - 1) << mbits) | ((1u << mbits) - 1);
  return (uint32_t(be) << mbits) | mi;
}

}  // namespace rslm
