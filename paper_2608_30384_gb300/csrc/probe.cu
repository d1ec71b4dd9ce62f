// probe.cu -- IVF probe (Sec. 5.5.1: the nprobe partitions with the largest
// <q, c_p>, ties to the lower p) on the tensor cores, without materialising
// the nq x nlist score matrix.
//
// For padded D <= 128 and nlist >= 32 nprobe:
//   1. queries and centroids are scaled by powers of two (max |q| and max |c|
//      into [1024, 2048)) and split into fp16 parts, x = x_hi + x_lo + e with
//      x_hi = fp16(x) and x_lo = fp16(x - x_hi).
//        a1 = <q_hi, c_hi> is within delta1 = 2^-9 ||q|| max ||c|| of <q, c>
//          (each fp16 rounding is relative 2^-11, Cauchy-Schwarz bounds the
//          sum, fp32 accumulation adds far less);
//        a3 = <q_hi, c_hi> + <q_lo, c_hi> + <q_hi, c_lo> is within
//          delta3 = 2^-14 ||q|| max ||c||: the dropped parts (<q_lo, c_lo>,
//          the fp16 rounding of the lo parts) are below 2^-20, and the
//          tensor core's fp32 accumulation of 3 x 128 products stays below
//          about 384 x 2^-23 of sum |q_i c_i| <= ||q|| ||c||;
//   2. probe_kernel, per CTA of 256 queries, streams the centroid tiles
//      through tcgen05.mma twice.  Pass 1 (a1): the columns are split into
//      ceil(nprobe / j) disjoint groups of whole 32-column chunks, and each
//      group contributes the j-th largest of its chunk maxima of a1 (j in
//      {1, 2, 4, 8}, a template parameter), which j distinct centroids of
//      the group reach; the smallest
//      contribution B1 is therefore reached by at least nprobe centroids, so
//      the nprobe-th largest <q, c> is at least B1 - delta1.  Pass 2 (a3)
//      appends every centroid with a3 >= B1 - delta1 - delta3, which includes
//      every centroid of the exact top nprobe, with a3, to the query's list;
//   3. probe_select_kernel takes the top nprobe of each list by
//      (a3 desc, p asc) and returns <q, c> = a3 / (2^sq 2^sC).  A list that
//      overflowed its capacity (many centroids tied at the bound) goes to
//      probe_exact_kernel, which scores every centroid in fp32.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math_constants.h>

#include <algorithm>
#include <climits>

#include "device_common.cuh"
#include "launch.h"
#include "tcgen05.cuh"

namespace rslm {
namespace {

constexpr int kPRows = 128;       // rows (queries or centroids) per operand tile
constexpr int kPQ = 2 * kPRows;   // queries per CTA (two M blocks)
constexpr int kPStages = 3;       // centroid tiles in flight
constexpr int kPEpiWarps = 16;    // (M block, column half, TMEM lane quarter)
// then one TMA warp and one MMA-issuing warp per M block: the tensor core
// queues only about two MMAs, so a lone issuer's barrier waits would leave
// it idle; two issuers cover each other's waits
constexpr int kPThreads = (kPEpiWarps + 3) * 32;
constexpr int kPTmaWarp = kPEpiWarps, kPMmaWarp0 = kPEpiWarps + 1;
constexpr uint32_t kPCols = 512;  // TMEM: (M block, buffer) accumulators of 128 columns
constexpr int kListCapMin = 1024;  // listed centroids per query (at least 8 nprobe) before the exact fallback

__host__ __device__ constexpr int tile_bytes(int Kp) { return kPRows * Kp * 2; }

// Byte offset of element (row r, dim k) of a K-major no-swizzle operand tile
// with Kp dims: core matrices of 8 rows x 16 bytes, K-adjacent ones 128 bytes
// apart, 8-row groups (Kp / 8) * 128 bytes apart.
__device__ __forceinline__ uint32_t ptile_off(int r, int k, int Kp) {
  return uint32_t((r >> 3) * (Kp / 8) * 128 + (k >> 3) * 128 + (r & 7) * 16 + (k & 7) * 2);
}

__device__ __forceinline__ int pow2_exp_for(float m) {
  int e = 0;
  if (m > 0.0f) frexpf(m, &e);  // m in [2^(e-1), 2^e)
  return 11 - e;                // m * 2^s in [1024, 2048)
}

// x = hi + lo with hi = fp16(x), lo = fp16(x - hi) (x - hi is exact in fp32).
__device__ __forceinline__ void split_half(float x, __half& hi, __half& lo) {
  hi = __float2half_rn(x);
  lo = __float2half_rn(x - __half2float(hi));
}

// meta[0] = max |c|, meta[1] = max ||c||^2 over the centroids (one block).
__global__ void centroid_stats_kernel(const float* __restrict__ C, int64_t n, int D, float* __restrict__ meta) {
  __shared__ float sa[32], sb[32];
  float am = 0.0f, nm = 0.0f;
  for (int64_t p = threadIdx.x; p < n; p += blockDim.x) {
    float s2 = 0.0f;
    for (int d = 0; d < D; ++d) {
      const float v = C[p * D + d];
      am = fmaxf(am, fabsf(v));
      s2 = fmaf(v, v, s2);
    }
    nm = fmaxf(nm, s2);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    am = fmaxf(am, __shfl_xor_sync(kFull, am, o));
    nm = fmaxf(nm, __shfl_xor_sync(kFull, nm, o));
  }
  if ((threadIdx.x & 31) == 0) {
    sa[threadIdx.x >> 5] = am;
    sb[threadIdx.x >> 5] = nm;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < int(blockDim.x >> 5); ++w) {
      am = fmaxf(am, sa[w]);
      nm = fmaxf(nm, sb[w]);
    }
    meta[0] = am;
    meta[1] = nm;
  }
}

// Centroid operand tiles: c * 2^sC split into fp16 hi (tiles 0 .. ntiles-1)
// and lo (tiles ntiles .. 2 ntiles-1), 128 centroids per tile (rows beyond
// nlist and dims beyond D are zero).  meta[2] = 2^sC, meta[3] = max ||c|| 2^sC.
__global__ void centroid_tiles_kernel(const float* __restrict__ C, int nlist, int D, int Kp,
                                      float* __restrict__ meta, uint8_t* __restrict__ tiles) {
  const int s = pow2_exp_for(meta[0]);
  const float sc = ldexpf(1.0f, s);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    meta[2] = sc;
    meta[3] = sqrtf(meta[1]) * sc;
  }
  const int ntiles = (nlist + kPRows - 1) / kPRows;
  const int k8n = Kp / 8;
  const int64_t total = int64_t(ntiles) * kPRows * k8n;
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < total;
       i += int64_t(gridDim.x) * blockDim.x) {
    const int k8 = int(i % k8n);
    const int64_t p = i / k8n;
    __align__(16) __half h[8], l[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int d = k8 * 8 + j;
      split_half((p < nlist && d < D) ? C[p * D + d] * sc : 0.0f, h[j], l[j]);
    }
    const int64_t t = p / kPRows;
    const int r = int(p % kPRows);
    const uint32_t off = ptile_off(r, k8 * 8, Kp);
    *reinterpret_cast<uint4*>(tiles + t * tile_bytes(Kp) + off) = *reinterpret_cast<const uint4*>(h);
    *reinterpret_cast<uint4*>(tiles + (ntiles + t) * tile_bytes(Kp) + off) = *reinterpret_cast<const uint4*>(l);
  }
}

// Query operand tiles, four per CTA of 256 queries: hi of M block 0 and 1,
// then lo of M block 0 and 1 (q * 2^sq split like the centroids; queries
// beyond nq are zero).  Per query: dthr = (delta1 + delta3) in the scaled
// units of a1 and a3, with a 1.001 margin for its own rounding, and
// qinv = 1 / (2^sq 2^sC), which maps a3 back to <q, c>.
__global__ void query_tiles_kernel(const float* __restrict__ Q, int64_t nq, int64_t nqp, int D, int Kp,
                                   const float* __restrict__ meta, uint8_t* __restrict__ tiles,
                                   float* __restrict__ dthr, float* __restrict__ qinv) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, W = blockDim.x >> 5;
  for (int64_t q = int64_t(blockIdx.x) * W + warp; q < nqp; q += int64_t(gridDim.x) * W) {
    float m = 0.0f, s2 = 0.0f;
    if (q < nq) {
      for (int d = lane; d < D; d += 32) {
        const float v = Q[q * D + d];
        m = fmaxf(m, fabsf(v));
        s2 = fmaf(v, v, s2);
      }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      m = fmaxf(m, __shfl_xor_sync(kFull, m, o));
      s2 += __shfl_xor_sync(kFull, s2, o);
    }
    const int sq = pow2_exp_for(m);
    const float sc = ldexpf(1.0f, sq);
    const int64_t cta = q / kPQ;
    const int mb = int((q / kPRows) % 2), r = int(q % kPRows);
    uint8_t* hi_tile = tiles + (cta * 4 + mb) * tile_bytes(Kp);
    uint8_t* lo_tile = tiles + (cta * 4 + 2 + mb) * tile_bytes(Kp);
    for (int k8 = lane; k8 < Kp / 8; k8 += 32) {
      __align__(16) __half h[8], l[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int d = k8 * 8 + j;
        split_half((q < nq && d < D) ? Q[q * D + d] * sc : 0.0f, h[j], l[j]);
      }
      const uint32_t off = ptile_off(r, k8 * 8, Kp);
      *reinterpret_cast<uint4*>(hi_tile + off) = *reinterpret_cast<const uint4*>(h);
      *reinterpret_cast<uint4*>(lo_tile + off) = *reinterpret_cast<const uint4*>(l);
    }
    if (lane == 0 && q < nq) {
      dthr[q] = (ldexpf(1.0f, -9) + ldexpf(1.0f, -14)) * sqrtf(s2) * sc * meta[3] * 1.001f;
      qinv[q] = ldexpf(1.0f, -sq) / meta[2];
    }
  }
}

// Largest of 32 values by a depth-4 tree of 3-input maxima.
__device__ __forceinline__ float max32(const float* v) {
  float a[11];
#pragma unroll
  for (int j = 0; j < 10; ++j) a[j] = fmax3(v[3 * j], v[3 * j + 1], v[3 * j + 2]);
  a[10] = fmaxf(v[30], v[31]);
  return fmax3(fmax3(a[0], a[1], a[2]), fmax3(a[3], a[4], a[5]), fmax3(a[6], a[7], fmax3(a[8], a[9], a[10])));
}

// v[i] for a lane-varying i in [0, 32) without leaving registers: a select
// tree on the bits of i.
__device__ __forceinline__ float pick32(const float* v, int i) {
  float a[16], b[8], c[4];
#pragma unroll
  for (int j = 0; j < 16; ++j) a[j] = (i & 1) ? v[2 * j + 1] : v[2 * j];
#pragma unroll
  for (int j = 0; j < 8; ++j) b[j] = (i & 2) ? a[2 * j + 1] : a[2 * j];
#pragma unroll
  for (int j = 0; j < 4; ++j) c[j] = (i & 4) ? b[2 * j + 1] : b[2 * j];
  const float d0 = (i & 8) ? c[1] : c[0], d1 = (i & 8) ? c[3] : c[2];
  return (i & 16) ? d1 : d0;
}

// Bit b of a chunk's hit mask stands for column 4 (b mod 8) + b / 8.
__host__ __device__ constexpr int mask_bit_col(int b) { return 4 * (b & 7) + (b >> 3); }

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
  return d;
}

// Mask of the columns of a 32-column chunk below thr, in mask-bit order: the
// signs of v - thr (paired fp32 arithmetic; exact zero for v == thr), their
// sign bytes gathered four at a time by byte permutes (selector nibbles with
// bit 3 set replicate a byte's sign), one bit of each kept.
__device__ __forceinline__ uint32_t miss_mask(const float* v, float thr) {
  const uint64_t one2 = f2pack(1.0f, 1.0f), nthr2 = f2pack(-thr, -thr);
  uint32_t miss = 0;
#pragma unroll
  for (int g = 0; g < 8; ++g) {
    float d[4];
    f2unpack(fma2(f2pack(v[4 * g], v[4 * g + 1]), one2, nthr2), d[0], d[1]);
    f2unpack(fma2(f2pack(v[4 * g + 2], v[4 * g + 3]), one2, nthr2), d[2], d[3]);
    const uint32_t s01 = prmt(__float_as_uint(d[0]), __float_as_uint(d[1]), 0x00fbu);
    const uint32_t s23 = prmt(__float_as_uint(d[2]), __float_as_uint(d[3]), 0x00fbu);
    miss |= prmt(s01, s23, 0x5410u) & (0x01010101u << g);  // column 4g + k at bit 8k + g
  }
  return miss;
}

// List entry: larger key = better (a3 desc, then p asc); keys are unique.
__device__ __forceinline__ uint64_t list_key(float a, int p) {
  return (uint64_t(float_order_key(a)) << 32) | uint64_t(~uint32_t(p));
}

struct ProbeArgs {
  const uint8_t* qtiles;
  const uint8_t* ctiles;
  const float* dthr;
  int64_t nq;
  // bound groups: the whole 32-column chunks (index < nlist / 32) of column
  // half h (chunks 2h and 2h + 1 of every tile), in order, form ngr[h]
  // groups of mch[h] chunks; a group contributes its JTH-largest chunk
  // maximum, and JTH (ngr[0] + ngr[1]) >= nprobe
  int nlist, Kp, ntiles, nprobe;
  int mch[2], ngr[2];
  int cap;
  uint64_t* keys;  // [nq][cap]: list_key of the centroids listed by half 0, then (at cap / 2) half 1
  int* cnt;        // [nq][2]: entries listed by each half (more than cap / 2: overflow)
  int* err;
};

template <int JTH>
__global__ void __launch_bounds__(kPThreads, 1) probe_kernel(const __grid_constant__ ProbeArgs a) {
  extern __shared__ __align__(128) uint8_t sm[];
  __shared__ __align__(8) uint64_t bars[1 + 2 * kPStages + 8];
  __shared__ uint32_t tmem_base_sh;
  __shared__ float half_bound[2][kPQ];  // pass-1 bound of each query from each column half
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int TB = tile_bytes(a.Kp);
  uint8_t* A0 = sm;            // query tiles: hi M0, hi M1, lo M0, lo M1
  uint8_t* B0 = sm + 4 * TB;   // kPStages centroid tiles
  const uint32_t bar0 = uint32_t(__cvta_generic_to_shared(&bars[0]));
  const uint32_t a_full = bar0;
  auto b_full = [&](uint32_t s) { return bar0 + 8u * (1 + s); };
  auto b_empty = [&](uint32_t s) { return bar0 + 8u * (1 + kPStages + s); };
  // accumulator (M block m, buffer b): MMAs done / read by the epilogue
  auto mma_done = [&](int m, uint32_t b) { return bar0 + 8u * (1 + 2 * kPStages + 2 * m + b); };
  auto acc_empty = [&](int m, uint32_t b) { return bar0 + 8u * (5 + 2 * kPStages + 2 * m + b); };
  if (tid == 0) {
    mbar_init(a_full, 1);
    for (uint32_t s = 0; s < kPStages; ++s) {
      mbar_init(b_full(s), 1);
      mbar_init(b_empty(s), 2);  // one commit per MMA-issuing warp
    }
    for (int m = 0; m < 2; ++m)
      for (uint32_t b = 0; b < 2; ++b) {
        mbar_init(mma_done(m, b), 1);
        mbar_init(acc_empty(m, b), kPEpiWarps / 2);
      }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();  // warp 0 again converged: tcgen05.alloc is .sync.aligned
  if (warp == 0) {
    const uint32_t dst = uint32_t(__cvta_generic_to_shared(&tmem_base_sh));
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst), "r"(kPCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = tmem_base_sh;
  const uint32_t a_addr = uint32_t(__cvta_generic_to_shared(A0));
  const uint32_t b_addr = uint32_t(__cvta_generic_to_shared(B0));
  const int T = a.ntiles;
  const int nload = 3 * T;  // centroid tiles loaded: T hi (pass 1), then hi and lo of each tile (pass 2)
  auto acc_col = [&](int m, uint32_t b) { return uint32_t((m * 2 + int(b)) * 128); };

  if (warp == kPTmaWarp) {
    // ---------------- TMA: the CTA's query tiles, then the centroid tiles
    if (lane == 0) {
      mbar_arrive_expect(a_full, uint32_t(4 * TB));
      bulk_copy_1d(a_addr, a.qtiles + size_t(blockIdx.x) * 4 * TB, uint32_t(4 * TB), a_full);
      int j = 0;
      for (; j < nload; ++j) {
        const uint32_t s = uint32_t(j % kPStages), u = uint32_t(j / kPStages);
        if (u > 0 && !mbar_wait(b_empty(s), (u - 1) & 1)) {
          set_device_error(a.err, kErrTimeout);
          break;
        }
        const int r = j - T;
        const int tile = j < T ? j : (r >> 1) + ((r & 1) ? T : 0);
        mbar_arrive_expect(b_full(s), uint32_t(TB));
        bulk_copy_1d(b_addr + s * uint32_t(TB), a.ctiles + size_t(tile) * TB, uint32_t(TB), b_full(s));
      }
      // no copy may still be landing when the CTA exits
      mbar_wait(a_full, 0);
      for (int s = 0; s < kPStages && s < j; ++s)
        mbar_wait(b_full(uint32_t(s)), uint32_t((j - 1 - s) / kPStages) & 1);
    }
    __syncwarp();
  } else if (warp >= kPMmaWarp0) {
    // ---------------- MMA issue: M block m against each centroid tile
    const int m = warp - kPMmaWarp0;
    if (lane == 0) {
      const uint32_t idesc = f16_idesc(kPRows, kPRows);
      const uint32_t sbo = uint32_t(a.Kp / 8) * 128;
      const int nks = a.Kp / 16;
      bool ok = mbar_wait(a_full, 0);
      int j = 0, last = -1;
      // acc(m, b) (+)= A tile `at + m` times the centroid tile in stage s
      auto mma_tile = [&](int at, uint32_t s, uint32_t b, bool acc) {
        for (int ks = 0; ks < nks; ++ks)
          umma_f16(tmem + acc_col(m, b), smem_desc(a_addr + uint32_t((at + m) * TB + ks * 256), 128, sbo),
                   smem_desc(b_addr + s * uint32_t(TB) + uint32_t(ks * 256), 128, sbo), idesc,
                   (acc || ks > 0) ? 1u : 0u);
      };
      // wait for centroid load j; its stage in s
      auto next_b = [&](uint32_t& s) {
        s = uint32_t(j % kPStages);
        const bool r = mbar_wait(b_full(s), uint32_t(j / kPStages) & 1);
        fence_after_sync();
        return r;
      };
      for (int gt = 0; ok && gt < 2 * T; ++gt) {
        const uint32_t b = uint32_t(gt & 1), ub = uint32_t(gt >> 1);
        uint32_t s = 0;
        if ((ub > 0 && !mbar_wait(acc_empty(m, b), (ub - 1) & 1)) || !next_b(s)) {
          ok = false;
          break;
        }
        mma_tile(0, s, b, false);  // <q_hi, c_hi>
        if (gt >= T) mma_tile(2, s, b, true);  // + <q_lo, c_hi>
        umma_commit(b_empty(s));
        ++j;
        if (gt >= T) {
          if (!next_b(s)) {
            ok = false;
            break;
          }
          mma_tile(0, s, b, true);  // + <q_hi, c_lo>
          umma_commit(b_empty(s));
          ++j;
        }
        umma_commit(mma_done(m, b));
        last = gt;
      }
      if (!ok) set_device_error(a.err, kErrTimeout);
      // no MMA may still be running when TMEM is freed: this warp's last
      // commit tracks every MMA it issued
      if (last >= 0) mbar_wait(mma_done(m, uint32_t(last & 1)), uint32_t(last >> 1) & 1);
    }
    __syncwarp();
  } else {
    // ---------------- epilogue: thread = one query row of M block m, 64
    // columns (column half h) of every tile
    const int m = warp >> 3, h = (warp >> 2) & 1, qd = warp & 3;
    const int row = m * kPRows + qd * 32 + lane;  // query within the CTA
    const int64_t q = int64_t(blockIdx.x) * kPQ + row;
    const bool valid = q < a.nq;
    const uint32_t lane_base = uint32_t(qd * 32) << 16;
    const int nwhole = a.nlist / 32;                 // whole chunks
    const int ngroups_chunks = a.ngr[h] * a.mch[h];  // this half's chunks that form its groups
    const int mch = a.mch[h];
    float top[JTH];  // the group's largest chunk maxima, descending
#pragma unroll
    for (int j = 0; j < JTH; ++j) top[j] = -CUDART_INF_F;
    float bound = CUDART_INF_F, thr = CUDART_INF_F;
    int n = 0, in_group = 0;  // chunks of the current bound group seen
    bool dead = false;        // a wait timed out: skip the work, keep the barrier
    uint64_t* out = a.keys + (valid ? q : 0) * int64_t(a.cap) + h * (a.cap / 2);  // this half's segment
    for (int gt = 0; gt < 2 * T; ++gt) {
      if (gt == T) {
        // B1 of the query: the smaller of the two halves' bounds
        half_bound[h][row] = bound;
        asm volatile("bar.sync 1, %0;" ::"n"(kPEpiWarps * 32) : "memory");
        bound = fminf(half_bound[0][row], half_bound[1][row]);
        thr = bound - (valid ? a.dthr[q] : 0.0f);
      }
      if (dead) continue;
      const uint32_t b = uint32_t(gt & 1), ub = uint32_t(gt >> 1);
      if (!mbar_wait_warp(mma_done(m, b), ub & 1)) {
        set_device_error(a.err, kErrTimeout);
        dead = true;
        continue;
      }
      fence_after_sync();
      const bool pass1 = gt < T;
      const int t = pass1 ? gt : gt - T;
      // this half's 64 columns in one load, then release the accumulator
      float vt[64];
      tmem_ld64(tmem + lane_base + acc_col(m, b) + uint32_t(h * 64), vt);
      fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty(m, b));
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const float* v = vt + c * 32;
        const int gc = t * (kPRows / 32) + 2 * h + c;  // 32-column chunk index
        if (pass1) {
          if (gc < nwhole && 2 * t + c < ngroups_chunks) {
            float x = max32(v);
#pragma unroll
            for (int j = 0; j < JTH; ++j) {
              const float hi = fmaxf(top[j], x);
              x = fminf(top[j], x);
              top[j] = hi;
            }
            if (++in_group == mch) {
              // at least JTH centroids of this group reach top[JTH - 1]
              bound = fminf(bound, top[JTH - 1]);
#pragma unroll
              for (int j = 0; j < JTH; ++j) top[j] = -CUDART_INF_F;
              in_group = 0;
            }
          }
        } else if (valid) {
          // append the columns at or above thr
          const int col0 = gc * 32;
          uint32_t hit = ~miss_mask(v, thr);
          float vp[32];  // the chunk in mask-bit order
#pragma unroll
          for (int b = 0; b < 32; ++b) vp[b] = v[mask_bit_col(b)];
          while (hit) {
            const int b = __ffs(hit) - 1;
            hit &= hit - 1;
            const int col = col0 + mask_bit_col(b);
            if (col < a.nlist) {  // columns beyond nlist are padding
              if (n < a.cap / 2) out[n] = list_key(pick32(vp, b), col);
              ++n;
            }
          }
        }
      }
    }
    if (valid) a.cnt[2 * q + h] = n;
  }
  __syncthreads();
  if (warp == 0) {
    fence_after_sync();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kPCols) : "memory");
  }
}

// Sort the warp's n (a power of two, <= 256) keys in shared memory into
// descending order.
__device__ __forceinline__ void warp_sort_desc(uint64_t* key, int n) {
  const int lane = threadIdx.x & 31;
  for (int size = 2; size <= n; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = lane; i < (n >> 1); i += 32) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool desc = (lo & size) == 0;
        const uint64_t klo = key[lo], khi = key[hi];
        if (desc ? khi > klo : klo > khi) {
          key[lo] = khi;
          key[hi] = klo;
        }
      }
      __syncwarp();
    }
  }
}

// The keys >= the k-th largest of a warp's list, the list held as J keys
// per lane (element lane + 32 j; 0 beyond the list, smaller than any real
// key), compacted into out[0, k).  T is found bit by bit, first over the
// high words below their common prefix, then, only if the k-th largest
// high word is tied, over the low words; the search stops as soon as
// exactly k keys are >= T.
template <int J>
__device__ __forceinline__ void select_top_regs(const uint64_t (&r)[J], int n, int k, uint64_t* out) {
  const int lane = threadIdx.x & 31;
  const unsigned lt = (1u << lane) - 1u;
  uint32_t hmax = 0u, hmin = ~0u;
#pragma unroll
  for (int j = 0; j < J; ++j) {
    if (lane + 32 * j < n) {
      const uint32_t h = uint32_t(r[j] >> 32);
      hmax = max(hmax, h);
      hmin = min(hmin, h);
    }
  }
  hmax = __reduce_max_sync(kFull, hmax);
  hmin = __reduce_min_sync(kFull, hmin);
  const int L = __clz(hmax ^ hmin);  // bits shared by every high word
  uint32_t Th = L == 0 ? 0u : (hmax & (~0u << (32 - L)));
  int cT = n;  // keys with high word >= Th
  for (int bit = 31 - L; bit >= 0 && cT > k; --bit) {
    const uint32_t t = Th | (1u << bit);
    int c = 0;
#pragma unroll
    for (int j = 0; j < J; ++j) c += uint32_t(r[j] >> 32) >= t ? 1 : 0;
    c = int(__reduce_add_sync(kFull, uint32_t(c)));
    if (c >= k) {
      Th = t;
      cT = c;
    }
  }
  uint64_t T = uint64_t(Th) << 32;
  for (int bit = 31; bit >= 0 && cT > k; --bit) {
    const uint64_t t = T | (uint64_t(1) << bit);
    int c = 0;
#pragma unroll
    for (int j = 0; j < J; ++j) c += r[j] >= t ? 1 : 0;
    c = int(__reduce_add_sync(kFull, uint32_t(c)));
    if (c >= k) {
      T = t;
      cT = c;
    }
  }
  int m = 0;
#pragma unroll
  for (int j = 0; j < J; ++j) {
    const bool keep = lane + 32 * j < n && r[j] >= T;
    const unsigned bal = __ballot_sync(kFull, keep);
    if (keep) out[m + __popc(bal & lt)] = r[j];
    m += __popc(bal);
  }
}

// Top nprobe of each query's list (the two column halves' segments) by its
// unique keys, sorted.  Lists of up to 256 entries are selected in
// registers; longer ones by the same bit search over the list in global
// memory.  A list with an overflowed segment (or, defensively, fewer than
// nprobe entries) is queued for probe_exact_kernel.  One warp per query.
constexpr int kSelWarpsPerBlock = 4;
__global__ void __launch_bounds__(kSelWarpsPerBlock * 32) probe_select_kernel(
    int64_t nq, const uint64_t* __restrict__ keys, const int* __restrict__ cnt, int cap, int k,
    const float* __restrict__ qinv, int* __restrict__ nexact, int32_t* __restrict__ exact_q,
    unsigned long long* __restrict__ ctr, int32_t* __restrict__ out_probes, float* __restrict__ out_cs) {
  __shared__ uint64_t ss[kSelWarpsPerBlock][256];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const unsigned lt = (1u << lane) - 1u;
  const int64_t nw = int64_t(gridDim.x) * kSelWarpsPerBlock;
  int p2 = 1;
  while (p2 < k) p2 <<= 1;
  for (int64_t q = int64_t(blockIdx.x) * kSelWarpsPerBlock + w; q < nq; q += nw) {
    const int half = cap / 2, n0 = cnt[2 * q], n1 = cnt[2 * q + 1], n = n0 + n1;
    if (n0 > half || n1 > half || n < k) {
      if (lane == 0) {
        exact_q[atomicAdd(nexact, 1)] = int32_t(q);
        atomicAdd(&ctr[kCtrProbeExact], 1ull);
      }
      continue;
    }
    // entry e of the list: the first n0 from half 0's segment, then half 1's
    const uint64_t* lk = keys + q * int64_t(cap);
    auto entry = [&](int e) { return __ldg(lk + (e < n0 ? e : half + e - n0)); };
    if (n <= 128) {
      uint64_t r[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) r[j] = lane + 32 * j < n ? entry(lane + 32 * j) : 0;
      select_top_regs<4>(r, n, k, ss[w]);
    } else if (n <= 256) {
      uint64_t r[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) r[j] = lane + 32 * j < n ? entry(lane + 32 * j) : 0;
      select_top_regs<8>(r, n, k, ss[w]);
    } else {
      uint64_t T = 0;
      int cT = n;  // keys >= T
      for (int bit = 63; bit >= 0 && cT > k; --bit) {
        const uint64_t t = T | (uint64_t(1) << bit);
        int c0 = 0;
        for (int i = lane; i < n; i += 32) c0 += entry(i) >= t ? 1 : 0;
        const int c = int(__reduce_add_sync(kFull, uint32_t(c0)));
        if (c >= k) {
          T = t;
          cT = c;
        }
      }
      // exactly k keys are >= T
      int m = 0;
      for (int base = 0; base < n; base += 32) {
        const int i = base + lane;
        const uint64_t key = i < n ? entry(i) : 0;
        const bool keep = i < n && key >= T;
        const unsigned bal = __ballot_sync(kFull, keep);
        if (keep) ss[w][m + __popc(bal & lt)] = key;
        m += __popc(bal);
      }
    }
    for (int i = k + lane; i < p2; i += 32) ss[w][i] = 0;
    __syncwarp();
    warp_sort_desc(ss[w], p2);
    const float inv = qinv[q];
    for (int i = lane; i < k; i += 32) {
      const uint64_t key = ss[w][i];
      out_probes[q * k + i] = int32_t(~uint32_t(key));
      out_cs[q * k + i] = float_from_order_key(uint32_t(key >> 32)) * inv;
    }
    __syncwarp();
  }
}

// Centroids again as fp32 rows of Kp floats (zero padded), so every row is
// 16-byte aligned for the exact scoring below.
__global__ void centroid_rows_kernel(const float* __restrict__ C, int nlist, int D, int Kp,
                                     float* __restrict__ out) {
  const int64_t total = int64_t(nlist) * Kp;
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < total;
       i += int64_t(gridDim.x) * blockDim.x) {
    const int d = int(i % Kp);
    out[i] = d < D ? C[(i / Kp) * D + d] : 0.0f;
  }
}

// Exact top-nprobe of the queued queries: fp32 <q, c> of every centroid, the
// nprobe-th largest order key T bit by bit, the centroids above T plus the
// lowest-index ones at T, sorted by (score desc, p asc).  One warp per
// query; the warp scores eight centroids per step (four groups of eight
// lanes, two centroids each, a lane holding Kp / 8 dims).  Keys live in the
// warp's global scratch row of nlist keys.
constexpr int kExactWarpsPerBlock = 4;
__global__ void __launch_bounds__(kExactWarpsPerBlock * 32) probe_exact_kernel(
    const float* __restrict__ Q, int D, const float* __restrict__ Cp, int Kp, int nlist,
    const int* __restrict__ nexact, const int32_t* __restrict__ exact_q, int k, uint32_t* __restrict__ scratch,
    int32_t* __restrict__ out_probes, float* __restrict__ out_cs) {
  __shared__ uint64_t ss[kExactWarpsPerBlock][256];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int grp = lane >> 3, sub = lane & 7;
  const unsigned lt = (1u << lane) - 1u;
  const int64_t gw = int64_t(blockIdx.x) * kExactWarpsPerBlock + w;
  const int64_t nw = int64_t(gridDim.x) * kExactWarpsPerBlock;
  const int nf = Kp / 4;  // float4 of a row; lane sub takes f = sub + 8 j (Kp <= 128)
  uint32_t* keys = scratch + gw * int64_t(nlist);
  const int nx = *nexact;
  int p2 = 1;
  while (p2 < k) p2 <<= 1;
  for (int64_t e = gw; e < nx; e += nw) {
    const int64_t q = exact_q[e];
    float4 qv[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      float v[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int d = (sub + 8 * j) * 4 + c;
        v[c] = (sub + 8 * j < nf && d < D) ? Q[q * D + d] : 0.0f;
      }
      qv[j] = make_float4(v[0], v[1], v[2], v[3]);
    }
    for (int i0 = 0; i0 < nlist; i0 += 8) {
      float acc[2];
      int idx[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        idx[u] = i0 + 4 * u + grp;
        const int p = idx[u] < nlist ? idx[u] : 0;
        const float4* c4 = reinterpret_cast<const float4*>(Cp + int64_t(p) * Kp);
        float s = 0.0f;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          if (sub + 8 * j < nf) {
            const float4 c = __ldg(c4 + sub + 8 * j);
            s = fmaf(qv[j].x, c.x, s);
            s = fmaf(qv[j].y, c.y, s);
            s = fmaf(qv[j].z, c.z, s);
            s = fmaf(qv[j].w, c.w, s);
          }
        }
        acc[u] = s;
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
#pragma unroll
        for (int o = 4; o; o >>= 1) acc[u] += __shfl_xor_sync(kFull, acc[u], o);
        if (sub == 0 && idx[u] < nlist) keys[idx[u]] = float_order_key(acc[u]);
      }
    }
    __syncwarp();
    // T = the k-th largest key
    uint32_t T = 0u;
    for (int bit = 31; bit >= 0; --bit) {
      const uint32_t t = T | (1u << bit);
      int c0 = 0;
      for (int i = lane; i < nlist; i += 32) c0 += keys[i] >= t ? 1 : 0;
      if (int(__reduce_add_sync(kFull, uint32_t(c0))) >= k) T = t;
    }
    // keys above T (fewer than k), then the lowest-index keys equal to T
    int ngt = 0, neq = 0, ngt_tot = 0;
    for (int base = 0; base < nlist; base += 32) {
      const int i = base + lane;
      ngt_tot += __popc(__ballot_sync(kFull, i < nlist && keys[i] > T));
    }
    for (int base = 0; base < nlist; base += 32) {
      const int i = base + lane;
      const uint32_t key = i < nlist ? keys[i] : 0u;
      const bool gtr = i < nlist && key > T, eq = i < nlist && key == T;
      const unsigned bg = __ballot_sync(kFull, gtr), be = __ballot_sync(kFull, eq);
      if (gtr) ss[w][ngt + __popc(bg & lt)] = (uint64_t(key) << 32) | uint64_t(~uint32_t(i));
      if (eq) {
        const int at = ngt_tot + neq + __popc(be & lt);
        if (at < k) ss[w][at] = (uint64_t(key) << 32) | uint64_t(~uint32_t(i));
      }
      ngt += __popc(bg);
      neq += __popc(be);
    }
    for (int i = k + lane; i < p2; i += 32) ss[w][i] = 0;
    __syncwarp();
    warp_sort_desc(ss[w], p2);
    for (int i = lane; i < k; i += 32) {
      const uint64_t key = ss[w][i];
      out_probes[q * k + i] = int32_t(~uint32_t(key));
      out_cs[q * k + i] = float_from_order_key(uint32_t(key >> 32));
    }
    __syncwarp();
  }
}

// ------------------------------------------------------------ probe GEMM
// For every other shape (padded D > 128, or fewer than 32 nprobe
// centroids) the probe scores form the matrix S = Q C^T, nq x nlist, which
// probe_gemm_kernel computes on the tensor cores and the row selection
// kernels then reduce to the top nprobe of each row.  Operands are split
// like the fused probe's (x = x_hi + x_lo, scaled by powers of two) and
// S = (<q_hi, c_hi> + <q_lo, c_hi> + <q_hi, c_lo>) / (2^sq 2^sC), within
// delta3 = 2^-14 ||q|| max ||c|| of <q, c> (the bound of the fused probe's
// second pass; the accumulation runs over K chunks of 32 dims instead of
// one chunk of up to 128).
//
// Pre-tiled operand blocks, one 1-D bulk copy each: for every tile of
// kGM = 128 queries (kGN = 256 centroids) and every K chunk of kGK = 32
// dims, the hi block then the lo block, each K-major without swizzle (core
// matrices of 8 rows x 16 bytes; K-adjacent ones 128 bytes apart, 8-row
// groups 512 bytes apart).
constexpr int kGM = 128, kGN = 256, kGK = 32;
constexpr int kGStages = 4;
constexpr int kGSbo = (kGK / 8) * 128;                  // bytes between 8-row groups
constexpr int kGBlockA = 2 * kGM * kGK * 2;             // hi + lo of a query block (16 KB)
constexpr int kGBlockB = 2 * kGN * kGK * 2;             // hi + lo of a centroid block (32 KB)
constexpr int kGStageBytes = kGBlockA + kGBlockB;
constexpr int kGEpiWarps = 8;                           // (lane quadrant, column half of 128)
constexpr int kGTmaWarp = kGEpiWarps, kGMmaWarp = kGEpiWarps + 1;
constexpr int kGThreads = (kGEpiWarps + 2) * 32;
constexpr uint32_t kGCols = 512;                        // two accumulators of 256 columns

__host__ __device__ constexpr int gemm_kchunks(int D) { return (D + kGK - 1) / kGK; }

__device__ __forceinline__ uint32_t gblock_off(int r, int k) {
  return uint32_t((r >> 3) * kGSbo + (k >> 3) * 128 + (r & 7) * 16 + (k & 7) * 2);
}

// Centroid blocks [N tile][K chunk] of c * 2^sC (meta[2] = 2^sC, set by
// centroid_tiles_meta_kernel); rows beyond nlist and dims beyond D are zero.
__global__ void centroid_gemm_blocks_kernel(const float* __restrict__ C, int nlist, int D,
                                            const float* __restrict__ meta, uint8_t* __restrict__ out) {
  const float sc = meta[2];
  const int nkc = gemm_kchunks(D), ntn = (nlist + kGN - 1) / kGN;
  const int64_t total = int64_t(ntn) * kGN * nkc * (kGK / 8);
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < total;
       i += int64_t(gridDim.x) * blockDim.x) {
    const int k8 = int(i % (nkc * (kGK / 8)));  // 8-dim group of the row
    const int64_t p = i / (nkc * (kGK / 8));
    __align__(16) __half h[8], l[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int d = k8 * 8 + j;
      split_half((p < nlist && d < D) ? C[p * D + d] * sc : 0.0f, h[j], l[j]);
    }
    const int kc = k8 / (kGK / 8), kk = (k8 % (kGK / 8)) * 8;
    uint8_t* blk = out + (size_t(p / kGN) * nkc + kc) * kGBlockB;
    const uint32_t off = gblock_off(int(p % kGN), kk);
    *reinterpret_cast<uint4*>(blk + off) = *reinterpret_cast<const uint4*>(h);
    *reinterpret_cast<uint4*>(blk + kGBlockB / 2 + off) = *reinterpret_cast<const uint4*>(l);
  }
}

// 2^sC from the centroids' largest |c| (meta[0]), as centroid_tiles_kernel
// does for the fused probe.
__global__ void centroid_tiles_meta_kernel(float* __restrict__ meta) {
  const float sc = ldexpf(1.0f, pow2_exp_for(meta[0]));
  meta[2] = sc;
  meta[3] = sqrtf(meta[1]) * sc;
}

// Query blocks [M tile][K chunk] of q * 2^sq for the nq queries (rows up to
// the next multiple of kGM are zero); qinv[q] = 1 / (2^sq 2^sC).
__global__ void query_gemm_blocks_kernel(const float* __restrict__ Q, int64_t nq, int D,
                                         const float* __restrict__ meta, uint8_t* __restrict__ out,
                                         float* __restrict__ qinv) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, W = blockDim.x >> 5;
  const int nkc = gemm_kchunks(D);
  const int64_t nqp = (nq + kGM - 1) / kGM * kGM;
  for (int64_t q = int64_t(blockIdx.x) * W + warp; q < nqp; q += int64_t(gridDim.x) * W) {
    float m = 0.0f;
    if (q < nq)
      for (int d = lane; d < D; d += 32) m = fmaxf(m, fabsf(Q[q * D + d]));
#pragma unroll
    for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(kFull, m, o));
    const int sq = pow2_exp_for(m);
    const float sc = ldexpf(1.0f, sq);
    const int r = int(q % kGM);
    for (int k8 = lane; k8 < nkc * (kGK / 8); k8 += 32) {
      __align__(16) __half h[8], l[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int d = k8 * 8 + j;
        split_half((q < nq && d < D) ? Q[q * D + d] * sc : 0.0f, h[j], l[j]);
      }
      const int kc = k8 / (kGK / 8), kk = (k8 % (kGK / 8)) * 8;
      uint8_t* blk = out + (size_t(q / kGM) * nkc + kc) * kGBlockA;
      const uint32_t off = gblock_off(r, kk);
      *reinterpret_cast<uint4*>(blk + off) = *reinterpret_cast<const uint4*>(h);
      *reinterpret_cast<uint4*>(blk + kGBlockA / 2 + off) = *reinterpret_cast<const uint4*>(l);
    }
    if (lane == 0 && q < nq) qinv[q] = ldexpf(1.0f, -sq) / meta[2];
  }
}

struct GemmArgs {
  const uint8_t* qblk;  // query blocks of this call's nq queries
  const uint8_t* cblk;  // centroid blocks of the index
  const float* qinv;
  int64_t nq;
  int nlist, nkc, ntm, ntn;
  float* S;    // [nq][ld] fp32 scores
  int64_t ld;  // row stride of S, a multiple of 4
  int* err;
};

// Persistent CTAs, one per SM, take the (M tile, N tile) units in M-major
// order (CTAs running at the same time share query blocks in L2).  Roles:
//   warp 8  lane 0 streams each unit's (query, centroid) block pairs of all K
//           chunks through kGStages shared-memory stages;
//   warp 9  lane 0 issues three 128 x 256 x 16 MMAs per 16 dims into one of
//           two 256-column TMEM accumulators (the epilogue of one unit
//           overlaps the next unit's MMAs);
//   warps 0-7 read their lane quadrant's 128 columns, scale each row by its
//           qinv and store the scores.
// Every wait is bounded; a timeout sets the error flag and ends every role.
__global__ void __launch_bounds__(kGThreads, 1) probe_gemm_kernel(const __grid_constant__ GemmArgs a) {
  extern __shared__ __align__(128) uint8_t gsm[];
  __shared__ __align__(8) uint64_t bars[2 * kGStages + 5];
  __shared__ uint32_t tmem_base_sh;
  __shared__ int s_fail;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t bar0 = uint32_t(__cvta_generic_to_shared(&bars[0]));
  auto full = [&](uint32_t s) { return bar0 + 8u * s; };
  auto empty = [&](uint32_t s) { return bar0 + 8u * (kGStages + s); };
  auto acc_full = [&](uint32_t b) { return bar0 + 8u * (2 * kGStages + b); };
  auto acc_empty = [&](uint32_t b) { return bar0 + 8u * (2 * kGStages + 2 + b); };
  const uint32_t drain = bar0 + 8u * (2 * kGStages + 4);  // every MMA of the CTA completed
  if (tid == 0) {
    s_fail = 0;
    mbar_init(drain, 1);
    for (uint32_t s = 0; s < kGStages; ++s) {
      mbar_init(full(s), 1);
      mbar_init(empty(s), 1);
    }
    for (uint32_t b = 0; b < 2; ++b) {
      mbar_init(acc_full(b), 1);
      mbar_init(acc_empty(b), kGEpiWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();  // warp 0 again converged: tcgen05.alloc is .sync.aligned
  if (warp == 0) {
    const uint32_t dst = uint32_t(__cvta_generic_to_shared(&tmem_base_sh));
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst), "r"(kGCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = tmem_base_sh;
  const uint32_t sm_addr = uint32_t(__cvta_generic_to_shared(gsm));
  const int64_t nunits = int64_t(a.ntm) * a.ntn;
  auto failed = [&]() { return *reinterpret_cast<volatile int*>(&s_fail) != 0; };
  auto fail = [&]() {
    set_device_error(a.err, kErrTimeout);
    atomicExch(&s_fail, 1);
  };

  if (warp == kGTmaWarp) {
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int64_t u = blockIdx.x; ok && u < nunits && !failed(); u += gridDim.x) {
        const int64_t mt = u / a.ntn, nt = u % a.ntn;
        for (int kc = 0; kc < a.nkc; ++kc, ++it) {
          const uint32_t s = it % kGStages, use = it / kGStages;
          if (use > 0 && !mbar_wait(empty(s), (use - 1) & 1)) {
            fail();
            ok = false;
            break;
          }
          const uint32_t dst = sm_addr + s * uint32_t(kGStageBytes);
          mbar_arrive_expect(full(s), uint32_t(kGStageBytes));
          bulk_copy_1d(dst, a.qblk + (size_t(mt) * a.nkc + kc) * kGBlockA, uint32_t(kGBlockA), full(s));
          bulk_copy_1d(dst + kGBlockA, a.cblk + (size_t(nt) * a.nkc + kc) * kGBlockB, uint32_t(kGBlockB), full(s));
        }
      }
      // no copy may still be landing when the CTA exits
      for (uint32_t s = 0; s < kGStages && s < it; ++s) mbar_wait(full(s), ((it - 1 - s) / kGStages) & 1);
    }
    __syncwarp();
  } else if (warp == kGMmaWarp) {
    if (lane == 0) {
      const uint32_t idesc = f16_idesc(kGM, kGN);
      uint32_t it = 0, nb = 0;
      bool ok = true;
      for (int64_t u = blockIdx.x; ok && u < nunits && !failed(); u += gridDim.x, ++nb) {
        const uint32_t b = nb & 1, ub = nb >> 1;
        if (ub > 0 && !mbar_wait(acc_empty(b), (ub - 1) & 1)) {
          fail();
          break;
        }
        fence_after_sync();
        const uint32_t acc = tmem + b * uint32_t(kGN);
        for (int kc = 0; kc < a.nkc; ++kc, ++it) {
          const uint32_t s = it % kGStages;
          if (!mbar_wait(full(s), (it / kGStages) & 1)) {
            fail();
            ok = false;
            break;
          }
          fence_after_sync();
          const uint32_t ahi = sm_addr + s * uint32_t(kGStageBytes), alo = ahi + kGBlockA / 2;
          const uint32_t bhi = ahi + kGBlockA, blo = bhi + kGBlockB / 2;
#pragma unroll
          for (int ks = 0; ks < kGK / 16; ++ks) {
            const uint32_t o = uint32_t(ks * 256);
            umma_f16(acc, smem_desc(ahi + o, 128, kGSbo), smem_desc(bhi + o, 128, kGSbo), idesc,
                     (kc > 0 || ks > 0) ? 1u : 0u);
            umma_f16(acc, smem_desc(alo + o, 128, kGSbo), smem_desc(bhi + o, 128, kGSbo), idesc, 1u);
            umma_f16(acc, smem_desc(ahi + o, 128, kGSbo), smem_desc(blo + o, 128, kGSbo), idesc, 1u);
          }
          umma_commit(empty(s));
        }
        if (!ok) break;
        umma_commit(acc_full(b));
      }
      // no MMA may still be running when TMEM is freed (also after a timeout):
      // a commit tracks every MMA this thread issued
      umma_commit(drain);
      mbar_wait(drain, 0);
    }
    __syncwarp();
  } else {
    // epilogue: rows of quadrant warp % 4, columns (warp / 4) * 128 ..
    const int quad = warp & 3, ch = warp >> 2;
    const int row = quad * 32 + lane;
    uint32_t nb = 0;
    for (int64_t u = blockIdx.x; u < nunits && !failed(); u += gridDim.x, ++nb) {
      const int64_t mt = u / a.ntn, nt = u % a.ntn;
      const uint32_t b = nb & 1, ub = nb >> 1;
      if (!mbar_wait_warp(acc_full(b), ub & 1)) {
        fail();
        break;
      }
      fence_after_sync();
      const int64_t q = mt * kGM + row;
      const bool valid = q < a.nq;
      const float inv = valid ? a.qinv[q] : 0.0f;
      float* dst = a.S + (valid ? q : 0) * a.ld;
#pragma unroll 1
      for (int c = 0; c < 4; ++c) {
        float v[32];
        tmem_ld32(tmem + (uint32_t(quad * 32) << 16) + b * uint32_t(kGN) + uint32_t(ch * 128 + c * 32), v);
        const int64_t col0 = nt * kGN + ch * 128 + c * 32;
        if (valid) {
#pragma unroll
          for (int j = 0; j < 32; j += 4)
            if (col0 + j < a.ld)
              *reinterpret_cast<float4*>(dst + col0 + j) =
                  make_float4(v[j] * inv, v[j + 1] * inv, v[j + 2] * inv, v[j + 3] * inv);
        }
      }
      fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty(b));
    }
  }
  __syncthreads();
  if (warp == 0) {
    fence_after_sync();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kGCols) : "memory");
  }
}

}  // namespace

bool probe_fused_supported(const rslm_index* ix, int nprobe) {
  return ix->ctiles != nullptr && nprobe <= 256 && int64_t(ix->nlist) >= int64_t(32) * nprobe;
}

cudaError_t probe_prepare(rslm_index* ix, cudaStream_t s) {
  // centroid statistics and scale (both probes)
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(&ix->cmeta), 4 * sizeof(float));
  if (e != cudaSuccess) return e;
  ix->device_bytes += 16;
  centroid_stats_kernel<<<1, 1024, 0, s>>>(ix->centroids, ix->nlist, ix->D, ix->cmeta);
  centroid_tiles_meta_kernel<<<1, 1, 0, s>>>(ix->cmeta);
  // probe GEMM operand (every shape)
  const size_t gbytes = size_t((ix->nlist + kGN - 1) / kGN) * gemm_kchunks(ix->D) * kGBlockB;
  e = cudaMalloc(reinterpret_cast<void**>(&ix->cgemm), gbytes);
  if (e != cudaSuccess) return e;
  ix->device_bytes += int64_t(gbytes);
  centroid_gemm_blocks_kernel<<<152 * 4, 256, 0, s>>>(ix->centroids, ix->nlist, ix->D, ix->cmeta, ix->cgemm);
  const int Kp = (ix->D + 15) / 16 * 16;
  if (Kp > 128) return cudaGetLastError();  // the fused probe keeps whole rows in one K chunk
  const int ntiles = (ix->nlist + kPRows - 1) / kPRows;
  e = cudaMalloc(reinterpret_cast<void**>(&ix->ctiles), size_t(2) * ntiles * tile_bytes(Kp));
  if (e != cudaSuccess) return e;
  e = cudaMalloc(reinterpret_cast<void**>(&ix->crows), size_t(ix->nlist) * Kp * sizeof(float));
  if (e != cudaSuccess) return e;
  ix->device_bytes += int64_t(2) * ntiles * tile_bytes(Kp) + int64_t(ix->nlist) * Kp * 4;
  centroid_rows_kernel<<<152 * 4, 256, 0, s>>>(ix->centroids, ix->nlist, ix->D, Kp, ix->crows);
  centroid_tiles_kernel<<<152 * 4, 256, 0, s>>>(ix->centroids, ix->nlist, ix->D, Kp, ix->cmeta, ix->ctiles);
  return cudaGetLastError();
}

cudaError_t launch_probe_gemm(const rslm_index* ix, const float* queries, int64_t nq, int nprobe,
                              int32_t* out_probes, float* out_cs, cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  const int nkc = gemm_kchunks(ix->D);
  const int64_t ld = (int64_t(ix->nlist) + 3) & ~int64_t(3);  // row stride of S, a 16-byte multiple
  const int64_t budget = int64_t(64) << 20;                   // floats of S per query chunk (256 MB)
  int64_t qc = std::max<int64_t>(kGM, budget / ld / kGM * kGM);
  qc = std::min(qc, (nq + kGM - 1) / kGM * kGM);
  size_t bytes = 0;
  auto take = [&](size_t n) {
    size_t at = bytes;
    bytes += (n + 255) / 256 * 256;
    return at;
  };
  const size_t o_S = take(size_t(qc) * ld * 4), o_flags = take(size_t(qc) * 4),
               o_qb = take(size_t(qc / kGM) * nkc * kGBlockA), o_inv = take(size_t(qc) * 4);
  uint8_t* ws = nullptr;
  cudaError_t e = cudaMallocAsync(reinterpret_cast<void**>(&ws), bytes, s);
  if (e != cudaSuccess) return e;
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const size_t smem = size_t(kGStages) * kGStageBytes;
  e = cudaFuncSetAttribute(probe_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  for (int64_t q0 = 0; q0 < nq && e == cudaSuccess; q0 += qc) {
    const int64_t n = std::min(qc, nq - q0);
    const int64_t nqp = (n + kGM - 1) / kGM * kGM;
    query_gemm_blocks_kernel<<<unsigned(std::min<int64_t>((nqp + 7) / 8, int64_t(sms) * 64)), 256, 0, s>>>(
        queries + q0 * ix->D, n, ix->D, ix->cmeta, ws + o_qb, reinterpret_cast<float*>(ws + o_inv));
    GemmArgs a;
    a.qblk = ws + o_qb;
    a.cblk = ix->cgemm;
    a.qinv = reinterpret_cast<const float*>(ws + o_inv);
    a.nq = n;
    a.nlist = ix->nlist;
    a.nkc = nkc;
    a.ntm = int(nqp / kGM);
    a.ntn = (ix->nlist + kGN - 1) / kGN;
    a.S = reinterpret_cast<float*>(ws + o_S);
    a.ld = ld;
    a.err = ix->d_err;
    const int64_t units = int64_t(a.ntm) * a.ntn;
    probe_gemm_kernel<<<unsigned(std::min<int64_t>(units, sms)), kGThreads, smem, s>>>(a);
    e = cudaGetLastError();
    if (e == cudaSuccess)
      e = launch_select_topn(a.S, n, ld, ix->nlist, nprobe, out_probes + q0 * nprobe, out_cs + q0 * nprobe,
                             reinterpret_cast<int*>(ws + o_flags), s);
  }
  cudaError_t f = cudaFreeAsync(ws, s);
  return e != cudaSuccess ? e : f;
}

cudaError_t launch_probe_fused(const rslm_index* ix, const float* queries, int64_t nq, int nprobe,
                               int32_t* out_probes, float* out_cs, cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  const int Kp = (ix->D + 15) / 16 * 16;
  const int ntiles = (ix->nlist + kPRows - 1) / kPRows;
  const int64_t nblk = (nq + kPQ - 1) / kPQ;
  const int64_t nqp = nblk * kPQ;  // queries padded to whole CTAs
  const int cap = std::max(kListCapMin, 8 * nprobe);
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int sel_blocks = sms * 8, exact_blocks = sms * 2;
  size_t bytes = 0;
  auto take = [&](size_t n) {
    size_t at = bytes;
    bytes += (n + 255) / 256 * 256;
    return at;
  };
  const size_t o_qt = take(size_t(nblk) * 4 * tile_bytes(Kp)), o_d = take(size_t(nq) * 4),
               o_inv = take(size_t(nq) * 4), o_keys = take(size_t(nq) * cap * 8), o_cnt = take(size_t(nq) * 8),
               o_nx = take(4), o_xq = take(size_t(nq) * 4),
               o_scr = take(size_t(exact_blocks) * kExactWarpsPerBlock * ix->nlist * 4);
  uint8_t* ws = nullptr;
  cudaError_t e = cudaMallocAsync(reinterpret_cast<void**>(&ws), bytes, s);
  if (e != cudaSuccess) return e;
  int* nexact = reinterpret_cast<int*>(ws + o_nx);
  e = cudaMemsetAsync(nexact, 0, sizeof(int), s);
  if (e == cudaSuccess) {
    query_tiles_kernel<<<unsigned((nqp + 7) / 8 < 152 * 64 ? (nqp + 7) / 8 : 152 * 64), 256, 0, s>>>(
        queries, nq, nqp, ix->D, Kp, ix->cmeta, ws + o_qt, reinterpret_cast<float*>(ws + o_d),
        reinterpret_cast<float*>(ws + o_inv));
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) {
    ProbeArgs a;
    a.qtiles = ws + o_qt;
    a.ctiles = ix->ctiles;
    a.dthr = reinterpret_cast<const float*>(ws + o_d);
    a.nq = nq;
    a.nlist = ix->nlist;
    a.Kp = Kp;
    a.ntiles = ntiles;
    a.nprobe = nprobe;
    // whole chunks of each column half (chunk g is in half (g mod 4) / 2),
    // then the largest jth in {8, 4, 2, 1} for which ceil(nprobe / jth)
    // groups of at least jth chunks fit in the two halves, split evenly
    const int nch = ix->nlist / 32;
    const int hc[2] = {2 * (nch / 4) + std::min(nch % 4, 2), 2 * (nch / 4) + std::max(nch % 4 - 2, 0)};
    int jth = 1;
    for (int j = 8; j >= 1; j >>= 1) {
      const int G = (nprobe + j - 1) / j, f0 = hc[0] / j, f1 = hc[1] / j;
      if (f0 + f1 >= G || j == 1) {
        jth = j;
        a.ngr[0] = std::min(f0, std::max(G - f1, (G + 1) / 2));
        a.ngr[1] = G - a.ngr[0];
        for (int h = 0; h < 2; ++h) a.mch[h] = a.ngr[h] > 0 ? hc[h] / a.ngr[h] : 1;
        break;
      }
    }
    a.cap = cap;
    a.keys = reinterpret_cast<uint64_t*>(ws + o_keys);
    a.cnt = reinterpret_cast<int*>(ws + o_cnt);
    a.err = ix->d_err;
    // at least 116 KB, so one CTA per SM: each CTA holds all 512 TMEM columns
    const size_t smem = std::max(size_t(4 + kPStages) * tile_bytes(Kp), size_t(116) * 1024);
    auto kern = jth == 8 ? probe_kernel<8> : jth == 4 ? probe_kernel<4> : jth == 2 ? probe_kernel<2> : probe_kernel<1>;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e == cudaSuccess) {
      kern<<<unsigned(nblk), kPThreads, smem, s>>>(a);
      e = cudaGetLastError();
    }
  }
  if (e == cudaSuccess) {
    probe_select_kernel<<<unsigned(sel_blocks), kSelWarpsPerBlock * 32, 0, s>>>(
        nq, reinterpret_cast<const uint64_t*>(ws + o_keys), reinterpret_cast<const int*>(ws + o_cnt), cap,
        nprobe, reinterpret_cast<const float*>(ws + o_inv), nexact, reinterpret_cast<int32_t*>(ws + o_xq),
        ix->d_counters, out_probes, out_cs);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) {
    probe_exact_kernel<<<unsigned(exact_blocks), kExactWarpsPerBlock * 32, 0, s>>>(
        queries, ix->D, ix->crows, Kp, ix->nlist, nexact, reinterpret_cast<const int32_t*>(ws + o_xq), nprobe,
        reinterpret_cast<uint32_t*>(ws + o_scr), out_probes, out_cs);
    e = cudaGetLastError();
  }
  cudaError_t f = cudaFreeAsync(ws, s);
  return e != cudaSuccess ? e : f;
}

}  // namespace rslm
