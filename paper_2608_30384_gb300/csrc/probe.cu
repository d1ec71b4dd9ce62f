// probe.cu -- IVF probe (Sec. 5.5.1: the nprobe partitions with the largest
// <q, c_p>, ties to the lower p) on the tensor cores, without materialising
// the nq x nlist score matrix.
//
// For padded D <= 128 and nlist >= 32 nprobe:
//   1. queries and centroids are scaled by powers of two (max |q| and max |c|
//      into [1024, 2048)) and rounded to fp16 ("hi"); a = <q_hi, c_hi> is
//      within delta = 2^-9 ||q|| max ||c|| of <q, c> (each fp16 rounding is
//      relative 2^-11, Cauchy-Schwarz bounds the sum, fp32 accumulation adds
//      far less);
//   2. probe_kernel, per CTA of 256 queries, streams all centroid tiles
//      through tcgen05.mma twice.  Pass 1: the columns are split into
//      ceil(nprobe / j) disjoint groups of whole 32-column chunks, and each
//      group contributes the j-th largest of its chunk maxima of a (j <= 8),
//      which j distinct centroids of the group reach; the smallest
//      contribution is therefore reached by at least nprobe centroids, and
//      B = that value - delta is at most the nprobe-th largest true score.
//      Pass 2 appends every centroid with a >= B - delta (which includes
//      every centroid whose true score is >= B), with its a, to the query's
//      list in increasing index order;
//   3. probe_finish_kernel computes the exact fp32 <q, c> of the listed
//      centroids (all centroids when a list overflowed) and takes the top
//      nprobe by (score desc, p asc).
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
constexpr int kPThreads = 10 * 32;  // warps 0-7 epilogue, 8 TMA, 9 MMA
constexpr int kPEpiWarps = 8;
constexpr uint32_t kPCols = 512;  // TMEM: (M block, buffer) accumulators of 128 columns

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
  am = fmaxf(am, __shfl_xor_sync(kFull, am, 16));
  nm = fmaxf(nm, __shfl_xor_sync(kFull, nm, 16));
#pragma unroll
  for (int o = 8; o; o >>= 1) {
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

// Centroid operand: c * 2^sC rounded to fp16, one tile per 128 centroids
// (rows beyond nlist and dims beyond D are zero).  meta[2] = 2^sC,
// meta[3] = max ||c|| * 2^sC.
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
    __align__(16) __half h[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int d = k8 * 8 + j;
      const float v = (p < nlist && d < D) ? C[p * D + d] * sc : 0.0f;
      h[j] = __float2half_rn(v);
    }
    const int64_t t = p / kPRows;
    const int r = int(p % kPRows);
    *reinterpret_cast<uint4*>(tiles + t * tile_bytes(Kp) + ptile_off(r, k8 * 8, Kp)) =
        *reinterpret_cast<const uint4*>(h);
  }
}

// Query operand tiles (q * 2^sq in fp16, 128 queries per tile, nqb tiles,
// queries beyond nq zero) and 2 delta per query in the scaled units of
// <q_hi, c_hi>: 2 * 2^-9 ||q|| 2^sq * max ||c|| 2^sC.
__global__ void query_tiles_kernel(const float* __restrict__ Q, int64_t nq, int64_t nqp, int D, int Kp,
                                   const float* __restrict__ meta, uint8_t* __restrict__ tiles,
                                   float* __restrict__ delta2) {
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
    const float sc = ldexpf(1.0f, pow2_exp_for(m));
    const int64_t t = q / kPRows;
    const int r = int(q % kPRows);
    for (int k8 = lane; k8 < Kp / 8; k8 += 32) {
      __align__(16) __half h[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int d = k8 * 8 + j;
        h[j] = __float2half_rn((q < nq && d < D) ? Q[q * D + d] * sc : 0.0f);
      }
      *reinterpret_cast<uint4*>(tiles + t * tile_bytes(Kp) + ptile_off(r, k8 * 8, Kp)) =
          *reinterpret_cast<const uint4*>(h);
    }
    if (lane == 0 && q < nq) delta2[q] = 2.0f * ldexpf(1.0f, -9) * sqrtf(s2) * sc * meta[3] * 1.001f;
  }
}

struct ProbeArgs {
  const uint8_t* qtiles;
  const uint8_t* ctiles;
  const float* delta2;
  int64_t nq;
  // bound groups: ngr groups of mch consecutive 32-column chunks; a group
  // contributes its jth-largest chunk maximum (jth <= 8, jth * ngr >= nprobe)
  int nlist, Kp, ntiles, nprobe, mch, ngr, jth;
  int cap;
  int32_t* cand;  // [nq * cap] listed centroids
  float* cval;    // [nq * cap] their a = <q_hi, c_hi>
  int* cnt;       // [nq]
  int* err;
};

__global__ void __launch_bounds__(kPThreads, 1) probe_kernel(const __grid_constant__ ProbeArgs a) {
  extern __shared__ __align__(128) uint8_t sm[];
  __shared__ __align__(8) uint64_t bars[1 + 2 * kPStages + 4];
  __shared__ uint32_t tmem_base_sh;
  __shared__ int s_fail;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int TB = tile_bytes(a.Kp);
  uint8_t* A0 = sm;                 // two query tiles
  uint8_t* B0 = sm + 2 * TB;        // kPStages centroid tiles, then the value stage
  const uint32_t bar0 = uint32_t(__cvta_generic_to_shared(&bars[0]));
  const uint32_t a_full = bar0;
  auto b_full = [&](uint32_t s) { return bar0 + 8u * (1 + s); };
  auto b_empty = [&](uint32_t s) { return bar0 + 8u * (1 + kPStages + s); };
  auto mma_done = [&](uint32_t b) { return bar0 + 8u * (1 + 2 * kPStages + b); };
  auto acc_empty = [&](uint32_t b) { return bar0 + 8u * (3 + 2 * kPStages + b); };
  if (tid == 0) {
    s_fail = 0;
    mbar_init(a_full, 1);
    for (uint32_t s = 0; s < kPStages; ++s) {
      mbar_init(b_full(s), 1);
      mbar_init(b_empty(s), 1);
    }
    for (uint32_t b = 0; b < 2; ++b) {
      mbar_init(mma_done(b), 1);
      mbar_init(acc_empty(b), kPEpiWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
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
  const int ngt = 2 * a.ntiles;  // tiles of both passes
  auto fail = [&]() {
    set_device_error(a.err, kErrTimeout);
    atomicExch(&s_fail, 1);
  };
  auto acc_col = [&](int m, uint32_t b) { return uint32_t((m * 2 + int(b)) * 128); };

  if (warp == 8) {
    // ---------------- TMA: the CTA's two query tiles, then every centroid tile twice
    if (lane == 0) {
      mbar_arrive_expect(a_full, uint32_t(2 * TB));
      bulk_copy_1d(a_addr, a.qtiles + size_t(blockIdx.x) * 2 * TB, uint32_t(2 * TB), a_full);
      int gt = 0;
      for (; gt < ngt; ++gt) {
        const uint32_t s = uint32_t(gt % kPStages), u = uint32_t(gt / kPStages);
        if (u > 0 && !mbar_wait(b_empty(s), (u - 1) & 1)) {
          fail();
          break;
        }
        const int t = gt % a.ntiles;
        mbar_arrive_expect(b_full(s), uint32_t(TB));
        bulk_copy_1d(b_addr + s * uint32_t(TB), a.ctiles + size_t(t) * TB, uint32_t(TB), b_full(s));
      }
      // no copy may still be landing when the CTA exits
      mbar_wait(a_full, 0);
      for (int s = 0; s < kPStages && s < gt; ++s) mbar_wait(b_full(uint32_t(s)), uint32_t((gt - 1 - s) / kPStages) & 1);
    }
    __syncwarp();
  } else if (warp == 9) {
    // ---------------- MMA issue: both M blocks against each centroid tile
    if (lane == 0) {
      const uint32_t idesc = f16_idesc(kPRows, kPRows);
      const uint32_t sbo = uint32_t(a.Kp / 8) * 128;
      bool ok = mbar_wait(a_full, 0);
      if (!ok) fail();
      int gt = 0;
      for (; ok && gt < ngt; ++gt) {
        const uint32_t s = uint32_t(gt % kPStages), u = uint32_t(gt / kPStages);
        const uint32_t b = uint32_t(gt & 1), ub = uint32_t(gt >> 1);
        if (!mbar_wait(b_full(s), u & 1) || (ub > 0 && !mbar_wait(acc_empty(b), (ub - 1) & 1))) {
          fail();
          break;
        }
        fence_after_sync();
        for (int m = 0; m < 2; ++m)
          for (int ks = 0; ks < a.Kp / 16; ++ks)
            umma_f16(tmem + acc_col(m, b), smem_desc(a_addr + uint32_t(m * TB + ks * 256), 128, sbo),
                     smem_desc(b_addr + s * uint32_t(TB) + uint32_t(ks * 256), 128, sbo), idesc,
                     ks > 0 ? 1u : 0u);
        umma_commit(b_empty(s));
        umma_commit(mma_done(b));
      }
      // no MMA may still be running when TMEM is freed
      if (gt > 0) mbar_wait(mma_done(uint32_t((gt - 1) & 1)), uint32_t(((gt - 1) >> 1) & 1));
    }
    __syncwarp();
  } else {
    // ---------------- epilogue: thread = one query row of M block m
    const int m = warp >> 2, qd = warp & 3;
    const int64_t q = int64_t(blockIdx.x) * kPQ + m * kPRows + qd * 32 + lane;
    const bool valid = q < a.nq;
    const uint32_t lane_base = uint32_t(qd * 32) << 16;
    const int ngroups_chunks = a.ngr * a.mch;  // chunks that form the bound groups
    float top[8];  // the group's largest chunk maxima, descending
#pragma unroll
    for (int j = 0; j < 8; ++j) top[j] = -CUDART_INF_F;
    float bound = CUDART_INF_F, thr = CUDART_INF_F;
    int n = 0, in_group = 0;  // chunks of the current bound group seen
    // this thread's row of the value stage: value i of a chunk at word i * kPThreads + tid
    float* stage = reinterpret_cast<float*>(sm + (2 + kPStages) * size_t(TB)) + tid;
    int32_t* out = a.cand + (valid ? q : 0) * int64_t(a.cap);
    float* outv = a.cval + (valid ? q : 0) * int64_t(a.cap);
    for (int gt = 0; gt < ngt; ++gt) {
      const uint32_t b = uint32_t(gt & 1), ub = uint32_t(gt >> 1);
      if (!mbar_wait(mma_done(b), ub & 1)) {
        fail();
        break;
      }
      fence_after_sync();
      const bool pass1 = gt < a.ntiles;
      const int t = pass1 ? gt : gt - a.ntiles;
      if (gt == a.ntiles) thr = bound - (valid ? a.delta2[q] : 0.0f);
      // the tile's 128 columns in one load (a TMEM load issued while the
      // tensor core is busy has a long latency), then release the accumulator
      float vt[kPRows];
      tmem_ld128(tmem + lane_base + acc_col(m, b), vt);
      fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty(b));
#pragma unroll
      for (int c = 0; c < kPRows / 32; ++c) {
        float v[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = vt[c * 32 + i];
        float mx = -CUDART_INF_F;
#pragma unroll
        for (int i = 0; i < 32; i += 2) mx = fmax3(mx, v[i], v[i + 1]);
        const int gc = t * (kPRows / 32) + c;  // 32-column chunk index
        if (pass1) {
          if (gc < ngroups_chunks) {
            float x = mx;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float hi = fmaxf(top[j], x);
              x = fminf(top[j], x);
              top[j] = hi;
            }
            if (++in_group == a.mch) {
              // at least jth centroids of this group reach top[jth - 1]
              float tj = top[0];
#pragma unroll
              for (int j = 1; j < 8; ++j) tj = j == a.jth - 1 ? top[j] : tj;
              bound = fminf(bound, tj);
#pragma unroll
              for (int j = 0; j < 8; ++j) top[j] = -CUDART_INF_F;
              in_group = 0;
            }
          }
        } else if (mx >= thr && valid) {
          // append the columns at or above thr, in increasing index order
          const int col0 = gc * 32;
          uint32_t hit = 0;
#pragma unroll
          for (int i = 0; i < 32; ++i) hit |= (v[i] >= thr ? 1u : 0u) << i;
          const int nreal = max(0, min(32, a.nlist - col0));  // columns beyond nlist are padding
          hit &= nreal == 32 ? ~0u : ((1u << nreal) - 1u);
          if (hit) {
#pragma unroll
            for (int i = 0; i < 32; ++i) stage[i * kPThreads] = v[i];
          }
          while (hit) {
            const int i = __ffs(hit) - 1;
            hit &= hit - 1;
            if (n < a.cap) {
              out[n] = col0 + i;
              outv[n] = stage[i * kPThreads];
            }
            ++n;
          }
        }
      }
    }
    if (valid) a.cnt[q] = n;
  }
  __syncthreads();
  if (warp == 0) {
    fence_after_sync();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kPCols) : "memory");
  }
}

// Centroids again as fp32 rows of Kp floats (zero padded), so every row is
// 16-byte aligned for the exact rescoring below.
__global__ void centroid_rows_kernel(const float* __restrict__ C, int nlist, int D, int Kp,
                                     float* __restrict__ out) {
  const int64_t total = int64_t(nlist) * Kp;
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < total;
       i += int64_t(gridDim.x) * blockDim.x) {
    const int d = int(i % Kp);
    out[i] = d < D ? C[(i / Kp) * D + d] : 0.0f;
  }
}

// Exact top-nprobe of every query from its list: fp32 <q, c> of the listed
// centroids (every centroid when the list overflowed), the nprobe-th largest
// order key T bit by bit, the centroids above T plus the lowest-index ones at
// T, sorted by (score desc, p asc).  One warp per query; the warp scores
// eight candidates per step (four groups of eight lanes, two candidates each,
// a lane holding Kp / 8 dims).  Keys of a list live in shared memory; an
// overflowed list uses the warp's global scratch row of nlist keys.
constexpr int kFinWarpsPerBlock = 4;
constexpr int kFinCap = 1024;
__global__ void __launch_bounds__(kFinWarpsPerBlock * 32) probe_finish_kernel(
    const float* __restrict__ Q, int64_t nq, int D, const float* __restrict__ Cp, int Kp, int nlist,
    const int32_t* __restrict__ cand, const float* __restrict__ cval, const float* __restrict__ delta2,
    const int* __restrict__ cnt, int cap, int k, uint32_t* __restrict__ scratch,
    int32_t* __restrict__ out_probes, float* __restrict__ out_cs) {
  __shared__ uint32_t skeys[kFinWarpsPerBlock][kFinCap];
  __shared__ int32_t sids[kFinWarpsPerBlock][kFinCap];
  __shared__ uint32_t sk[kFinWarpsPerBlock][256];
  __shared__ int32_t si[kFinWarpsPerBlock][256];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int grp = lane >> 3, sub = lane & 7;
  const int64_t gw = int64_t(blockIdx.x) * kFinWarpsPerBlock + w;
  const int64_t nw = int64_t(gridDim.x) * kFinWarpsPerBlock;
  const int nf = Kp / 4;  // float4 of a row; lane sub takes f = sub + 8 j (Kp <= 128)
  for (int64_t q = gw; q < nq; q += nw) {
    float4 qv[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      float e[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int d = (sub + 8 * j) * 4 + c;
        e[c] = (sub + 8 * j < nf && d < D) ? Q[q * D + d] : 0.0f;
      }
      qv[j] = make_float4(e[0], e[1], e[2], e[3]);
    }
    const int nc = cnt[q];
    const bool all = nc > cap;
    const int32_t* cl = cand + q * int64_t(cap);
    uint32_t* keys = all ? scratch + gw * int64_t(nlist) : skeys[w];
    int n = all ? nlist : nc;
    if (!all) {
      // Keep only the listed centroids whose a is within 2 delta of the k-th
      // largest a (A_k): the k centroids at or above A_k score at least
      // A_k - delta, so no centroid below A_k - 2 delta is in the top k.
      const float* cv = cval + q * int64_t(cap);
      for (int i = lane; i < n; i += 32) keys[i] = float_order_key(cv[i]);
      __syncwarp();
      uint32_t Ak = 0u;
      for (int bit = 31; bit >= 0; --bit) {
        const uint32_t t = Ak | (1u << bit);
        int c0 = 0;
        for (int i = lane; i < n; i += 32) c0 += keys[i] >= t ? 1 : 0;
        if (int(__reduce_add_sync(kFull, uint32_t(c0))) >= k) Ak = t;
      }
      const uint32_t lim = float_order_key(float_from_order_key(Ak) - delta2[q]);
      const unsigned lt = (1u << lane) - 1u;
      int m = 0;
      for (int base = 0; base < n; base += 32) {
        const int i = base + lane;
        const bool keep = i < n && keys[i] >= lim;
        const unsigned bal = __ballot_sync(kFull, keep);
        const int id = keep ? cl[i] : 0;
        __syncwarp();
        if (keep) sids[w][m + __popc(bal & lt)] = id;
        m += __popc(bal);
      }
      __syncwarp();
      cl = sids[w];
      n = m;
    }
    for (int i0 = 0; i0 < n; i0 += 8) {
      float acc[2];
      int idx[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        idx[u] = i0 + 4 * u + grp;
        const int p = idx[u] < n ? (all ? idx[u] : cl[idx[u]]) : 0;
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
        if (sub == 0 && idx[u] < n) keys[idx[u]] = float_order_key(acc[u]);
      }
    }
    __syncwarp();
    // T = the k-th largest key
    uint32_t T = 0u;
    for (int bit = 31; bit >= 0; --bit) {
      const uint32_t t = T | (1u << bit);
      int c0 = 0;
      for (int i = lane; i < n; i += 32) c0 += keys[i] >= t ? 1 : 0;
      if (int(__reduce_add_sync(kFull, uint32_t(c0))) >= k) T = t;
    }
    // keys above T (fewer than k), then the lowest-index keys equal to T
    const unsigned lt = (1u << lane) - 1u;
    int ngt = 0, neq = 0, ngt_tot = 0;
    for (int base = 0; base < n; base += 32) {
      const int i = base + lane;
      ngt_tot += __popc(__ballot_sync(kFull, i < n && keys[i] > T));
    }
    for (int base = 0; base < n; base += 32) {
      const int i = base + lane;
      const uint32_t key = i < n ? keys[i] : 0u;
      const bool gtr = i < n && key > T, eq = i < n && key == T;
      const unsigned bg = __ballot_sync(kFull, gtr), be = __ballot_sync(kFull, eq);
      const int p = i < n ? (all ? i : cl[i]) : 0;
      if (gtr) {
        const int at = ngt + __popc(bg & lt);
        sk[w][at] = key;
        si[w][at] = p;
      }
      if (eq) {
        const int at = ngt_tot + neq + __popc(be & lt);
        if (at < k) {
          sk[w][at] = key;
          si[w][at] = p;
        }
      }
      ngt += __popc(bg);
      neq += __popc(be);
    }
    int p2 = 1;
    while (p2 < k) p2 <<= 1;
    for (int i = k + lane; i < p2; i += 32) {
      sk[w][i] = 0u;
      si[w][i] = INT_MAX;
    }
    __syncwarp();
    for (int size = 2; size <= p2; size <<= 1) {
      for (int stride = size >> 1; stride > 0; stride >>= 1) {
        for (int i = lane; i < (p2 >> 1); i += 32) {
          const int lo = 2 * i - (i & (stride - 1));
          const int hi = lo + stride;
          const bool asc = (lo & size) == 0;
          const uint32_t klo = sk[w][lo], khi = sk[w][hi];
          const int32_t ilo = si[w][lo], ihi = si[w][hi];
          const bool swap = asc ? better(khi, ihi, klo, ilo) : better(klo, ilo, khi, ihi);
          if (swap) {
            sk[w][lo] = khi;
            sk[w][hi] = klo;
            si[w][lo] = ihi;
            si[w][hi] = ilo;
          }
        }
        __syncwarp();
      }
    }
    for (int i = lane; i < k; i += 32) {
      out_probes[q * k + i] = si[w][i];
      out_cs[q * k + i] = float_from_order_key(sk[w][i]);
    }
    __syncwarp();
  }
}

}  // namespace

bool probe_fused_supported(const rslm_index* ix, int nprobe) {
  return ix->ctiles != nullptr && nprobe <= 256 && int64_t(ix->nlist) >= int64_t(32) * nprobe;
}

cudaError_t probe_prepare(rslm_index* ix, cudaStream_t s) {
  const int Kp = (ix->D + 15) / 16 * 16;
  if (Kp > 128) return cudaSuccess;  // the fused probe keeps whole rows in one K chunk
  const int ntiles = (ix->nlist + kPRows - 1) / kPRows;
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(&ix->ctiles), size_t(ntiles) * tile_bytes(Kp));
  if (e != cudaSuccess) return e;
  e = cudaMalloc(reinterpret_cast<void**>(&ix->cmeta), 4 * sizeof(float));
  if (e != cudaSuccess) return e;
  e = cudaMalloc(reinterpret_cast<void**>(&ix->crows), size_t(ix->nlist) * Kp * sizeof(float));
  if (e != cudaSuccess) return e;
  ix->device_bytes += int64_t(ntiles) * tile_bytes(Kp) + 16 + int64_t(ix->nlist) * Kp * 4;
  centroid_rows_kernel<<<152 * 4, 256, 0, s>>>(ix->centroids, ix->nlist, ix->D, Kp, ix->crows);
  centroid_stats_kernel<<<1, 1024, 0, s>>>(ix->centroids, ix->nlist, ix->D, ix->cmeta);
  centroid_tiles_kernel<<<152 * 4, 256, 0, s>>>(ix->centroids, ix->nlist, ix->D, Kp, ix->cmeta, ix->ctiles);
  return cudaGetLastError();
}

cudaError_t launch_probe_fused(const rslm_index* ix, const float* queries, int64_t nq, int nprobe,
                               int32_t* out_probes, float* out_cs, cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  const int Kp = (ix->D + 15) / 16 * 16;
  const int ntiles = (ix->nlist + kPRows - 1) / kPRows;
  const int64_t nblk = (nq + kPQ - 1) / kPQ;
  const int64_t nqp = nblk * kPQ;  // queries padded to whole CTAs
  const int cap = kFinCap;
  int sms = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int fin_blocks = sms * 8;
  const int64_t scratch_row = ix->nlist;
  size_t bytes = 0;
  auto take = [&](size_t n) {
    size_t at = bytes;
    bytes += (n + 255) / 256 * 256;
    return at;
  };
  const size_t o_qt = take(size_t(nblk) * 2 * tile_bytes(Kp)), o_d = take(size_t(nq) * 4),
               o_cand = take(size_t(nq) * cap * 4), o_cval = take(size_t(nq) * cap * 4),
               o_cnt = take(size_t(nq) * 4),
               o_scr = take(size_t(fin_blocks) * kFinWarpsPerBlock * scratch_row * 4);
  uint8_t* ws = nullptr;
  cudaError_t e = cudaMallocAsync(reinterpret_cast<void**>(&ws), bytes, s);
  if (e != cudaSuccess) return e;
  query_tiles_kernel<<<unsigned((nqp + 7) / 8 < 152 * 64 ? (nqp + 7) / 8 : 152 * 64), 256, 0, s>>>(
      queries, nq, nqp, ix->D, Kp, ix->cmeta, ws + o_qt, reinterpret_cast<float*>(ws + o_d));
  e = cudaGetLastError();
  if (e == cudaSuccess) {
    ProbeArgs a;
    a.qtiles = ws + o_qt;
    a.ctiles = ix->ctiles;
    a.delta2 = reinterpret_cast<const float*>(ws + o_d);
    a.nq = nq;
    a.nlist = ix->nlist;
    a.Kp = Kp;
    a.ntiles = ntiles;
    a.nprobe = nprobe;
    // the largest jth in {8, 4, 2, 1} whose ceil(nprobe / jth) groups of at
    // least jth chunks fit in the nlist / 32 whole chunks
    const int nch = ix->nlist / 32;
    for (int j = 8; j >= 1; j >>= 1) {
      const int ng = (nprobe + j - 1) / j;
      if (nch / ng >= j || j == 1) {
        a.jth = j;
        a.ngr = ng;
        a.mch = nch / ng;
        break;
      }
    }
    a.cap = cap;
    a.cand = reinterpret_cast<int32_t*>(ws + o_cand);
    a.cval = reinterpret_cast<float*>(ws + o_cval);
    a.cnt = reinterpret_cast<int*>(ws + o_cnt);
    a.err = ix->d_err;
    // at least 116 KB, so one CTA per SM: each CTA holds all 512 TMEM columns
    const size_t smem = std::max(size_t(2 + kPStages) * tile_bytes(Kp) + size_t(32) * kPThreads * 4,
                                 size_t(116) * 1024);
    e = cudaFuncSetAttribute(probe_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e == cudaSuccess) {
      probe_kernel<<<unsigned(nblk), kPThreads, smem, s>>>(a);
      e = cudaGetLastError();
    }
  }
  if (e == cudaSuccess) {
    probe_finish_kernel<<<unsigned(fin_blocks), kFinWarpsPerBlock * 32, 0, s>>>(
        queries, nq, ix->D, ix->crows, Kp, ix->nlist, reinterpret_cast<const int32_t*>(ws + o_cand),
        reinterpret_cast<const float*>(ws + o_cval), reinterpret_cast<const float*>(ws + o_d),
        reinterpret_cast<const int*>(ws + o_cnt), cap, nprobe, reinterpret_cast<uint32_t*>(ws + o_scr),
        out_probes, out_cs);
    e = cudaGetLastError();
  }
  cudaError_t f = cudaFreeAsync(ws, s);
  return e != cudaSuccess ? e : f;
}

}  // namespace rslm
