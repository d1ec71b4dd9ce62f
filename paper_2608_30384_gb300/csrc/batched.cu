// batched.cu -- partition-major scan for query batches that share partitions.
//
// When many queries probe the same partition (nq * nprobe / nlist large), the
// per-row dot products <R q, uhat_j> of Sec. 3.5 form a dense contraction:
// (rows of a partition x D) decoded codewords times (D x queries) rotated
// queries.  This path
//   1. inverts the probe lists into per-partition query lists,
//   2. takes a per-query lower bound theta_q on the k-th best score from a
//      one-partition pass of the single-query scan (the k-th best score of
//      any subset of the candidates is <= the k-th best of all of them),
//   3. for every (partition, tile of up to 128 of its queries) decodes the
//      codes of 128-row tiles once into shared memory as fp16 (the codebook
//      components are binary16-exact) and multiplies them on the tensor cores
//      with the queries split into fp16 hi + lo parts (fp32 accumulation: the
//      split keeps about 22 significant bits of the query), then applies
//      s = G (cs + L dot) and appends only the candidates with s >= theta_q to
//      a per-query buffer,
//   4. takes the exact top-k of every buffer, ordered by (score desc, id asc);
//      a query whose buffer overflowed is re-scanned by the single-query path.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math_constants.h>

#include <algorithm>
#include <cmath>
#include <climits>

#include "device_common.cuh"
#include "launch.h"
#include "tcgen05.cuh"

namespace rslm {
namespace {

constexpr int kNQ = 128;    // queries per work item
constexpr int kMR = 128;    // rows per tile
constexpr int kKC = 128;    // dimensions per K chunk held in shared memory

// ------------------------------------------------------ probe-list inversion
// Pairs (query q, probe slot j < eff) of probe lists with rows `stride` long.
__global__ void count_pairs_kernel(const int32_t* __restrict__ probes, int64_t nq, int stride, int eff,
                                   int nlist, int* __restrict__ cnt, int* err) {
  const int64_t npairs = nq * eff;
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < npairs;
       i += int64_t(gridDim.x) * blockDim.x) {
    const int p = probes[(i / eff) * stride + i % eff];
    if (p >= 0 && p < nlist) atomicAdd(&cnt[p], 1);
    else set_device_error(err, kErrBadProbe);
  }
}

// Single block: off[p] = exclusive prefix of cnt; items[p] = prefix of
// ceil(cnt / kNQ); off[nlist], items[nlist] = totals.
__global__ void scan_lists_kernel(const int* __restrict__ cnt, int nlist, int* __restrict__ off,
                                  int* __restrict__ items) {
  __shared__ int scratch[32];
  int run_o = 0, run_i = 0;
  for (int base = 0; base < nlist; base += blockDim.x) {
    const int p = base + threadIdx.x;
    const int c = p < nlist ? cnt[p] : 0;
    int tot_o, tot_i;
    const int eo = block_exclusive_scan(c, scratch, &tot_o);
    const int ei = block_exclusive_scan((c + kNQ - 1) / kNQ, scratch, &tot_i);
    if (p < nlist) {
      off[p] = run_o + eo;
      items[p] = run_i + ei;
    }
    run_o += tot_o;
    run_i += tot_i;
  }
  if (threadIdx.x == 0) {
    off[nlist] = run_o;
    items[nlist] = run_i;
  }
}

// item_p[i] = the partition of work item i (items[p] <= i < items[p + 1]).
__global__ void item_part_kernel(const int* __restrict__ items, int nlist, int* __restrict__ item_p) {
  for (int p = blockIdx.x * blockDim.x + threadIdx.x; p < nlist; p += gridDim.x * blockDim.x)
    for (int i = items[p]; i < items[p + 1]; ++i) item_p[i] = p;
}

__global__ void scatter_pairs_kernel(const int32_t* __restrict__ probes, const float* __restrict__ cs,
                                     int64_t nq, int stride, int eff, int nlist,
                                     const int* __restrict__ off, int* __restrict__ fill,
                                     int32_t* __restrict__ lq, float* __restrict__ lcs) {
  const int64_t npairs = nq * eff;
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < npairs;
       i += int64_t(gridDim.x) * blockDim.x) {
    const int64_t src = (i / eff) * stride + i % eff;
    const int p = probes[src];
    if (p < 0 || p >= nlist) continue;
    const int at = off[p] + atomicAdd(&fill[p], 1);
    lq[at] = int32_t(i / eff);
    lcs[at] = cs ? cs[src] : 0.0f;  // no cs: full-vector codes
  }
}

// The same inversion without a global atomic per pair, for nlist small
// enough for a shared-memory histogram: block b takes the pairs
// [b chunk, (b + 1) chunk) and writes their per-partition counts to row b of
// ghist; hist_prefix_kernel turns every column into its exclusive prefix over
// blocks (cnt[p] = the total); scatter_hist_kernel places block b's pairs of
// partition p at off[p] + ghist[b][p] + their rank inside the block.
constexpr int kHistBlocks = 2 * 152;
constexpr int kHistMaxList = 24576;  // shared-memory histogram: nlist ints
__global__ void __launch_bounds__(1024) hist_pairs_kernel(const int32_t* __restrict__ probes, int64_t nq,
                                                          int stride, int eff, int nlist, int64_t chunk,
                                                          int* __restrict__ ghist, int* err) {
  extern __shared__ int h[];
  for (int p = threadIdx.x; p < nlist; p += blockDim.x) h[p] = 0;
  __syncthreads();
  const int64_t npairs = nq * eff;
  const int64_t lo = blockIdx.x * chunk, hi = min(npairs, lo + chunk);
  for (int64_t i = lo + threadIdx.x; i < hi; i += blockDim.x) {
    const int p = probes[(i / eff) * stride + i % eff];
    if (p >= 0 && p < nlist) atomicAdd(&h[p], 1);
    else set_device_error(err, kErrBadProbe);
  }
  __syncthreads();
  for (int p = threadIdx.x; p < nlist; p += blockDim.x) ghist[int64_t(blockIdx.x) * nlist + p] = h[p];
}

// The column prefix in two steps over segments of kHistSeg rows, one thread
// per (column, segment): segment sums, then each segment's rows rewritten
// from the sum of the segments above it.
constexpr int kHistSeg = 16;
__global__ void hist_segsum_kernel(const int* __restrict__ ghist, int nb, int nlist, int* __restrict__ segsum) {
  const int p = blockIdx.x * blockDim.x + threadIdx.x, seg = blockIdx.y;
  if (p >= nlist) return;
  int sum = 0;
#pragma unroll
  for (int r = 0; r < kHistSeg; ++r) {
    const int b = seg * kHistSeg + r;
    if (b < nb) sum += ghist[int64_t(b) * nlist + p];
  }
  segsum[int64_t(seg) * nlist + p] = sum;
}

__global__ void hist_prefix_kernel(int* __restrict__ ghist, const int* __restrict__ segsum, int nb, int nlist,
                                   int* __restrict__ cnt) {
  const int p = blockIdx.x * blockDim.x + threadIdx.x, seg = blockIdx.y;
  if (p >= nlist) return;
  int run = 0;
  for (int s2 = 0; s2 < seg; ++s2) run += segsum[int64_t(s2) * nlist + p];
#pragma unroll
  for (int r = 0; r < kHistSeg; ++r) {
    const int b = seg * kHistSeg + r;
    if (b < nb) {
      const int v = ghist[int64_t(b) * nlist + p];
      ghist[int64_t(b) * nlist + p] = run;
      run += v;
    }
  }
  if (seg == int(gridDim.y) - 1) cnt[p] = run;
}

__global__ void __launch_bounds__(1024) scatter_hist_kernel(const int32_t* __restrict__ probes,
                                                            const float* __restrict__ cs, int64_t nq,
                                                            int stride, int eff, int nlist, int64_t chunk,
                                                            const int* __restrict__ off,
                                                            const int* __restrict__ ghist,
                                                            int32_t* __restrict__ lq, float* __restrict__ lcs) {
  extern __shared__ int base[];
  for (int p = threadIdx.x; p < nlist; p += blockDim.x)
    base[p] = off[p] + ghist[int64_t(blockIdx.x) * nlist + p];
  __syncthreads();
  const int64_t npairs = nq * eff;
  const int64_t lo = blockIdx.x * chunk, hi = min(npairs, lo + chunk);
  for (int64_t i = lo + threadIdx.x; i < hi; i += blockDim.x) {
    const int64_t src = (i / eff) * stride + i % eff;
    const int p = probes[src];
    if (p < 0 || p >= nlist) continue;
    const int at = atomicAdd(&base[p], 1);
    lq[at] = int32_t(i / eff);
    lcs[at] = cs ? cs[src] : 0.0f;  // no cs: full-vector codes
  }
}

// --------------------------------------------------------- query operands
// q * 2^s (s puts max |q| in [1024, 2048)) split into fp16 hi + lo;
// inv = 2^-s.  Dimensions Dp..Dp16 are zero.
__global__ void split_queries_kernel(const float* __restrict__ qrot, int64_t nq, int Dp, int Dp16,
                                     __half* __restrict__ qhi, __half* __restrict__ qlo,
                                     float* __restrict__ qinv, float* __restrict__ qrho, float U) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, W = blockDim.x >> 5;
  for (int64_t q = int64_t(blockIdx.x) * W + warp; q < nq; q += int64_t(gridDim.x) * W) {
    const float* src = qrot + q * Dp;
    float m = 0.0f;
    for (int d = lane; d < Dp; d += 32) m = fmaxf(m, fabsf(src[d]));
#pragma unroll
    for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(kFull, m, o));
    int e = 0;
    if (m > 0.0f) frexpf(m, &e);  // m in [2^(e-1), 2^e)
    const int s = 11 - e;
    const float sc = ldexpf(1.0f, s);
    float l2 = 0.0f;  // ||v - hi||^2 (the exact remainder, before its own rounding)
    for (int d = lane; d < Dp16; d += 32) {
      const float v = d < Dp ? src[d] * sc : 0.0f;
      const __half h = __float2half_rn(v);
      const float r = v - __half2float(h);
      qhi[q * Dp16 + d] = h;
      qlo[q * Dp16 + d] = __float2half_rn(r);
      l2 = fmaf(r, r, l2);
    }
    if (qrho) {
#pragma unroll
      for (int o = 16; o; o >>= 1) l2 += __shfl_xor_sync(kFull, l2, o);
      // |<v - hi, uhat>| <= ||v - hi|| ||uhat||, ||uhat|| <= U; rounded up
      // against the float rounding of the norm
      if (lane == 0) qrho[q] = U * sqrtf(l2) * (1.0f + 1e-5f);
    }
    if (lane == 0) qinv[q] = ldexpf(1.0f, -s);
  }
}

// Radix select, by one block, of the k-th largest order key among n scores
// (n > k).  Returns the key; every thread gets it.
__device__ uint32_t block_kth_key(const float* s, int n, int k, uint32_t* hist, uint32_t* sh) {
  const int tid = threadIdx.x;
  uint32_t prefix = 0, mask = 0, rem = uint32_t(k);
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int i = tid; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int base = 0; base < n; base += blockDim.x) {
      const int i = base + tid;
      const uint32_t kk = i < n ? float_order_key(s[i]) : 0u;
      warp_hist_add(hist, (kk >> shift) & 255u, i < n && (kk & mask) == prefix);
    }
    __syncthreads();
    if (tid < 32) {
      // lane l holds bins 255 - 8 l .. 248 - 8 l (from the top); the first
      // bin, from the top, where the count reaches rem
      uint32_t c8[8], tot = 0u;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        c8[j] = hist[255 - 8 * tid - j];
        tot += c8[j];
      }
      uint32_t incl = tot;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(kFull, incl, o);
        if (tid >= o) incl += y;
      }
      const uint32_t excl = incl - tot;
      const unsigned hit = __ballot_sync(kFull, excl < rem && incl >= rem);
      if (tid == __ffs(hit) - 1) {
        uint32_t cum = excl;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (cum + c8[j] >= rem) {
            sh[0] = rem - cum;
            sh[1] = prefix | (uint32_t(255 - 8 * tid - j) << shift);
            break;
          }
          cum += c8[j];
        }
      }
    }
    __syncthreads();
    rem = sh[0];
    prefix = sh[1];
    mask |= 255u << shift;
    __syncthreads();
  }
  return prefix;
}

// theta_q bounds the query's k-th best score from below: k distinct
// candidates of its first probed partition (all of whose scores are in the
// buffer) reach the k-th largest of the maxima of 256 interleaved groups
// (element i in group i mod 256); lowered by a relative margin of 1e-6;
// -inf when that partition has fewer than k rows.  One warp per query; the
// k-th largest group maximum is found bit by bit.
__device__ __forceinline__ float theta_from(float t) { return t - 1e-6f * fabsf(t) - 1e-30f; }

__global__ void __launch_bounds__(256) theta_warp_kernel(const float* __restrict__ buf_s,
                                                         const int* __restrict__ cnt, int64_t nq, int cap,
                                                         int k, float* __restrict__ theta) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t q = int64_t(blockIdx.x) * 8 + w;
  if (q >= nq) return;
  const int n = min(cnt[q], cap);
  if (n < k) {
    if (lane == 0) theta[q] = -CUDART_INF_F;
    return;
  }
  const float* s = buf_s + q * cap;
  uint32_t gm[8];
#pragma unroll
  for (int c = 0; c < 8; ++c) gm[c] = 0u;
  for (int base = 0; base < n; base += 256) {
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      const int i = base + 32 * c + lane;
      if (i < n) gm[c] = max(gm[c], float_order_key(s[i]));
    }
  }
  // the largest t with #{gm >= t} >= k (groups without an element hold 0)
  uint32_t bound = 0u;
  for (int bit = 31; bit >= 0; --bit) {
    const uint32_t t = bound | (1u << bit);
    int c0 = 0;
#pragma unroll
    for (int c = 0; c < 8; ++c) c0 += gm[c] >= t ? 1 : 0;
    if (int(__reduce_add_sync(kFull, uint32_t(c0))) >= k) bound = t;
  }
  if (lane == 0) theta[q] = theta_from(float_from_order_key(bound));
}

struct BatchArgs {
  const uint8_t* codes;
  const uint32_t* scales;
  const int64_t* part_off;
  const int32_t* part_n;
  int nlist;
  int stride, chunk, g, Dp16, nkc;
  uint32_t cbbits[64];  // codebook components as binary16 bits, K x g
  int lite_h;            // Rslm4Lite: leading coordinates on the K = 8 levels (0: none)
  uint32_t cb8bits[8];   // their levels as binary16 bits
  const int* off;       // [nlist + 1] per-partition query list offsets
  const int* items;     // [nlist + 1] per-partition work-item offsets
  const int* item_p;    // [items[nlist]] partition of each work item
  const int32_t* lq;
  const float* lcs;
  const __half* qhi;
  const __half* qlo;
  const float* qinv;
  const float* qrho;  // hi-only mode: per query U ||q_lo||, scaled units (a bound on |<q_lo, uhat>|)
  float* buf_l;       // hi-only mode, pass 2: lower bound of each kept candidate's score
  const float* theta;  // nullptr: keep every candidate
  float* buf_s;
  int32_t* buf_p;
  int* cnt;
  int cap;
  int* work;
  int* err;
};

constexpr int kSBO = (kKC / 8) * 128;  // bytes between 8-row groups of an operand tile
constexpr int kTileBytes = kMR * kKC * 2;
// Codes of one K chunk of a tile: kKC / g positions of 4 bits per row.
__host__ __device__ constexpr int slab_bytes(int g) { return kMR * kKC / (2 * g); }

// Shared offset of element (row, k) of a K-major operand tile (core
// matrices of 8 rows x 8 halves, K-adjacent ones 128 bytes apart).
__device__ __forceinline__ uint32_t tile_off(int row, int k8) {
  return uint32_t((row >> 3) * kSBO + k8 * 128 + (row & 7) * 16);
}

// ------------------------------------------------ pipelined kernel (D <= 128)
// The same computation for a single K chunk (padded D <= 128), as one
// persistent CTA per SM whose warps each take one stage, overlapped across
// the 128-row tiles of an item and across items:
//   warps 22-23 load: fetch the next item (partition, up to 128 of its
//              queries) and stage its per-query epilogue constants and its B
//              operands (the queries' fp16 hi / lo parts in the no-swizzle
//              K-major layout) into one of two item slots while the other
//              slot's item computes;
//   warp 21    lane 0 streams each tile's codes (one contiguous slab of the
//              tile-interleaved layout) and its scales by TMA into rings
//              of kSlabs and kScaleStages buffers;
//   warps 0-3  decode: thread = row; take the row's codes from the slab,
//              decode them through the per-lane byte table (or the code
//              tables of the other formats) and store them into one of two
//              A operands in TMEM (tcgen05.st; lane = row, two halves per
//              32-bit column);
//   warp 20    lane 0 issues the MMAs (A from TMEM, B hi / lo from the item
//              slot, N = the item's query count rounded up to 16) into one
//              of three TMEM accumulators;
//   warps 4-19 epilogue: thread = (row, 32 of the query columns); read its
//              accumulator part, apply s = G (cs + L dot) and append the
//              candidates with s >= theta_q.
// A warp reaches only its TMEM lane quadrant (warp index mod 4), so the
// decode and epilogue roles span the four quadrants.  TMEM columns: three
// accumulators 0-127, 128-255, 256-383 (a tcgen05.ld issued while the
// tensor core is busy takes ~1.6k cycles, so the epilogue gets two tiles of
// MMA time per accumulator), A operands 384-447 and 448-511.
// mbarriers: item_full (loader -> all roles), item_empty (epilogue ->
// loader), slab_full / scale_full (TMA landed), slab_empty (decoders read
// the codes), scale_empty (epilogue read the scales), a_full
// (decoders wrote A), a_free (the MMAs reading an A buffer finished),
// acc_full (a tile's MMAs finished), acc_empty (epilogue read the
// accumulator).  Every wait
// is bounded; a timeout sets the error flag and every role leaves its loop.
constexpr int kDecWarps = 4, kEpiWarps = 16;  // decoders: warps 0-3, epilogue: warps 4-19
constexpr int kMmaWarp = 20, kTmaWarp = 21, kLoadWarp0 = 22;
constexpr int kLoadThreads = 64;
constexpr int kPipeThreads = (kLoadWarp0 * 32) + kLoadThreads;
constexpr int kSlabs = 6;        // code slabs in flight (released by the decoders)
constexpr int kScaleStages = 8;  // tile scales in flight (released by the epilogue, which lags)
constexpr uint32_t kPipeCols = 512;
constexpr uint32_t kAccBufs = 3;  // accumulators in flight (a TMEM load under MMA load is slow)
__device__ __forceinline__ uint32_t acc_col(uint32_t b) { return b * 128u; }       // accumulators
__device__ __forceinline__ uint32_t a_col(uint32_t b) { return 384u + b * 64u; }   // A operands

// One work item as staged by the loader.
struct ItemDesc {
  int64_t slot0;  // first row slot of the partition
  int p;          // partition; -1: no more items
  int q0;         // first entry of the item in the partition's query list
  int nqt;        // queries of the item (<= kNQ)
  int nrows;      // rows of the partition
};
// Item slot layout: B hi, B lo, (cs, theta) scaled by 2^s, 2^-s, query ids,
// descriptor.
constexpr int kOffBl = kTileBytes, kOffQct = 2 * kTileBytes, kOffQinv = kOffQct + kNQ * 8,
              kOffQid = kOffQinv + kNQ * 4, kOffDesc = kOffQid + kNQ * 4,
              kSlotBytes = (kOffDesc + int(sizeof(ItemDesc)) + 127) / 128 * 128;
constexpr int kScaleBytes = kMR * 4;  // a tile's (L | G << 16) words
// Hi-only mode (HI: 4-bit codes of one coordinate): the queries' fp16 hi
// parts alone are multiplied with the codes, and one more MMA (K = 16,
// bf16 operands: the fold MMA) adds, per (row, query),
//   hU + cs' / L - theta' / (G L)     (pass 1: -hU + cs' / L)
// so that the accumulator holds (G (cs' + L (v + hU)) - theta') / (G L): a
// candidate's upper bound reaches theta exactly when it is >= 0, and G L
// times it plus theta' is that upper bound.  hU >= |<q - q_hi, uhat>| + 1
// bounds the hi part's error (the + 1 covers the fold's rounding); the
// products 1/L cs' and -1/(G L) theta' are each formed from three-part
// bf16 splits (six partial products, within 2^-24 of the product).
// Columns of the fold operands (A: per row, written by the decoders; B: per
// query, staged by the loader):
//   0: 1 x hU;  1-6: (a1 a1 a2 a1 a2 a3) x (c1 c2 c1 c3 c2 c1) = cs' / L;
//   7-12: (b1 b1 b2 b1 b2 b3) x (t1 t2 t1 t3 t2 t1) = -theta' / (G L);
// a = 1 / L, b = -1 / (G L), c = cs', t = theta' split into bf16 parts.
// The lo region of an item slot holds the B operand and the margins:
constexpr int kOffBc = kOffBl;           // fold B: the item's queries x 16 bf16
constexpr int kOffKeep = kOffBl + 4096;  // columns whose theta is -inf (keep every row): 128-bit mask
constexpr int kOffHu = kOffBl + 8192;    // hU per query column, float
constexpr int kConstSBO = 256;         // 8-row groups of a K = 16 operand (two 128-byte core matrices)
// The hi-only kernel's item slot is the hi B operand, those operands and
// the per-query constants; its shared memory puts the code slabs, scales
// and small tables below shared address kHiTableAddr, a 64 KB per-lane byte
// table there (entry (byte, lane) at kHiTableAddr + 256 byte + 4 lane, so
// one byte permute forms a lookup's whole address), and the two item slots
// above the table.
constexpr int kHOffQct = kOffHu + kNQ * 4, kHOffQinv = kHOffQct + kNQ * 8, kHOffQid = kHOffQinv + kNQ * 4,
              kHOffDesc = kHOffQid + kNQ * 4,
              kHSlotBytes = (kHOffDesc + int(sizeof(ItemDesc)) + 127) / 128 * 128;
constexpr uint32_t kHiTableAddr = 0x10000u;
constexpr int kFoldABytes = kMR * 32;  // a tile's fold A operand (128 rows x 16 bf16), two buffers after the slots
constexpr uint32_t kHiLowReserve = 4096;  // static + reserved shared memory below the dynamic allocation, at most
__device__ __forceinline__ uint32_t const_off(int row, int k8) {
  return uint32_t((row >> 3) * kConstSBO + k8 * 128 + (row & 7) * 16);
}
// 4-bit codes decode a whole byte (two codes -> two halves) through a
// 256-entry table held once per lane (entry (byte, lane) at word byte * 32 +
// lane), so the 32 lookups of a warp always fall into 32 distinct banks.
constexpr int kByteTableBytes = 256 * 32 * 4;
// Rslm4Lite head bytes: (3-bit code | 3-bit code << 3) -> two halves, 64
// entries (the top bits, which hold the scale codes, are dropped)
constexpr int kLiteTableBytes = 64 * 4;
// Code formats of the scoring rows: codes of 4 bits (g = 1, 2, 4), the
// same with the Rslm4Lite head, and Rslm3's 3-bit stream (g = 1).  Rslm3
// decodes two codes (6 stream bits) per lookup through a 64-entry table
// held once per lane (entry (pair, lane) at word pair * 32 + lane), which
// takes the place of the 256-entry byte table.
constexpr int kFmtNibble = 0, kFmtLite = 1, kFmt3 = 2;
// Code words of one row in a K chunk of 128 coordinates.
__host__ __device__ constexpr int row_words(int g, int fmt) { return fmt == kFmt3 ? 12 : 16 / g; }
// Code bytes of klen (<= 128) coordinates of a row.
__host__ __device__ constexpr int row_bytes(int klen, int g, int fmt) {
  return fmt == kFmt3 ? (3 * klen + 7) / 8 : (klen + 2 * g - 1) / (2 * g);
}
__host__ __device__ constexpr size_t pipe_smem_bytes(int g) {
  return size_t(2) * kSlotBytes + size_t(kSlabs) * slab_bytes(g) + size_t(kScaleStages) * kScaleBytes + 32 * 4 +
         (g == 1 ? kByteTableBytes + kLiteTableBytes : 0);
}
// Hi-only kernel: the dynamic allocation starts at most kHiLowReserve bytes
// above shared address 0, so reserving everything up to the table suffices.
__host__ __device__ constexpr size_t hi_pipe_smem_bytes() {
  return size_t(kHiTableAddr) + 65536 + size_t(2) * kHSlotBytes + size_t(2) * kFoldABytes;
}
__host__ __device__ constexpr size_t hi_pipe_low_bytes() {
  return size_t(kSlabs) * slab_bytes(1) + size_t(kScaleStages) * kScaleBytes + 32 * 4;
}
static_assert(hi_pipe_low_bytes() + kHiLowReserve <= kHiTableAddr, "slabs and scales fit below the table");

// The NW code words of row r of a slab whose rows are interleaved in
// chunks of CH bytes (chunk c of row r at (c * kMR + r) * CH; CH is 16, 8
// or 4); words of the nch chunks present, zeros after them.  The branch
// picks a path with constant chunk arithmetic.
template <int NW>
__device__ __forceinline__ void load_row_words(const uint8_t* sl, int r, int CH, int nch, uint32_t (&wd)[NW]) {
  if (CH == 16) {
#pragma unroll
    for (int v = 0; v < NW / 4; ++v) {
      uint4 x = make_uint4(0, 0, 0, 0);
      if (v < nch) x = *reinterpret_cast<const uint4*>(sl + (v * kMR + r) * 16);
      wd[4 * v] = x.x;
      wd[4 * v + 1] = x.y;
      wd[4 * v + 2] = x.z;
      wd[4 * v + 3] = x.w;
    }
  } else if (CH == 8) {
#pragma unroll
    for (int v = 0; v < NW / 2; ++v) {
      uint2 x = make_uint2(0, 0);
      if (v < nch) x = *reinterpret_cast<const uint2*>(sl + (v * kMR + r) * 8);
      wd[2 * v] = x.x;
      wd[2 * v + 1] = x.y;
    }
  } else {
#pragma unroll
    for (int w = 0; w < NW; ++w) wd[w] = w < nch ? *reinterpret_cast<const uint32_t*>(sl + (w * kMR + r) * 4) : 0u;
  }
}

// Half dh (32 columns = 64 halves = 64 / G codes) of a row's A operand from
// the row's code words wd (G = 1: 16 words; byte -> column through the
// per-lane table t256; G = 2, 4: nibble -> halves through t32; Rslm3: 12
// words, three per 32 codes, code i of a group at its bits 3i .. 3i + 2, so
// column m of the group is its 6-bit field 6m .. 6m + 5, looked up in the
// per-lane pair table held in t256's place).
template <int G, int FMT>
__device__ __forceinline__ void decode_half(const uint32_t* wd, int dh, const uint32_t* t256,
                                            const uint32_t* t32, int lane, uint32_t (&av)[32],
                                            int lite_words, const uint32_t* t64) {
  if constexpr (FMT == kFmt3) {
    const uint32_t* tl = t256 + lane;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const uint32_t w0 = wd[6 * dh + 3 * j], w1 = wd[6 * dh + 3 * j + 1], w2 = wd[6 * dh + 3 * j + 2];
#pragma unroll
      for (int m = 0; m < 16; ++m) {
        const int bit = 6 * m, wi = bit >> 5, sh = bit & 31;
        const uint32_t lo = wi == 0 ? w0 : (wi == 1 ? w1 : w2);
        const uint32_t hi = wi == 0 ? w1 : w2;
        const uint32_t v = (sh <= 26 ? lo >> sh : __funnelshift_r(lo, hi, sh)) & 63u;
        av[16 * j + m] = tl[v << 5];
      }
    }
  } else if constexpr (G == 1) {
    // one byte (two codes) -> one 32-bit column (low half = even position)
    const uint32_t* tl = t256 + lane;
#pragma unroll
    for (int w = 0; w < 8; ++w)
#pragma unroll
      for (int bb = 0; bb < 4; ++bb) av[4 * w + bb] = tl[((wd[8 * dh + w] >> (8 * bb)) & 255u) << 5];
    // Rslm4Lite: the first lite_words (<= 4) words hold K = 8 codes under
    // the scale bits (static indices keep av in registers)
    if constexpr (FMT == kFmtLite) {
#pragma unroll
      for (int w = 0; w < 4; ++w)
        if (w < lite_words)
#pragma unroll
          for (int bb = 0; bb < 4; ++bb) {
            const uint32_t byte = (wd[8 * dh + w] >> (8 * bb)) & 255u;
            av[4 * w + bb] = t64[(byte & 7u) | ((byte >> 1) & 0x38u)];
          }
    }
  } else if constexpr (G == 2) {
#pragma unroll
    for (int w = 0; w < 4; ++w)
#pragma unroll
      for (int n = 0; n < 8; ++n) av[8 * w + n] = t32[(wd[4 * dh + w] >> (4 * n)) & 15u];
  } else {
#pragma unroll
    for (int w = 0; w < 2; ++w)
#pragma unroll
      for (int n = 0; n < 8; ++n) {
        const uint32_t c = (wd[2 * dh + w] >> (4 * n)) & 15u;
        av[16 * w + 2 * n] = t32[2 * c];
        av[16 * w + 2 * n + 1] = t32[2 * c + 1];
      }
  }
}

// x = b0 + b1 + b2 in bf16 parts (nearest at each step); the sum is within
// 2^-24 |x| of x.
__device__ __forceinline__ void bf16_split3(float x, uint32_t (&b)[3]) {
  float r = x;
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    const __nv_bfloat16 h = __float2bfloat16_rn(r);
    b[i] = __bfloat16_as_ushort(h);
    r -= __bfloat162float(h);
  }
}
__device__ __forceinline__ uint32_t bf16_pair(uint32_t lo, uint32_t hi) { return lo | (hi << 16); }
__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
// The margin hU of a query as the fold operands hold it (bf16, rounded up).
__device__ __forceinline__ float fold_margin(float rho) {
  return __bfloat162float(__float2bfloat16_ru(rho + 1.0f));
}

// Epilogue of one row (thread) over the warp's 32 query columns of a tile:
// DENSE stores every score at the row's place in the query's buffer;
// otherwise G (cs' + L acc) - theta' >= 0 decides and the hits are appended.
template <bool DENSE, bool HI = false>
__device__ __forceinline__ void epilogue_row(const BatchArgs& a, const float (&vall)[32], float L, float Gs,
                                             int row, int t, int nrows, int nqt, int eh, int32_t pos,
                                             const float* qpair, const float* qinv_s, const int* qid_s,
                                             const float* hu_s = nullptr) {
  constexpr int kPart = 16;
#pragma unroll
  for (int part = 0; part < 32 / kPart; ++part) {
    float v[kPart];
#pragma unroll
    for (int i = 0; i < kPart; ++i) v[i] = vall[part * kPart + i];
    const int cbase = eh * 32 + part * kPart;
    // (cs', cs'', -theta', -theta'') of columns cbase + 2i, + 2i + 1
    const float4* q4 = reinterpret_cast<const float4*>(qpair + 2 * cbase);
    if constexpr (DENSE) {
      // first pass: every score, at its row of the query's buffer
      float* dst = a.buf_s + int64_t(t) * kMR + row;
#pragma unroll
      for (int i = 0; i < kPart; ++i) {
        const float4 c = q4[i / 2];
        const int col = cbase + i;
        if (col < nqt) {
          const float sc = Gs * fmaf(L, v[i], (i & 1) ? c.y : c.x);
          dst[int64_t(qid_s[col]) * a.cap] = sc * qinv_s[col];
          if (t == 0 && row == 0) a.cnt[qid_s[col]] = nrows;
        }
      }
    } else {
      // y = G (cs' + L v) - theta' per column (packed pairs, each rounded
      // as fmaf); its maximum over the part's columns rules out most rows
      // at once, and the signs of the same y values give the hits
      const uint64_t L2 = f2pack(L, L), G2 = f2pack(Gs, Gs);
      float y[kPart];
      float m = -CUDART_INF_F;
#pragma unroll
      for (int i = 0; i < kPart; i += 2) {
        const float4 c = q4[i / 2];
        const uint64_t y2 = fma2(G2, fma2(L2, f2pack(v[i], v[i + 1]), f2pack(c.x, c.y)), f2pack(c.z, c.w));
        f2unpack(y2, y[i], y[i + 1]);
        m = fmax3(m, y[i], y[i + 1]);
      }
      if (m >= 0.0f) {
        uint32_t hit = 0;
#pragma unroll
        for (int i = 0; i < kPart; ++i) hit |= (y[i] >= 0.0f ? 1u : 0u) << i;
        while (hit) {
          const int i = __ffs(hit) - 1;
          hit &= hit - 1;
          float acc = 0.0f;
#pragma unroll
          for (int kk = 0; kk < kPart; ++kk) acc = kk == i ? v[kk] : acc;
          const int col = cbase + i;
          const int q = qid_s[col];
          if (q < 0) continue;
          const float csc = qpair[(col >> 1) * 4 + (col & 1)];
          const float sc = Gs * fmaf(L, acc, csc);  // score x 2^s (HI: its upper bound)
          const int at = atomicAdd(&a.cnt[q], 1);
          if (at < a.cap) {
            a.buf_s[int64_t(q) * a.cap + at] = sc * qinv_s[col];
            a.buf_p[int64_t(q) * a.cap + at] = pos;
            // HI: the lower bound, with the dot product's margin taken off twice
            if constexpr (HI) a.buf_l[int64_t(q) * a.cap + at] = Gs * fmaf(L, acc - 2.0f * hu_s[col], csc) * qinv_s[col];
          }
        }
      }
    }
  }
}

// Epilogue of one row in the hi-only mode, for a row with L > 0 and G > 0:
// the fold MMA left a = (G (cs' + L (v +- hU)) - theta') / (G L) per query
// column (pass 1, and columns whose theta is -inf: theta' = 0; pass 1:
// -hU).  DENSE stores G L a (the lower bound) for every column; otherwise
// a >= 0 (or a column of the keep mask) is a hit, with upper bound
// G L a + theta' and lower bound that minus 2 G L hU (scores x 2^s).
template <bool DENSE>
__device__ __forceinline__ void epilogue_row_fold(const BatchArgs& a, const float (&vall)[32], float GL, int row,
                                                  int t, int nrows, int nqt, int eh, int32_t pos,
                                                  const float* qpair, const float* qinv_s, const int* qid_s,
                                                  const float* hu_s, const uint32_t* keep_s) {
  constexpr int kPart = 16;
#pragma unroll
  for (int part = 0; part < 32 / kPart; ++part) {
    const int cbase = eh * 32 + part * kPart;
    if constexpr (DENSE) {
      float* dst = a.buf_s + int64_t(t) * kMR + row;
#pragma unroll
      for (int i = 0; i < kPart; ++i) {
        const int col = cbase + i;
        if (col < nqt) {
          dst[int64_t(qid_s[col]) * a.cap] = GL * vall[part * kPart + i] * qinv_s[col];
          if (t == 0 && row == 0) a.cnt[qid_s[col]] = nrows;
        }
      }
    } else {
      float m = -CUDART_INF_F;
#pragma unroll
      for (int i = 0; i < kPart; i += 2) m = fmax3(m, vall[part * kPart + i], vall[part * kPart + i + 1]);
      const uint32_t keep = (keep_s[cbase >> 5] >> (cbase & 31)) & 0xFFFFu;
      if (m >= 0.0f || keep) {
        uint32_t hit = keep;
#pragma unroll
        for (int i = 0; i < kPart; ++i) hit |= (vall[part * kPart + i] >= 0.0f ? 1u : 0u) << i;
        while (hit) {
          const int i = __ffs(hit) - 1;
          hit &= hit - 1;
          float acc = 0.0f;
#pragma unroll
          for (int kk = 0; kk < kPart; ++kk) acc = kk == i ? vall[part * kPart + kk] : acc;
          const int col = cbase + i;
          const int q = qid_s[col];
          if (q < 0) continue;
          const float thq = -qpair[(col >> 1) * 4 + 2 + (col & 1)];
          const float sup = fmaf(GL, acc, thq > -CUDART_INF_F ? thq : 0.0f);  // upper bound x 2^s
          const int at = atomicAdd(&a.cnt[q], 1);
          if (at < a.cap) {
            a.buf_s[int64_t(q) * a.cap + at] = sup * qinv_s[col];
            a.buf_p[int64_t(q) * a.cap + at] = pos;
            a.buf_l[int64_t(q) * a.cap + at] = fmaf(-2.0f * GL, hu_s[col], sup) * qinv_s[col];
          }
        }
      }
    }
  }
}

template <int G, bool DENSE, int FMT, bool HI = false>
__global__ void __launch_bounds__(kPipeThreads, 1) batched_pipe_kernel(const __grid_constant__ BatchArgs a) {
  static_assert(!HI || (G == 1 && FMT == kFmtNibble), "hi-only mode: 4-bit codes of one coordinate");
  extern __shared__ __align__(128) uint8_t psm[];
  // item slot layout (the hi-only kernel's slots are smaller and sit above
  // its byte table)
  constexpr int SlotB = HI ? kHSlotBytes : kSlotBytes;
  constexpr int OffQct = HI ? kHOffQct : kOffQct, OffQinv = HI ? kHOffQinv : kOffQinv,
                OffQid = HI ? kHOffQid : kOffQid, OffDesc = HI ? kHOffDesc : kOffDesc;
  const uint32_t dyn0 = uint32_t(__cvta_generic_to_shared(psm));
  uint8_t* slots = HI ? psm + (2 * kHiTableAddr - dyn0) : psm;
  uint8_t* slab0 = HI ? psm : psm + 2 * kSlotBytes;
  // the scales of the tile in scale stage b: scl0 + b * kMR
  uint32_t* scl0 = reinterpret_cast<uint32_t*>(slab0 + kSlabs * slab_bytes(G));
  // decode table: G = 1: code -> 1 half; G = 2: code -> 2 halves; G = 4: code -> 4 halves
  uint32_t* t32 = scl0 + kScaleStages * kMR;
  __shared__ __align__(8) uint64_t bars[8 + 2 * kSlabs + 2 * kAccBufs + 2 * kScaleStages];
  __shared__ uint32_t tmem_base_sh;
  __shared__ int s_fail;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int CH = a.chunk;

  uint32_t* t256 = t32 + 32;  // G = 1 only
  uint32_t* t64 = t256 + 256 * 32;  // G = 1 only: Rslm4Lite head
  if constexpr (HI) {
    if (dyn0 + uint32_t(hi_pipe_low_bytes()) > kHiTableAddr) {
      // more static shared memory than assumed: the slabs would overlap the table
      if (tid == 0) set_device_error(a.err, kErrSmemLayout);
      return;
    }
    // the per-lane byte table: low half = level of the low nibble (the even
    // code position), high half = level of the high nibble
    uint32_t* tb = reinterpret_cast<uint32_t*>(psm + (kHiTableAddr - dyn0));
    for (int e = tid; e < 256 * 32; e += blockDim.x) {
      const uint32_t byte = uint32_t(e) >> 5;
      tb[byte * 64 + (e & 31)] = a.cbbits[byte & 15u] | (a.cbbits[byte >> 4] << 16);
    }
  } else if (FMT == kFmt3) {
    for (int e = tid; e < 64 * 32; e += blockDim.x) {
      const uint32_t pair = uint32_t(e) >> 5;  // even code in the low 3 bits -> low half
      t256[e] = a.cbbits[pair & 7u] | (a.cbbits[pair >> 3] << 16);
    }
  } else if (G == 1) {
    for (int e = tid; e < 256 * 32; e += blockDim.x) {
      const uint32_t byte = uint32_t(e) >> 5;  // low nibble -> low half (even position)
      t256[e] = a.cbbits[byte & 15u] | (a.cbbits[byte >> 4] << 16);
    }
    for (int e = tid; e < 64; e += blockDim.x) t64[e] = a.cb8bits[e & 7] | (a.cb8bits[e >> 3] << 16);
  } else if (G == 2) {
    for (int c = tid; c < 16; c += blockDim.x) t32[c] = a.cbbits[2 * c] | (a.cbbits[2 * c + 1] << 16);
  } else {
    for (int c = tid; c < 16; c += blockDim.x) {
      t32[2 * c] = a.cbbits[4 * c] | (a.cbbits[4 * c + 1] << 16);
      t32[2 * c + 1] = a.cbbits[4 * c + 2] | (a.cbbits[4 * c + 3] << 16);
    }
  }
  // HI: the two fold A buffers (tile gt uses buffer gt & 1, like A)
  uint8_t* afold = slots + 2 * SlotB;
  const uint32_t bar0 = uint32_t(__cvta_generic_to_shared(&bars[0]));
  // mbarrier layout: item_full[2], item_empty[2], a_full[2], a_free[2],
  // slab_full / slab_empty[kSlabs], acc_full / acc_empty[kAccBufs],
  // scale_full / scale_empty[kScaleStages]
  auto item_full = [&](uint32_t s) { return bar0 + 8u * s; };
  auto item_empty = [&](uint32_t s) { return bar0 + 8u * (2 + s); };
  auto a_full = [&](uint32_t b) { return bar0 + 8u * (4 + b); };
  auto a_free = [&](uint32_t b) { return bar0 + 8u * (6 + b); };  // A buffer b read by its MMAs
  auto slab_full = [&](uint32_t b) { return bar0 + 8u * (8 + b); };
  auto slab_empty = [&](uint32_t b) { return bar0 + 8u * (8 + kSlabs + b); };
  auto acc_full = [&](uint32_t b) { return bar0 + 8u * (8 + 2 * kSlabs + b); };
  auto acc_empty = [&](uint32_t b) { return bar0 + 8u * (8 + 2 * kSlabs + kAccBufs + b); };
  auto scale_full = [&](uint32_t b) { return bar0 + 8u * (8 + 2 * kSlabs + 2 * kAccBufs + b); };
  auto scale_empty = [&](uint32_t b) {
    return bar0 + 8u * (8 + 2 * kSlabs + 2 * kAccBufs + kScaleStages + b);
  };
  if (tid == 0) {
    s_fail = 0;
    for (uint32_t b = 0; b < 2; ++b) {
      mbar_init(item_full(b), kLoadThreads);
      mbar_init(item_empty(b), kEpiWarps);
      mbar_init(a_full(b), kDecWarps);
      mbar_init(a_free(b), 1);
    }
    for (uint32_t b = 0; b < kSlabs; ++b) {
      mbar_init(slab_full(b), 1);
      mbar_init(slab_empty(b), kDecWarps);
    }
    for (uint32_t b = 0; b < kScaleStages; ++b) {
      mbar_init(scale_full(b), 1);
      mbar_init(scale_empty(b), kEpiWarps);
    }
    for (uint32_t b = 0; b < kAccBufs; ++b) {
      mbar_init(acc_full(b), 1);
      mbar_init(acc_empty(b), kEpiWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();  // warp 0 again converged: tcgen05.alloc is .sync.aligned
  if (warp == 0) {
    const uint32_t dst = uint32_t(__cvta_generic_to_shared(&tmem_base_sh));
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst),
                 "r"(kPipeCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = tmem_base_sh;
  const uint32_t slots_addr = uint32_t(__cvta_generic_to_shared(slots));
  const uint32_t afold_addr = uint32_t(__cvta_generic_to_shared(afold));
  const uint32_t slab_addr0 = uint32_t(__cvta_generic_to_shared(slab0));
  const uint32_t scl_addr0 = uint32_t(__cvta_generic_to_shared(scl0));
  const int n_items = a.items[a.nlist];
  const int klen = a.Dp16;  // single K chunk
  const int nbytes = row_bytes(klen, G, FMT);
  const int c1 = min((nbytes + CH - 1) / CH, a.stride / CH);  // code chunks of a row used
  const uint32_t slab_len = uint32_t(c1 * kMR * CH);
  auto slot = [&](uint32_t s) { return slots + s * SlotB; };
  auto desc = [&](uint32_t s) { return reinterpret_cast<const volatile ItemDesc*>(slot(s) + OffDesc); };
  auto failed = [&]() { return *reinterpret_cast<volatile int*>(&s_fail) != 0; };
  auto fail = [&]() {
    set_device_error(a.err, kErrTimeout);
    atomicExch(&s_fail, 1);
  };

  if (warp >= kLoadWarp0) {
    // ---------------- loader: one item per slot use
    const int lt = tid - kLoadWarp0 * 32;
    const int k8n = klen / 8;
    for (uint32_t seq = 0;; ++seq) {
      const uint32_t s = seq & 1, use = seq >> 1;
      bool ok = !(use > 0 && !mbar_wait_warp(item_empty(s), (use - 1) & 1));
      if (!ok) fail();
      fence_proxy_async();  // the MMAs' reads of this slot (async proxy) before its new generic stores
      uint8_t* sb = slot(s);
      ItemDesc* d = reinterpret_cast<ItemDesc*>(sb + OffDesc);
      if (lt == 0) {
        const int item = (ok && !failed()) ? atomicAdd(a.work, 1) : n_items;
        if (item < n_items) {
          const int lo = a.item_p[item];
          d->p = lo;
          d->q0 = a.off[lo] + (item - a.items[lo]) * kNQ;
          d->nqt = min(kNQ, a.off[lo + 1] - d->q0);
          d->nrows = a.part_n[lo];
          d->slot0 = a.part_off[lo];
        } else {
          d->p = -1;
        }
      }
      asm volatile("bar.sync 1, %0;" ::"n"(kLoadThreads) : "memory");
      const int p = d->p, q0 = d->q0, nqt = d->nqt;
      if (p >= 0) {
        float* qpair = reinterpret_cast<float*>(sb + OffQct);
        float* qinv = reinterpret_cast<float*>(sb + OffQinv);
        int* qid = reinterpret_cast<int*>(sb + OffQid);
        int qs[kNQ / kLoadThreads];
#pragma unroll
        for (int u = 0; u < kNQ / kLoadThreads; ++u) {
          const int j = lt + u * kLoadThreads;
          qs[u] = j < nqt ? __ldg(a.lq + q0 + j) : -1;
        }
#pragma unroll
        for (int u = 0; u < kNQ / kLoadThreads; ++u) {
          const int j = lt + u * kLoadThreads;
          const bool v = qs[u] >= 0;
          const float inv = v ? __ldg(a.qinv + qs[u]) : 1.0f;
          const float cs = v ? __ldg(a.lcs + q0 + j) : 0.0f;
          const float th = v ? (a.theta ? __ldg(a.theta + qs[u]) : -CUDART_INF_F) : CUDART_INF_F;
          // (cs', cs'', -theta', -theta'') of the column pair: exact, inv is a power of two
          qpair[(j >> 1) * 4 + (j & 1)] = cs / inv;
          qpair[(j >> 1) * 4 + 2 + (j & 1)] = -th / inv;
          qinv[j] = inv;
          qid[j] = qs[u];
          if constexpr (HI) {
            // fold B row: the margin hU (+ in pass 2: upper bounds; - in
            // pass 1: lower bounds, for theta), cs' and theta' in bf16 parts;
            // a column with theta = -inf folds theta' = 0 and is marked in
            // the keep mask; a padding column gets a margin of -1e30 (never
            // a hit)
            const float hu = v ? fold_margin(__ldg(a.qrho + qs[u])) : 0.0f;
            reinterpret_cast<float*>(sb + kOffHu)[j] = hu;
            uint32_t h0 = v ? uint32_t(__bfloat16_as_ushort(__float2bfloat16_rn(DENSE ? -hu : hu)))
                            : uint32_t(__bfloat16_as_ushort(__float2bfloat16_rn(-1e30f)));
            uint32_t c[3] = {0u, 0u, 0u}, t3[3] = {0u, 0u, 0u};
            const bool keep = v && !(th > -CUDART_INF_F);  // theta = -inf: every row is kept
            if (v) {
              bf16_split3(cs / inv, c);
              if (!DENSE && !keep) bf16_split3(th / inv, t3);
            }
            const unsigned km = __ballot_sync(kFull, keep);
            if ((lt & 31) == 0) reinterpret_cast<uint32_t*>(sb + kOffKeep)[j >> 5] = km;
            *reinterpret_cast<uint4*>(sb + kOffBc + const_off(j, 0)) =
                make_uint4(bf16_pair(h0, c[0]), bf16_pair(c[1], c[0]), bf16_pair(c[2], c[1]),
                           bf16_pair(c[0], t3[0]));
            *reinterpret_cast<uint4*>(sb + kOffBc + const_off(j, 1)) =
                make_uint4(bf16_pair(t3[1], t3[0]), bf16_pair(t3[2], t3[1]), bf16_pair(t3[0], 0u), 0u);
          }
        }
        // B rows: loads in batches of four 16-byte pieces, then shared stores
        // (lane = query row, so a warp's stores fill whole 128-byte
        // core-matrix rows); padding columns get zeros.  Plain stores plus
        // the proxy fence below: cp.async copies did not become reliably
        // visible to the tensor cores through the same fence.
#pragma unroll
        for (int u = 0; u < kNQ / kLoadThreads; ++u) {
          const int j = lt + u * kLoadThreads;
          const bool v = qs[u] >= 0;
          const int64_t base = int64_t(v ? qs[u] : 0) * a.Dp16;
          for (int k0 = 0; k0 < k8n; k0 += 4) {
            uint4 hv[4], lv[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              hv[e] = make_uint4(0, 0, 0, 0);
              lv[e] = make_uint4(0, 0, 0, 0);
              if (v && k0 + e < k8n) {
                hv[e] = __ldg(reinterpret_cast<const uint4*>(a.qhi + base + (k0 + e) * 8));
                if (!HI) lv[e] = __ldg(reinterpret_cast<const uint4*>(a.qlo + base + (k0 + e) * 8));
              }
            }
#pragma unroll
            for (int e = 0; e < 4; ++e)
              if (k0 + e < k8n) {
                *reinterpret_cast<uint4*>(sb + tile_off(j, k0 + e)) = hv[e];
                if (!HI) *reinterpret_cast<uint4*>(sb + kOffBl + tile_off(j, k0 + e)) = lv[e];
              }
          }
        }
        fence_proxy_async();  // B is read by the tensor cores (async proxy)
      }
      mbar_arrive(item_full(s));
      if (p < 0) break;
    }
  } else if (warp == kTmaWarp) {
    // ---------------- TMA: the code slab and the scales of every tile, kSlabs ahead
    if (lane == 0) {
      uint32_t gt = 0;
      bool ok = true;
      for (uint32_t seq = 0; ok; ++seq) {
        const uint32_t s = seq & 1;
        if (!mbar_wait(item_full(s), (seq >> 1) & 1)) {
          fail();
          break;
        }
        const int p = desc(s)->p;
        if (p < 0 || failed()) break;
        const int ntiles = (desc(s)->nrows + kMR - 1) / kMR;
        const int64_t slot0 = desc(s)->slot0;  // a multiple of kMR: scale blocks are 512-byte aligned
        const uint8_t* codes0 = a.codes + slot0 * a.stride;
        for (int t = 0; t < ntiles; ++t, ++gt) {
          const uint32_t sb = gt % kSlabs, u = gt / kSlabs;
          const uint32_t ss = gt % kScaleStages, us = gt / kScaleStages;
          if ((u > 0 && !mbar_wait(slab_empty(sb), (u - 1) & 1)) ||
              (us > 0 && !mbar_wait(scale_empty(ss), (us - 1) & 1))) {
            fail();
            ok = false;
            break;
          }
          mbar_arrive_expect(slab_full(sb), slab_len);
          bulk_copy_1d(slab_addr0 + sb * uint32_t(slab_bytes(G)), codes0 + size_t(t) * kMR * a.stride,
                       slab_len, slab_full(sb));
          mbar_arrive_expect(scale_full(ss), kScaleBytes);
          bulk_copy_1d(scl_addr0 + ss * uint32_t(kScaleBytes), a.scales + slot0 + int64_t(t) * kMR,
                       kScaleBytes, scale_full(ss));
        }
      }
      // no copy may still be landing when the CTA exits
      for (uint32_t sb = 0; sb < kSlabs && sb < gt; ++sb) {
        const uint32_t last = (gt - 1 - sb) / kSlabs;  // last use of buffer sb
        mbar_wait(slab_full(sb), last & 1);
      }
      for (uint32_t ss = 0; ss < kScaleStages && ss < gt; ++ss) {
        const uint32_t last = (gt - 1 - ss) / kScaleStages;
        mbar_wait(scale_full(ss), last & 1);
      }
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ---------------- MMA issue
    if (lane == 0) {
      uint32_t gt = 0;
      bool ok = true;
      for (uint32_t seq = 0; ok; ++seq) {
        const uint32_t s = seq & 1;
        if (!mbar_wait(item_full(s), (seq >> 1) & 1)) {
          fail();
          break;
        }
        const int p = desc(s)->p;
        if (p < 0 || failed()) break;
        const int ntiles = (desc(s)->nrows + kMR - 1) / kMR;
        const int nqt = desc(s)->nqt;
        const uint32_t idesc = f16_idesc(kMR, max(16, (nqt + 15) & ~15));
        const uint32_t bh_addr = slots_addr + s * SlotB, bl_addr = bh_addr + kOffBl;
        for (int t = 0; t < ntiles; ++t, ++gt) {
          const uint32_t b = gt & 1, u = gt >> 1;             // A buffer
          const uint32_t c = gt % kAccBufs, uc = gt / kAccBufs;  // accumulator
          if (!mbar_wait(a_full(b), u & 1) || (uc > 0 && !mbar_wait(acc_empty(c), (uc - 1) & 1))) {
            fail();
            ok = false;
            break;
          }
          fence_after_sync();
          for (int ks = 0; ks < klen / 16; ++ks) {
            const uint32_t at = tmem + a_col(b) + uint32_t(ks * 8);
            umma_f16_ts(tmem + acc_col(c), at, smem_desc(bh_addr + ks * 256, 128, kSBO), idesc,
                        ks > 0 ? 1u : 0u);
            if (!HI) umma_f16_ts(tmem + acc_col(c), at, smem_desc(bl_addr + ks * 256, 128, kSBO), idesc, 1u);
          }
          if (HI)  // the fold: margin, cs' / L and -theta' / (G L), bf16 operands
            umma_f16(tmem + acc_col(c), smem_desc(afold_addr + b * uint32_t(kFoldABytes), 128, kConstSBO),
                     smem_desc(bh_addr + kOffBc, 128, kConstSBO), idesc | kIdescBf16AB, 1u);
          umma_commit(a_free(b));
          umma_commit(acc_full(c));
        }
      }
      // no MMA may still be running when TMEM is freed
      if (gt > 0) mbar_wait(acc_full((gt - 1) % kAccBufs), ((gt - 1) / kAccBufs) & 1);
    }
    __syncwarp();
  } else if (warp < kDecWarps) {
    // ---------------- decoders: thread = row r of the tile (both column halves)
    const int r = warp * 32 + lane;
    uint32_t gt = 0;
    bool ok = true;
    for (uint32_t seq = 0; ok; ++seq) {
      const uint32_t s = seq & 1;
      if (!mbar_wait_warp(item_full(s), (seq >> 1) & 1)) {
        fail();
        break;
      }
      const int p = desc(s)->p;
      if (p < 0 || failed()) break;
      const int ntiles = (desc(s)->nrows + kMR - 1) / kMR;
      for (int t = 0; t < ntiles; ++t, ++gt) {
        const uint32_t sb = gt % kSlabs, us = gt / kSlabs;
        if (!mbar_wait_warp(slab_full(sb), us & 1)) {
          fail();
          ok = false;
          break;
        }
        // HI: the row's scale word, loaded now and used after the decode
        uint32_t swd = 0u;
        if constexpr (HI) {
          if (t * kMR + r < desc(s)->nrows) swd = __ldg(a.scales + desc(s)->slot0 + int64_t(t) * kMR + r);
        }
        // the code words of row r (half dh: words dh * NW / 2 ..)
        constexpr int NW = row_words(G, FMT);
        uint32_t wd[NW];
        load_row_words<NW>(slab0 + sb * slab_bytes(G), r, FMT == kFmt3 ? 4 : CH, c1, wd);
        fence_proxy_async();  // generic reads of the slab before the next bulk copy into it
        __syncwarp();
        if (lane == 0) mbar_arrive(slab_empty(sb));
        // A buffer b is free once the MMAs of tile gt - 2 have completed
        const uint32_t b = gt & 1, u = gt >> 1;
        if (u > 0 && !mbar_wait_warp(a_free(b), (u - 1) & 1)) {
          fail();
          ok = false;
          break;
        }
        __syncwarp();  // converged for the .sync.aligned tcgen05.st (also on a buffer's first use)
        fence_after_sync();
#pragma unroll
        for (int dh = 0; dh < 2; ++dh) {
          uint32_t av[32];
          if constexpr (HI) {
            // byte bb of word w -> one permute forms the entry's address
            // kHiTableAddr + 256 byte + 4 lane; one shared load
            const uint32_t tbl = kHiTableAddr | (uint32_t(lane) << 2);
#pragma unroll
            for (int w = 0; w < 8; ++w)
#pragma unroll
              for (int bb = 0; bb < 4; ++bb) {
                uint32_t v;
                asm volatile("ld.shared.b32 %0, [%1];"
                             : "=r"(v)
                             : "r"(__byte_perm(wd[8 * dh + w], tbl, 0x7604u | (uint32_t(bb) << 4))));
                av[4 * w + bb] = v;
              }
          } else {
            decode_half<G, FMT>(wd, dh, t256, t32, lane, av, dh == 0 ? a.lite_h / 8 : 0, t64);
          }
          tmem_st32(tmem + (uint32_t(warp * 32) << 16) + a_col(b) + uint32_t(dh * 32), av);
        }
        if constexpr (HI) {
          fence_proxy_async();  // the earlier MMAs' reads of this buffer before the new stores
          // fold A row: 1, then 1 / L and -1 / (G L) in bf16 parts; a row
          // past the partition's end or with L = 0 or G = 0 keeps the margin
          // column only (its epilogue uses the explicit formula)
          // (the hardware reciprocal: its ~2^-22 relative error is far
          // inside the margin's + 1)
          const float Lr = ue7m9_to_f32(swd & 0xffffu), Gr = ue4m12_to_f32(swd >> 16);
          uint32_t al[3] = {0u, 0u, 0u}, be[3] = {0u, 0u, 0u};
          if (Lr > 0.0f && Gr > 0.0f) {
            const float ra = rcp_approx(Lr);
            bf16_split3(ra, al);
            bf16_split3(-ra * rcp_approx(Gr), be);
          }
          uint8_t* fa = afold + b * kFoldABytes;
          *reinterpret_cast<uint4*>(fa + const_off(r, 0)) =
              make_uint4(bf16_pair(0x3F80u, al[0]), bf16_pair(al[0], al[1]), bf16_pair(al[0], al[1]),
                         bf16_pair(al[2], be[0]));
          *reinterpret_cast<uint4*>(fa + const_off(r, 1)) =
              make_uint4(bf16_pair(be[0], be[1]), bf16_pair(be[0], be[1]), bf16_pair(be[2], 0u), 0u);
          fence_proxy_async();  // generic stores, read by the tensor core
        }
        fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(a_full(b));
      }
    }
  } else {
    // ---------------- epilogue: thread = row of quadrant warp % 4, columns chunk * 32 ..
    const int quad = warp & 3;
    const int eh = (warp - kDecWarps) >> 2;
    const int row = quad * 32 + lane;
    uint32_t gt = 0;
    bool ok = true;
    for (uint32_t seq = 0; ok; ++seq) {
      const uint32_t s = seq & 1;
      if (!mbar_wait_warp(item_full(s), (seq >> 1) & 1)) {
        fail();
        break;
      }
      const int p = desc(s)->p;
      if (p < 0 || failed()) break;
      const int nrows = desc(s)->nrows, nqt = desc(s)->nqt;
      const int64_t slot0 = desc(s)->slot0;
      const int ntiles = (nrows + kMR - 1) / kMR;
      const float* qpair = reinterpret_cast<const float*>(slot(s) + OffQct);
      const float* qinv_s = reinterpret_cast<const float*>(slot(s) + OffQinv);
      const int* qid_s = reinterpret_cast<const int*>(slot(s) + OffQid);
      // the item's 32-column chunks: with one (two) of them the four warps
      // of a quadrant take every fourth (second) tile in turn, so that a
      // warp's TMEM load and epilogue get several tiles of time
      const int nch = (nqt + 31) >> 5;
      const int rot = nch <= 1 ? 4 : nch == 2 ? 2 : 1;
      const int chunk = nch <= 1 ? 0 : nch == 2 ? (eh & 1) : eh;
      const int phase = nch <= 1 ? eh : nch == 2 ? (eh >> 1) : 0;
      const bool has_cols = chunk * 32 < nqt;
      for (int t = 0; t < ntiles; ++t, ++gt) {
        const bool active = has_cols && int(gt % uint32_t(rot)) == phase;
        const uint32_t b = gt % kAccBufs, u = gt / kAccBufs;  // accumulator
        const int nvalid = min(kMR, nrows - t * kMR);
        const int32_t pos = int32_t(slot0 + int64_t(t) * kMR + row);
        // the tile's scales (scale stage ss)
        const uint32_t ss = gt % kScaleStages;
        if (!mbar_wait_warp(scale_full(ss), (gt / kScaleStages) & 1)) {
          fail();
          ok = false;
          break;
        }
        const uint32_t sc = scl0[ss * kMR + row];
        // the generic read must be ordered before the next bulk copy into
        // this stage (async proxy) that the release below allows
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(scale_empty(ss));
        float L = 0.0f, Gs = 0.0f;
        if (row < nvalid) {
          L = ue7m9_to_f32(sc & 0xffffu);
          Gs = ue4m12_to_f32(sc >> 16);
        }
        if (!mbar_wait_warp(acc_full(b), u & 1)) {
          fail();
          ok = false;
          break;
        }
        fence_after_sync();
        float vall[32];
        if (active) tmem_ld32(tmem + (uint32_t(quad * 32) << 16) + acc_col(b) + uint32_t(chunk * 32), vall);
        // the accumulator is in registers: release it to the next tile's MMAs
        fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(acc_empty(b));
        if (active && row < nvalid)
        {
          const float* hu_s = reinterpret_cast<const float*>(slot(s) + kOffHu);
          if (HI && L > 0.0f && Gs > 0.0f)
            epilogue_row_fold<DENSE>(a, vall, Gs * L, row, t, nrows, nqt, chunk, pos, qpair, qinv_s, qid_s, hu_s,
                                     reinterpret_cast<const uint32_t*>(slot(s) + kOffKeep));
          else
            epilogue_row<DENSE, HI>(a, vall, L, Gs, row, t, nrows, nqt, chunk, pos, qpair, qinv_s, qid_s, hu_s);
        }
      }
      __syncwarp();
      if (ok && lane == 0) mbar_arrive(item_empty(s));
    }
  }
  __syncthreads();
  if (warp == 0) {
    fence_after_sync();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kPipeCols)
                 : "memory");
  }
}

// ------------------------------------------- pipelined kernel, D > 128
// The same roles for several K chunks of 128 dims.  The query operands of
// a whole item no longer fit in shared memory, so the rows are taken in
// groups of kKR tiles (one TMEM accumulator each) and, per group, the K
// chunks in order: the loader streams each chunk's B operands (the item's
// queries, hi / lo, dims [128 kc, 128 kc + 128)) through a ring of two
// stages, each used by the kKR tiles of the group; the TMA warp brings the
// (tile, chunk) code slabs (a chunk's interleaved code bytes are contiguous)
// and each tile's scales; the MMAs of a tile accumulate over its chunks.
// Sequence per item: for group g, for chunk kc, for tile r of the group.
constexpr int kKR = 3;                                   // tiles per group = accumulators
// Roles of this kernel (768 threads, like the single-chunk one): decoders
// warps 0-3, epilogue warps 4-11 (64 query columns each, in two passes of
// 32), MMA warp 12, TMA warp 13, loader warps 14-23.  Staging a 64 KB B
// chunk for every K chunk of a group sets this kernel's pace, so it gets
// ten loader warps (the epilogue works once per group of K chunks).
constexpr int kKEpiWarps = 8, kKMmaWarp = 12, kKTmaWarp = 13, kKLoadWarp0 = 14;
constexpr int kKLoadThreads = kPipeThreads - kKLoadWarp0 * 32;
static_assert(kKLoadThreads >= 2 * kNQ && kKLoadThreads % 32 == 0, "the loader covers the B pieces");
static_assert(kDecWarps + kKEpiWarps == kKMmaWarp, "the roles are contiguous");
constexpr int kBStageBytes = 2 * kTileBytes;             // B hi + lo of one K chunk
constexpr int kKSlot = (kNQ * 16 + int(sizeof(ItemDesc)) + 127) / 128 * 128;  // constants + desc
constexpr int kKOffQinv = kNQ * 8, kKOffQid = kNQ * 12, kKOffDesc = kNQ * 16;
__host__ __device__ constexpr size_t kpipe_smem_bytes(int g) {
  return size_t(2) * kBStageBytes + size_t(2) * kKSlot + size_t(kSlabs) * slab_bytes(g) +
         size_t(kScaleStages) * kScaleBytes + 32 * 4 + (g == 1 ? kByteTableBytes + kLiteTableBytes : 0);
}

template <int G, bool DENSE, int FMT, bool HI = false>
__global__ void __launch_bounds__(kPipeThreads, 1) batched_kpipe_kernel(const __grid_constant__ BatchArgs a) {
  static_assert(!HI || FMT == kFmtNibble, "hi-only mode: 4-bit codes");
  extern __shared__ __align__(128) uint8_t psm[];
  uint8_t* bst0 = psm;                               // B ring
  uint8_t* islot0 = psm + 2 * kBStageBytes;          // item constants + descriptor
  uint8_t* slab0 = islot0 + 2 * kKSlot;
  uint32_t* scl0 = reinterpret_cast<uint32_t*>(slab0 + kSlabs * slab_bytes(G));
  uint32_t* t32 = scl0 + kScaleStages * kMR;
  uint32_t* t256 = t32 + 32;  // G = 1 only
  uint32_t* t64 = t256 + 256 * 32;  // G = 1 only: Rslm4Lite head
  __shared__ __align__(8) uint64_t bars[12 + 2 * kSlabs + 2 * kKR + 2 * kScaleStages];
  __shared__ uint32_t tmem_base_sh;
  __shared__ int s_fail;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int CH = a.chunk;
  if (FMT == kFmt3) {
    for (int e = tid; e < 64 * 32; e += blockDim.x) {
      const uint32_t pair = uint32_t(e) >> 5;
      t256[e] = a.cbbits[pair & 7u] | (a.cbbits[pair >> 3] << 16);
    }
  } else if (G == 1) {
    for (int e = tid; e < 256 * 32; e += blockDim.x) {
      const uint32_t byte = uint32_t(e) >> 5;
      t256[e] = a.cbbits[byte & 15u] | (a.cbbits[byte >> 4] << 16);
    }
    for (int e = tid; e < 64; e += blockDim.x) t64[e] = a.cb8bits[e & 7] | (a.cb8bits[e >> 3] << 16);
  } else if (G == 2) {
    for (int c = tid; c < 16; c += blockDim.x) t32[c] = a.cbbits[2 * c] | (a.cbbits[2 * c + 1] << 16);
  } else {
    for (int c = tid; c < 16; c += blockDim.x) {
      t32[2 * c] = a.cbbits[4 * c] | (a.cbbits[4 * c + 1] << 16);
      t32[2 * c + 1] = a.cbbits[4 * c + 2] | (a.cbbits[4 * c + 3] << 16);
    }
  }
  // HI: the lo half of each B ring stage is free; the first 4 KB of stage
  // 0's hold the margin MMA's A operand (1 in column 0 of every row, fp16),
  // and stage s's [4 KB, 8.5 KB) item slot s's margin B rows and margins
  auto margin_b = [&](uint32_t s) { return bst0 + s * kBStageBytes + kTileBytes + 4096; };
  auto margin_hu = [&](uint32_t s) { return reinterpret_cast<float*>(bst0 + s * kBStageBytes + kTileBytes + 8192); };
  if constexpr (HI) {
    for (int e = tid; e < kMR * 2; e += blockDim.x) {
      const int r = e >> 1, k8 = e & 1;
      *reinterpret_cast<uint4*>(bst0 + kTileBytes + const_off(r, k8)) = make_uint4(k8 == 0 ? 0x3C00u : 0u, 0u, 0u, 0u);
    }
    fence_proxy_async();
  }
  const uint32_t bar0 = uint32_t(__cvta_generic_to_shared(&bars[0]));
  // mbarriers: item_full[2], item_empty[2], b_full[2], b_empty[2], a_full[2],
  // a_free[2], slab_full / slab_empty[kSlabs], acc_full / acc_empty[kKR],
  // scale_full / scale_empty[kScaleStages]
  auto item_full = [&](uint32_t s) { return bar0 + 8u * s; };
  auto item_empty = [&](uint32_t s) { return bar0 + 8u * (2 + s); };
  auto b_full = [&](uint32_t s) { return bar0 + 8u * (4 + s); };
  auto b_empty = [&](uint32_t s) { return bar0 + 8u * (6 + s); };
  auto a_full = [&](uint32_t b) { return bar0 + 8u * (8 + b); };
  auto a_free = [&](uint32_t b) { return bar0 + 8u * (10 + b); };
  auto slab_full = [&](uint32_t b) { return bar0 + 8u * (12 + b); };
  auto slab_empty = [&](uint32_t b) { return bar0 + 8u * (12 + kSlabs + b); };
  auto acc_full = [&](uint32_t b) { return bar0 + 8u * (12 + 2 * kSlabs + b); };
  auto acc_empty = [&](uint32_t b) { return bar0 + 8u * (12 + 2 * kSlabs + kKR + b); };
  auto scale_full = [&](uint32_t b) { return bar0 + 8u * (12 + 2 * kSlabs + 2 * kKR + b); };
  auto scale_empty = [&](uint32_t b) { return bar0 + 8u * (12 + 2 * kSlabs + 2 * kKR + kScaleStages + b); };
  if (tid == 0) {
    s_fail = 0;
    for (uint32_t b = 0; b < 2; ++b) {
      mbar_init(item_full(b), kKLoadThreads);
      mbar_init(item_empty(b), kKEpiWarps);
      mbar_init(b_full(b), kKLoadThreads);
      mbar_init(b_empty(b), 1);
      mbar_init(a_full(b), kDecWarps);
      mbar_init(a_free(b), 1);
    }
    for (uint32_t b = 0; b < kSlabs; ++b) {
      mbar_init(slab_full(b), 1);
      mbar_init(slab_empty(b), kDecWarps);
    }
    for (uint32_t b = 0; b < kKR; ++b) {
      mbar_init(acc_full(b), 1);
      mbar_init(acc_empty(b), kKEpiWarps);
    }
    for (uint32_t b = 0; b < kScaleStages; ++b) {
      mbar_init(scale_full(b), 1);
      mbar_init(scale_empty(b), kKEpiWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();  // warp 0 again converged: tcgen05.alloc is .sync.aligned
  if (warp == 0) {
    const uint32_t dst = uint32_t(__cvta_generic_to_shared(&tmem_base_sh));
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst),
                 "r"(kPipeCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = tmem_base_sh;
  const uint32_t bst_addr0 = uint32_t(__cvta_generic_to_shared(bst0));
  const uint32_t slab_addr0 = uint32_t(__cvta_generic_to_shared(slab0));
  const uint32_t scl_addr0 = uint32_t(__cvta_generic_to_shared(scl0));
  const int n_items = a.items[a.nlist];
  const int nkc = a.nkc;
  // bytes of a full K chunk of a row; its code chunks [kc * cpk, kc * cpk + cpk)
  const int kc_bytes = row_bytes(kKC, G, FMT);
  const int cpk = kc_bytes / CH;
  const int nchunks_row = a.stride / CH;
  auto klen_of = [&](int kc) { return min(kKC, a.Dp16 - kc * kKC); };
  auto slot = [&](uint32_t s) { return islot0 + s * kKSlot; };
  auto desc = [&](uint32_t s) { return reinterpret_cast<const volatile ItemDesc*>(slot(s) + kKOffDesc); };
  auto failed = [&]() { return *reinterpret_cast<volatile int*>(&s_fail) != 0; };
  auto fail = [&]() {
    set_device_error(a.err, kErrTimeout);
    atomicExch(&s_fail, 1);
  };

  if (warp >= kKLoadWarp0) {
    // ---------------- loader: the item's constants, then its B chunks (group, chunk)
    const int lt = tid - kKLoadWarp0 * 32;
    uint32_t bseq = 0;
    bool ok = true;
    for (uint32_t seq = 0; ok; ++seq) {
      const uint32_t s = seq & 1, use = seq >> 1;
      if (use > 0 && !mbar_wait_warp(item_empty(s), (use - 1) & 1)) {
        fail();
        ok = false;
      }
      uint8_t* sb = slot(s);
      ItemDesc* d = reinterpret_cast<ItemDesc*>(sb + kKOffDesc);
      if (lt == 0) {
        const int item = (ok && !failed()) ? atomicAdd(a.work, 1) : n_items;
        if (item < n_items) {
          const int lo = a.item_p[item];
          d->p = lo;
          d->q0 = a.off[lo] + (item - a.items[lo]) * kNQ;
          d->nqt = min(kNQ, a.off[lo + 1] - d->q0);
          d->nrows = a.part_n[lo];
          d->slot0 = a.part_off[lo];
        } else {
          d->p = -1;
        }
      }
      asm volatile("bar.sync 1, %0;" ::"n"(kKLoadThreads) : "memory");
      const int p = d->p, q0 = d->q0, nqt = d->nqt, nrows = d->nrows;
      int* qid = reinterpret_cast<int*>(sb + kKOffQid);
      if (p >= 0 && lt < kNQ) {
        // thread lt: the constants of the item's query lt
        float* qpair = reinterpret_cast<float*>(sb);
        float* qinv = reinterpret_cast<float*>(sb + kKOffQinv);
        const int j = lt;
        const int qj = j < nqt ? __ldg(a.lq + q0 + j) : -1;
        const bool v = qj >= 0;
        const float inv = v ? __ldg(a.qinv + qj) : 1.0f;
        const float cs = v ? __ldg(a.lcs + q0 + j) : 0.0f;
        const float th = v ? (a.theta ? __ldg(a.theta + qj) : -CUDART_INF_F) : CUDART_INF_F;
        qpair[(j >> 1) * 4 + (j & 1)] = cs / inv;  // exact: inv is a power of two
        qpair[(j >> 1) * 4 + 2 + (j & 1)] = -th / inv;
        qinv[j] = inv;
        qid[j] = qj;
        if constexpr (HI) {
          // the margin hU >= |<q - q_hi, uhat>| (rounded up to fp16): + in
          // pass 2 (upper bounds), - in pass 1 (lower bounds, for theta)
          fence_proxy_async();  // the previous item's margin MMAs read these rows
          const __half hh = __float2half_ru(v ? __ldg(a.qrho + qj) : 0.0f);
          margin_hu(s)[j] = __half2float(hh);
          const uint32_t bits = uint32_t(__half_as_ushort(hh)) ^ (DENSE ? 0x8000u : 0u);
          *reinterpret_cast<uint4*>(margin_b(s) + const_off(j, 0)) = make_uint4(bits, 0u, 0u, 0u);
          *reinterpret_cast<uint4*>(margin_b(s) + const_off(j, 1)) = make_uint4(0u, 0u, 0u, 0u);
          fence_proxy_async();  // read by the tensor core
        }
      }
      asm volatile("bar.sync 1, %0;" ::"n"(kKLoadThreads) : "memory");
      // B work of thread lt < 2 kNQ: query lt % kNQ, the 16-byte pieces
      // [8 (lt / kNQ), + 8) of each K chunk (lanes take adjacent queries)
      const int bj = lt & (kNQ - 1), bh = lt / kNQ;
      const int bq = (p >= 0 && lt < 2 * kNQ) ? qid[bj] : -1;
      mbar_arrive(item_full(s));
      if (p < 0) break;
      // B chunks, one per (group, chunk), through the two-stage ring
      const int ntiles = (nrows + kMR - 1) / kMR;
      const int ngroups = (ntiles + kKR - 1) / kKR;
      for (int g = 0; g < ngroups && ok; ++g) {
        for (int kc = 0; kc < nkc; ++kc, ++bseq) {
          const uint32_t bs = bseq & 1, bu = bseq >> 1;
          if (bu > 0 && !mbar_wait_warp(b_empty(bs), (bu - 1) & 1)) {
            fail();
            ok = false;
            break;
          }
          fence_proxy_async();  // the MMAs' reads of this stage (async proxy) before its new generic stores
          uint8_t* dst = bst0 + bs * kBStageBytes;
          const int k8n = klen_of(kc) / 8;
          // one batch of 16 loads per thread (8 pieces of hi and of lo), then
          // shared stores (lane = query row: a warp's stores fill whole
          // 128-byte core-matrix rows)
          if (lt < 2 * kNQ) {
            const bool v = bq >= 0;
            const int64_t base = int64_t(v ? bq : 0) * a.Dp16 + kc * kKC;
            uint4 hv[8], lv[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const int k8 = 8 * bh + e;
              hv[e] = make_uint4(0, 0, 0, 0);
              lv[e] = make_uint4(0, 0, 0, 0);
              if (v && k8 < k8n) {
                hv[e] = __ldg(reinterpret_cast<const uint4*>(a.qhi + base + k8 * 8));
                if (!HI) lv[e] = __ldg(reinterpret_cast<const uint4*>(a.qlo + base + k8 * 8));
              }
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const int k8 = 8 * bh + e;
              if (k8 < k8n) {
                *reinterpret_cast<uint4*>(dst + tile_off(bj, k8)) = hv[e];
                if (!HI) *reinterpret_cast<uint4*>(dst + kTileBytes + tile_off(bj, k8)) = lv[e];
              }
            }
          }
          fence_proxy_async();  // B is read by the tensor cores (async proxy)
          mbar_arrive(b_full(bs));
        }
      }
    }
  } else if (warp == kKTmaWarp) {
    // ---------------- TMA: (tile, chunk) code slabs in the group order, and each tile's scales
    if (lane == 0) {
      uint32_t sseq = 0, cseq = 0;
      bool ok = true;
      for (uint32_t seq = 0; ok; ++seq) {
        const uint32_t s = seq & 1;
        if (!mbar_wait(item_full(s), (seq >> 1) & 1)) {
          fail();
          break;
        }
        const int p = desc(s)->p;
        if (p < 0 || failed()) break;
        const int ntiles = (desc(s)->nrows + kMR - 1) / kMR;
        const int64_t slot0 = desc(s)->slot0;  // a multiple of kMR: scale blocks are 512-byte aligned
        const uint8_t* codes0 = a.codes + slot0 * a.stride;
        for (int g0 = 0; g0 < ntiles && ok; g0 += kKR) {
          const int R = min(kKR, ntiles - g0);
          for (int kc = 0; kc < nkc && ok; ++kc) {
            const int c_lo = kc * cpk, c_n = min(cpk, nchunks_row - c_lo);
            for (int r = 0; r < R; ++r, ++sseq) {
              const int t = g0 + r;
              const uint32_t sb = sseq % kSlabs, u = sseq / kSlabs;
              if (u > 0 && !mbar_wait(slab_empty(sb), (u - 1) & 1)) {
                fail();
                ok = false;
                break;
              }
              const uint32_t len = uint32_t(c_n * kMR * CH);
              mbar_arrive_expect(slab_full(sb), len);
              bulk_copy_1d(slab_addr0 + sb * uint32_t(slab_bytes(G)),
                           codes0 + size_t(t) * kMR * a.stride + size_t(c_lo) * kMR * CH, len, slab_full(sb));
              if (kc == 0) {
                const uint32_t ss = cseq % kScaleStages, us = cseq / kScaleStages;
                ++cseq;
                if (us > 0 && !mbar_wait(scale_empty(ss), (us - 1) & 1)) {
                  fail();
                  ok = false;
                  break;
                }
                mbar_arrive_expect(scale_full(ss), kScaleBytes);
                bulk_copy_1d(scl_addr0 + ss * uint32_t(kScaleBytes), a.scales + slot0 + int64_t(t) * kMR,
                             kScaleBytes, scale_full(ss));
              }
            }
          }
        }
      }
      // no copy may still be landing when the CTA exits
      for (uint32_t sb = 0; sb < kSlabs && sb < sseq; ++sb) mbar_wait(slab_full(sb), ((sseq - 1 - sb) / kSlabs) & 1);
      for (uint32_t ss = 0; ss < kScaleStages && ss < cseq; ++ss)
        mbar_wait(scale_full(ss), ((cseq - 1 - ss) / kScaleStages) & 1);
    }
    __syncwarp();
  } else if (warp == kKMmaWarp) {
    // ---------------- MMA issue: per group, per chunk, per tile
    if (lane == 0) {
      uint32_t bseq = 0, aseq = 0, accu[kKR] = {0, 0, 0}, last_acc = 0;
      bool ok = true, any = false;
      for (uint32_t seq = 0; ok; ++seq) {
        const uint32_t s = seq & 1;
        if (!mbar_wait(item_full(s), (seq >> 1) & 1)) {
          fail();
          break;
        }
        const int p = desc(s)->p;
        if (p < 0 || failed()) break;
        const int ntiles = (desc(s)->nrows + kMR - 1) / kMR;
        const int nqt = desc(s)->nqt;
        const uint32_t idesc = f16_idesc(kMR, max(16, (nqt + 15) & ~15));
        for (int g0 = 0; g0 < ntiles && ok; g0 += kKR) {
          const int R = min(kKR, ntiles - g0);
          for (int kc = 0; kc < nkc && ok; ++kc, ++bseq) {
            const uint32_t bs = bseq & 1;
            if (!mbar_wait(b_full(bs), (bseq >> 1) & 1)) {
              fail();
              ok = false;
              break;
            }
            const uint32_t bh = bst_addr0 + bs * uint32_t(kBStageBytes), bl = bh + uint32_t(kTileBytes);
            const int nks = klen_of(kc) / 16;
            for (int r = 0; r < R; ++r, ++aseq) {
              const uint32_t ab = aseq & 1;
              if (!mbar_wait(a_full(ab), (aseq >> 1) & 1) ||
                  (kc == 0 && accu[r] > 0 && !mbar_wait(acc_empty(r), (accu[r] - 1) & 1))) {
                fail();
                ok = false;
                break;
              }
              fence_after_sync();
              for (int ks = 0; ks < nks; ++ks) {
                const uint32_t at = tmem + a_col(ab) + uint32_t(ks * 8);
                umma_f16_ts(tmem + acc_col(r), at, smem_desc(bh + ks * 256, 128, kSBO), idesc,
                            (kc > 0 || ks > 0) ? 1u : 0u);
                if (!HI) umma_f16_ts(tmem + acc_col(r), at, smem_desc(bl + ks * 256, 128, kSBO), idesc, 1u);
              }
              umma_commit(a_free(ab));
            }
            if (!ok) break;
            umma_commit(b_empty(bs));
          }
          if (!ok) break;
          if (HI) {
            // + (or, pass 1, -) the margin hU of every query column
            const uint32_t mb = uint32_t(__cvta_generic_to_shared(margin_b(s)));
            for (int r = 0; r < R; ++r)
              umma_f16(tmem + acc_col(r), smem_desc(bst_addr0 + uint32_t(kTileBytes), 128, kConstSBO),
                       smem_desc(mb, 128, kConstSBO), idesc, 1u);
          }
          for (int r = 0; r < R; ++r) {
            umma_commit(acc_full(r));
            ++accu[r];
            last_acc = r;
            any = true;
          }
        }
      }
      // no MMA may still be running when TMEM is freed
      if (any) mbar_wait(acc_full(last_acc), (accu[last_acc] - 1) & 1);
    }
    __syncwarp();
  } else if (warp < kDecWarps) {
    // ---------------- decoders: thread = row r of the tile, one (tile, chunk) at a time
    const int row = warp * 32 + lane;
    uint32_t sseq = 0, aseq = 0;
    bool ok = true;
    for (uint32_t seq = 0; ok; ++seq) {
      const uint32_t s = seq & 1;
      if (!mbar_wait_warp(item_full(s), (seq >> 1) & 1)) {
        fail();
        break;
      }
      const int p = desc(s)->p;
      if (p < 0 || failed()) break;
      const int ntiles = (desc(s)->nrows + kMR - 1) / kMR;
      for (int g0 = 0; g0 < ntiles && ok; g0 += kKR) {
        const int R = min(kKR, ntiles - g0);
        for (int kc = 0; kc < nkc && ok; ++kc) {
          const int c_n = min(cpk, nchunks_row - kc * cpk);  // code chunks of this K chunk
          for (int r = 0; r < R; ++r, ++sseq, ++aseq) {
            const uint32_t sb = sseq % kSlabs;
            if (!mbar_wait_warp(slab_full(sb), (sseq / kSlabs) & 1)) {
              fail();
              ok = false;
              break;
            }
            constexpr int NW = row_words(G, FMT);
            uint32_t wd[NW];
            load_row_words<NW>(slab0 + sb * slab_bytes(G), row, FMT == kFmt3 ? 4 : CH, c_n, wd);
            fence_proxy_async();  // generic reads of the slab before the next bulk copy into it
            __syncwarp();
            if (lane == 0) mbar_arrive(slab_empty(sb));
            const uint32_t ab = aseq & 1, au = aseq >> 1;
            if (au > 0 && !mbar_wait_warp(a_free(ab), (au - 1) & 1)) {
              fail();
              ok = false;
              break;
            }
            __syncwarp();  // converged for the .sync.aligned tcgen05.st (also on a buffer's first use)
            fence_after_sync();
#pragma unroll
            for (int dh = 0; dh < 2; ++dh) {
              uint32_t av[32];
              decode_half<G, FMT>(wd, dh, t256, t32, lane, av, (kc == 0 && dh == 0) ? a.lite_h / 8 : 0,
                                   t64);
              tmem_st32(tmem + (uint32_t(warp * 32) << 16) + a_col(ab) + uint32_t(dh * 32), av);
            }
            fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(a_full(ab));
          }
        }
      }
    }
  } else {
    // ---------------- epilogue: thread = row of quadrant warp % 4, columns
    // eh * 64 .. eh * 64 + 63 in two passes of 32
    const int quad = warp & 3;
    const int eh = (warp - kDecWarps) >> 2;
    const int row = quad * 32 + lane;
    uint32_t cseq = 0, accu[kKR] = {0, 0, 0};
    bool ok = true;
    for (uint32_t seq = 0; ok; ++seq) {
      const uint32_t s = seq & 1;
      if (!mbar_wait_warp(item_full(s), (seq >> 1) & 1)) {
        fail();
        break;
      }
      const int p = desc(s)->p;
      if (p < 0 || failed()) break;
      const int nrows = desc(s)->nrows, nqt = desc(s)->nqt;
      const int64_t slot0 = desc(s)->slot0;
      const int ntiles = (nrows + kMR - 1) / kMR;
      const float* qpair = reinterpret_cast<const float*>(slot(s));
      const float* qinv_s = reinterpret_cast<const float*>(slot(s) + kKOffQinv);
      const int* qid_s = reinterpret_cast<const int*>(slot(s) + kKOffQid);
      for (int t = 0; t < ntiles && ok; ++t, ++cseq) {
        const int r = t % kKR;
        const int nvalid = min(kMR, nrows - t * kMR);
        const int32_t pos = int32_t(slot0 + int64_t(t) * kMR + row);
        const uint32_t ss = cseq % kScaleStages;
        if (!mbar_wait_warp(scale_full(ss), (cseq / kScaleStages) & 1)) {
          fail();
          ok = false;
          break;
        }
        const uint32_t sc = scl0[ss * kMR + row];
        // the generic read must be ordered before the next bulk copy into
        // this stage (async proxy) that the release below allows
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(scale_empty(ss));
        float L = 0.0f, Gs = 0.0f;
        if (row < nvalid) {
          L = ue7m9_to_f32(sc & 0xffffu);
          Gs = ue4m12_to_f32(sc >> 16);
        }
        if (!mbar_wait_warp(acc_full(r), accu[r] & 1)) {
          fail();
          ok = false;
          break;
        }
        ++accu[r];
        fence_after_sync();
#pragma unroll 1
        for (int c2 = 0; c2 < 2; ++c2) {
          const int ec = 2 * eh + c2;  // 32-column group
          const bool active = ec * 32 < nqt;
          float vall[32];
          if (active) tmem_ld32(tmem + (uint32_t(quad * 32) << 16) + acc_col(r) + uint32_t(ec * 32), vall);
          if (c2 == 1) {
            // the accumulator is in registers: release it to the next group's MMAs
            fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(acc_empty(r));
          }
          if (active && row < nvalid)
            epilogue_row<DENSE, HI>(a, vall, L, Gs, row, t, nrows, nqt, ec, pos, qpair, qinv_s, qid_s,
                                    margin_hu(s));
          __syncwarp();
        }
      }
      __syncwarp();
      if (ok && lane == 0) mbar_arrive(item_empty(s));
    }
  }
  __syncthreads();
  if (warp == 0) {
    fence_after_sync();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kPipeCols)
                 : "memory");
  }
}

// ---------------------------------------------------------------- finalize
// Exact top-k of a query's buffer by (score desc, id asc).  A buffer that
// overflowed marks the query for the single-query re-scan.
__global__ void finalize_kernel(const float* __restrict__ buf_s, const int32_t* __restrict__ buf_p,
                                const int* __restrict__ cnt, int cap, const int64_t* __restrict__ ids,
                                int k, const int* __restrict__ qlist, const int* __restrict__ qcount,
                                int64_t* __restrict__ out_ids, float* __restrict__ out_scores) {
  extern __shared__ __align__(16) uint8_t fsm[];
  __shared__ uint32_t hist[256];
  __shared__ uint32_t sh_prefix[2];
  __shared__ uint32_t sh_n;
  const int nlisted = *qcount;
  for (int e = blockIdx.x; e < nlisted; e += gridDim.x) {
  const int64_t q = qlist[e];
  const int tid = threadIdx.x;
  const int n = cnt[q];
  int p2 = 1;
  while (p2 < k + 64) p2 <<= 1;
  float* key = reinterpret_cast<float*>(fsm);
  int64_t* idv = reinterpret_cast<int64_t*>(fsm + size_t(p2) * 4);
  const float* s = buf_s + q * cap;
  const int32_t* pp = buf_p + q * cap;
  // Threshold T: the k-th largest order key (everything kept when n <= k).
  uint32_t T = 0;
  if (n > k) {
    T = block_kth_key(s, n, k, hist, sh_prefix);
  }
  if (tid == 0) sh_n = 0;
  __syncthreads();
  for (int i = tid; i < n; i += blockDim.x) {
    if (float_order_key(s[i]) >= T) {
      const uint32_t at = atomicAdd(&sh_n, 1u);
      if (at < uint32_t(p2)) {
        key[at] = s[i];
        idv[at] = ids[pp[i]];
      }
    }
  }
  __syncthreads();
  const int m = min(int(sh_n), p2);
  for (int i = m + tid; i < p2; i += blockDim.x) {
    key[i] = -CUDART_INF_F;
    idv[i] = LLONG_MAX;
  }
  block_bitonic_sort(key, idv, p2);
  for (int i = tid; i < k; i += blockDim.x) {
    const bool ok = i < m && idv[i] != LLONG_MAX;
    out_ids[q * k + i] = ok ? idv[i] : -1;
    out_scores[q * k + i] = ok ? key[i] : -CUDART_INF_F;
  }
  __syncthreads();  // the next listed query reuses the shared buffers
  }
}

// The same result by one warp per query for buffers of at most kFinCap
// candidates: sort them in shared memory by (score desc, id asc).  A longer
// buffer is listed for finalize_kernel, an overflowed one (more than cap
// candidates) for the single-query re-scan.  So is a buffer with fewer than
// k candidates under a finite theta: k candidates of the first probed list
// reach theta, so pass 2 must keep at least k, and a shorter list means the
// two passes disagreed; the exact re-scan answers it and ctr counts it.
constexpr int kFinCap = 512;
constexpr int kFinWarps = 4;
__global__ void __launch_bounds__(kFinWarps * 32) finalize_warp_kernel(
    const float* __restrict__ buf_s, const int32_t* __restrict__ buf_p, const int* __restrict__ cnt,
    int64_t nq, int cap, const int64_t* __restrict__ ids, int k, const float* __restrict__ theta,
    int* __restrict__ ovf_list, int* __restrict__ blk_list, int* __restrict__ counts,
    unsigned long long* __restrict__ ctr, int64_t* __restrict__ out_ids, float* __restrict__ out_scores) {
  __shared__ uint32_t fk[kFinWarps][kFinCap];
  __shared__ int64_t fi[kFinWarps][kFinCap];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t q = int64_t(blockIdx.x) * kFinWarps + w;
  if (q >= nq) return;
  const int n = cnt[q];
  const bool short_list = n < k && theta[q] > -CUDART_INF_F;
  if (n > cap || n > kFinCap || short_list) {
    // counts[0]: queries for the exact re-scan, counts[1]: queries for the block kernel
    if (lane == 0) {
      if (n > cap || short_list) {
        ovf_list[atomicAdd(&counts[0], 1)] = int(q);
        atomicAdd(&ctr[short_list ? kCtrBatchedShort : kCtrBatchedOverflow], 1ull);
      } else {
        blk_list[atomicAdd(&counts[1], 1)] = int(q);
      }
    }
    return;
  }
  int p2 = 1;
  while (p2 < n || p2 < k) p2 <<= 1;
  const float* s = buf_s + q * cap;
  const int32_t* pp = buf_p + q * cap;
  for (int i = lane; i < p2; i += 32) {
    fk[w][i] = i < n ? float_order_key(s[i]) : 0u;
    fi[w][i] = i < n ? ids[pp[i]] : LLONG_MAX;
  }
  __syncwarp();
  for (int size = 2; size <= p2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = lane; i < (p2 >> 1); i += 32) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool asc = (lo & size) == 0;
        const uint32_t klo = fk[w][lo], khi = fk[w][hi];
        const int64_t ilo = fi[w][lo], ihi = fi[w][hi];
        const bool swap = asc ? better(khi, ihi, klo, ilo) : better(klo, ilo, khi, ihi);
        if (swap) {
          fk[w][lo] = khi;
          fk[w][hi] = klo;
          fi[w][lo] = ihi;
          fi[w][hi] = ilo;
        }
      }
      __syncwarp();
    }
  }
  for (int i = lane; i < k; i += 32) {
    const bool ok = i < n && fi[w][i] != LLONG_MAX;
    out_ids[q * k + i] = ok ? fi[w][i] : -1;
    out_scores[q * k + i] = ok ? float_from_order_key(fk[w][i]) : -CUDART_INF_F;
  }
}

// Hi-only mode: pass 2 kept every candidate whose upper bound reached theta,
// with its upper bound s_up (buf_s) and lower bound s_lo (buf_l).  Per
// query, T = the k-th largest s_lo bounds the exact k-th best score from
// below, so only candidates with s_up >= T can be in the top k; their exact
// scores are s_up + G L (<r, uhat> - hU) 2^-s (r = 2^s q - q_hi, exact in
// fp32; the MMAs added the margin hU instead of <r, uhat>), from the row's
// codes (4-bit codes of g coordinates, tile-interleaved chunks), and the top
// k of those by (score desc, id asc) is the result; T comes from a warp
// radix select over all the candidates.  Buffers that overflowed, came out
// short under a finite theta, or leave more than fcap candidates above T go
// to the exact single-query re-scan, as in finalize_warp_kernel.
struct FinHiArgs {
  const float* buf_s;
  const float* buf_l;
  const int32_t* buf_p;
  const int* cnt;
  int64_t nq;
  int cap;
  const int64_t* ids;
  int k;
  const float* theta;
  const float* qrot;  // rotated queries, nq x Dp
  int Dp;
  const float* qrho;
  int fold;              // the margin as the fold MMA holds it (else the fp16 margin MMA's)
  const uint8_t* codes;  // 4-bit codes of g coordinates each, tile-interleaved chunks
  const uint32_t* scales;
  int stride, chunk, g;
  int npos;  // coordinates covered by a row's codes: 2 g stride
  int fcap;  // candidates per query in shared memory (a power of two >= 512)
  int tbl;   // block kernel: score window rows through the per-query code table
  uint32_t* tq;  // block kernel: T per query (finalize_hi_select_kernel)
  uint32_t zero;  // 0: makes the table lookups depend on a row's loads (all issued first)
  float cb[64];
  int* ovf_list;
  int* counts;
  unsigned long long* ctr;
  int64_t* out_ids;
  float* out_scores;
};
__host__ __device__ constexpr size_t fin_hi_warp_bytes(int fcap, int npos) {
  return size_t(fcap) * 12 + 256 * 4 + size_t(npos) * 4;  // window, radix histogram, r
}
// codebook, window (ids, keys, candidate indices), then r (npos floats) or
// the code table (npos / g groups x 16 codes)
__host__ __device__ constexpr size_t fin_hi_block_bytes(int fcap, int npos, int g, bool tbl) {
  return 256 + size_t(fcap) * 16 + (tbl ? size_t(npos / g) * 64 : size_t(npos) * 4);
}

// <r, uhat> of the row at slot pos (r in shared memory, codebook cb:
// component j of codeword c at cb[G c + j]).
template <int G>
__device__ __forceinline__ float fin_word_dot(uint32_t wd, const float* rv, const float* cb, float dot) {
#pragma unroll
  for (int nb = 0; nb < 8; ++nb) {
    const float* cv = cb + G * ((wd >> (4 * nb)) & 15u);
#pragma unroll
    for (int j = 0; j < G; ++j) dot = fmaf(cv[j], rv[G * nb + j], dot);
  }
  return dot;
}
template <int G>
__device__ __forceinline__ float fin_row_dot(const FinHiArgs& a, int32_t pos, const float* rq, const float* cb) {
  const int r = pos & (kMR - 1);
  const uint8_t* tile = a.codes + int64_t(pos - r) * a.stride;
  const int CH = a.chunk;
  float dot = 0.0f;
  if (CH == 16) {
    // eight 16-byte loads in flight, four partial sums
    const int nch = a.stride / 16;
    float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    int c = 0;
    for (; c + 8 <= nch; c += 8) {
      uint4 wv[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) wv[u] = __ldg(reinterpret_cast<const uint4*>(tile + (size_t(c + u) * kMR + r) * 16));
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const float* rv = rq + G * 32 * (c + u);
        float& d = acc[u & 3];
        d = fin_word_dot<G>(wv[u].x, rv, cb, d);
        d = fin_word_dot<G>(wv[u].y, rv + 8 * G, cb, d);
        d = fin_word_dot<G>(wv[u].z, rv + 16 * G, cb, d);
        d = fin_word_dot<G>(wv[u].w, rv + 24 * G, cb, d);
      }
    }
    for (; c < nch; ++c) {
      const uint4 wv = __ldg(reinterpret_cast<const uint4*>(tile + (size_t(c) * kMR + r) * 16));
      const float* rv = rq + G * 32 * c;
      float& d = acc[c & 3];
      d = fin_word_dot<G>(wv.x, rv, cb, d);
      d = fin_word_dot<G>(wv.y, rv + 8 * G, cb, d);
      d = fin_word_dot<G>(wv.z, rv + 16 * G, cb, d);
      d = fin_word_dot<G>(wv.w, rv + 24 * G, cb, d);
    }
    return (acc[0] + acc[1]) + (acc[2] + acc[3]) + dot;
  }
  for (int c = 0; c < a.stride / CH; ++c) {
    const uint8_t* chp = tile + (size_t(c) * kMR + r) * CH;
    for (int w = 0; w < CH / 4; ++w)
      dot = fin_word_dot<G>(__ldg(reinterpret_cast<const uint32_t*>(chp) + w), rq + G * 2 * (c * CH + 4 * w), cb,
                            dot);
  }
  return dot;
}

// <r, uhat> of the row at slot pos through the query's code table T:
// T[16 i + c] = <r restricted to group i, codeword c>, so a code costs one
// shared load and one add (four partial sums, eight 16-byte loads in
// flight for 16-byte chunks).
__device__ __forceinline__ float fin_row_dot_t(const FinHiArgs& a, int32_t pos, const float* T) {
  const int r = pos & (kMR - 1);
  const uint8_t* tile = a.codes + int64_t(pos - r) * a.stride;
  const int CH = a.chunk;
  float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
  auto word = [&](const float* Tw, uint32_t wd, int gi, float& d) {  // gi: group of the word's first code
#pragma unroll
    for (int nb = 0; nb < 8; ++nb) d += Tw[((gi + nb) << 4) | ((wd >> (4 * nb)) & 15u)];
  };
  if (CH == 16) {
    const int nch = a.stride / 16;
    int c = 0;
    for (; c + 8 <= nch; c += 8) {
      uint4 wv[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) wv[u] = __ldg(reinterpret_cast<const uint4*>(tile + (size_t(c + u) * kMR + r) * 16));
      // the lookups' base depends on every word (a.zero = 0), so the eight
      // loads are all issued before the first lookup
      uint32_t dep = 0u;
#pragma unroll
      for (int u = 0; u < 8; ++u) dep |= wv[u].x | wv[u].y | wv[u].z | wv[u].w;
      const float* Tb = T + (dep & a.zero);
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int gi = 32 * (c + u);
        word(Tb, wv[u].x, gi, acc[u & 3]);
        word(Tb, wv[u].y, gi + 8, acc[u & 3]);
        word(Tb, wv[u].z, gi + 16, acc[u & 3]);
        word(Tb, wv[u].w, gi + 24, acc[u & 3]);
      }
    }
    for (; c < nch; ++c) {
      const uint4 wv = __ldg(reinterpret_cast<const uint4*>(tile + (size_t(c) * kMR + r) * 16));
      const int gi = 32 * c;
      word(T, wv.x, gi, acc[c & 3]);
      word(T, wv.y, gi + 8, acc[c & 3]);
      word(T, wv.z, gi + 16, acc[c & 3]);
      word(T, wv.w, gi + 24, acc[c & 3]);
    }
  } else {
    for (int c = 0; c < a.stride / CH; ++c) {
      const uint8_t* chp = tile + (size_t(c) * kMR + r) * CH;
      for (int w = 0; w < CH / 4; ++w)
        word(T, __ldg(reinterpret_cast<const uint32_t*>(chp) + w), 2 * (c * CH + 4 * w), acc[w & 3]);
    }
  }
  return (acc[0] + acc[1]) + (acc[2] + acc[3]);
}

// The k-th largest order key of s[0 .. n) (n > k) by one warp: four 8-bit
// radix passes over a 256-bin histogram in shared memory.
__device__ uint32_t warp_kth_key(const float* s, int n, int k, uint32_t* hist) {
  const int lane = threadIdx.x & 31;
  uint32_t prefix = 0u, mask = 0u;
  int rem = k;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int i = lane; i < 256; i += 32) hist[i] = 0u;
    __syncwarp();
    for (int base = 0; base < n; base += 128) {  // four loads in flight per lane
      uint32_t key[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = base + 32 * u + lane;
        key[u] = i < n ? float_order_key(__ldg(s + i)) : 0u;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = base + 32 * u + lane;
        warp_hist_add(hist, (key[u] >> shift) & 255u, i < n && (key[u] & mask) == prefix);
      }
    }
    __syncwarp();
    // lane l holds bins 255 - 8 l .. 248 - 8 l (from the top); the first
    // bin, from the top, where the count reaches rem
    uint32_t c8[8], tot = 0u;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      c8[j] = hist[255 - 8 * lane - j];
      tot += c8[j];
    }
    uint32_t incl = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += y;
    }
    const uint32_t excl = incl - tot;
    const unsigned hit = __ballot_sync(kFull, excl < uint32_t(rem) && incl >= uint32_t(rem));
    const int src = __ffs(hit) - 1;
    int bin = 0, newrem = rem;
    if (lane == src) {
      uint32_t cum = excl;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (cum + c8[j] >= uint32_t(rem)) {
          bin = 255 - 8 * lane - j;
          newrem = rem - int(cum);
          break;
        }
        cum += c8[j];
      }
    }
    bin = __shfl_sync(kFull, bin, src);
    rem = __shfl_sync(kFull, newrem, src);
    prefix |= uint32_t(bin) << shift;
    mask |= 255u << shift;
    __syncwarp();
  }
  return prefix;
}

// One warp per query (the shorter rows: window decode is cheap, the select
// and sort dominate).
template <int G>
__global__ void __launch_bounds__(128) finalize_hi_warp_kernel(const __grid_constant__ FinHiArgs a) {
  extern __shared__ __align__(16) uint8_t fsm_hi[];
  float* cbs = reinterpret_cast<float*>(fsm_hi);
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, W = blockDim.x >> 5;
  const int fcap = a.fcap;
  uint8_t* wb = fsm_hi + 256 + size_t(w) * fin_hi_warp_bytes(fcap, a.npos);
  int64_t* fi = reinterpret_cast<int64_t*>(wb);
  uint32_t* fk = reinterpret_cast<uint32_t*>(wb + size_t(fcap) * 8);
  uint32_t* hist = fk + fcap;  // 256 bins
  float* rq = reinterpret_cast<float*>(hist + 256);
  if (threadIdx.x < 64) cbs[threadIdx.x] = a.cb[threadIdx.x];
  __syncthreads();
  const int64_t q = int64_t(blockIdx.x) * W + w;
  if (q >= a.nq) return;
  const int n = a.cnt[q];
  const int k = a.k;
  const bool short_list = n < k && a.theta[q] > -CUDART_INF_F;
  if (n > a.cap || short_list) {
    if (lane == 0) {
      a.ovf_list[atomicAdd(&a.counts[0], 1)] = int(q);
      atomicAdd(&a.ctr[short_list ? kCtrBatchedShort : kCtrBatchedOverflow], 1ull);
    }
    return;
  }
  // the query's scaling 2^s (max |q| 2^s in [1024, 2048)) and remainder r
  const float* src = a.qrot + q * a.Dp;
  float m = 0.0f;
  for (int d = lane; d < a.Dp; d += 32) m = fmaxf(m, fabsf(src[d]));
#pragma unroll
  for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(kFull, m, o));
  int e2 = 0;
  if (m > 0.0f) frexpf(m, &e2);
  const float sc = ldexpf(1.0f, 11 - e2), inv = ldexpf(1.0f, e2 - 11);
  for (int d = lane; d < a.npos; d += 32) {
    const float v = d < a.Dp ? src[d] * sc : 0.0f;
    rq[d] = v - __half2float(__float2half_rn(v));
  }
  __syncwarp();  // rq is read by every lane below
  // the margin the MMAs added
  const float hu = a.fold ? fold_margin(a.qrho[q]) : __half2float(__float2half_ru(a.qrho[q]));
  const float* su = a.buf_s + q * a.cap;
  const int32_t* pp = a.buf_p + q * a.cap;
  // T: the k-th largest lower bound (all candidates when n <= k)
  const uint32_t T = n > k ? warp_kth_key(a.buf_l + q * a.cap, n, k, hist) : 0u;
  // the candidates that can be in the top k, with their exact scores
  int mcnt = 0;
  // the window's candidate indices (four loads in flight per lane), then
  // their exact scores in place
  for (int base = 0; base < n; base += 128) {
    float sv[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = base + 32 * u + lane;
      sv[u] = i < n ? su[i] : 0.0f;
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = base + 32 * u + lane;
      const bool in = i < n && float_order_key(sv[u]) >= T;
      const unsigned bm = __ballot_sync(kFull, in);
      const int at = mcnt + __popc(bm & ((1u << lane) - 1u));
      if (in && at < fcap) fk[at] = uint32_t(i);
      mcnt += __popc(bm);
    }
  }
  if (mcnt > fcap) {
    if (lane == 0) {
      a.ovf_list[atomicAdd(&a.counts[0], 1)] = int(q);
      atomicAdd(&a.ctr[kCtrBatchedOverflow], 1ull);
    }
    return;
  }
  __syncwarp();
  for (int w = lane; w < mcnt; w += 32) {
    const int i = int(fk[w]);
    const int32_t pos = pp[i];
    const uint32_t swd = __ldg(a.scales + pos);
    const int64_t id = a.ids[pos];
    const float dot = fin_row_dot<G>(a, pos, rq, cbs);
    const float Gs = ue4m12_to_f32(swd >> 16), L = ue7m9_to_f32(swd & 0xffffu);
    fk[w] = float_order_key(su[i] + Gs * L * (dot - hu) * inv);
    fi[w] = id;
  }
  if (lane == 0) atomicAdd(&a.ctr[kCtrHiExact], (unsigned long long)mcnt);
  __syncwarp();
  int p2 = 1;
  while (p2 < mcnt || p2 < k) p2 <<= 1;
  for (int i = mcnt + lane; i < p2; i += 32) {
    fk[i] = 0u;
    fi[i] = LLONG_MAX;
  }
  __syncwarp();
  for (int size = 2; size <= p2; size <<= 1)
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = lane; i < (p2 >> 1); i += 32) {
        const int lo = 2 * i - (i & (stride - 1)), hi = lo + stride;
        const bool asc = (lo & size) == 0;
        const uint32_t klo = fk[lo], khi = fk[hi];
        const int64_t ilo = fi[lo], ihi = fi[hi];
        const bool swap = asc ? better(khi, ihi, klo, ilo) : better(klo, ilo, khi, ihi);
        if (swap) {
          fk[lo] = khi;
          fk[hi] = klo;
          fi[lo] = ihi;
          fi[hi] = ilo;
        }
      }
      __syncwarp();
    }
  for (int i = lane; i < k; i += 32) {
    const bool ok = i < mcnt && fi[i] != LLONG_MAX;
    a.out_ids[q * k + i] = ok ? fi[i] : -1;
    a.out_scores[q * k + i] = ok ? float_from_order_key(fk[i]) : -CUDART_INF_F;
  }
}

// T per query by one warp (a radix select over the candidates' lower
// bounds), then one block of kFinHiThreads per query (grid-strided): the
// remainder r (or its code table) and the window live in the block's shared
// memory, every thread scores window rows, and each row's rank among them
// is its place in the result.
constexpr uint32_t kFinSkip = 0xffffffffu;  // T of a query listed for the exact re-scan
__global__ void __launch_bounds__(128) finalize_hi_select_kernel(const __grid_constant__ FinHiArgs a) {
  __shared__ uint32_t hist[4][256];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t q = int64_t(blockIdx.x) * 4 + w;
  if (q >= a.nq) return;
  const int n = a.cnt[q], k = a.k;
  const bool short_list = n < k && a.theta[q] > -CUDART_INF_F;
  if (n > a.cap || short_list) {
    if (lane == 0) {
      a.ovf_list[atomicAdd(&a.counts[0], 1)] = int(q);
      atomicAdd(&a.ctr[short_list ? kCtrBatchedShort : kCtrBatchedOverflow], 1ull);
      a.tq[q] = kFinSkip;
    }
    return;
  }
  const uint32_t T = n > k ? warp_kth_key(a.buf_l + q * a.cap, n, k, hist[w]) : 0u;
  if (lane == 0) a.tq[q] = T;
}

constexpr int kFinHiThreads = 256;
template <int G>
__global__ void __launch_bounds__(kFinHiThreads) finalize_hi_block_kernel(const __grid_constant__ FinHiArgs a) {
  extern __shared__ __align__(16) uint8_t fsm_hi[];
  const int fcap = a.fcap;
  float* cbs = reinterpret_cast<float*>(fsm_hi);                 // 64 floats
  int64_t* fi = reinterpret_cast<int64_t*>(fsm_hi + 256);        // fcap ids
  uint32_t* fk = reinterpret_cast<uint32_t*>(fi + fcap);         // fcap keys
  int* wl = reinterpret_cast<int*>(fk + fcap);                   // fcap window indices
  float* rq = reinterpret_cast<float*>(wl + fcap);               // npos (r), or the code table
  __shared__ int sh_m;
  __shared__ float sh_max[kFinHiThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  if (tid < 64) cbs[tid] = a.cb[tid];
  const int k = a.k;
  for (int64_t q = blockIdx.x; q < a.nq; q += gridDim.x) {
    __syncthreads();  // the previous query's buffers are read
    // T (finalize_hi_select_kernel): the k-th largest lower bound, 0 when
    // n <= k, kFinSkip for a query already listed for the exact re-scan
    const uint32_t T = a.tq[q];
    if (T == kFinSkip) continue;
    const int n = a.cnt[q];
    // the query's scaling 2^s (max |q| 2^s in [1024, 2048)) and remainder r
    const float* src = a.qrot + q * a.Dp;
    float m = 0.0f;
    for (int d = tid; d < a.Dp; d += kFinHiThreads) m = fmaxf(m, fabsf(src[d]));
#pragma unroll
    for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(kFull, m, o));
    if (lane == 0) sh_max[w] = m;
    if (tid == 0) sh_m = 0;
    __syncthreads();
    m = sh_max[0];
#pragma unroll
    for (int i = 1; i < kFinHiThreads / 32; ++i) m = fmaxf(m, sh_max[i]);
    int e2 = 0;
    if (m > 0.0f) frexpf(m, &e2);
    const float sc = ldexpf(1.0f, 11 - e2), inv = ldexpf(1.0f, e2 - 11);
    if (a.tbl) {
      // the code table: group gi's remainder r_gi against each codeword
      for (int gi = tid; gi < a.npos / G; gi += kFinHiThreads) {
        float rv[G];
#pragma unroll
        for (int j = 0; j < G; ++j) {
          const int d = G * gi + j;
          const float v = d < a.Dp ? src[d] * sc : 0.0f;
          rv[j] = v - __half2float(__float2half_rn(v));
        }
        float4* tg = reinterpret_cast<float4*>(rq + 16 * gi);
#pragma unroll
        for (int c4 = 0; c4 < 4; ++c4) {
          float e[4];
#pragma unroll
          for (int x = 0; x < 4; ++x) {
            float t = 0.0f;
#pragma unroll
            for (int j = 0; j < G; ++j) t = fmaf(cbs[G * (4 * c4 + x) + j], rv[j], t);
            e[x] = t;
          }
          tg[c4] = make_float4(e[0], e[1], e[2], e[3]);
        }
      }
    } else {
      for (int d = tid; d < a.npos; d += kFinHiThreads) {
        const float v = d < a.Dp ? src[d] * sc : 0.0f;
        rq[d] = v - __half2float(__float2half_rn(v));
      }
    }
    __syncthreads();  // r or the code table is written
    // the margin the MMAs added
    const float hu = a.fold ? fold_margin(a.qrho[q]) : __half2float(__float2half_ru(a.qrho[q]));
    const float* su = a.buf_s + q * a.cap;
    const int32_t* pp = a.buf_p + q * a.cap;
    // the window: the candidates that can be in the top k (upper bound >= T),
    // listed with four loads in flight per thread
    for (int i0 = tid; i0 < n; i0 += 4 * kFinHiThreads) {
      float sv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * kFinHiThreads;
        sv[u] = i < n ? su[i] : 0.0f;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + u * kFinHiThreads;
        if (i < n && float_order_key(sv[u]) >= T) {
          const int at = atomicAdd(&sh_m, 1);
          if (at < fcap) wl[at] = i;
        }
      }
    }
    __syncthreads();
    const int mcnt = sh_m;
    if (mcnt > fcap) {
      if (tid == 0) {
        a.ovf_list[atomicAdd(&a.counts[0], 1)] = int(q);
        atomicAdd(&a.ctr[kCtrBatchedOverflow], 1ull);
      }
      continue;
    }
    // their exact scores
    for (int w = tid; w < mcnt; w += kFinHiThreads) {
      const int i = wl[w];
      const int32_t pos = pp[i];
      const uint32_t swd = __ldg(a.scales + pos);
      const int64_t id = a.ids[pos];
      const float dot = a.tbl ? fin_row_dot_t(a, pos, rq) : fin_row_dot<G>(a, pos, rq, cbs);
      const float Gs = ue4m12_to_f32(swd >> 16), L = ue7m9_to_f32(swd & 0xffffu);
      fk[w] = float_order_key(su[i] + Gs * L * (dot - hu) * inv);
      fi[w] = id;
    }
    __syncthreads();
    if (tid == 0) atomicAdd(&a.ctr[kCtrHiExact], (unsigned long long)mcnt);
    // the top k by rank: (score desc, id asc) is a strict order, so each
    // window entry's count of better entries is its place
    for (int i = tid; i < mcnt; i += kFinHiThreads) {
      const uint32_t ki = fk[i];
      const int64_t ii = fi[i];
      int rank = 0;
      for (int j = 0; j < mcnt; ++j) rank += better(fk[j], fi[j], ki, ii) ? 1 : 0;
      if (rank < k) {
        a.out_ids[q * k + rank] = ii;
        a.out_scores[q * k + rank] = float_from_order_key(ki);
      }
    }
    for (int i = mcnt + tid; i < k; i += kFinHiThreads) {
      a.out_ids[q * k + i] = -1;
      a.out_scores[q * k + i] = -CUDART_INF_F;
    }
  }
}

int blocks_for(int64_t n, int per, int maxb) {
  int64_t b = (n + per - 1) / per;
  if (b < 1) b = 1;
  return int(b < maxb ? b : maxb);
}

}  // namespace

namespace {

// Per-partition query lists of the probe pairs (q, j < eff).
struct Lists {
  int* cnt;
  int* fill;   // global-atomic path only
  int* ghist;   // shared-memory histogram path: kHistBlocks x nlist (shared by both lists)
  int* segsum;  // and its segment sums: kHistBlocks / kHistSeg (rounded up) x nlist
  int* off;
  int* items;
  int32_t* lq;
  float* lcs;
  int* item_p;
};

cudaError_t build_lists(const rslm_index* ix, const int32_t* probes, const float* cs, int64_t nq,
                        int stride, int eff, const Lists& L, cudaStream_t s) {
  const int nlist = ix->nlist;
  const int64_t npairs = nq * eff;
  if (nlist <= kHistMaxList) {
    const int64_t chunk = std::max<int64_t>(2048, (npairs + kHistBlocks - 1) / kHistBlocks);
    const int nb = int(std::max<int64_t>(1, (npairs + chunk - 1) / chunk));
    const size_t hs = size_t(nlist) * 4;
    cudaError_t e = cudaFuncSetAttribute(hist_pairs_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(hs));
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(scatter_hist_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(hs));
    if (e != cudaSuccess) return e;
    hist_pairs_kernel<<<nb, 1024, hs, s>>>(probes, nq, stride, eff, nlist, chunk, L.ghist, ix->d_err);
    const dim3 pg((nlist + 255) / 256, (nb + kHistSeg - 1) / kHistSeg);
    hist_segsum_kernel<<<pg, 256, 0, s>>>(L.ghist, nb, nlist, L.segsum);
    hist_prefix_kernel<<<pg, 256, 0, s>>>(L.ghist, L.segsum, nb, nlist, L.cnt);
    scan_lists_kernel<<<1, 1024, 0, s>>>(L.cnt, nlist, L.off, L.items);
    item_part_kernel<<<blocks_for(nlist, 256, 152 * 4), 256, 0, s>>>(L.items, nlist, L.item_p);
    scatter_hist_kernel<<<nb, 1024, hs, s>>>(probes, cs, nq, stride, eff, nlist, chunk, L.off, L.ghist, L.lq,
                                              L.lcs);
    return cudaGetLastError();
  }
  cudaError_t e = cudaMemsetAsync(L.cnt, 0, size_t(nlist) * 4, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(L.fill, 0, size_t(nlist) * 4, s);
  if (e != cudaSuccess) return e;
  count_pairs_kernel<<<blocks_for(npairs, 256, 152 * 8), 256, 0, s>>>(probes, nq, stride, eff, nlist,
                                                                      L.cnt, ix->d_err);
  scan_lists_kernel<<<1, 1024, 0, s>>>(L.cnt, nlist, L.off, L.items);
  item_part_kernel<<<blocks_for(nlist, 256, 152 * 4), 256, 0, s>>>(L.items, nlist, L.item_p);
  scatter_pairs_kernel<<<blocks_for(npairs, 256, 152 * 8), 256, 0, s>>>(
      probes, cs, nq, stride, eff, nlist, L.off, L.fill, L.lq, L.lcs);
  return cudaGetLastError();
}

cudaError_t run_batched(const rslm_index* ix, const Lists& L, const __half* qhi, const __half* qlo,
                        const float* qinv, int Dp16, const float* theta, float* bs, int32_t* bp, int* bc,
                        int cap, int* work, bool profile, cudaStream_t s, const float* qrho = nullptr,
                        float* bl = nullptr) {
  const CodecSpec& c1 = ix->cs1;
  BatchArgs b;
  b.codes = ix->codes1;
  b.scales = ix->scales1;
  b.part_off = ix->part_off;
  b.part_n = ix->part_n;
  b.nlist = ix->nlist;
  b.stride = c1.stride;
  b.chunk = c1.chunk;
  b.g = c1.g;
  b.Dp16 = Dp16;
  b.nkc = (Dp16 + kKC - 1) / kKC;
  for (int i = 0; i < 64; ++i) b.cbbits[i] = __half_as_ushort(__float2half_rn(c1.cbf[i]));
  b.lite_h = c1.lite_h;
  for (int i = 0; i < 8; ++i) b.cb8bits[i] = __half_as_ushort(__float2half_rn(c1.cb8f[i]));
  b.off = L.off;
  b.items = L.items;
  b.item_p = L.item_p;
  b.lq = L.lq;
  b.lcs = L.lcs;
  b.qhi = qhi;
  b.qlo = qlo;
  b.qinv = qinv;
  b.qrho = qrho;
  b.buf_l = bl;
  b.theta = theta;
  b.buf_s = bs;
  b.buf_p = bp;
  b.cnt = bc;
  b.cap = cap;
  b.work = work;
  b.err = ix->d_err;
  cudaError_t e = cudaMemsetAsync(work, 0, 4, s);
  if (e != cudaSuccess) return e;
  const int g = c1.g;
  int sms = 152;
  int dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // padded D <= 128: the whole K range per item (B once per item);
  // otherwise K chunks of 128 with B streamed per group of tiles
  const bool one = b.nkc == 1;
  const size_t smem = one ? (qrho ? hi_pipe_smem_bytes() : pipe_smem_bytes(g)) : kpipe_smem_bytes(g);
  using K = void (*)(BatchArgs);
  K pk;
  if (one && qrho)  // hi-only mode (4-bit codes of one coordinate)
    pk = theta ? batched_pipe_kernel<1, false, kFmtNibble, true> : batched_pipe_kernel<1, true, kFmtNibble, true>;
  else if (one)
    pk = c1.bits == 3 ? (theta ? batched_pipe_kernel<1, false, kFmt3> : batched_pipe_kernel<1, true, kFmt3>)
         : b.lite_h   ? (theta ? batched_pipe_kernel<1, false, kFmtLite> : batched_pipe_kernel<1, true, kFmtLite>)
         : theta      ? (g == 1   ? batched_pipe_kernel<1, false, kFmtNibble>
                         : g == 2 ? batched_pipe_kernel<2, false, kFmtNibble>
                                  : batched_pipe_kernel<4, false, kFmtNibble>)
                      : (g == 1   ? batched_pipe_kernel<1, true, kFmtNibble>
                         : g == 2 ? batched_pipe_kernel<2, true, kFmtNibble>
                                  : batched_pipe_kernel<4, true, kFmtNibble>);
  else if (qrho)  // hi-only mode, K chunks of 128 (4-bit codes, no Rslm4Lite head)
    pk = theta ? (g == 1   ? batched_kpipe_kernel<1, false, kFmtNibble, true>
                  : g == 2 ? batched_kpipe_kernel<2, false, kFmtNibble, true>
                           : batched_kpipe_kernel<4, false, kFmtNibble, true>)
               : (g == 1   ? batched_kpipe_kernel<1, true, kFmtNibble, true>
                  : g == 2 ? batched_kpipe_kernel<2, true, kFmtNibble, true>
                           : batched_kpipe_kernel<4, true, kFmtNibble, true>);
  else
    pk = c1.bits == 3 ? (theta ? batched_kpipe_kernel<1, false, kFmt3> : batched_kpipe_kernel<1, true, kFmt3>)
         : b.lite_h   ? (theta ? batched_kpipe_kernel<1, false, kFmtLite> : batched_kpipe_kernel<1, true, kFmtLite>)
         : theta      ? (g == 1   ? batched_kpipe_kernel<1, false, kFmtNibble>
                         : g == 2 ? batched_kpipe_kernel<2, false, kFmtNibble>
                                  : batched_kpipe_kernel<4, false, kFmtNibble>)
                      : (g == 1   ? batched_kpipe_kernel<1, true, kFmtNibble>
                         : g == 2 ? batched_kpipe_kernel<2, true, kFmtNibble>
                                  : batched_kpipe_kernel<4, true, kFmtNibble>);
  e = cudaFuncSetAttribute(pk, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  cudaEvent_t stop =
      profile ? prof_start(ix, s, b.nkc == 1 ? "batched_pipe_kernel" : "batched_kpipe_kernel") : nullptr;
  pk<<<sms, kPipeThreads, smem, s>>>(b);
  prof_stop(stop, s);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_scan_batched(const rslm_index* ix, const float* qrot, int64_t nq,
                                const int32_t* probes, const float* cs, int nprobe, int k,
                                int64_t* out_ids, float* out_scores, cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  const CodecSpec& c1 = ix->cs1;
  const int Dp16 = (c1.Dp + 15) / 16 * 16;
  const int nlist = ix->nlist;
  const int cap = 16 * k + 1024;                       // per-query candidate buffer
  const int capA = ix->max_part_n > 0 ? ix->max_part_n : 1;  // first pass: a whole partition
  const int64_t npairs = nq * nprobe;
  size_t bytes = 0;
  auto take = [&](size_t n) {
    size_t at = bytes;
    bytes += (n + 255) / 256 * 256;
    return at;
  };
  size_t oL[2][7];
  const size_t o_ghist = take(nlist <= kHistMaxList ? size_t(kHistBlocks) * nlist * 4 : 4);
  const size_t o_segsum =
      take(nlist <= kHistMaxList ? size_t((kHistBlocks + kHistSeg - 1) / kHistSeg) * nlist * 4 : 4);
  for (int l = 0; l < 2; ++l) {
    const int64_t np = l ? npairs : nq;
    oL[l][0] = take(size_t(nlist) * 4);
    oL[l][1] = take(size_t(nlist) * 4);
    oL[l][2] = take(size_t(nlist + 1) * 4);
    oL[l][3] = take(size_t(nlist + 1) * 4);
    oL[l][4] = take(size_t(np) * 4);
    oL[l][5] = take(size_t(np) * 4);
    oL[l][6] = take(size_t(np / kNQ + nlist + 1) * 4);  // at most sum of ceil(cnt / kNQ) items
  }
  // hi-only mode: 4-bit codes (of g = 1, 2 or 4 coordinates), no Rslm4Lite
  // head; padded D <= 128 (the fold kernel) needs 16-byte chunks of one
  // coordinate, larger D (the margin MMA in the K-chunk kernel) any of them
  const bool hi = c1.bits != 3 && c1.lite_h == 0 &&
                  (Dp16 <= kKC ? (c1.g == 1 && c1.chunk == 16) : true);
  const size_t o_qrho = take(hi ? size_t(nq) * 4 : 4), o_bl = take(hi ? size_t(nq) * cap * 4 : 4);
  const size_t o_qhi = take(size_t(nq) * Dp16 * 2), o_qlo = take(size_t(nq) * Dp16 * 2),
               o_qinv = take(size_t(nq) * 4), o_theta = take(size_t(nq) * 4),
               o_as = take(size_t(nq) * capA * 4), o_ap = take(size_t(nq) * capA * 4),
               o_ac = take(size_t(nq) * 4), o_bs = take(size_t(nq) * cap * 4),
               o_bp = take(size_t(nq) * cap * 4), o_bc = take(size_t(nq) * 4),
               o_ovf = take(size_t(nq) * 4), o_work = take(4), o_fcounts = take(8),
               o_tq = take(hi ? size_t(nq) * 4 : 4);
  uint8_t* ws = nullptr;
  cudaError_t e = cudaMallocAsync(reinterpret_cast<void**>(&ws), bytes, s);
  if (e != cudaSuccess) return e;
  Lists L[2];
  for (int l = 0; l < 2; ++l)
    L[l] = Lists{reinterpret_cast<int*>(ws + oL[l][0]), reinterpret_cast<int*>(ws + oL[l][1]),
                 reinterpret_cast<int*>(ws + o_ghist), reinterpret_cast<int*>(ws + o_segsum),
                 reinterpret_cast<int*>(ws + oL[l][2]), reinterpret_cast<int*>(ws + oL[l][3]),
                 reinterpret_cast<int32_t*>(ws + oL[l][4]), reinterpret_cast<float*>(ws + oL[l][5]),
                 reinterpret_cast<int*>(ws + oL[l][6])};
  __half* qhi = reinterpret_cast<__half*>(ws + o_qhi);
  __half* qlo = reinterpret_cast<__half*>(ws + o_qlo);
  float* qinv = reinterpret_cast<float*>(ws + o_qinv);
  float* theta = reinterpret_cast<float*>(ws + o_theta);
  float* as = reinterpret_cast<float*>(ws + o_as);
  int32_t* ap = reinterpret_cast<int32_t*>(ws + o_ap);
  int* ac = reinterpret_cast<int*>(ws + o_ac);
  float* bs = reinterpret_cast<float*>(ws + o_bs);
  int32_t* bp = reinterpret_cast<int32_t*>(ws + o_bp);
  int* bc = reinterpret_cast<int*>(ws + o_bc);
  int* ovf = reinterpret_cast<int*>(ws + o_ovf);
  int* work = reinterpret_cast<int*>(ws + o_work);
  int* fcounts = reinterpret_cast<int*>(ws + o_fcounts);
  float* qrho = hi ? reinterpret_cast<float*>(ws + o_qrho) : nullptr;
  float* bl = hi ? reinterpret_cast<float*>(ws + o_bl) : nullptr;
  // ||uhat|| <= sqrt(codes per row x max ||codeword||^2) bounds the dot
  // product with the remainder
  float maxcw = 0.0f;
  for (int c = 0; c < 16; ++c) {
    float n2 = 0.0f;
    for (int j = 0; j < c1.g; ++j) n2 += c1.cbf[c1.g * c + j] * c1.cbf[c1.g * c + j];
    maxcw = std::max(maxcw, n2);
  }
  const int ncodes = (c1.Dp + c1.g - 1) / c1.g;
  const float U = std::sqrt(float(ncodes) * maxcw) * (1.0f + 1e-5f);

  // lists: L[0] the first probe of every query, L[1] all probe pairs
  const float* lcs = (ix->flags & RSLM_FULL_VECTOR) ? nullptr : cs;  // full-vector codes: no <q, c> term
  e = build_lists(ix, probes, lcs, nq, nprobe, 1, L[0], s);
  if (e == cudaSuccess) e = build_lists(ix, probes, lcs, nq, nprobe, nprobe, L[1], s);
  if (e == cudaSuccess) {
    split_queries_kernel<<<blocks_for(nq, 8, 152 * 32), 256, 0, s>>>(qrot, nq, c1.Dp, Dp16, qhi, qlo,
                                                                      qinv, qrho, U);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaMemsetAsync(ac, 0, size_t(nq) * 4, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(bc, 0, size_t(nq) * 4, s);
  // Pass 1: every candidate of each query's first probed partition; k of
  // them reach theta, which bounds the query's k-th best score from below.
  if (e == cudaSuccess)
    e = run_batched(ix, L[0], qhi, qlo, qinv, Dp16, nullptr, as, ap, ac, capA, work, false, s, qrho);
  if (e == cudaSuccess) {
    theta_warp_kernel<<<unsigned((nq + 7) / 8), 256, 0, s>>>(as, ac, nq, capA, k, theta);
    e = cudaGetLastError();
  }
  // Pass 2: all probed partitions, keeping candidates >= theta.
  if (e == cudaSuccess)
    e = run_batched(ix, L[1], qhi, qlo, qinv, Dp16, theta, bs, bp, bc, cap, work, true, s, qrho, bl);
  if (e == cudaSuccess) {
    int p2 = 1;
    while (p2 < k + 64) p2 <<= 1;
    const size_t smem = size_t(p2) * 12;
    e = cudaFuncSetAttribute(finalize_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e == cudaSuccess) {
      // ac (the first pass's counts) is free again: it lists the queries
      // handed to the block kernel; ovf lists the overflowed ones
      e = cudaMemsetAsync(fcounts, 0, 2 * sizeof(int), s);
      if (e == cudaSuccess && hi) {
        FinHiArgs fa;
        fa.buf_s = bs;
        fa.buf_l = bl;
        fa.buf_p = bp;
        fa.cnt = bc;
        fa.nq = nq;
        fa.cap = cap;
        fa.ids = ix->ids;
        fa.k = k;
        fa.theta = theta;
        fa.qrot = qrot;
        fa.Dp = c1.Dp;
        fa.qrho = qrho;
        fa.fold = Dp16 <= kKC ? 1 : 0;
        fa.codes = ix->codes1;
        fa.scales = ix->scales1;
        fa.stride = c1.stride;
        fa.chunk = c1.chunk;
        fa.g = c1.g;
        fa.npos = 2 * c1.g * c1.stride;
        int fcap = 512;
        while (fcap < 4 * k) fcap <<= 1;
        fa.fcap = fcap;
        for (int i = 0; i < 64; ++i) fa.cb[i] = c1.cbf[i];
        fa.ovf_list = ovf;
        fa.counts = fcounts;
        fa.ctr = ix->d_counters;
        fa.out_ids = out_ids;
        fa.out_scores = out_scores;
        fa.tq = reinterpret_cast<uint32_t*>(ws + o_tq);
        fa.zero = 0u;
        // rows of at most 256 coordinates: one warp per query; longer rows:
        // one block per query, whose threads share the window's row decode
        using FK = void (*)(FinHiArgs);
        const bool per_warp = fa.npos <= 256;
        const int fw = 4;  // warps (queries) per block of the per-warp kernel
        int dev = 0, sms = 152, optin = 0;
        if (cudaGetDevice(&dev) == cudaSuccess) {
          cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
          cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
        }
        fa.tbl = fin_hi_block_bytes(fcap, fa.npos, c1.g, true) <= size_t(optin) / 2 ? 1 : 0;
        const size_t fsm = per_warp ? 256 + size_t(fw) * fin_hi_warp_bytes(fcap, fa.npos)
                                    : fin_hi_block_bytes(fcap, fa.npos, c1.g, fa.tbl != 0);
        const FK fk = per_warp ? (c1.g == 1   ? finalize_hi_warp_kernel<1>
                                  : c1.g == 2 ? finalize_hi_warp_kernel<2>
                                              : finalize_hi_warp_kernel<4>)
                               : (c1.g == 1   ? finalize_hi_block_kernel<1>
                                  : c1.g == 2 ? finalize_hi_block_kernel<2>
                                              : finalize_hi_block_kernel<4>);
        e = cudaFuncSetAttribute(fk, cudaFuncAttributeMaxDynamicSharedMemorySize, int(fsm));
        if (e == cudaSuccess) {
          if (per_warp)
            fk<<<unsigned((nq + fw - 1) / fw), fw * 32, fsm, s>>>(fa);
          else {
            finalize_hi_select_kernel<<<unsigned((nq + 3) / 4), 128, 0, s>>>(fa);
            // as many blocks as stay resident (each strides over the queries)
            int per_sm = 1;
            if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fk, kFinHiThreads, fsm) != cudaSuccess ||
                per_sm < 1)
              per_sm = 1;
            fk<<<unsigned(std::min<int64_t>(nq, int64_t(sms) * per_sm)), kFinHiThreads, fsm, s>>>(fa);
          }
          e = cudaGetLastError();
        }
      } else if (e == cudaSuccess) {
        finalize_warp_kernel<<<unsigned((nq + kFinWarps - 1) / kFinWarps), kFinWarps * 32, 0, s>>>(
            bs, bp, bc, nq, cap, ix->ids, k, theta, ovf, ac, fcounts, ix->d_counters, out_ids, out_scores);
        finalize_kernel<<<unsigned(std::min<int64_t>(nq, 2 * 152)), 256, smem, s>>>(
            bs, bp, bc, cap, ix->ids, k, ac, fcounts + 1, out_ids, out_scores);
        e = cudaGetLastError();
      }
    }
  }
  // Queries whose buffer overflowed (or came out short): exact single-query scan of all probes.
  if (e == cudaSuccess)
    e = launch_scan_listed(ix, qrot, nq, probes, nprobe, cs, nprobe, k, out_ids, out_scores, ovf, fcounts,
                           s);
  cudaError_t f = cudaFreeAsync(ws, s);
  return e != cudaSuccess ? e : f;
}

}  // namespace rslm
