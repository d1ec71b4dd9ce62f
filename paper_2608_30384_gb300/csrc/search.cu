// search.cu -- probe selection, code scan with per-query top-k, rescoring.
//
// Scan (Sec. 5.5.1 step 3 with the scores of Sec. 3.5): one CTA per query.
// The query, already rotated (Sec. 5.4), becomes a lookup table
// T[group][code] = <q_group, codeword_code> in shared memory, so that the
// dot product <R q, uhat> of a row is the sum of one table entry per 4-bit
// code; per code the work is one byte permute (its table address), one
// shared-memory load and one add.  Warps stream 128-row tiles of the probed partitions; every lane
// owns 4 rows of a tile and reads 16-byte chunks that are contiguous across
// the warp (tile-interleaved layout).  The epilogue applies the scales,
// s = G (cs + L dot) (Sec. 3.5.2), and feeds a per-warp top-k list; the
// lists are merged by a block sort at the end.
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

// ------------------------------------------------------------ probe select
// Top-kk of one row of S per block.  STAGED: the row's order keys are first
// copied to shared memory so the radix passes read it from there.
template <bool STAGED>
__global__ void select_topn_kernel(const float* __restrict__ S, int64_t ld, int n, int kk,
                                   int32_t* __restrict__ out_idx, float* __restrict__ out_val,
                                   const int* __restrict__ only_if) {
  if (only_if && only_if[blockIdx.x] == 0) return;
  extern __shared__ uint32_t xsm[];
  __shared__ uint32_t hist[256];
  __shared__ int scratch[32];
  __shared__ uint32_t sh_prefix, sh_rem, sh_gt;
  int p2 = 1;
  while (p2 < kk) p2 <<= 1;
  const int sbuf = p2 >= 1024 ? p2 : 1024;  // candidate buffer entries
  uint32_t* skey = xsm;
  int32_t* sidx = reinterpret_cast<int32_t*>(xsm + sbuf);
  uint32_t* rowk = xsm + 2 * sbuf;
  const float* s = S + int64_t(blockIdx.x) * ld;
  const int tid = threadIdx.x;
  if (STAGED) {
    for (int i = tid; i < n; i += blockDim.x) rowk[i] = float_order_key(s[i]);
    __syncthreads();
  }
  auto key_at = [&](int i) { return STAGED ? rowk[i] : float_order_key(s[i]); };

  // Fast path.  Split the row into kk groups; the smallest of the kk group
  // maxima is at most the kk-th largest key (the maxima are kk distinct
  // elements), so every element of the top kk is >= it.  Collect those
  // elements (usually a few times kk) and sort them.
  {
    __shared__ uint32_t gmax_sh[kMaxNprobe];
    __shared__ uint32_t sh_bound, sh_cnt;
    const int gs = (n + kk - 1) / kk;  // group size
    for (int g = tid; g < kk; g += blockDim.x) gmax_sh[g] = 0u;
    if (tid == 0) {
      sh_bound = 0xffffffffu;
      sh_cnt = 0;
    }
    __syncthreads();
    for (int base = 0; base < n; base += blockDim.x) {
      const int i = base + tid;
      const uint32_t key = i < n ? key_at(i) : 0u;
      const int g = (i < n ? i : n - 1) / gs;
      // lanes of a warp mostly share a group: reduce them first
      const unsigned same = __match_any_sync(kFull, g);
      const uint32_t m = __reduce_max_sync(same, key);
      if ((tid & 31) == __ffs(same) - 1) atomicMax(&gmax_sh[g], m);
    }
    __syncthreads();
    const int ng = (n + gs - 1) / gs;  // groups that hold elements
    for (int g = tid; g < ng; g += blockDim.x) atomicMin(&sh_bound, gmax_sh[g]);
    __syncthreads();
    // fewer than kk non-empty groups: no bound, every element is a candidate
    const uint32_t bound = ng >= kk ? sh_bound : 0u;
    const int cap = p2 >= 1024 ? p2 : 1024;  // candidates that fit skey / sidx
    for (int base = 0; base < n; base += blockDim.x) {
      const int i = base + tid;
      const bool c = i < n && key_at(i) >= bound;
      const unsigned bal = __ballot_sync(kFull, c);
      uint32_t at0 = 0;
      if ((tid & 31) == 0 && bal) at0 = atomicAdd(&sh_cnt, uint32_t(__popc(bal)));
      at0 = __shfl_sync(kFull, at0, 0);
      if (c) {
        const uint32_t at = at0 + uint32_t(__popc(bal & ((1u << (tid & 31)) - 1)));
        if (at < uint32_t(cap)) {
          skey[at] = key_at(i);
          sidx[at] = i;
        }
      }
    }
    __syncthreads();
    const int m = int(sh_cnt);
    if (m <= cap) {
      int q2 = 1;
      while (q2 < m) q2 <<= 1;
      for (int i = m + tid; i < q2; i += blockDim.x) {
        skey[i] = 0;
        sidx[i] = INT_MAX;
      }
      block_bitonic_sort(skey, sidx, q2);
      for (int i = tid; i < kk; i += blockDim.x) {
        out_idx[int64_t(blockIdx.x) * kk + i] = sidx[i];
        out_val[int64_t(blockIdx.x) * kk + i] = float_from_order_key(skey[i]);
      }
      return;
    }
    __syncthreads();
  }

  // Radix select of the kk-th largest order key, 8 bits at a time.
  uint32_t prefix = 0, mask = 0, rem = uint32_t(kk);
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int i = tid; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int base = 0; base < n; base += blockDim.x) {
      const int i = base + tid;
      const uint32_t key = i < n ? key_at(i) : 0u;
      warp_hist_add(hist, (key >> shift) & 255u, i < n && (key & mask) == prefix);
    }
    __syncthreads();
    if (tid == 0) {
      uint32_t cum = 0;
      int b = 255;
      for (; b > 0; --b) {
        if (cum + hist[b] >= rem) break;
        cum += hist[b];
      }
      sh_rem = rem - cum;
      sh_prefix = prefix | (uint32_t(b) << shift);
    }
    __syncthreads();
    rem = sh_rem;
    prefix = sh_prefix;
    mask |= 255u << shift;
    __syncthreads();
  }
  // prefix is now the kk-th largest key; rem of its copies are taken.
  const uint32_t T = prefix;
  const int ngt = kk - int(rem);
  if (tid == 0) sh_gt = 0;
  __syncthreads();
  for (int i = tid; i < n; i += blockDim.x) {
    const uint32_t key = key_at(i);
    if (key > T) {
      const uint32_t slot = atomicAdd(&sh_gt, 1u);
      skey[slot] = key;
      sidx[slot] = i;
    }
  }
  // Copies of T in column order (lower column first).
  int taken = 0;
  for (int base = 0; base < n && taken < int(rem); base += blockDim.x) {
    const int i = base + tid;
    const int e = (i < n && key_at(i) == T) ? 1 : 0;
    int tot;
    const int ex = block_exclusive_scan(e, scratch, &tot);
    if (e && taken + ex < int(rem)) {
      skey[ngt + taken + ex] = T;
      sidx[ngt + taken + ex] = i;
    }
    taken += tot;
  }
  for (int i = kk + tid; i < p2; i += blockDim.x) {
    skey[i] = 0;
    sidx[i] = INT_MAX;
  }
  block_bitonic_sort(skey, sidx, p2);
  for (int i = tid; i < kk; i += blockDim.x) {
    out_idx[int64_t(blockIdx.x) * kk + i] = sidx[i];
    out_val[int64_t(blockIdx.x) * kk + i] = float_from_order_key(skey[i]);
  }
}

// Warp-per-row top-kk (kk <= 256) of rows with a stride ld % 4 == 0.  Each
// lane reads two float4 per 256-element step, so element i belongs to one of
// 256 interleaved groups (i mod 256).  The kk-th largest of the 256 group
// maxima is at most the kk-th largest key (kk groups, each with a distinct
// element at or above it), so the top kk are among the elements >= that
// bound -- usually about kk, for scores in random order.  They are compacted
// into a per-warp buffer of kSelCap entries and sorted by the warp; a row
// with more sets need_cta[row] for select_topn_kernel.
constexpr int kSelCap = 512;
constexpr int kSelWarps = 8;

__device__ __forceinline__ void keys_at(const float* s, int j, int n, uint32_t (&k)[8], int lane) {
  // Elements 4 (lane + 32 h) + c + 256 j for h = 0, 1 and c = 0..3.
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int i0 = j * 256 + 4 * (lane + 32 * h);
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i0 < n) v = __ldg(reinterpret_cast<const float4*>(s + i0));
    k[4 * h + 0] = i0 + 0 < n ? float_order_key(v.x) : 0u;
    k[4 * h + 1] = i0 + 1 < n ? float_order_key(v.y) : 0u;
    k[4 * h + 2] = i0 + 2 < n ? float_order_key(v.z) : 0u;
    k[4 * h + 3] = i0 + 3 < n ? float_order_key(v.w) : 0u;
  }
}

__global__ void __launch_bounds__(kSelWarps * 32) select_warp_kernel(
    const float* __restrict__ S, int64_t rows, int64_t ld, int n, int kk, int32_t* __restrict__ out_idx,
    float* __restrict__ out_val, int* __restrict__ need_cta) {
  __shared__ uint32_t ckey[kSelWarps][kSelCap];
  __shared__ int32_t cidx[kSelWarps][kSelCap];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t row = int64_t(blockIdx.x) * kSelWarps + w;
  if (row >= rows) return;
  const float* s = S + row * ld;
  const int steps = (n + 255) / 256;
  uint32_t gm[8];
#pragma unroll
  for (int c = 0; c < 8; ++c) gm[c] = 0u;
  for (int j = 0; j < steps; ++j) {
    uint32_t k[8];
    keys_at(s, j, n, k, lane);
#pragma unroll
    for (int c = 0; c < 8; ++c) gm[c] = max(gm[c], k[c]);
  }
  // Bound = kk-th largest of the 256 group maxima (empty groups hold 0),
  // found bit by bit: the largest t with #{gm >= t} >= kk.
  uint32_t bound = 0u;
  for (int bit = 31; bit >= 0; --bit) {
    const uint32_t t = bound | (1u << bit);
    int c0 = 0;
#pragma unroll
    for (int c = 0; c < 8; ++c) c0 += gm[c] >= t ? 1 : 0;
    if (int(__reduce_add_sync(kFull, uint32_t(c0))) >= kk) bound = t;
  }
  const unsigned lt = (1u << lane) - 1u;
  int cnt = 0;
  for (int j = 0; j < steps; ++j) {
    uint32_t k[8];
    keys_at(s, j, n, k, lane);
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      const int i = j * 256 + 4 * (lane + 32 * (c >> 2)) + (c & 3);
      const bool hit = i < n && k[c] >= bound;
      const unsigned bal = __ballot_sync(kFull, hit);
      const int at = cnt + __popc(bal & lt);
      if (hit && at < kSelCap) {
        ckey[w][at] = k[c];
        cidx[w][at] = i;
      }
      cnt += __popc(bal);
    }
  }
  if (cnt > kSelCap) {
    if (lane == 0) need_cta[row] = 1;
    return;
  }
  if (lane == 0) need_cta[row] = 0;
  int p2 = 1;
  while (p2 < cnt) p2 <<= 1;
  for (int i = cnt + lane; i < p2; i += 32) {
    ckey[w][i] = 0u;
    cidx[w][i] = INT_MAX;
  }
  __syncwarp();
  for (int size = 2; size <= p2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = lane; i < (p2 >> 1); i += 32) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool asc = (lo & size) == 0;
        const uint32_t klo = ckey[w][lo], khi = ckey[w][hi];
        const int32_t ilo = cidx[w][lo], ihi = cidx[w][hi];
        const bool swap = asc ? better(khi, ihi, klo, ilo) : better(klo, ilo, khi, ihi);
        if (swap) {
          ckey[w][lo] = khi;
          ckey[w][hi] = klo;
          cidx[w][lo] = ihi;
          cidx[w][hi] = ilo;
        }
      }
      __syncwarp();
    }
  }
  for (int i = lane; i < kk; i += 32) {
    out_idx[row * kk + i] = cidx[w][i];
    out_val[row * kk + i] = float_from_order_key(ckey[w][i]);
  }
}

// ------------------------------------------------------------------- scan
struct ScanArgs {
  const float* qrot;
  int Dp;
  const int32_t* probes;
  const float* cs;
  int nprobe;        // probes scanned per query (the first nprobe of each list)
  int probe_stride;  // row stride of probes / cs
  const int* only_if;  // optional: scan query q only if only_if[q] != 0
  // optional: scan the queries qlist[0 .. *qcount) instead, blocks striding
  const int* qlist;
  const int* qcount;
  int k;
  int out_k;
  const uint8_t* codes;
  const uint32_t* scales;
  const int64_t* ids;
  const int64_t* part_off;
  const int32_t* part_n;
  int nlist;
  int stride;
  int lut_groups;  // 2 * stride: one table row per nibble position of a row
  int ngroups;
  int g;
  float cb[64];
  int lite_h;    // Rslm4Lite: leading coordinates on the K = 8 levels (0: none);
  float cb8[8];  // their levels; the scale codes are read from the codes' top bits
  int64_t* out_ids;
  float* out_scores;
  int* err;
  int lut_region;  // bytes of the table / merge region
  int parts;       // scan_bt_kernel: work units per query, each over a contiguous range of its probes
  int stages;      // scan_bt_kernel: shared-memory stages of tiles (kBtStages when it runs)
  int stages_pre;  // scan_bt_kernel: stages placed below the byte table
  int64_t nq;      // scan_bt_kernel: queries (unlisted)
};

template <int CH>
__device__ __forceinline__ void load_chunk(const uint8_t* p, uint32_t (&w)[CH / 4]) {
  if constexpr (CH == 16) {
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(p));
    w[0] = v.x;
    w[1] = v.y;
    w[2] = v.z;
    w[3] = v.w;
  } else if constexpr (CH == 8) {
    const uint2 v = __ldg(reinterpret_cast<const uint2*>(p));
    w[0] = v.x;
    w[1] = v.y;
  } else {
    w[0] = __ldg(reinterpret_cast<const uint32_t*>(p));
  }
}

__device__ __forceinline__ float lds_f32(uint32_t addr) {
  float v;
  asm("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(addr));
  return v;
}

// Insert (s, p) into a warp's list sorted by (score desc, position asc).
// Every lane calls with the same (s, p).
__device__ __forceinline__ void warp_insert(float* sc, int* ps, int& cnt, int k, float s, int p,
                                            int lane) {
  int at = 0;
  for (int base = 0; base < cnt; base += 32) {
    const int i = base + lane;
    bool b = false;
    if (i < cnt) {
      const float v = sc[i];
      b = v > s || (v == s && ps[i] < p);
    }
    at += __popc(__ballot_sync(kFull, b));
  }
  if (at >= k) return;
  const int newcnt = cnt + 1 < k ? cnt + 1 : k;
  for (int end = newcnt - 1; end > at; end -= 32) {
    const int i = end - lane;
    const bool act = i > at;
    float v = 0.0f;
    int pp = 0;
    if (act) {
      v = sc[i - 1];
      pp = ps[i - 1];
    }
    __syncwarp();
    if (act) {
      sc[i] = v;
      ps[i] = pp;
    }
    __syncwarp();
  }
  if (lane == 0) {
    sc[at] = s;
    ps[at] = p;
  }
  __syncwarp();
  cnt = newcnt;
}

// The top bits of a word's eight 4-bit codes, code k's at bit k.
__device__ __forceinline__ uint32_t nibble_tops(uint32_t w) {
  uint32_t t = (w >> 3) & 0x11111111u;
  t = (t | (t >> 3)) & 0x03030303u;
  t = (t | (t >> 6)) & 0x000F000Fu;
  return (t | (t >> 12)) & 0xFFu;
}

template <int CH, bool B3>
__global__ void __launch_bounds__(256) scan_kernel(const __grid_constant__ ScanArgs a) {
  extern __shared__ __align__(16) uint8_t ssm[];
  __shared__ int scratch[32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, W = blockDim.x >> 5;
  const int nrun = a.qlist ? *a.qcount : 1;
  for (int run0 = a.qlist ? int(blockIdx.x) : 0; run0 < nrun; run0 += a.qlist ? int(gridDim.x) : 1) {
  const int64_t q = a.qlist ? int64_t(a.qlist[run0]) : int64_t(blockIdx.x);
  if (a.only_if && a.only_if[q] == 0) return;
  // The table starts on a 256-byte boundary of the shared window (up to 255
  // bytes of padding are reserved by the launcher).
  const uint32_t ssm_addr = uint32_t(__cvta_generic_to_shared(ssm));
  const uint32_t lut_pad = (256u - (ssm_addr & 255u)) & 255u;
  float* lut = reinterpret_cast<float*>(ssm + lut_pad);
  const uint32_t lut_block0 = (ssm_addr + lut_pad) >> 8;
  float* wsc = reinterpret_cast<float*>(ssm + 256 + a.lut_region);
  int* wps = reinterpret_cast<int*>(wsc + W * a.k);
  int* wcnt = wps + W * a.k;
  int* pid = wcnt + W;
  int* tpref = pid + a.nprobe;

  // Query lookup table T[position][code] = <q_group, C[code]>, one entry per
  // (4-bit code position of a row, code value).  Layout: the 8 positions of
  // each 32-bit code word w go to two 256-byte blocks, even positions in
  // block 2w and odd ones in block 2w + 1, position 2k (+1) at byte 64 k.  A
  // code's shared-memory address is then (block << 8) | (64 k + 4 code):
  // one byte permute per code builds it (see the scan loop).
  const float* qr = a.qrot + q * a.Dp;
  if constexpr (B3) {
    // Rslm3: T[position][code] at lut[8 position + code]
    for (int e = tid; e < a.lut_groups * 8; e += blockDim.x) {
      const int pos = e >> 3;
      lut[e] = pos < a.ngroups ? qr[pos] * a.cb[e & 7] : 0.0f;
    }
  }
  for (int e = tid; !B3 && e < a.lut_groups * 16; e += blockDim.x) {
    const int grp = e >> 4, code = e & 15;
    float v = 0.0f;
    if (grp < a.lite_h)
      v = qr[grp] * a.cb8[code & 7];  // the top bit is a scale bit (g = 1)
    else if (grp < a.ngroups)
      for (int j = 0; j < a.g; ++j) v = fmaf(qr[grp * a.g + j], a.cb[code * a.g + j], v);
    lut[(2 * (grp >> 3) + (grp & 1)) * 64 + ((grp & 7) >> 1) * 16 + code] = v;
  }
  // Probe list -> tiles to visit.
  int run = 0;
  for (int base = 0; base < a.nprobe; base += blockDim.x) {
    const int j = base + tid;
    int nt = 0;
    if (j < a.nprobe) {
      const int p = a.probes[q * a.probe_stride + j];
      if (p < 0 || p >= a.nlist) {
        set_device_error(a.err, kErrBadProbe);
        pid[j] = -1;
      } else {
        pid[j] = p;
        nt = (a.part_n[p] + kTile - 1) / kTile;
      }
    }
    int tot;
    const int ex = block_exclusive_scan(nt, scratch, &tot);
    if (j < a.nprobe) tpref[j] = run + ex;
    run += tot;
  }
  if (tid == 0) tpref[a.nprobe] = run;
  if (tid < W) wcnt[tid] = 0;
  __syncthreads();

  const int total = tpref[a.nprobe];
  int cnt = 0;
  float thr = -CUDART_INF_F;
  int thr_pos = INT_MAX;
  float* msc = wsc + warp * a.k;
  int* mps = wps + warp * a.k;
  const int nch = a.stride / CH;
  int j = 0;
  for (int it = warp; it < total; it += W) {
    while (tpref[j + 1] <= it) ++j;
    const int p = pid[j];
    const int t = it - tpref[j];
    const int64_t slot0 = a.part_off[p] + int64_t(t) * kTile;
    const int nvalid = min(kTile, a.part_n[p] - t * kTile);
    const float csj = a.cs ? a.cs[q * a.probe_stride + j] : 0.0f;  // no cs: full-vector codes
    const uint8_t* tp = a.codes + slot0 * a.stride;
    float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    uint32_t hb[4] = {0u, 0u, 0u, 0u};  // Rslm4Lite: UE7M9 | UE4M12 << 16 from the top bits
    if constexpr (B3) {
      // Rslm3: 32 codes per three words (chunks of 4 bytes), code k at bits
      // 3k .. 3k + 2 of the 96-bit group
      for (int g3 = 0; g3 < nch / 3; ++g3) {
        uint32_t w[4][3];
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int t = 0; t < 3; ++t)
            w[r][t] = __ldg(reinterpret_cast<const uint32_t*>(tp + (size_t(3 * g3 + t) * kTile + r * 32 + lane) * 4));
        const float* lg = lut + g3 * 32 * 8;
#pragma unroll
        for (int kk = 0; kk < 32; ++kk) {
          const int bit = 3 * kk, wi = bit >> 5, sh = bit & 31;
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            const uint32_t code = sh <= 29 ? (w[r][wi] >> sh) & 7u : __funnelshift_r(w[r][wi], w[r][wi + 1], sh) & 7u;
            acc[r] += lg[kk * 8 + int(code)];
          }
        }
      }
    }
    for (int c = 0; !B3 && c < nch; ++c) {
      uint32_t w[4][CH / 4];
#pragma unroll
      for (int r = 0; r < 4; ++r)
        load_chunk<CH>(tp + (size_t(c) * kTile + r * 32 + lane) * CH, w[r]);
      if (c * CH < a.lite_h / 2) {
        // word wi of the row holds codes 8 wi .. 8 wi + 7: their top bits are
        // bits 8 wi .. 8 wi + 7 of the scale pair
#pragma unroll
        for (int v = 0; v < CH / 4; ++v) {
          const int wi = c * (CH / 4) + v;
          if (wi < a.lite_h / 8)
#pragma unroll
            for (int r = 0; r < 4; ++r) hb[r] |= nibble_tops(w[r][v]) << (8 * wi);
        }
      }
#pragma unroll
      for (int v = 0; v < CH / 4; ++v) {
        // bits 8.. of the addresses of this word's even / odd positions
        const uint32_t blk_even = (lut_block0 + 2u * uint32_t(c * (CH / 4) + v)) << 8;
        const uint32_t blk_odd = blk_even + 256u;
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          // byte k of ev (od) = 64 k + 4 * code of position 2k (2k + 1)
          const uint32_t ev = ((w[r][v] << 2) & 0x3C3C3C3Cu) | 0xC0804000u;
          const uint32_t od = ((w[r][v] >> 2) & 0x3C3C3C3Cu) | 0xC0804000u;
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            acc[r] += lds_f32(__byte_perm(ev, blk_even, 0x7650u + k));
            acc[r] += lds_f32(__byte_perm(od, blk_odd, 0x7650u + k));
          }
        }
      }
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int row = r * 32 + lane;
      const bool valid = row < nvalid;
      const int pos = int(slot0) + row;
      float s = -CUDART_INF_F;
      if (valid) {
        const uint32_t sc = a.lite_h ? (a.lite_h == 32 ? hb[r] : (hb[r] | (7u << 28))) : __ldg(a.scales + slot0 + row);
        s = ue4m12_to_f32(sc >> 16) * fmaf(ue7m9_to_f32(sc & 0xffffu), acc[r], csj);
      }
      const bool cand = valid && (cnt < a.k || s > thr || (s == thr && pos < thr_pos));
      unsigned m = __ballot_sync(kFull, cand);
      while (m) {
        const int src = __ffs(m) - 1;
        m &= m - 1;
        const float s2 = __shfl_sync(kFull, s, src);
        const int p2 = __shfl_sync(kFull, pos, src);
        if (cnt < a.k || s2 > thr || (s2 == thr && p2 < thr_pos)) {
          warp_insert(msc, mps, cnt, a.k, s2, p2, lane);
          if (cnt == a.k) {
            thr = msc[a.k - 1];
            thr_pos = mps[a.k - 1];
          }
        }
      }
    }
  }
  if (lane == 0) wcnt[warp] = cnt;
  __syncthreads();

  // Merge the warp lists: block sort by (score desc, row id asc).
  const int tot = W * a.k;
  int np2 = 1;
  while (np2 < tot) np2 <<= 1;
  float* mkey = lut;
  int64_t* mid = reinterpret_cast<int64_t*>(reinterpret_cast<uint8_t*>(lut) +
                                            ((size_t(np2) * 4 + 15) & ~size_t(15)));
  for (int e = tid; e < np2; e += blockDim.x) {
    float kv = -CUDART_INF_F;
    int64_t iv = LLONG_MAX;
    if (e < tot) {
      const int w = e / a.k, i = e - w * a.k;
      if (i < wcnt[w]) {
        kv = wsc[w * a.k + i];
        iv = a.ids[wps[w * a.k + i]];
      }
    }
    mkey[e] = kv;
    mid[e] = iv;
  }
  block_bitonic_sort(mkey, mid, np2);
  for (int e = tid; e < a.out_k; e += blockDim.x) {
    const int64_t id = mid[e];
    const bool ok = id != LLONG_MAX;
    a.out_ids[q * a.out_k + e] = ok ? id : -1;
    a.out_scores[q * a.out_k + e] = ok ? mkey[e] : -CUDART_INF_F;
  }
  __syncthreads();  // the next listed query rebuilds the shared tables
  }
}

// ------------------------------------------------ single-query scan, 4-bit
// The single-query scan for 4-bit codes of one coordinate each (g = 1, no
// Rslm4Lite head, 16-byte chunks, padded D <= 128).  The dot products
// <R q, uhat_j> of 16 rows at a time run on the warp-level tensor-core
// instruction mma.sync.m16n8k16 (fp16 operands, fp32 accumulation), used
// here as the multiply-add engine of a memory-bound loop (a 16 x 16 x 2
// product per instruction; tcgen05 would need the decoded codes staged in
// shared or tensor memory, which doubles the shared-memory traffic that
// bounds this loop):
//   A (16 rows x 16 code positions) = decoded codes.  A query-independent
//     table maps a code byte (two codes) to its two codebook levels as an
//     fp16 pair (the levels are binary16-exact), one copy per lane: entry
//     (byte, lane) at shared address kBtTableAddr + 256 byte + 4 lane, so
//     one byte permute of a code word forms the whole address and the 32
//     lanes of a read hit 32 distinct banks; the pair is one A register.
//   B (16 x 8) = the query scaled by 2^s (max |q| 2^s in [1024, 2048)) and
//     split into q_hi = fp16(q) (column 0) and q_lo = fp16(q - q_hi)
//     (column 1); the other columns are zero.
//   D column 0 + column 1 = 2^s <q, uhat> to about 22 bits of the query.
// The dot product is order-free in its positions, so each lane takes the
// codes that ldmatrix hands it: one ldmatrix.x4 reads four 8-row x 16-byte
// blocks of a staged tile (rows 16 P .. + 7 and + 8 .. + 15 of two chunk
// columns; each block is one conflict-free 128-byte row of banks) and gives
// lane (g, t) = (lane / 4, lane % 4) word t of rows g and g + 8 of each
// chunk column.  In the MMAs of chunk c the lane supplies bytes (0, 1), then
// (2, 3), of its words -- code positions 32 c + 8 t + 4 m .. + 3 for MMA m
// -- as the fragment columns (2 t, 2 t + 1) and (2 t + 8, 2 t + 9).  The B
// fragment of lane (g, t) holds the same positions of column g, so a lane's
// query fragments depend only on t and stay in registers.  Per code byte
// that is one permute and one 4-byte shared read, and one MMA per 256
// codes.
//
// Streaming: one persistent CTA of 16 warps per SM (four per SM
// sub-partition, so 128 registers per thread).  Its producer warp turns
// each work unit (a query, or a contiguous part of its probe list) into a
// list of 128-row tiles, keeping each probe's row offset, row count and cs
// in the unit's shared-memory descriptor (double-buffered); then 15 of its
// lanes copy the tiles -- the codes (a contiguous slab of the
// tile-interleaved layout) and the scale words -- into 15 shared-memory
// stages with 1-D bulk copies (one issuing thread sustains only about one
// copy per 600 cycles).  Tile T of the CTA's sequence goes to stage T mod
// 15, issued by producer lane T mod 15 and scored by consumer warp T mod
// 15: every stage has one issuing lane and one consumer warp, which use its
// phases in order (an mbarrier parity wait is only sound for the current
// phase), and no warp waits behind another's copies.  A consumer warp reads
// its tile's codes into registers (ldmatrix), releases the stage, and
// scores the 128 rows in 8 passes of 16; after each pass the row dots sit
// in lanes t = 0, and a shuffle hands pass P's dots to lanes t = P mod 4,
// so that after each 4 passes every lane holds two rows and the epilogue
// (scales, s = G (cs + L dot), per-warp top-k list) runs on all 32 lanes.
// At the end of a unit each warp writes its own list (no barrier between
// the consumer warps); merge_parts_kernel merges the 15 lists of every unit
// of a query (a query has `parts` > 1 units when the batch is too small to
// fill the SMs).
constexpr int kBtTableBytes = 256 * 256;
constexpr uint32_t kBtTableAddr = 0x10000u;
constexpr uint32_t kBtLowReserve = 4096;  // static + reserved shared memory below the dynamic allocation, at most
constexpr int kBtWarps = 15;                     // consumer warps
constexpr int kBtThreads = (kBtWarps + 1) * 32;  // + the producer warp: 4 warps per SM sub-partition
constexpr int kBtStages = kBtWarps;              // stage w: consumer warp w, issuing lane w
constexpr int kBtMaxChunks = 4;                  // padded D <= 128
constexpr int kBtHalf = kTile / 2;

__device__ __forceinline__ void mma_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                          uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Byte-table entry of byte KB (0..3) of code word w for this lane.  The
// table sits at shared address kBtTableAddr (64 KB aligned) and tbl holds
// kBtTableAddr | 4 lane, so one byte permute forms the entry's whole
// address kBtTableAddr + 256 byte + 4 lane (bytes: 4 lane, the code byte,
// then the table's upper address bytes).
template <int KB>
__device__ __forceinline__ uint32_t bt_entry(uint32_t w, uint32_t tbl) {
  uint32_t v;
  asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(__byte_perm(w, tbl, 0x7604u | (uint32_t(KB) << 4))));
  return v;
}

// The 8 MMAs of four chunk columns: word t of rows g and g + 8 of column
// c in w0[c] / w1[c], query fragments bq[2 c + m][0..1]; even and odd MMAs
// accumulate separately.
__device__ __forceinline__ void bt_group_mma(uint32_t tbl, const uint32_t (&w0)[4],
                                             const uint32_t (&w1)[4], const uint32_t (&bq)[8][2], float (&d)[4],
                                             float (&e)[4]) {
#pragma unroll
  for (int wi = 0; wi < 4; ++wi) {
    // MMA 2 wi: bytes 0, 1 of the column's words; MMA 2 wi + 1: bytes 2, 3
    mma_16816(d, bt_entry<0>(w0[wi], tbl), bt_entry<0>(w1[wi], tbl), bt_entry<1>(w0[wi], tbl),
              bt_entry<1>(w1[wi], tbl), bq[2 * wi][0], bq[2 * wi][1]);
    mma_16816(e, bt_entry<2>(w0[wi], tbl), bt_entry<2>(w1[wi], tbl), bt_entry<3>(w0[wi], tbl),
              bt_entry<3>(w1[wi], tbl), bq[2 * wi + 1][0], bq[2 * wi + 1][1]);
  }
}

// A work unit as the producer publishes it (double-buffered).  Per probe
// j of the unit the same buffer holds, after this header: the partition's
// first row slot off[j] (int64), its rows n[j], cs[j] and the prefix tile
// count tpref[j] (tpref[np] = total).
struct BtUnit {
  int64_t q;     // the query
  int64_t orow;  // output row: the query, or its part
  int np;        // probes of the unit
  int total;     // tiles of the unit
  int valid;     // 0: no more units
};
constexpr int kBtUnitHead = 32;
static_assert(sizeof(BtUnit) <= kBtUnitHead, "unit header");
__host__ __device__ constexpr int bt_unit_bytes(int nprobe) { return (kBtUnitHead + 20 * nprobe + 4 + 15) & ~15; }

__global__ void __launch_bounds__(kBtThreads, 1) scan_bt_kernel(const __grid_constant__ ScanArgs a) {
  extern __shared__ __align__(128) uint8_t bsm[];
  __shared__ __align__(8) uint64_t bars[2 * kBtStages + 4];
  __shared__ int s_fail;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nch = a.stride / 16;
  const uint32_t stage_bytes = uint32_t(nch) * 2048u + 512u;
  // dynamic shared memory: stages 0 .. stages_pre - 1, the byte table at
  // shared address kBtTableAddr, the other stages, the unit descriptors and
  // the warps' lists
  const uint32_t dyn0 = uint32_t(__cvta_generic_to_shared(bsm));
  uint8_t* table = bsm + (kBtTableAddr - dyn0);
  uint8_t* stage_hi = table + kBtTableBytes;
  const int npre = a.stages_pre;
  auto stage_at = [&](uint32_t s) {
    return int(s) < npre ? bsm + size_t(s) * stage_bytes : stage_hi + size_t(int(s) - npre) * stage_bytes;
  };
  const int ubytes = bt_unit_bytes(a.nprobe);
  uint8_t* ubuf0 = stage_hi + size_t(kBtStages - npre) * stage_bytes;
  if (dyn0 + uint32_t(npre) * stage_bytes > kBtTableAddr) {
    // the stages below the table would overlap it (more static shared
    // memory than the host assumed): nothing is scanned
    if (tid == 0) set_device_error(a.err, kErrSmemLayout);
    return;
  }
  float* wsc = reinterpret_cast<float*>(ubuf0 + 2 * ubytes);  // the warps' top-k lists
  int* wps = reinterpret_cast<int*>(wsc + kBtWarps * a.k);
  const uint32_t bar0 = uint32_t(__cvta_generic_to_shared(&bars[0]));
  auto stage_full = [&](uint32_t s) { return bar0 + 8u * s; };
  auto stage_empty = [&](uint32_t s) { return bar0 + 8u * (kBtStages + s); };
  auto unit_full = [&](int b) { return bar0 + 8u * (2 * kBtStages + b); };
  auto unit_empty = [&](int b) { return bar0 + 8u * (2 * kBtStages + 2 + b); };
  // unit buffer b: header, off[nprobe], n[nprobe], cs[nprobe], tpref[nprobe + 1]
  auto unit_at = [&](int b) { return ubuf0 + b * ubytes; };
  auto u_off = [&](int b) { return reinterpret_cast<int64_t*>(unit_at(b) + kBtUnitHead); };
  auto u_n = [&](int b) { return reinterpret_cast<int*>(u_off(b) + a.nprobe); };
  auto u_cs = [&](int b) { return reinterpret_cast<float*>(u_n(b) + a.nprobe); };
  auto u_tpref = [&](int b) { return reinterpret_cast<int*>(u_cs(b) + a.nprobe); };
  auto failed = [&]() { return *reinterpret_cast<volatile int*>(&s_fail) != 0; };
  auto fail = [&]() {
    set_device_error(a.err, kErrTimeout);
    atomicExch(&s_fail, 1);
  };
  {
    // the byte table: low half = level of the low nibble (the even code
    // position), high half = level of the high nibble
    uint32_t* tb = reinterpret_cast<uint32_t*>(table);
    for (int e = tid; e < 256 * 32; e += blockDim.x) {
      const int byte = e >> 5, ln = e & 31;
      const uint32_t lo = __half_as_ushort(__float2half_rn(a.cb[byte & 15]));
      const uint32_t hi = __half_as_ushort(__float2half_rn(a.cb[byte >> 4]));
      tb[byte * 64 + ln] = lo | (hi << 16);
    }
  }
  if (tid == 0) {
    s_fail = 0;
    for (int s = 0; s < kBtStages; ++s) {
      mbar_init(stage_full(s), 1);
      mbar_init(stage_empty(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(unit_full(b), 1);
      mbar_init(unit_empty(b), kBtWarps);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const int parts = a.parts;
  const int64_t nunits = a.nq * parts;

  if (warp == kBtWarps) {
    // ---------------- producer: unit descriptors, then the unit's tiles by bulk copy
    uint32_t T = 0;     // tiles of the units so far
    uint32_t tend = 0;  // this lane: 1 + the last tile it issued
    for (int ui = 0;; ++ui) {
      const int ub = ui & 1;
      if (ui >= 2 && !mbar_wait_warp(unit_empty(ub), ((ui >> 1) - 1) & 1)) {
        fail();
        break;
      }
      BtUnit* hd = reinterpret_cast<BtUnit*>(unit_at(ub));
      int64_t* uoff = u_off(ub);
      int* un = u_n(ub);
      float* ucs = u_cs(ub);
      int* tpref = u_tpref(ub);
      const int64_t u = int64_t(blockIdx.x) + int64_t(ui) * gridDim.x;
      const bool more = u < nunits && !failed();
      int run = 0;
      if (more) {
        const int64_t q = u / parts;
        const int part = int(u % parts);
        const int j0 = int(int64_t(part) * a.nprobe / parts), j1 = int(int64_t(part + 1) * a.nprobe / parts);
        const int np = j1 - j0;
        // probes [j0, j1) -> tiles (a warp-wide running prefix sum)
        for (int base = 0; base < np; base += 32) {
          const int jj = base + lane;
          int nt = 0;
          if (jj < np) {
            const int p = a.probes[q * a.probe_stride + j0 + jj];
            int64_t off = 0;
            int n = 0;
            if (p < 0 || p >= a.nlist) {
              set_device_error(a.err, kErrBadProbe);
            } else {
              off = a.part_off[p];
              n = a.part_n[p];
              nt = (n + kTile - 1) / kTile;
            }
            uoff[jj] = off;
            un[jj] = n;
            ucs[jj] = a.cs ? a.cs[q * a.probe_stride + j0 + jj] : 0.0f;  // no cs: full-vector codes
          }
          int x = nt;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(kFull, x, o);
            if (lane >= o) x += y;
          }
          if (jj < np) tpref[jj] = run + x - nt;
          run += __shfl_sync(kFull, x, 31);
        }
        if (lane == 0) {
          tpref[np] = run;
          hd->q = q;
          hd->orow = u;
          hd->np = np;
          hd->total = run;
          hd->valid = 1;
        }
      } else if (lane == 0) {
        hd->valid = 0;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(unit_full(ub));
      if (!more) break;
      int ok = 1;
      if (lane < kBtWarps) {
        // lane L issues the unit's tiles T with T mod kBtStages = L, into stage L
        int jc = 0;
        const uint32_t s = uint32_t(lane);
        const uint32_t dst = uint32_t(__cvta_generic_to_shared(stage_at(s)));
        for (int i = int((s + kBtStages - T % kBtStages) % kBtStages); i < run; i += kBtStages) {
          while (tpref[jc + 1] <= i) ++jc;
          const int t = i - tpref[jc];
          const int64_t slot0 = uoff[jc] + int64_t(t) * kTile;  // the tile's first row slot
          const bool both = un[jc] - t * kTile > kBtHalf;      // rows in its second half
          const uint32_t Ti = T + uint32_t(i);
          const uint32_t n = Ti / kBtStages;
          if (n > 0 && !mbar_wait(stage_empty(s), (n - 1) & 1)) {
            fail();
            ok = 0;
            break;
          }
          // the codes (when the partition ends in the first half, up to the
          // end of the last chunk column's first half), then the scales
          const uint32_t cbytes = both ? uint32_t(nch) * 2048u : uint32_t(nch - 1) * 2048u + 1024u;
          const uint32_t sbytes = both ? 512u : 256u;
          mbar_arrive_expect(stage_full(s), cbytes + sbytes);
          bulk_copy_1d(dst, a.codes + slot0 * a.stride, cbytes, stage_full(s));
          bulk_copy_1d(dst + uint32_t(nch) * 2048u, a.scales + slot0, sbytes, stage_full(s));
          tend = Ti + 1;
        }
      }
      T += uint32_t(run);
      if (__any_sync(kFull, ok == 0)) break;
    }
    // no copy may still be landing when the CTA exits: each lane waits for
    // the last phase of its stage (the phases before it completed before
    // that copy was issued)
    if (lane < kBtWarps && tend > uint32_t(lane))
      mbar_wait(stage_full(uint32_t(lane)), ((tend - 1 - uint32_t(lane)) / kBtStages) & 1);
    __syncwarp();
  } else {
    // ---------------- consumers: warp w scores the tiles T with T mod kBtStages = w, from stage w
    const int cw = warp;
    const uint32_t lane4 = uint32_t(lane) * 4u;
    const uint32_t tbl = kBtTableAddr | lane4;
    const int tq = lane & 3, gq = lane >> 2;
    const uint8_t* st = stage_at(uint32_t(cw));
    const uint32_t st_addr = uint32_t(__cvta_generic_to_shared(st));
    float* msc = wsc + cw * a.k;
    int* mps = wps + cw * a.k;
    uint32_t T0 = 0;  // sequence number of the unit's first tile
    for (int ui = 0;; ++ui) {
      const int ub = ui & 1;
      const bool got = mbar_wait_warp(unit_full(ub), (ui >> 1) & 1);
      const BtUnit* hd = reinterpret_cast<const BtUnit*>(unit_at(ub));
      if (!got) fail();
      if (!got || failed() || hd->valid == 0) break;
      const int64_t* uoff = u_off(ub);
      const int* un = u_n(ub);
      const float* ucs = u_cs(ub);
      const int* tpref = u_tpref(ub);
      const int64_t q = hd->q, orow = hd->orow;
      const int total = hd->total;
      const float* qr = a.qrot + q * a.Dp;
      // 2^s with max |q| 2^s in [1024, 2048)
      float m = 0.0f;
      for (int d = lane; d < a.Dp; d += 32) m = fmaxf(m, fabsf(qr[d]));
#pragma unroll
      for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(kFull, m, o));
      int ex = 0;
      if (m > 0.0f) frexpf(m, &ex);
      const float qsc = ldexpf(1.0f, 11 - ex), qinv = ldexpf(1.0f, ex - 11);
      // this lane's query fragments: column gq (0: hi, 1: lo, else 0); for
      // MMA m of chunk column c (index 2 c + m) the positions
      // 32 c + 8 tq + 4 m + {0, 1} (register 0) and + {2, 3} (register 1)
      uint32_t bq[8][2];
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int c = i >> 1;
          uint32_t wv = 0;
          if (gq < 2 && c < nch) {
            const int k0 = 32 * c + 8 * tq + 4 * (i & 1) + 2 * r;
            __half h2[2];
#pragma unroll
            for (int x = 0; x < 2; ++x) {
              const float v = (k0 + x < a.Dp ? __ldg(qr + k0 + x) : 0.0f) * qsc;
              const __half hi = __float2half_rn(v);
              h2[x] = gq == 0 ? hi : __float2half_rn(v - __half2float(hi));
            }
            wv = uint32_t(__half_as_ushort(h2[0])) | (uint32_t(__half_as_ushort(h2[1])) << 16);
          }
          bq[i][r] = wv;
        }
      int cnt = 0;
      float thr = -CUDART_INF_F;
      int thr_pos = INT_MAX;
      // candidates (s, pos) of the lane's rows -> the warp's top-k list
      auto offer = [&](float sc, int pos, bool valid) {
        const bool cand = valid && (cnt < a.k || sc > thr || (sc == thr && pos < thr_pos));
        unsigned mk = __ballot_sync(kFull, cand);
        while (mk) {
          const int src = __ffs(mk) - 1;
          mk &= mk - 1;
          const float s2 = __shfl_sync(kFull, sc, src);
          const int p2 = __shfl_sync(kFull, pos, src);
          if (cnt < a.k || s2 > thr || (s2 == thr && p2 < thr_pos)) {
            warp_insert(msc, mps, cnt, a.k, s2, p2, lane);
            if (cnt == a.k) {
              thr = msc[a.k - 1];
              thr_pos = mps[a.k - 1];
            }
          }
        }
      };
      int jc = 0;
      for (int i = int((uint32_t(cw) + kBtStages - T0 % kBtStages) % kBtStages); i < total; i += kBtStages) {
        const uint32_t T = T0 + uint32_t(i);
        while (tpref[jc + 1] <= i) ++jc;
        const int t = i - tpref[jc];
        const int nvalid = min(kTile, un[jc] - t * kTile);
        const bool two = nvalid > kBtHalf;  // rows in the second half
        const int pos0 = int(uoff[jc]) + t * kTile;
        const float csj = ucs[jc];
        if (!mbar_wait_warp(stage_full(uint32_t(cw)), (T / kBtStages) & 1)) {
          fail();
          break;
        }
        // this lane's rows: 16 tq + gq and + 8 of each half
        const int ra = 16 * tq + gq, rb = ra + 8;
        const uint32_t* scl = reinterpret_cast<const uint32_t*>(st + nch * 2048);
        uint32_t sw[2][2];
        sw[0][0] = scl[ra];
        sw[0][1] = scl[rb];
        sw[1][0] = two ? scl[kBtHalf + ra] : 0u;
        sw[1][1] = two ? scl[kBtHalf + rb] : 0u;
        // the tile's code words by ldmatrix: for pass P (rows 16 P .. + 15)
        // and chunk columns (2 x, 2 x + 1), word tq of rows gq and gq + 8
        uint32_t w[8][2][4];
        auto load_pass = [&](int P) {
#pragma unroll
          for (int x = 0; x < 2; ++x) {
            int c = 2 * x + (lane >> 4);
            c = c < nch ? c : 0;  // a column past the row's codes: any staged bytes (the query is 0 there)
            const int r = 16 * P + 8 * ((lane >> 3) & 1) + (lane & 7);
            asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                         : "=r"(w[P][0][2 * x]), "=r"(w[P][1][2 * x]), "=r"(w[P][0][2 * x + 1]),
                           "=r"(w[P][1][2 * x + 1])
                         : "r"(st_addr + uint32_t(c * kTile + r) * 16u)
                         : "memory");
          }
        };
#pragma unroll
        for (int P = 0; P < 4; ++P) load_pass(P);
        if (two) {
#pragma unroll
          for (int P = 4; P < 8; ++P) load_pass(P);
        }
        // the stage has been read: release it to the producer (the generic
        // reads before the next bulk copy into it)
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(stage_empty(uint32_t(cw)));
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          if (hh == 1 && !two) break;
          float da = 0.0f, db = 0.0f;
#pragma unroll
          for (int pp = 0; pp < 4; ++pp) {
            const int P = 4 * hh + pp;
            float d[4] = {0.0f, 0.0f, 0.0f, 0.0f}, e[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            bt_group_mma(tbl, w[P][0], w[P][1], bq, d, e);
            // lanes tq = 0: (hi, lo) of rows 16 P + gq (d0, d1) and + 8 (d2, d3)
            const float x0 = __shfl_sync(kFull, (d[0] + e[0]) + (d[1] + e[1]), lane & ~3);
            const float x1 = __shfl_sync(kFull, (d[2] + e[2]) + (d[3] + e[3]), lane & ~3);
            if (tq == pp) {
              da = x0;
              db = x1;
            }
          }
          // epilogue of the half's 64 rows: two per lane
          const int hv = nvalid - kBtHalf * hh;
          const bool va = ra < hv, vb = rb < hv;
          const uint32_t swa = sw[hh][0], swb = sw[hh][1];
          const float sa = va ? ue4m12_to_f32(swa >> 16) * fmaf(ue7m9_to_f32(swa & 0xffffu), da * qinv, csj)
                              : -CUDART_INF_F;
          const float sb = vb ? ue4m12_to_f32(swb >> 16) * fmaf(ue7m9_to_f32(swb & 0xffffu), db * qinv, csj)
                              : -CUDART_INF_F;
          offer(sa, pos0 + kBtHalf * hh + ra, va);
          offer(sb, pos0 + kBtHalf * hh + rb, vb);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(unit_empty(ub));  // the unit's descriptor is no longer read
      T0 += uint32_t(total);
      // this warp's list of the unit -> its row of the partial lists (k
      // entries, -1 / -inf padded); merge_parts_kernel merges the rows
      const int64_t prow = orow * kBtWarps + cw;
      for (int e = lane; e < a.k; e += 32) {
        const bool ok = e < cnt;
        a.out_ids[prow * a.k + e] = ok ? a.ids[mps[e]] : -1;
        a.out_scores[prow * a.k + e] = ok ? msc[e] : -CUDART_INF_F;
      }
      __syncwarp();  // the list is read before the next unit's inserts
    }
  }
  __syncthreads();
}

// Top out_k of a query's `parts` partial lists (k entries each, sorted by
// (score desc, id asc), -1 / -inf padded): one block per query.
__global__ void merge_parts_kernel(const int64_t* __restrict__ pid, const float* __restrict__ psc, int64_t nq,
                                   int parts, int k, int out_k, int64_t* __restrict__ out_ids,
                                   float* __restrict__ out_scores) {
  extern __shared__ __align__(16) uint8_t msm[];
  const int n = parts * k;
  int np2 = 1;
  while (np2 < n) np2 <<= 1;
  float* key = reinterpret_cast<float*>(msm);
  int64_t* idv = reinterpret_cast<int64_t*>(msm + ((size_t(np2) * 4 + 15) & ~size_t(15)));
  for (int64_t q = blockIdx.x; q < nq; q += gridDim.x) {
    for (int e = threadIdx.x; e < np2; e += blockDim.x) {
      const int64_t id = e < n ? pid[q * n + e] : -1;
      key[e] = id >= 0 ? psc[q * n + e] : -CUDART_INF_F;
      idv[e] = id >= 0 ? id : LLONG_MAX;
    }
    block_bitonic_sort(key, idv, np2);
    for (int e = threadIdx.x; e < out_k; e += blockDim.x) {
      const bool ok = idv[e] != LLONG_MAX;
      out_ids[q * out_k + e] = ok ? idv[e] : -1;
      out_scores[q * out_k + e] = ok ? key[e] : -CUDART_INF_F;
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------- rescore
struct RescoreArgs {
  const float* qrot2;
  int Dp2;
  const int64_t* cand_ids;
  const float* cand_scores;
  int k;
  int kf;
  const int32_t* slot_of_row;
  int64_t n_rows;
  const uint8_t* codes2;
  const uint32_t* scales2;
  int stride2;
  int code_bytes2;
  float lv[16];
  // <q, a2>: reading B the stage-1 score; reading A <R2 q, R2 c> of the row's
  // partition (crot2, assign); 0 for full-vector codes (zero_a)
  const float* crot2;
  const int32_t* assign;
  int zero_a;
  int64_t* out_ids;
  float* out_scores;
  int* err;
  // rescore_mma_kernel: queries, warps whose region sits below the byte
  // table, bytes per warp region
  int64_t nq;
  int warps_pre;
  int region;
  uint32_t zero;  // 0: makes the table lookups depend on a segment pair's loads (all issued first)
};

__global__ void __launch_bounds__(256) rescore_kernel(const __grid_constant__ RescoreArgs a) {
  extern __shared__ __align__(16) uint8_t rsm2[];
  __shared__ float lv[16];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, W = blockDim.x >> 5;
  const int64_t q = blockIdx.x;
  int np2 = 1;
  while (np2 < a.k) np2 <<= 1;
  const int qlen = 2 * a.stride2;
  float* q2 = reinterpret_cast<float*>(rsm2);
  float* key = q2 + qlen;
  int64_t* idv = reinterpret_cast<int64_t*>(rsm2 + ((size_t(qlen + np2) * 4 + 15) & ~size_t(15)));
  if (tid < 16) lv[tid] = a.lv[tid];
  for (int d = tid; d < qlen; d += blockDim.x) q2[d] = d < a.Dp2 ? a.qrot2[q * a.Dp2 + d] : 0.0f;
  __syncthreads();
  for (int j = warp; j < np2; j += W) {
    float s2 = -CUDART_INF_F;
    int64_t id = LLONG_MAX;
    if (j < a.k) {
      const int64_t cid = a.cand_ids[q * a.k + j];
      if (cid >= a.n_rows || cid < -1) set_device_error(a.err, kErrBadCandidate);
      if (cid >= 0 && cid < a.n_rows) {
        const int64_t slot = a.slot_of_row[cid];
        const uint8_t* row = a.codes2 + slot * a.stride2;
        float acc = 0.0f;
        for (int b = lane * 4; b < a.code_bytes2; b += 128) {
          const uint32_t w = __ldg(reinterpret_cast<const uint32_t*>(row + b));
#pragma unroll
          for (int n = 0; n < 8; ++n) acc = fmaf(lv[(w >> (4 * n)) & 15u], q2[2 * b + n], acc);
        }
        acc = warp_sum(acc);
        const uint32_t sc = __ldg(a.scales2 + slot);
        float a2 = a.cand_scores[q * a.k + j];  // reading B: <q, a2> = s1
        if (a.zero_a) {
          a2 = 0.0f;
        } else if (a.crot2) {
          const float* cr = a.crot2 + int64_t(a.assign[cid]) * a.Dp2;
          float c = 0.0f;
          for (int d = lane; d < a.Dp2; d += 32) c = fmaf(q2[d], __ldg(cr + d), c);
          a2 = warp_sum(c);
        }
        s2 = ue4m12_to_f32(sc >> 16) * fmaf(ue7m9_to_f32(sc & 0xffffu), acc, a2);
        id = cid;
      }
    }
    if (lane == 0) {
      key[j] = s2;
      idv[j] = id;
    }
  }
  block_bitonic_sort(key, idv, np2);
  for (int e = tid; e < a.kf; e += blockDim.x) {
    const bool ok = idv[e] != LLONG_MAX;
    a.out_ids[q * a.kf + e] = ok ? idv[e] : -1;
    a.out_scores[q * a.kf + e] = ok ? key[e] : -CUDART_INF_F;
  }
}

// Rescoring on the tensor cores, for 4-bit rescoring codes of one
// coordinate each scored by reading B (<q, a2> = the stage-1 score) or as
// full-vector codes: one warp per query in persistent CTAs of up to
// kRsWarps warps, one CTA per SM.  The warp-level MMA m16n8k16 (fp16
// operands, fp32 accumulation) is the multiply-add engine, as in the
// single-query scan:
//   A (16 candidate rows x 16 code positions) = the codes' levels, looked
//     up through the per-lane byte table at kBtTableAddr (a byte = two codes
//     -> their two binary16-exact levels, one A register);
//   B (16 x 8) = the rotated query scaled by 2^s (max |q| 2^s in [1024,
//     2048)) and split into q_hi = fp16(q) (column 0) and q_lo = fp16(q -
//     q_hi) (column 1);
//   D column 0 + column 1 = 2^s <R2 q, u2hat> of each row.
// A rescoring row is contiguous (stride2 bytes, a multiple of 16).  Lane (g,
// t) = (lane / 4, lane % 4) loads bytes 64 J + 16 t .. + 15 of rows g and g
// + 8 of a 16-row group: code positions 128 J + 32 t + 8 w + {0..7} in its
// word w, and MMA i = 2 w + m of segment J takes bytes 2 m and 2 m + 1 of
// word w, i.e. positions 128 J + 32 t + 4 i + {0..3}.  The dot product is
// order-free, so the B fragment of lane (g, t) holds those same positions of
// column g; the warp's query block keeps them as one 16-byte entry (J, i,
// t) = (hi, lo) halves of the four positions, so the eight lanes that read
// an entry set touch 64 contiguous bytes.  A pass scores 32 candidates (two
// 16-row groups share the B fragments); s2 = G2 (<q, a2> + L2 <R2 q,
// u2hat>) (Sec. 3.5, Sec. 5.2) is stored in place of the stage-1 score, and
// a warp bitonic sort of the query's k candidates by (score desc, id asc)
// gives the top k_final.  Per warp: the query block (stride2 x 8 bytes
// rounded to 512), then np2 keys and np2 ids.
constexpr int kRsWarps = 16;


__device__ __forceinline__ void warp_bitonic_sort(float* key, int64_t* id, int n) {
  const int lane = threadIdx.x & 31;
  for (int size = 2; size <= n; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      __syncwarp();
      for (int i = lane; i < (n >> 1); i += 32) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool asc = (lo & size) == 0;
        const float klo = key[lo], khi = key[hi];
        const int64_t ilo = id[lo], ihi = id[hi];
        const bool swap = asc ? better(khi, ihi, klo, ilo) : better(klo, ilo, khi, ihi);
        if (swap) {
          key[lo] = khi;
          key[hi] = klo;
          id[lo] = ihi;
          id[hi] = ilo;
        }
      }
    }
  }
  __syncwarp();
}

__global__ void __launch_bounds__(kRsWarps * 32, 1) rescore_mma_kernel(const __grid_constant__ RescoreArgs a) {
  extern __shared__ __align__(128) uint8_t rsm[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
  const uint32_t dyn0 = uint32_t(__cvta_generic_to_shared(rsm));
  uint8_t* table = rsm + (kBtTableAddr - dyn0);
  if (dyn0 + uint32_t(a.warps_pre) * uint32_t(a.region) > kBtTableAddr) {
    // the regions below the table would overlap it (more static shared
    // memory than the host assumed): nothing is rescored
    if (tid == 0) set_device_error(a.err, kErrSmemLayout);
    return;
  }
  {
    // the byte table: low half = level of the low nibble (the even code
    // position), high half = level of the high nibble
    uint32_t* tb = reinterpret_cast<uint32_t*>(table);
    for (int e = tid; e < 256 * 32; e += blockDim.x) {
      const int byte = e >> 5, ln = e & 31;
      const uint32_t lo = __half_as_ushort(__float2half_rn(a.lv[byte & 15]));
      const uint32_t hi = __half_as_ushort(__float2half_rn(a.lv[byte >> 4]));
      tb[byte * 64 + ln] = lo | (hi << 16);
    }
  }
  __syncthreads();
  uint8_t* reg = warp < a.warps_pre ? rsm + size_t(warp) * a.region
                                    : table + kBtTableBytes + size_t(warp - a.warps_pre) * a.region;
  const int nj = (a.stride2 + 63) / 64;
  int np2 = 2;
  while (np2 < a.k) np2 <<= 1;
  const uint8_t* qblk = reg;
  float* key = reinterpret_cast<float*>(reg + size_t(nj) * 512);
  int64_t* idv = reinterpret_cast<int64_t*>(key + np2);
  const uint32_t tbl = kBtTableAddr | (uint32_t(lane) * 4u);
  const int t = lane & 3, g = lane >> 2;
  const int64_t nwt = int64_t(gridDim.x) * nw;
  for (int64_t q = int64_t(blockIdx.x) * nw + warp; q < a.nq; q += nwt) {
    // 2^s with max |q| 2^s in [1024, 2048)
    const float* qr = a.qrot2 + q * a.Dp2;
    float m = 0.0f;
    for (int d = lane; d < a.Dp2; d += 32) m = fmaxf(m, fabsf(__ldg(qr + d)));
#pragma unroll
    for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(kFull, m, o));
    int ex = 0;
    if (m > 0.0f) frexpf(m, &ex);
    const float qsc = ldexpf(1.0f, 11 - ex), qinv = ldexpf(1.0f, ex - 11);
    // the query block: entry (J, i, t) at 16 ((8 J + i) 4 + t) holds the hi
    // halves, then the lo halves, of positions 128 J + 32 t + 4 i + {0..3}
    for (int e = lane; e < nj * 32; e += 32) {
      const int p = 128 * (e >> 5) + 32 * (e & 3) + 4 * ((e >> 2) & 7);
      uint32_t h2[2], l2[2];
#pragma unroll
      for (int x = 0; x < 2; ++x) {
        __half hh[2], ll[2];
#pragma unroll
        for (int y = 0; y < 2; ++y) {
          const int d = p + 2 * x + y;
          const float v = d < a.Dp2 ? __ldg(qr + d) * qsc : 0.0f;
          hh[y] = __float2half_rn(v);
          ll[y] = __float2half_rn(v - __half2float(hh[y]));
        }
        h2[x] = uint32_t(__half_as_ushort(hh[0])) | (uint32_t(__half_as_ushort(hh[1])) << 16);
        l2[x] = uint32_t(__half_as_ushort(ll[0])) | (uint32_t(__half_as_ushort(ll[1])) << 16);
      }
      *reinterpret_cast<uint4*>(reg + size_t(e) * 16) = make_uint4(h2[0], h2[1], l2[0], l2[1]);
    }
    // the candidates: ids (LLONG_MAX: none) and <q, a2>
    for (int j = lane; j < np2; j += 32) {
      int64_t id = LLONG_MAX;
      float s1 = -CUDART_INF_F;
      if (j < a.k) {
        const int64_t cid = a.cand_ids[q * a.k + j];
        if (cid >= a.n_rows || cid < -1) set_device_error(a.err, kErrBadCandidate);
        if (cid >= 0 && cid < a.n_rows) {
          id = cid;
          s1 = a.zero_a ? 0.0f : a.cand_scores[q * a.k + j];
        }
      }
      idv[j] = id;
      key[j] = s1;
    }
    __syncwarp();
    for (int j0 = 0; j0 < a.k; j0 += 32) {
      // this lane's rows j0 + g + 8 h (h = 0, 1: group 0; 2, 3: group 1),
      // at its 16-byte column of each 64-byte segment
      const uint8_t* rp[4];
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        const int j = j0 + g + 8 * h;
        const int64_t id = j < a.k ? idv[j] : LLONG_MAX;
        rp[h] = id != LLONG_MAX ? a.codes2 + int64_t(__ldg(a.slot_of_row + id)) * a.stride2 + 16 * t : nullptr;
      }
      float d0[4] = {0.0f, 0.0f, 0.0f, 0.0f}, e0[4] = {0.0f, 0.0f, 0.0f, 0.0f};
      float d1[4] = {0.0f, 0.0f, 0.0f, 0.0f}, e1[4] = {0.0f, 0.0f, 0.0f, 0.0f};
      // two 64-byte segments per step: their eight loads are issued together
      // (the lookups' table address depends on all of them; a.zero = 0)
      for (int J = 0; J < nj; J += 2) {
        uint4 w[2][4];
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
          const bool in = J + jj < nj && 64 * (J + jj) + 16 * t < a.stride2;  // rows are whole 16-byte columns
#pragma unroll
          for (int h = 0; h < 4; ++h)
            w[jj][h] = rp[h] != nullptr && in ? __ldg(reinterpret_cast<const uint4*>(rp[h] + 64 * (J + jj)))
                                              : make_uint4(0u, 0u, 0u, 0u);
        }
        uint32_t dep = 0u;
#pragma unroll
        for (int jj = 0; jj < 2; ++jj)
#pragma unroll
          for (int h = 0; h < 4; ++h) dep |= w[jj][h].x | w[jj][h].y | w[jj][h].z | w[jj][h].w;
        const uint32_t tblj = tbl | (dep & a.zero);
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
          if (J + jj >= nj) break;
          uint32_t bq[8][2];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            uint2 v = make_uint2(0u, 0u);
            if (g < 2) v = *reinterpret_cast<const uint2*>(qblk + ((8 * (J + jj) + i) * 4 + t) * 16 + 8 * g);
            bq[i][0] = v.x;
            bq[i][1] = v.y;
          }
          const uint32_t w0[4] = {w[jj][0].x, w[jj][0].y, w[jj][0].z, w[jj][0].w};
          const uint32_t w1[4] = {w[jj][1].x, w[jj][1].y, w[jj][1].z, w[jj][1].w};
          const uint32_t w2[4] = {w[jj][2].x, w[jj][2].y, w[jj][2].z, w[jj][2].w};
          const uint32_t w3[4] = {w[jj][3].x, w[jj][3].y, w[jj][3].z, w[jj][3].w};
          bt_group_mma(tblj, w0, w1, bq, d0, e0);
          bt_group_mma(tblj, w2, w3, bq, d1, e1);
        }
      }
      // lanes t = 0 hold (hi, lo) of rows g, g + 8 (group 0) and g + 16,
      // g + 24 (group 1); lane L takes row j0 + L
      const float r0 = (d0[0] + e0[0]) + (d0[1] + e0[1]), r1 = (d0[2] + e0[2]) + (d0[3] + e0[3]);
      const float r2 = (d1[0] + e1[0]) + (d1[1] + e1[1]), r3 = (d1[2] + e1[2]) + (d1[3] + e1[3]);
      const int src = 4 * (lane & 7), part = lane >> 3;
      const float x0 = __shfl_sync(kFull, r0, src), x1 = __shfl_sync(kFull, r1, src);
      const float x2 = __shfl_sync(kFull, r2, src), x3 = __shfl_sync(kFull, r3, src);
      const float dot = part == 0 ? x0 : part == 1 ? x1 : part == 2 ? x2 : x3;
      const int j = j0 + lane;
      if (j < a.k && idv[j] != LLONG_MAX) {
        const uint32_t sc = __ldg(a.scales2 + __ldg(a.slot_of_row + idv[j]));
        key[j] = ue4m12_to_f32(sc >> 16) * fmaf(ue7m9_to_f32(sc & 0xffffu), dot * qinv, key[j]);
      }
    }
    warp_bitonic_sort(key, idv, np2);
    for (int e = lane; e < a.kf; e += 32) {
      const bool ok = idv[e] != LLONG_MAX;
      a.out_ids[q * a.kf + e] = ok ? idv[e] : -1;
      a.out_scores[q * a.kf + e] = ok ? key[e] : -CUDART_INF_F;
    }
    __syncwarp();  // the region is read before the next query's stores
  }
}
template <int CH, bool B3>
cudaError_t launch_scan_ch(const rslm_index* ix, const ScanArgs& a, int64_t nq, size_t smem,
                           cudaStream_t s) {
  // listed queries: a fixed grid strides over the list, whose length is on the device
  const int64_t grid = a.qlist ? (nq < 2 * 152 ? nq : 2 * 152) : nq;
  cudaError_t e = cudaFuncSetAttribute(scan_kernel<CH, B3>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       int(smem));
  if (e != cudaSuccess) return e;
  cudaEvent_t stop =
      a.only_if == nullptr && a.qlist == nullptr && a.nprobe > 1 ? prof_start(ix, s, "scan_kernel") : nullptr;
  scan_kernel<CH, B3><<<unsigned(grid), 256, smem, s>>>(a);
  prof_stop(stop, s);
  return cudaGetLastError();
}

// Shared memory of scan_bt_kernel for a's k and nprobe: sets a.stages
// (kBtStages, or 0 when they do not fit) and returns the bytes.
size_t plan_scan_bt(ScanArgs& a, int dev) {
  const int k = a.k;
  const size_t stage_bytes = size_t(a.stride / 16) * 2048 + 512;
  const size_t ubytes = size_t(bt_unit_bytes(a.nprobe));
  // below the table: the stages that fit when static and reserved shared
  // memory take at most kBtLowReserve bytes (the kernel checks); the
  // dynamic allocation starts at most that far above 0, so reserving the
  // full 64 KB below the table always suffices
  const int pre = std::min(kBtStages, int((kBtTableAddr - kBtLowReserve) / stage_bytes));
  const size_t bytes = size_t(kBtTableAddr) + size_t(kBtTableBytes) + size_t(kBtStages - pre) * stage_bytes +
                       2 * ubytes + size_t(kBtWarps) * k * 8;
  int optin = 0;
  if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) optin = 0;
  const bool fits = bytes + kBtLowReserve <= size_t(optin);
  a.stages = fits ? kBtStages : 0;
  a.stages_pre = fits ? pre : 0;
  return fits ? bytes : 0;
}

// scan_bt_kernel over nq queries, after plan_scan_bt.  Every (unit, consumer
// warp) writes a k-entry list into a stream-ordered workspace; batches too
// small to give every SM several units split each query's probe list into
// `parts` units.  merge_parts_kernel merges the kBtWarps * parts lists of
// each query into its top out_k.
cudaError_t launch_scan_bt(const rslm_index* ix, ScanArgs a, int64_t nq, size_t smem, int sms, cudaStream_t s) {
  const int k = a.k;
  int parts = 1;
  const int64_t want = int64_t(4) * sms;  // units: about four per SM
  if (nq < want) parts = int(std::min<int64_t>(a.nprobe, (want + nq - 1) / nq));
  parts = std::max(1, std::min(parts, 4096 / (kBtWarps * k)));  // the merge sorts its lists in shared memory
  a.parts = parts;
  a.nq = nq;
  cudaError_t e = cudaFuncSetAttribute(scan_bt_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  const int nl = parts * kBtWarps;  // lists per query
  const size_t n = size_t(nq) * nl * k;
  void* ws = nullptr;
  e = cudaMallocAsync(&ws, n * 12, s);
  if (e != cudaSuccess) return e;
  int64_t* pids = reinterpret_cast<int64_t*>(ws);
  float* pscs = reinterpret_cast<float*>(pids + n);
  const int out_k = a.out_k;
  int64_t* final_ids = a.out_ids;
  float* final_sc = a.out_scores;
  a.out_ids = pids;
  a.out_scores = pscs;
  a.out_k = k;
  const int64_t grid = std::min<int64_t>(nq * parts, sms);
  cudaEvent_t stop = a.nprobe > 1 ? prof_start(ix, s, "scan_bt_kernel") : nullptr;
  scan_bt_kernel<<<unsigned(grid), kBtThreads, smem, s>>>(a);
  prof_stop(stop, s);
  e = cudaGetLastError();
  if (e == cudaSuccess) {
    int mp2 = 1;
    while (mp2 < nl * k) mp2 <<= 1;
    const size_t msm = ((size_t(mp2) * 4 + 15) & ~size_t(15)) + size_t(mp2) * 8;
    e = cudaFuncSetAttribute(merge_parts_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(msm));
    if (e == cudaSuccess) {
      merge_parts_kernel<<<unsigned(std::min<int64_t>(nq, int64_t(8) * sms)), 256, msm, s>>>(
          pids, pscs, nq, nl, k, out_k, final_ids, final_sc);
      e = cudaGetLastError();
    }
  }
  cudaError_t f = cudaFreeAsync(ws, s);
  return e == cudaSuccess ? f : e;
}

}  // namespace

cudaError_t launch_select_topn(const float* S, int64_t rows, int64_t ld, int n, int kk,
                               int32_t* out_idx, float* out_val, int* flags, cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  int p2 = 1;
  while (p2 < kk) p2 <<= 1;
  const int* only_if = nullptr;
  cudaError_t e;
  if (kk <= 256 && flags && ld % 4 == 0 && (reinterpret_cast<uintptr_t>(S) & 15) == 0) {
    select_warp_kernel<<<unsigned((rows + kSelWarps - 1) / kSelWarps), kSelWarps * 32, 0, s>>>(
        S, rows, ld, n, kk, out_idx, out_val, flags);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    only_if = flags;  // rows whose candidates overflowed the warp buffer
  }
  const size_t base = size_t(p2 >= 1024 ? p2 : 1024) * 8;
  const size_t staged = base + size_t(n) * 4;
  if (staged <= size_t(160) * 1024) {
    e = cudaFuncSetAttribute(select_topn_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             int(staged));
    if (e != cudaSuccess) return e;
    select_topn_kernel<true><<<unsigned(rows), 256, staged, s>>>(S, ld, n, kk, out_idx, out_val, only_if);
  } else {
    e = cudaFuncSetAttribute(select_topn_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             int(base));
    if (e != cudaSuccess) return e;
    select_topn_kernel<false><<<unsigned(rows), 256, base, s>>>(S, ld, n, kk, out_idx, out_val, only_if);
  }
  return cudaGetLastError();
}

cudaError_t launch_scan(const rslm_index* ix, const float* qrot, int64_t nq, const int32_t* probes,
                        const float* cs, int nprobe, int k, int out_k, int64_t* out_ids,
                        float* out_scores, cudaStream_t s) {
  return launch_scan_strided(ix, qrot, nq, probes, nprobe, cs, nprobe, k, out_k, out_ids, out_scores,
                             nullptr, s);
}

namespace {
cudaError_t launch_scan_impl(const rslm_index* ix, const float* qrot, int64_t nq, const int32_t* probes,
                             int probe_stride, const float* cs, int nprobe, int k, int out_k,
                             int64_t* out_ids, float* out_scores, const int* only_if, const int* qlist,
                             const int* qcount, cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  ScanArgs a;
  a.qlist = qlist;
  a.qcount = qcount;
  a.qrot = qrot;
  a.Dp = ix->cs1.Dp;
  a.probes = probes;
  a.cs = (ix->flags & RSLM_FULL_VECTOR) ? nullptr : cs;
  a.nprobe = nprobe;
  a.probe_stride = probe_stride;
  a.only_if = only_if;
  a.k = k;
  a.out_k = out_k;
  a.codes = ix->codes1;
  a.scales = ix->scales1;
  a.ids = ix->ids;
  a.part_off = ix->part_off;
  a.part_n = ix->part_n;
  a.nlist = ix->nlist;
  a.stride = ix->cs1.stride;
  const bool b3 = ix->cs1.bits == 3;
  a.lut_groups = b3 ? (ix->cs1.ngroups + 31) / 32 * 32 : 2 * ix->cs1.stride;
  a.ngroups = ix->cs1.ngroups;
  a.g = ix->cs1.g;
  for (int i = 0; i < 64; ++i) a.cb[i] = ix->cs1.cbf[i];
  a.lite_h = ix->cs1.lite_h;
  for (int i = 0; i < 8; ++i) a.cb8[i] = ix->cs1.cb8f[i];
  a.out_ids = out_ids;
  a.out_scores = out_scores;
  a.err = ix->d_err;
  const int W = 8;
  int np2 = 1;
  while (np2 < W * k) np2 <<= 1;
  a.parts = 1;
  // 4-bit codes of one coordinate in 16-byte chunks, padded D <= 128: the tensor-core form
  if (!b3 && ix->cs1.g == 1 && ix->cs1.lite_h == 0 && ix->cs1.chunk == 16 &&
      ix->cs1.stride <= 16 * kBtMaxChunks && only_if == nullptr && qlist == nullptr) {
    int dev = 0, sms = 152;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    ScanArgs b = a;
    const size_t bsmem = plan_scan_bt(b, dev);
    if (b.stages > 0) return launch_scan_bt(ix, b, nq, bsmem, sms, s);
  }
  const size_t lut_bytes = size_t(a.lut_groups) * (b3 ? 8 : 16) * 4;
  const size_t merge_bytes = ((size_t(np2) * 4 + 15) & ~size_t(15)) + size_t(np2) * 8;
  size_t region = lut_bytes > merge_bytes ? lut_bytes : merge_bytes;
  region = (region + 15) & ~size_t(15);
  a.lut_region = int(region);
  const size_t smem = 256 + region + size_t(W) * k * 8 + size_t(W) * 4 + size_t(2 * nprobe + 1) * 4;
  if (b3) return launch_scan_ch<4, true>(ix, a, nq, smem, s);
  switch (ix->cs1.chunk) {
    case 16: return launch_scan_ch<16, false>(ix, a, nq, smem, s);
    case 8: return launch_scan_ch<8, false>(ix, a, nq, smem, s);
    default: return launch_scan_ch<4, false>(ix, a, nq, smem, s);
  }
}
}  // namespace

cudaError_t launch_scan_strided(const rslm_index* ix, const float* qrot, int64_t nq,
                                const int32_t* probes, int probe_stride, const float* cs, int nprobe,
                                int k, int out_k, int64_t* out_ids, float* out_scores,
                                const int* only_if, cudaStream_t s) {
  return launch_scan_impl(ix, qrot, nq, probes, probe_stride, cs, nprobe, k, out_k, out_ids, out_scores,
                          only_if, nullptr, nullptr, s);
}

cudaError_t launch_scan_listed(const rslm_index* ix, const float* qrot, int64_t nq, const int32_t* probes,
                               int probe_stride, const float* cs, int nprobe, int k, int64_t* out_ids,
                               float* out_scores, const int* qlist, const int* qcount, cudaStream_t s) {
  return launch_scan_impl(ix, qrot, nq, probes, probe_stride, cs, nprobe, k, k, out_ids, out_scores, nullptr,
                          qlist, qcount, s);
}

cudaError_t launch_rescore(const rslm_index* ix, const float* qrot2, int64_t nq,
                           const int64_t* cand_ids, const float* cand_scores, int k, int k_final,
                           int64_t* out_ids, float* out_scores, cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  RescoreArgs a;
  a.qrot2 = qrot2;
  a.Dp2 = ix->cs2.Dp;
  a.cand_ids = cand_ids;
  a.cand_scores = cand_scores;
  a.k = k;
  a.kf = k_final;
  a.slot_of_row = ix->slot_of_row;
  a.n_rows = ix->n_rows;
  a.codes2 = ix->codes2;
  a.scales2 = ix->scales2;
  a.stride2 = ix->cs2.stride;
  a.code_bytes2 = ix->cs2.code_bytes;
  for (int i = 0; i < 16; ++i) a.lv[i] = ix->cs2.cbf[i];
  const bool reading_a = (ix->flags & RSLM_RESCORE_READING_A) != 0;
  a.zero_a = reading_a && (ix->flags & RSLM_FULL_VECTOR) ? 1 : 0;
  a.crot2 = reading_a ? ix->crot2 : nullptr;
  a.assign = ix->assign;
  a.out_ids = out_ids;
  a.out_scores = out_scores;
  a.err = ix->d_err;
  if (a.crot2 == nullptr && ix->cs2.g == 1 && ix->cs2.stride % 16 == 0 && k <= 256) {
    // the tensor-core kernel: per-warp regions below and above the byte table
    int np2m = 2;
    while (np2m < k) np2m <<= 1;
    const size_t region =
        (size_t((ix->cs2.stride + 63) / 64) * 512 + size_t(np2m) * 12 + 15) & ~size_t(15);
    int dev = 0, optin = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const int pre = int(std::min<size_t>(kRsWarps, (kBtTableAddr - kBtLowReserve) / region));
    const long above = long(optin) - long(kBtLowReserve) - long(kBtTableAddr) - long(kBtTableBytes);
    const int post = above > 0 ? int(std::min<long>(kRsWarps - pre, above / long(region))) : 0;
    const int nw = pre + post;
    if (nw >= 4) {
      a.nq = nq;
      a.zero = 0u;
      a.warps_pre = pre;
      a.region = int(region);
      const size_t bytes = size_t(kBtTableAddr) + size_t(kBtTableBytes) + size_t(post) * region;
      e = cudaFuncSetAttribute(rescore_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(bytes));
      if (e != cudaSuccess) return e;
      const int64_t grid = std::min<int64_t>(sms, (nq + nw - 1) / nw);
      rescore_mma_kernel<<<unsigned(grid), unsigned(nw * 32), bytes, s>>>(a);
      return cudaGetLastError();
    }
  }
  int np2 = 1;
  while (np2 < k) np2 <<= 1;
  const size_t smem = ((size_t(2 * a.stride2 + np2) * 4 + 15) & ~size_t(15)) + size_t(np2) * 8;
  cudaError_t e = cudaFuncSetAttribute(rescore_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       int(smem));
  if (e != cudaSuccess) return e;
  rescore_kernel<<<unsigned(nq), 256, smem, s>>>(a);
  return cudaGetLastError();
}

}  // namespace rslm
