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
  int bt_bytes;    // byte-table form: bytes of the per-lane byte table at the start of shared memory (else 0)
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

// Byte-table form (4-bit codes with one coordinate per code, BT): instead of
// the per-query table, a query-independent table maps a code byte (two
// codes) to its two codebook levels as an fp16 pair, one copy per lane
// (entry (byte, lane) at byte 256 * byte + 4 * lane: the 32 lanes of a read
// always hit 32 distinct banks).  The levels are exact in fp16; each byte
// then costs one table read, two conversions and one paired fp32 FMA with
// the query pair (q[2j], q[2j + 1]) -- half the shared-memory traffic of a
// 4-byte table entry per code.
constexpr int kByteTableBytes = 256 * 256;

template <int CH, bool B3, bool BT = false>
__global__ void __launch_bounds__(256) scan_kernel(const __grid_constant__ ScanArgs a) {
  extern __shared__ __align__(16) uint8_t ssm_all[];
  __shared__ int scratch[32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, W = blockDim.x >> 5;
  if constexpr (BT) {
    // the byte table, once per CTA: low half = level of the low nibble
    // (the even code position), high half = level of the high nibble
    uint32_t* tb = reinterpret_cast<uint32_t*>(ssm_all);
    for (int e = tid; e < 256 * 32; e += blockDim.x) {
      const int byte = e >> 5, ln = e & 31;
      const uint32_t lo = __half_as_ushort(__float2half_rn(a.cb[byte & 15]));
      const uint32_t hi = __half_as_ushort(__float2half_rn(a.cb[byte >> 4]));
      tb[byte * 64 + ln] = lo | (hi << 16);
    }
  }
  uint8_t* ssm = ssm_all + a.bt_bytes;
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
  if constexpr (BT) {
    // the query itself, zero beyond Dp, one float per code position
    for (int e = tid; e < a.lut_groups; e += blockDim.x) lut[e] = e < a.Dp ? qr[e] : 0.0f;
  }
  if constexpr (B3) {
    // Rslm3: T[position][code] at lut[8 position + code]
    for (int e = tid; e < a.lut_groups * 8; e += blockDim.x) {
      const int pos = e >> 3;
      lut[e] = pos < a.ngroups ? qr[pos] * a.cb[e & 7] : 0.0f;
    }
  }
  for (int e = tid; !B3 && !BT && e < a.lut_groups * 16; e += blockDim.x) {
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
    if constexpr (BT) {
      // fp32 pairs (even positions, odd positions) per row
      uint64_t acc2[4] = {0ull, 0ull, 0ull, 0ull};
      const uint32_t lane4 = uint32_t(lane) * 4u;
#pragma unroll 1
      for (int c = 0; c < nch; ++c) {
        uint32_t w[4][4];
#pragma unroll
        for (int r = 0; r < 4; ++r) load_chunk<16>(tp + (size_t(c) * kTile + r * 32 + lane) * 16, w[r]);
        // the 32 query values of this chunk's positions, as 16 (even, odd) pairs
        const ulonglong2* qc = reinterpret_cast<const ulonglong2*>(lut + 32 * c);
        uint64_t qp[16];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const ulonglong2 v = qc[i];
          qp[2 * i] = v.x;
          qp[2 * i + 1] = v.y;
        }
#pragma unroll
        for (int v = 0; v < 4; ++v)
#pragma unroll
          for (int k = 0; k < 4; ++k)
#pragma unroll
            for (int r = 0; r < 4; ++r) {
              // entry (byte k of word v, lane): byte 0 = 4 lane, byte 1 = the code byte
              const uint32_t off = __byte_perm(w[r][v], lane4, 0x5504u + 0x10u * k);
              const uint32_t h2 = *reinterpret_cast<const uint32_t*>(ssm_all + off);
              const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&h2));
              acc2[r] = fma2(f2pack(f.x, f.y), qp[4 * v + k], acc2[r]);
            }
      }
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        float e, o;
        f2unpack(acc2[r], e, o);
        acc[r] = e + o;
      }
    }
    for (int c = 0; !B3 && !BT && c < nch; ++c) {
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

template <int CH, bool B3, bool BT = false>
cudaError_t launch_scan_ch(const rslm_index* ix, const ScanArgs& a, int64_t nq, size_t smem,
                           cudaStream_t s) {
  // listed queries: a fixed grid strides over the list, whose length is on the device
  const int64_t grid = a.qlist ? (nq < 2 * 152 ? nq : 2 * 152) : nq;
  cudaError_t e = cudaFuncSetAttribute(scan_kernel<CH, B3, BT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       int(smem));
  if (e != cudaSuccess) return e;
  cudaEvent_t stop =
      a.only_if == nullptr && a.qlist == nullptr && a.nprobe > 1 ? prof_start(ix, s, "scan_kernel") : nullptr;
  scan_kernel<CH, B3, BT><<<unsigned(grid), 256, smem, s>>>(a);
  prof_stop(stop, s);
  return cudaGetLastError();
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
  // byte-table form for 4-bit codes of one coordinate in 16-byte chunks
  const bool bt = !b3 && ix->cs1.g == 1 && ix->cs1.lite_h == 0 && ix->cs1.chunk == 16;
  const size_t lut_bytes = size_t(a.lut_groups) * (bt ? 1 : b3 ? 8 : 16) * 4;
  const size_t merge_bytes = ((size_t(np2) * 4 + 15) & ~size_t(15)) + size_t(np2) * 8;
  size_t region = lut_bytes > merge_bytes ? lut_bytes : merge_bytes;
  region = (region + 15) & ~size_t(15);
  a.lut_region = int(region);
  a.bt_bytes = bt ? kByteTableBytes : 0;
  const size_t smem =
      size_t(a.bt_bytes) + 256 + region + size_t(W) * k * 8 + size_t(W) * 4 + size_t(2 * nprobe + 1) * 4;
  if (b3) return launch_scan_ch<4, true>(ix, a, nq, smem, s);
  if (bt) return launch_scan_ch<16, false, true>(ix, a, nq, smem, s);
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
