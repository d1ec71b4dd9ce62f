// device_common.cuh -- device helpers shared by the librslm kernels.
#pragma once

#include <cuda_runtime.h>
#include <math_constants.h>
#include <stdint.h>

#include "rslm_internal.h"

namespace rslm {

constexpr unsigned kFull = 0xffffffffu;

template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

__device__ __forceinline__ double warp_max(double v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmax(v, __shfl_xor_sync(kFull, v, o));
  return v;
}

// Rotation tables staged in shared memory (Sec. 3.1.2).
struct RotTables {
  uint32_t s1[8];
  uint32_t s2[8];
  uint8_t perm[128];
};

__device__ __forceinline__ void load_rot_tables(RotTables* t, const RotSpec& rs) {
  for (int i = threadIdx.x; i < 8; i += blockDim.x) {
    t->s1[i] = rs.s1[i];
    t->s2[i] = rs.s2[i];
  }
  for (int i = threadIdx.x; i < 128; i += blockDim.x) t->perm[i] = rs.perm[i];
}

__device__ __forceinline__ bool sign_neg(const uint32_t* bits, int i) {
  const int j = i & 255;
  return (bits[j >> 5] >> (j & 31)) & 1u;
}

// Orthonormal FWHT H_B = Hhat_B / sqrt(B) of one block (Sec. 3.1.1), in
// place, by one warp: log2(B) butterfly stages, then the 1/sqrt(B) scale.
// In float (the query rotation), blocks of 32, 64 or 128 run in registers:
// lane l holds x[32 j + l] (j < B / 32); the stages of span h < 32 pair
// lanes l and l ^ h (warp shuffles), the spans 32 and 64 pair the lane's own
// values j and j ^ h / 32.  The stages are Kronecker factors of Hhat_B and
// commute, so their order is free.  Smaller blocks, and float64 (the
// encoder, where a shuffle moves two 32-bit halves and measured slower), go
// through shared memory stage by stage.
template <typename T>
__device__ __forceinline__ void warp_fwht(T* x, int B, int logB, T scale, int lane) {
  if (sizeof(T) == 4 && B >= 32) {
    const int J = B >> 5;
    T v[4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (j < J) v[j] = x[32 * j + lane];
#pragma unroll
    for (int h = 1; h < 32; h <<= 1) {
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (j < J) {
          const T o = __shfl_xor_sync(kFull, v[j], h);
          v[j] = (lane & h) ? o - v[j] : v[j] + o;
        }
    }
#pragma unroll
    for (int hj = 1; hj < 4; hj <<= 1)
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (j < J && hj < J && !(j & hj)) {
          const T a = v[j], b = v[j | hj];
          v[j] = a + b;
          v[j | hj] = a - b;
        }
    __syncwarp();  // every lane has read its block values before any is overwritten
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (j < J) x[32 * j + lane] = v[j] * scale;
    __syncwarp();
    return;
  }
  for (int s = 0; s < logB; ++s) {
    const int h = 1 << s;
    for (int t = lane; t < (B >> 1); t += 32) {
      const int i = ((t >> s) << (s + 1)) | (t & (h - 1));
      const T a = x[i], b = x[i + h];
      x[i] = a + b;
      x[i + h] = a - b;
    }
    __syncwarp();
  }
  for (int t = lane; t < B; t += 32) x[t] *= scale;
  __syncwarp();
}

template <typename T>
__device__ __forceinline__ void warp_signs(T* x, int D, const uint32_t* bits, int lane) {
  for (int i = lane; i < D; i += 32)
    if (sign_neg(bits, i)) x[i] = -x[i];
  __syncwarp();
}

// Block-wise FWHT of a whole vector: full blocks, then the overlapping last
// block [D - B, D) (Sec. 3.1.1); `reverse` applies them in the opposite
// order (the inverse, since every block transform is an involution).
template <typename T>
__device__ __forceinline__ void warp_blocks(T* x, const RotSpec& rs, bool reverse, int lane) {
  const T sc = T(rs.inv_sqrt_B);
  if (!reverse) {
    for (int m = 0; m < rs.M; ++m) warp_fwht(x + m * rs.B, rs.B, rs.logB, sc, lane);
    if (rs.overlap >= 0) warp_fwht(x + rs.overlap, rs.B, rs.logB, sc, lane);
  } else {
    if (rs.overlap >= 0) warp_fwht(x + rs.overlap, rs.B, rs.logB, sc, lane);
    for (int m = rs.M - 1; m >= 0; --m) warp_fwht(x + m * rs.B, rs.B, rs.logB, sc, lane);
  }
}

// Rotation R of Sec. 3.1.3 (or its inverse R^T) of the vector x[0, D) held
// in shared memory, by one warp.  tmp: shared scratch of D elements.
// Two-pass: S1, FWHT, x'[k M + b] = x[b B + P(k)], S2, FWHT.
template <typename T>
__device__ void warp_rotate(T* x, T* tmp, const RotSpec& rs, const RotTables& tb, bool inverse,
                            int lane) {
  const int D = rs.D, M = rs.M, MB = rs.M * rs.B;
  if (!inverse) {
    warp_signs(x, D, tb.s1, lane);
    warp_blocks(x, rs, false, lane);
    if (rs.two_pass) {
      for (int i = lane; i < MB; i += 32) {
        const int k = i / M, b = i - k * M;
        tmp[i] = x[b * rs.B + tb.perm[k]];
      }
      __syncwarp();
      for (int i = lane; i < MB; i += 32) x[i] = tmp[i];
      __syncwarp();
      warp_signs(x, D, tb.s2, lane);
      warp_blocks(x, rs, false, lane);
    }
  } else {
    if (rs.two_pass) {
      warp_blocks(x, rs, true, lane);
      warp_signs(x, D, tb.s2, lane);
      for (int i = lane; i < MB; i += 32) {
        const int k = i / M, b = i - k * M;
        tmp[b * rs.B + tb.perm[k]] = x[i];
      }
      __syncwarp();
      for (int i = lane; i < MB; i += 32) x[i] = tmp[i];
      __syncwarp();
    }
    warp_blocks(x, rs, true, lane);
    warp_signs(x, D, tb.s1, lane);
  }
}

// Unsigned float scale codes (Sec. 3.3.1 UE7M9, Sec. 3.5.2 UE4M12): code 0
// (exponent field 0) is 0, otherwise 2^(e - bias) (1 + m / 2^mbits); round
// to nearest even; flush below the smallest normal; saturate above the max.
__device__ __forceinline__ uint32_t ue_encode(double v, int ebits, int mbits) {
  if (!(v > 0.0)) return 0;
  int k;
  const double f = frexp(v, &k);
  int e = k - 1;
  uint32_t m = uint32_t(rint((2.0 * f - 1.0) * double(1 << mbits)));
  if (m == (1u << mbits)) {
    m = 0;
    e += 1;
  }
  const int be = e + (1 << (ebits - 1)) - 1;
  if (be <= 0) return 0;
  if (be > (1 << ebits) - 1) return (((1u << ebits) - 1) << mbits) | ((1u << mbits) - 1);
  return (uint32_t(be) << mbits) | m;
}

__device__ __forceinline__ double ue_decode(uint32_t u, int ebits, int mbits) {
  const int e = int(u >> mbits);
  if (e == 0) return 0.0;
  const double m = double(u & ((1u << mbits) - 1)) / double(1 << mbits);
  return ldexp(1.0 + m, e - ((1 << (ebits - 1)) - 1));
}

// Binary32 from the 16-bit codes by rebiasing the exponent: UE7M9 bias 63 ->
// 127 adds 64 to the exponent field; UE4M12 bias 7 -> 127 adds 120.
__device__ __forceinline__ float ue7m9_to_f32(uint32_t u) {
  return (u >> 9) ? __uint_as_float((u << 14) + (64u << 23)) : 0.0f;
}
__device__ __forceinline__ float ue4m12_to_f32(uint32_t u) {
  return (u >> 12) ? __uint_as_float((u << 11) + (120u << 23)) : 0.0f;
}

// Order "a before b": larger key first, then smaller id.
template <typename K, typename I>
__device__ __forceinline__ bool better(K ka, I ia, K kb, I ib) {
  return ka > kb || (ka == kb && ia < ib);
}

// Bitonic sort of n (a power of two) pairs in shared memory into "better
// first" order.  Called by every thread of the block.
template <typename K, typename I>
__device__ void block_bitonic_sort(K* key, I* id, int n) {
  for (int size = 2; size <= n; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      __syncthreads();
      for (int i = threadIdx.x; i < (n >> 1); i += blockDim.x) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool asc = (lo & size) == 0;
        const K klo = key[lo], khi = key[hi];
        const I ilo = id[lo], ihi = id[hi];
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
  __syncthreads();
}

// Exclusive prefix sum of v over the block; *total receives the sum.
// scratch: shared int[32].  Called by every thread of the block.
__device__ __forceinline__ int block_exclusive_scan(int v, int* scratch, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFull, x, o);
    if (lane >= o) x += y;
  }
  __syncthreads();
  if (lane == 31) scratch[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nw ? scratch[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, w, o);
      if (lane >= o) w += y;
    }
    scratch[lane] = w;
  }
  __syncthreads();
  const int before = (warp ? scratch[warp - 1] : 0) + x - v;
  *total = scratch[nw - 1];
  __syncthreads();
  return before;
}

__device__ __forceinline__ uint32_t float_order_key(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float float_from_order_key(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// hist[bin] += 1 for this lane's bin when `active`; lanes of a warp with
// the same bin are combined into one shared-memory atomic (radix-select
// histograms are dominated by a few bins, which would serialise).
__device__ __forceinline__ void warp_hist_add(uint32_t* hist, uint32_t bin, bool active) {
  const unsigned act = __ballot_sync(kFull, active);
  if (!active) return;
  const unsigned peers = __match_any_sync(act, bin);
  if ((threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&hist[bin], uint32_t(__popc(peers)));
}

__device__ __forceinline__ void set_device_error(int* err, int code) {
  if (err) atomicCAS(err, 0, code);
}

}  // namespace rslm
