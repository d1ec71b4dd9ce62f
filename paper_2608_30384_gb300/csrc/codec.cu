// codec.cu -- query rotation, residual encoding, code export / import.
//
// Encoding (Sec. 3.4 applied to the residual of Sec. 3.5) runs one warp per
// row with the row staged in shared memory in float64, so that codes and
// scale codes reproduce the exact definition except where a coordinate sits
// within rounding distance of a decision threshold.  Query rotation (once per
// query, Sec. 5.4) runs in float32.
#include <cuda_runtime.h>

#include "device_common.cuh"
#include "launch.h"

namespace rslm {
namespace {

struct RotateArgs {
  RotSpec rot;
  const float* in;   // [n * D]
  float* out;        // [n * Dp]
  int64_t n;
  int Dp;
  int buflen;
};

__global__ void rotate_rows_kernel(const __grid_constant__ RotateArgs a) {
  extern __shared__ float rsm[];
  __shared__ RotTables tb;
  load_rot_tables(&tb, a.rot);
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, W = blockDim.x >> 5;
  float* x = rsm + size_t(warp) * 2 * a.buflen;
  float* tmp = x + a.buflen;
  const int D = a.rot.D;
  for (int64_t r = int64_t(blockIdx.x) * W + warp; r < a.n; r += int64_t(gridDim.x) * W) {
    const float* src = a.in + r * D;
    for (int d = lane; d < D; d += 32) x[d] = src[d];
    __syncwarp();
    warp_rotate(x, tmp, a.rot, tb, false, lane);
    float* dst = a.out + r * a.Dp;
    for (int d = lane; d < a.Dp; d += 32) dst[d] = d < D ? x[d] : 0.0f;
    __syncwarp();
  }
}

struct EncodeArgs {
  RotSpec rot1, rot2;
  CodecSpec cs1, cs2;
  const float* x;          // [rows * D] rows row_begin ..
  int64_t row_begin, rows;
  const float* centroids;  // [nlist * D]
  const int32_t* assign;   // [n_rows]
  const int32_t* slot_of_row;
  uint8_t* codes1;         // tile-interleaved
  uint32_t* scales1;
  uint8_t* codes2;         // row-major
  uint32_t* scales2;
  int64_t* ids;
  int D;
  int global_scale;
  int stage2;
  int full_vector;  // approximation 0 instead of the centroid (Sec. 3.5)
  int reading_a;    // stage 2 against the stage-1 approximation, not its reconstruction
  int buflen;
};

struct CodecTables {
  double cb[64];
  double thr[15];
  double cb8[8];  // Rslm4Lite head (K = 8)
  double thr8[7];
};

// Nearest codeword of the group starting at u (Sec. 3.2): 1-D by the count
// of thresholds <= u (a value on a threshold goes up); multi-D by the
// smallest squared distance, accumulated in coordinate order, lowest index on
// ties.
__device__ __forceinline__ int nearest_code(const double* u, const CodecSpec& cs,
                                            const CodecTables& t) {
  if (cs.g == 1) {
    int c = 0;
    for (int i = 0; i < cs.K - 1; ++i) c += (u[0] >= t.thr[i]);
    return c;
  }
  int best = 0;
  double bd = 0.0;
  for (int k = 0; k < cs.K; ++k) {
    double d = (u[0] - t.cb[k * cs.g]) * (u[0] - t.cb[k * cs.g]);
    for (int j = 1; j < cs.g; ++j) d = d + (u[j] - t.cb[k * cs.g + j]) * (u[j] - t.cb[k * cs.g + j]);
    if (k == 0 || d < bd) {
      bd = d;
      best = k;
    }
  }
  return best;
}

// One quantization stage on the residual held in A[0, D) (Sec. 3.2, 3.3):
// rotate, EVT-normalise, nearest codeword per group, local scale.  Writes the
// code bytes through `put(byte_index, value)`.  On return A holds the chosen
// codewords uhat on [0, D) (zero beyond) and the UE7M9 code of L is returned.
template <typename Put>
__device__ uint32_t quantize_stage(double* A, double* tmp, const RotSpec& rs, const RotTables& tb,
                                   const CodecSpec& cs, const CodecTables& ct, double nr2, int lane,
                                   Put put, double* Lhat) {
  const int D = rs.D;
  warp_rotate(A, tmp, rs, tb, false, lane);
  double m = 0.0;
  for (int d = lane; d < D; d += 32) m = fmax(m, fabs(A[d]));
  m = warp_max(m);
  const double f = m > 0.0 ? cs.emax / m : 0.0;
  for (int d = lane; d < cs.Dp; d += 32) A[d] = d < D ? A[d] * f : 0.0;
  __syncwarp();
  if (cs.bits == 3) {
    // Rslm3 (g = 1, K = 8): eight codes per 3 bytes, code i at stream bits 3i ..
    for (int o = lane; o * 8 < cs.ngroups; o += 32) {
      uint32_t v = 0;
      for (int i = 0; i < 8; ++i) {
        const int gi = 8 * o + i;
        if (gi < cs.ngroups) {
          const int c = nearest_code(A + gi, cs, ct);
          v |= uint32_t(c) << (3 * i);
          A[gi] = ct.cb[c];
        }
      }
      for (int t = 0; t < 3; ++t)
        if (3 * o + t < cs.code_bytes) put(3 * o + t, (v >> (8 * t)) & 255u);
    }
  }
  for (int b = lane; cs.bits != 3 && b < cs.code_bytes; b += 32) {
    const int g0 = 2 * b, g1 = 2 * b + 1;
    if (g0 < cs.lite_h) {
      // Rslm4Lite head (g = 1, lite_h even): the K = 8 levels; the top bits
      // stay clear for the scale codes
      int c0 = 0, c1 = 0;
      for (int i = 0; i < 7; ++i) {
        c0 += (A[g0] >= ct.thr8[i]);
        c1 += (A[g1] >= ct.thr8[i]);
      }
      put(b, uint32_t(c0 | (c1 << 4)));
      A[g0] = ct.cb8[c0];
      A[g1] = ct.cb8[c1];
      continue;
    }
    const int c0 = nearest_code(A + g0 * cs.g, cs, ct);
    const int c1 = g1 < cs.ngroups ? nearest_code(A + g1 * cs.g, cs, ct) : 0;
    put(b, uint32_t(c0 | (c1 << 4)));
    for (int j = 0; j < cs.g; ++j) {
      A[g0 * cs.g + j] = ct.cb[c0 * cs.g + j];
      if (g1 < cs.ngroups) A[g1 * cs.g + j] = ct.cb[c1 * cs.g + j];
    }
  }
  __syncwarp();
  double nu2 = 0.0;
  for (int d = lane; d < cs.Dp; d += 32) {
    if (d >= D) A[d] = 0.0;
    else nu2 += A[d] * A[d];
  }
  nu2 = warp_sum(nu2);
  __syncwarp();
  const double L = nu2 > 0.0 ? sqrt(nr2) / sqrt(nu2) : 0.0;
  const uint32_t Lu = ue_encode(L, 7, 9);
  *Lhat = ue_decode(Lu, 7, 9);
  return Lu;
}

__global__ void encode_kernel(const __grid_constant__ EncodeArgs a) {
  extern __shared__ double esm[];
  __shared__ RotTables tb1, tb2;
  __shared__ CodecTables ct1, ct2;
  load_rot_tables(&tb1, a.rot1);
  load_rot_tables(&tb2, a.rot2);
  for (int i = threadIdx.x; i < 64; i += blockDim.x) {
    ct1.cb[i] = a.cs1.cbd[i];
    ct2.cb[i] = a.cs2.cbd[i];
  }
  for (int i = threadIdx.x; i < 15; i += blockDim.x) {
    ct1.thr[i] = a.cs1.thr[i];
    ct2.thr[i] = a.cs2.thr[i];
  }
  for (int i = threadIdx.x; i < 8; i += blockDim.x) {
    ct1.cb8[i] = a.cs1.cb8d[i];
    if (i < 7) ct1.thr8[i] = a.cs1.thr8[i];
  }
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, W = blockDim.x >> 5;
  double* A = esm + size_t(warp) * 3 * a.buflen;
  double* T = A + a.buflen;
  double* Ap = T + a.buflen;  // stage-2 approximation a2
  const int D = a.D;
  const uint32_t one_ue4m12 = 7u << 12;

  for (int64_t i = int64_t(blockIdx.x) * W + warp; i < a.rows; i += int64_t(gridDim.x) * W) {
    const int64_t gid = a.row_begin + i;
    const int p = a.assign[gid];
    const int64_t slot = a.slot_of_row[gid];
    const float* x = a.x + i * D;
    // the stage-1 approximation: the centroid, or 0 for full-vector codes
    const float* c = a.centroids + int64_t(p) * D;
    const double cw = a.full_vector ? 0.0 : 1.0;

    // ---- stage 1: residual against the centroid (Sec. 3.5, Sec. 5.5.1)
    double nr2 = 0.0, nx2 = 0.0;
    for (int d = lane; d < D; d += 32) {
      const double xv = x[d], cv = cw * c[d];
      const double r = xv - cv;
      A[d] = r;
      nr2 += r * r;
      nx2 += xv * xv;
    }
    nr2 = warp_sum(nr2);
    nx2 = warp_sum(nx2);
    __syncwarp();
    uint8_t* tile = a.codes1 + (slot >> 7) * kTile * a.cs1.stride;
    const int rin = int(slot & 127);
    const int ch = a.cs1.chunk;
    double Lh1;
    const uint32_t Lu1 = quantize_stage(
        A, T, a.rot1, tb1, a.cs1, ct1, nr2, lane,
        [&](int b, uint32_t v) { tile[((b / ch) * kTile + rin) * ch + (b % ch)] = uint8_t(v); }, &Lh1);
    uint32_t Gu1 = one_ue4m12;
    double Gh1 = 1.0;
    if (a.global_scale || (a.stage2 && !a.reading_a)) {
      warp_rotate(A, T, a.rot1, tb1, true, lane);  // A = R^T uhat
    }
    if (a.global_scale) {
      // Sec. 3.5.2: G = ||x|| / ||c + Lhat R^T uhat||
      double na2 = 0.0;
      for (int d = lane; d < D; d += 32) {
        const double v = cw * double(c[d]) + Lh1 * A[d];
        na2 += v * v;
      }
      na2 = warp_sum(na2);
      const double G = na2 > 0.0 ? sqrt(nx2) / sqrt(na2) : 0.0;
      Gu1 = ue_encode(G, 4, 12);
      Gh1 = ue_decode(Gu1, 4, 12);
    }
    if (a.cs1.lite_h) {
      // Rslm4Lite: bit i of the UE7M9 code into the top bit of code i, and
      // of the UE4M12 code into that of code 16 + i (lite_h = 32); code j
      // is the low (even j) or high (odd j) nibble of byte j / 2
      __syncwarp();
      if (lane < a.cs1.lite_h / 2) {
        const int b = lane;
        uint8_t* pb = tile + ((b / ch) * kTile + rin) * ch + (b % ch);
        auto bit = [&](int j) { return j < 16 ? (Lu1 >> j) & 1u : (Gu1 >> (j - 16)) & 1u; };
        *pb = uint8_t(*pb | (bit(2 * b) << 3) | (bit(2 * b + 1) << 7));
      }
    }
    if (lane == 0) {
      a.scales1[slot] = Lu1 | (Gu1 << 16);
      a.ids[slot] = gid;
    }
    if (!a.stage2) continue;

    // ---- stage 2: residual against the full stage-1 reconstruction (Sec.
    // 5.2), or against the stage-1 approximation itself (reading A)
    double nr2b = 0.0;
    for (int d = lane; d < D; d += 32) {
      const double ap = a.reading_a ? cw * double(c[d]) : Gh1 * (cw * double(c[d]) + Lh1 * A[d]);
      Ap[d] = ap;
      const double r = double(x[d]) - ap;
      A[d] = r;
      nr2b += r * r;
    }
    nr2b = warp_sum(nr2b);
    __syncwarp();
    uint8_t* row2 = a.codes2 + slot * a.cs2.stride;
    double Lh2;
    const uint32_t Lu2 = quantize_stage(
        A, T, a.rot2, tb2, a.cs2, ct2, nr2b, lane, [&](int b, uint32_t v) { row2[b] = uint8_t(v); },
        &Lh2);
    uint32_t Gu2 = one_ue4m12;
    if (a.global_scale) {
      warp_rotate(A, T, a.rot2, tb2, true, lane);
      double na2 = 0.0;
      for (int d = lane; d < D; d += 32) {
        const double v = Ap[d] + Lh2 * A[d];
        na2 += v * v;
      }
      na2 = warp_sum(na2);
      const double G = na2 > 0.0 ? sqrt(nx2) / sqrt(na2) : 0.0;
      Gu2 = ue_encode(G, 4, 12);
    }
    if (lane == 0) a.scales2[slot] = Lu2 | (Gu2 << 16);
    __syncwarp();
  }
}

// Decompression (Sec. 4, the inverse of the codec): the reconstruction
// Ghat (a + Lhat R^T uhat) of each row from its stored codes and scales, in
// float64 like the encoder, written as float32.  Stage 1: a = the centroid
// (0 for full-vector codes).  Stage 2: a = the stage-1 reconstruction
// (reading B) or the stage-1 approximation (reading A).  One warp per row.
struct DecompArgs {
  RotSpec rot1, rot2;
  CodecSpec cs1, cs2;
  int64_t row_begin, rows;
  const float* centroids;
  const int32_t* assign;
  const int32_t* slot_of_row;
  const uint8_t* codes1;  // tile-interleaved
  const uint32_t* scales1;
  const uint8_t* codes2;  // row-major
  const uint32_t* scales2;
  int D, which, full_vector, reading_a, buflen;
  float* out;             // [rows * D]
};

// Codewords of a stored row into u[0, Dp) (zero beyond D); `byte(b)` reads
// code byte b.
template <typename Byte>
__device__ __forceinline__ void decode_codewords(double* u, const CodecSpec& cs, int D, int lane, Byte byte) {
  for (int g = lane; g < cs.ngroups; g += 32) {
    uint32_t code;
    if (cs.bits == 3) {  // Rslm3: bits 3g .. 3g + 2 of the byte stream
      const int bit = 3 * g, b0 = bit >> 3;
      const uint32_t two = uint32_t(byte(b0)) | (b0 + 1 < cs.code_bytes ? uint32_t(byte(b0 + 1)) << 8 : 0u);
      code = (two >> (bit & 7)) & 7u;
    } else {
      code = (uint32_t(byte(g >> 1)) >> (4 * (g & 1))) & 15u;
    }
    if (g < cs.lite_h) {
      u[g] = cs.cb8d[code & 7u];  // Rslm4Lite head: the top bit is a scale bit
    } else {
      for (int j = 0; j < cs.g; ++j) {
        const int d = g * cs.g + j;
        u[d] = d < D ? cs.cbd[code * cs.g + j] : 0.0;
      }
    }
  }
}

__global__ void decompress_kernel(const __grid_constant__ DecompArgs a) {
  extern __shared__ double dsm[];
  __shared__ RotTables tb1, tb2;
  load_rot_tables(&tb1, a.rot1);
  load_rot_tables(&tb2, a.rot2);
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, W = blockDim.x >> 5;
  double* U = dsm + size_t(warp) * 3 * a.buflen;
  double* T = U + a.buflen;
  double* R1 = T + a.buflen;  // stage-1 reconstruction
  const int D = a.D;
  const double cw = a.full_vector ? 0.0 : 1.0;
  for (int64_t i = int64_t(blockIdx.x) * W + warp; i < a.rows; i += int64_t(gridDim.x) * W) {
    const int64_t gid = a.row_begin + i;
    const int64_t slot = a.slot_of_row[gid];
    const float* c = a.centroids + int64_t(a.assign[gid]) * D;
    const uint8_t* tile = a.codes1 + (slot >> 7) * kTile * a.cs1.stride;
    const int rin = int(slot & 127), ch = a.cs1.chunk;
    decode_codewords(U, a.cs1, D, lane,
                     [&](int b) { return tile[((b / ch) * kTile + rin) * ch + (b % ch)]; });
    __syncwarp();
    warp_rotate(U, T, a.rot1, tb1, true, lane);  // R^T uhat
    const uint32_t sc1 = a.scales1[slot];
    const double Lh1 = ue_decode(sc1 & 0xffffu, 7, 9), Gh1 = ue_decode(sc1 >> 16, 4, 12);
    for (int d = lane; d < D; d += 32) R1[d] = Gh1 * (cw * double(c[d]) + Lh1 * U[d]);
    __syncwarp();
    if (a.which == 1) {
      for (int d = lane; d < D; d += 32) a.out[i * D + d] = float(R1[d]);
      __syncwarp();
      continue;
    }
    const uint8_t* row2 = a.codes2 + slot * a.cs2.stride;
    decode_codewords(U, a.cs2, D, lane, [&](int b) { return row2[b]; });
    __syncwarp();
    warp_rotate(U, T, a.rot2, tb2, true, lane);
    const uint32_t sc2 = a.scales2[slot];
    const double Lh2 = ue_decode(sc2 & 0xffffu, 7, 9), Gh2 = ue_decode(sc2 >> 16, 4, 12);
    for (int d = lane; d < D; d += 32) {
      const double a2 = a.reading_a ? cw * double(c[d]) : R1[d];
      a.out[i * D + d] = float(Gh2 * (a2 + Lh2 * U[d]));
    }
    __syncwarp();
  }
}

struct ExportArgs {
  const int32_t* slot_of_row;
  int64_t row_begin, rows;
  uint8_t* layout;      // device layout of the codes
  uint32_t* scales;
  int code_bytes, stride, chunk;  // chunk 0: row-major layout
  uint8_t* codes;       // canonical [rows * code_bytes]
  uint16_t* lscale;
  uint16_t* gscale;
  int64_t* ids;         // import: slot -> row id
  int import;
};

__global__ void export_import_kernel(const __grid_constant__ ExportArgs a) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, W = blockDim.x >> 5;
  for (int64_t i = int64_t(blockIdx.x) * W + warp; i < a.rows; i += int64_t(gridDim.x) * W) {
    const int64_t gid = a.row_begin + i;
    const int64_t slot = a.slot_of_row[gid];
    for (int b = lane; b < a.code_bytes; b += 32) {
      uint8_t* p;
      if (a.chunk) {
        p = a.layout + (slot >> 7) * kTile * a.stride +
            ((b / a.chunk) * kTile + (slot & 127)) * a.chunk + (b % a.chunk);
      } else {
        p = a.layout + slot * a.stride + b;
      }
      if (a.import) *p = a.codes[i * a.code_bytes + b];
      else a.codes[i * a.code_bytes + b] = *p;
    }
    if (lane == 0) {
      if (a.import) {
        a.scales[slot] = uint32_t(a.lscale[i]) | (uint32_t(a.gscale[i]) << 16);
        if (a.ids) a.ids[slot] = gid;
      } else {
        a.lscale[i] = uint16_t(a.scales[slot] & 0xffffu);
        a.gscale[i] = uint16_t(a.scales[slot] >> 16);
      }
    }
  }
}

int grid_for(int64_t items, int per_block, int max_blocks) {
  int64_t g = (items + per_block - 1) / per_block;
  if (g < 1) g = 1;
  if (g > max_blocks) g = max_blocks;
  return int(g);
}

}  // namespace

cudaError_t launch_rotate_rows(const RotSpec& rot, const float* in, int64_t n, float* out, int Dp,
                               cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  RotateArgs a;
  a.rot = rot;
  a.in = in;
  a.out = out;
  a.n = n;
  a.Dp = Dp;
  a.buflen = (rot.D + 3) / 4 * 4;
  const int warps = 8;
  const size_t smem = size_t(warps) * 2 * a.buflen * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(rotate_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       int(smem));
  if (e != cudaSuccess) return e;
  rotate_rows_kernel<<<grid_for(n, warps, 152 * 32), warps * 32, smem, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_encode(const rslm_index* ix, const float* x, int64_t row_begin, int64_t rows,
                          cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  EncodeArgs a;
  a.rot1 = ix->rot1;
  a.rot2 = ix->rescore_bits ? ix->rot2 : ix->rot1;
  a.cs1 = ix->cs1;
  a.cs2 = ix->rescore_bits ? ix->cs2 : ix->cs1;
  a.x = x;
  a.row_begin = row_begin;
  a.rows = rows;
  a.centroids = ix->centroids;
  a.assign = ix->assign;
  a.slot_of_row = ix->slot_of_row;
  a.codes1 = ix->codes1;
  a.scales1 = ix->scales1;
  a.codes2 = ix->codes2;
  a.scales2 = ix->scales2;
  a.ids = ix->ids;
  a.D = ix->D;
  a.global_scale = (ix->flags & RSLM_GLOBAL_SCALE) ? 1 : 0;
  a.stage2 = ix->rescore_bits ? 1 : 0;
  a.full_vector = (ix->flags & RSLM_FULL_VECTOR) ? 1 : 0;
  a.reading_a = (ix->flags & RSLM_RESCORE_READING_A) ? 1 : 0;
  int len = ix->D;
  if (ix->cs1.Dp > len) len = ix->cs1.Dp;
  if (ix->rescore_bits && ix->cs2.Dp > len) len = ix->cs2.Dp;
  a.buflen = (len + 3) / 4 * 4;
  const size_t per_warp = size_t(3) * a.buflen * sizeof(double);
  int warps = int((96 * 1024) / per_warp);
  if (warps > 8) warps = 8;
  if (warps < 1) warps = 1;
  const size_t smem = per_warp * warps;
  cudaError_t e =
      cudaFuncSetAttribute(encode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  encode_kernel<<<grid_for(rows, warps, 152 * 16), warps * 32, smem, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_decompress(const rslm_index* ix, int which, int64_t row_begin, int64_t rows, float* out,
                              cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  DecompArgs a;
  a.rot1 = ix->rot1;
  a.rot2 = ix->rescore_bits ? ix->rot2 : ix->rot1;
  a.cs1 = ix->cs1;
  a.cs2 = ix->rescore_bits ? ix->cs2 : ix->cs1;
  a.row_begin = row_begin;
  a.rows = rows;
  a.centroids = ix->centroids;
  a.assign = ix->assign;
  a.slot_of_row = ix->slot_of_row;
  a.codes1 = ix->codes1;
  a.scales1 = ix->scales1;
  a.codes2 = ix->codes2;
  a.scales2 = ix->scales2;
  a.D = ix->D;
  a.which = which;
  a.full_vector = (ix->flags & RSLM_FULL_VECTOR) ? 1 : 0;
  a.reading_a = (ix->flags & RSLM_RESCORE_READING_A) ? 1 : 0;
  a.out = out;
  int len = ix->D;
  if (ix->cs1.Dp > len) len = ix->cs1.Dp;
  if (ix->rescore_bits && ix->cs2.Dp > len) len = ix->cs2.Dp;
  a.buflen = (len + 3) / 4 * 4;
  const size_t per_warp = size_t(3) * a.buflen * sizeof(double);
  int warps = int((96 * 1024) / per_warp);
  if (warps > 8) warps = 8;
  if (warps < 1) warps = 1;
  const size_t smem = per_warp * warps;
  cudaError_t e =
      cudaFuncSetAttribute(decompress_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  decompress_kernel<<<grid_for(rows, warps, 152 * 16), warps * 32, smem, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_export_import(const rslm_index* ix, int which, int64_t row_begin, int64_t rows,
                                 uint8_t* codes, uint16_t* lscale, uint16_t* gscale, bool import,
                                 cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  ExportArgs a;
  const CodecSpec& cs = which == 1 ? ix->cs1 : ix->cs2;
  a.slot_of_row = ix->slot_of_row;
  a.row_begin = row_begin;
  a.rows = rows;
  a.layout = which == 1 ? ix->codes1 : ix->codes2;
  a.scales = which == 1 ? ix->scales1 : ix->scales2;
  a.code_bytes = cs.code_bytes;
  a.stride = cs.stride;
  a.chunk = which == 1 ? cs.chunk : 0;
  a.codes = codes;
  a.lscale = lscale;
  a.gscale = gscale;
  a.ids = (import && which == 1) ? ix->ids : nullptr;
  a.import = import ? 1 : 0;
  export_import_kernel<<<grid_for(rows, 8, 152 * 16), 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace rslm
