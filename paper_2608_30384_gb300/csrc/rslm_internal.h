// rslm_internal.h -- types shared by the host code and the kernels of librslm.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>
#include <string>
#include <utility>
#include <vector>

#include "rslm.h"

namespace rslm {

constexpr int kTile = 128;      // rows per layout tile (partitions start on tiles)
constexpr int kMaxDim = 4096;
constexpr int kMaxK = 256;
constexpr int kMaxNprobe = 4096;
constexpr int kBatchMinQueries = 16;  // rslm_search: batched scan above this queries/partition

// Event counters of an index (rslm_counters): queries that a search path
// handed to an exact fallback, and the hi-only finalize's exact rescores.
enum Counter : int {
  kCtrBatchedShort = 0,     // pass 2 kept fewer than k candidates under a finite threshold
  kCtrBatchedOverflow = 1,  // the pass-2 candidate buffer overflowed
  kCtrProbeExact = 2,       // a fused-probe candidate list overflowed
  kCtrHiExact = 3,          // rows whose exact score the hi-only finalize recomputed
  kNumCounters = 4,
};

// Device error codes written to the index's sticky flag.
enum DeviceError : int {
  kErrNone = 0,
  kErrBadProbe = 1,      // partition id out of range in a probe list
  kErrBadCandidate = 2,  // candidate id out of range in rescoring
  kErrBadAssignment = 3,
  kErrTimeout = 4,       // a bounded wait on the tensor-core pipeline gave up
  kErrSmemLayout = 5,    // a kernel's shared-memory layout did not fit its launch
};

// Block-wise cascaded FWHT rotation (Sec. 3.1.1-3.1.3).
struct RotSpec {
  int D;          // vector length
  int B;          // block size (128, or the largest power of two <= D)
  int logB;
  int M;          // floor(D / B) full blocks
  int overlap;    // start of the overlapping last block, or -1
  int two_pass;   // 1: S1, FWHT, permute+transpose, S2, FWHT; 0: S1, FWHT
  double inv_sqrt_B;
  uint32_t s1[8];  // bit i set: sign of coordinate i (mod 256) is -1
  uint32_t s2[8];
  uint8_t perm[128];  // in-block permutation P(k)
};

// A bit rate's codebook (Sec. 3.2) and EVT constant.
struct CodecSpec {
  int bits;
  int g;          // coordinates per code
  int K;          // codewords (16)
  int ngroups;    // ceil(D / g)
  int Dp;         // g * ngroups
  int code_bytes; // ceil(ngroups / 2) canonical bytes per row
  int stride;     // bytes per row in the device layout (>= code_bytes)
  int chunk;      // bytes per interleaved chunk (scoring layout): 16, 8 or 4
  double emax;    // E_max(D)
  float cbf[64];  // K x g codewords (binary16-exact)
  double cbd[64];
  double thr[15]; // 1-D decision thresholds (midpoints of adjacent levels)
  // Rslm4Lite (Sec. 3.4): the first lite_h coordinates (0, 16 or 32) take
  // the K=8 levels; the UE7M9 code sits in the top bits of codes 0-15 and,
  // with lite_h = 32, the UE4M12 code in those of codes 16-31
  int lite_h;
  double cb8d[8];
  float cb8f[8];
  double thr8[7];
};

// Host-side tables (tables.cpp).
void rotation_tables(int8_t s1[256], int32_t perm[128]);
RotSpec make_rot_spec(int D, int bits);
bool make_codec_spec(int bits, int D, bool interleaved, CodecSpec* out);
double e_max(int D);
uint32_t ue_encode_host(double v, int ebits, int mbits);

// Record the calling thread's rslm_last_error() message and return `st`.
rslm_status set_last_error(rslm_status st, const std::string& msg);

// Timing of the dominant scan kernel (rslm_profile_enable / rslm_profile_read):
// prof_start records a start event on `s` and returns the stop event to record
// after the launch (nullptr when profiling is off).
cudaEvent_t prof_start(const rslm_index* ix, cudaStream_t s, const char* kernel);
void prof_stop(cudaEvent_t stop, cudaStream_t s);

}  // namespace rslm

// Index state (host object; arrays are device pointers).
struct rslm_index {
  int device = 0;
  int D = 0, nlist = 0, bits = 0, rescore_bits = 0;
  uint32_t flags = 0;
  rslm::RotSpec rot1{}, rot2{};
  rslm::CodecSpec cs1{}, cs2{};
  float* centroids = nullptr;   // [nlist * D]
  int64_t n_rows = 0, n_slots = 0;
  int32_t max_part_n = 0;       // rows of the largest partition
  int64_t* part_off = nullptr;  // [nlist + 1] first slot of each partition
  int32_t* part_n = nullptr;    // [nlist] rows in each partition
  int32_t* assign = nullptr;    // [n_rows]
  int32_t* slot_of_row = nullptr;  // [n_rows]
  int64_t* ids = nullptr;       // [n_slots] row id of each slot, -1 for padding
  uint8_t* codes1 = nullptr;    // scoring codes, tile-interleaved
  uint32_t* scales1 = nullptr;  // [n_slots] UE7M9 | UE4M12 << 16
  uint8_t* codes2 = nullptr;    // rescoring codes, row-major by slot
  uint32_t* scales2 = nullptr;
  int* d_err = nullptr;         // sticky device error flag
  unsigned long long* d_counters = nullptr;  // [kNumCounters] event counters
  uint8_t* ctiles = nullptr;    // fused probe: centroids * 2^sC as fp16 operand tiles (D <= 128)
  float* cmeta = nullptr;       // fused probe: max|c|, max||c||^2, 2^sC, max||c|| 2^sC
  float* crows = nullptr;       // fused probe: centroids as fp32 rows of Kp floats
  float* crot2 = nullptr;       // rescoring reading A: R2 c of every centroid [nlist * Dp2]
  uint8_t* cgemm = nullptr;     // probe GEMM: centroids * 2^sC as fp16 hi / lo operand blocks
  int64_t device_bytes = 0;
  // profiling of the dominant scan kernel
  mutable std::mutex prof_mu;
  mutable std::vector<std::pair<cudaEvent_t, cudaEvent_t>> prof_events;
  mutable std::string prof_kernel;
  int profile = 0;
};
