// probe_noalloc.cu -- rslm_probe_noalloc: the probe step without device allocation.
//
// rslm_probe keeps its working buffers (query operands, candidate lists or a
// <query, centroid> score chunk) in temporary memory from the stream-ordered
// allocator.
// Some callers cannot allocate on the query path: applications whose device
// memory is entirely owned by another allocator (a framework's caching
// allocator, or a fixed budget handed out up front), and latency-critical
// serving loops that forbid cudaMalloc / cudaFree because those calls can
// synchronize the device.  This variant keeps its scratch in a fixed
// file-scope device array instead, computes the dot products with its own
// kernel, and allocates nothing.
//
// The scratch array (kScratchFloats floats = 16 MiB) exists on every GPU that
// loads the library, for the life of the process.  Its device address is
// looked up once per device, on the first call made with that device's
// index, with that device current (cudaGetSymbolAddress); make that first
// call before any stream capture.  Every call on a device shares the one
// array: calls whose work overlaps on the GPU (different streams, or host
// threads without ordering between them) race on it and must be serialised
// by the caller.  Each chunk's scores are fully rewritten before they are
// read, so nothing left by an earlier call is ever used.
#include <cuda_runtime.h>

#include <mutex>
#include <string>

#include "launch.h"
#include "rslm_internal.h"

namespace rslm {
namespace {

constexpr size_t kScratchFloats = size_t(4) << 20;  // 16 MiB of <q, c> scores
constexpr int kMaxDevices = 64;

static __device__ __align__(256) float g_probe_scratch[kScratchFloats];

std::mutex g_scratch_mu;
float* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_probe_scratch on `dev`, which must be the current
// device: the address is cached per device, so a lookup made with another
// device current would poison every later call on `dev`.
cudaError_t scratch_address(int dev, float** out) {
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    int cur = -1;
    cudaError_t e0 = cudaGetDevice(&cur);
    if (e0 != cudaSuccess) return e0;
    if (cur != dev) return cudaErrorInvalidDevice;
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_probe_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = static_cast<float*>(p);
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

// S[q, p] = <Q[q], C[p]> for q < nq, p < nlist: 64 x 64 output tile per
// block of 256 threads, 4 x 4 outputs per thread, float32 accumulation.
__global__ void __launch_bounds__(256) probe_scores_kernel(const float* __restrict__ Q, int nq,
                                                           const float* __restrict__ C, int nlist,
                                                           int D, float* __restrict__ S) {
  __shared__ float qs[32][65];
  __shared__ float cs[32][65];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int q0 = blockIdx.y * 64, p0 = blockIdx.x * 64;
  float acc[4][4] = {};
  for (int d0 = 0; d0 < D; d0 += 32) {
    for (int e = threadIdx.x; e < 64 * 32; e += 256) {
      const int r = e >> 5, d = e & 31;
      const int q = q0 + r, p = p0 + r, dd = d0 + d;
      qs[d][r] = (q < nq && dd < D) ? Q[int64_t(q) * D + dd] : 0.0f;
      cs[d][r] = (p < nlist && dd < D) ? C[int64_t(p) * D + dd] : 0.0f;
    }
    __syncthreads();
#pragma unroll 8
    for (int d = 0; d < 32; ++d) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = qs[d][ty + 16 * i];
        b[i] = cs[d][tx + 16 * i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int q = q0 + ty + 16 * i;
    if (q >= nq) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int p = p0 + tx + 16 * j;
      if (p < nlist) S[int64_t(q) * nlist + p] = acc[i][j];
    }
  }
}

}  // namespace
}  // namespace rslm

using namespace rslm;

extern "C" rslm_status rslm_probe_noalloc(const rslm_index* ix, const float* queries, int64_t nq,
                                          int32_t nprobe, int32_t* out_probes, float* out_cs,
                                          void* stream) {
  if (!ix) return set_last_error(RSLM_ERR_INVALID_ARG, "index is NULL");
  if (nq < 0 || nq >= (int64_t(1) << 31))
    return set_last_error(RSLM_ERR_INVALID_ARG, "nq out of range [0, 2^31)");
  if (nprobe < 1 || nprobe > ix->nlist || nprobe > kMaxNprobe)
    return set_last_error(RSLM_ERR_INVALID_ARG, "nprobe must be in [1, min(nlist, 4096)]");
  if (size_t(ix->nlist) > kScratchFloats)
    return set_last_error(RSLM_ERR_INVALID_ARG,
                          "nlist = " + std::to_string(ix->nlist) + " exceeds the " +
                              std::to_string(kScratchFloats) +
                              " scores one query needs in the fixed no-allocation scratch");
  if (nq > 0 && !(queries && out_probes && out_cs))
    return set_last_error(RSLM_ERR_INVALID_ARG, "NULL array");
  if (ix->device < 0 || ix->device >= kMaxDevices)
    return set_last_error(RSLM_ERR_INVALID_ARG, "device ordinal beyond the scratch table");
  if (nq == 0) return RSLM_OK;
  int prev = -1;
  cudaError_t e = cudaGetDevice(&prev);
  if (e != cudaSuccess)
    return set_last_error(RSLM_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (prev != ix->device) {
    e = cudaSetDevice(ix->device);
    if (e != cudaSuccess)
      return set_last_error(RSLM_ERR_CUDA, std::string("cudaSetDevice: ") + cudaGetErrorString(e));
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  rslm_status st = RSLM_OK;
  float* S = nullptr;
  e = scratch_address(ix->device, &S);
  if (e != cudaSuccess) {
    st = set_last_error(RSLM_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
  }
  int64_t qc = int64_t(kScratchFloats) / ix->nlist;  // >= 1 by the check above
  if (qc > (int64_t(1) << 21)) qc = int64_t(1) << 21;  // grid.y = qc / 64 stays below 65536
  for (int64_t q0 = 0; st == RSLM_OK && q0 < nq; q0 += qc) {
    const int n = int(nq - q0 < qc ? nq - q0 : qc);
    dim3 grid(unsigned((ix->nlist + 63) / 64), unsigned((n + 63) / 64));
    probe_scores_kernel<<<grid, 256, 0, s>>>(queries + q0 * ix->D, n, ix->centroids, ix->nlist, ix->D, S);
    e = cudaGetLastError();
    if (e == cudaSuccess)
      e = launch_select_topn(S, n, ix->nlist, ix->nlist, nprobe, out_probes + q0 * nprobe,
                             out_cs + q0 * nprobe, nullptr, s);
    if (e != cudaSuccess)
      st = set_last_error(RSLM_ERR_CUDA, std::string("probe_noalloc launch: ") + cudaGetErrorString(e));
  }
  if (prev >= 0 && prev != ix->device) cudaSetDevice(prev);
  return st;
}
