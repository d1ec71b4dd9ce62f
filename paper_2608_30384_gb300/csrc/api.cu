// api.cu -- the extern "C" entry points of librslm (declared in include/rslm.h).
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "launch.h"
#include "rslm_internal.h"

using namespace rslm;

namespace {

thread_local std::string g_last_error;

rslm_status fail(rslm_status st, const std::string& msg) {
  g_last_error = msg;
  return st;
}

rslm_status cuda_fail(cudaError_t e, const char* what) {
  cudaGetLastError();  // clear a non-sticky error
  return fail(e == cudaErrorMemoryAllocation ? RSLM_ERR_OUT_OF_MEMORY : RSLM_ERR_CUDA,
              std::string(what) + ": " + cudaGetErrorString(e));
}

#define RSLM_CK(expr, what)                          \
  do {                                               \
    cudaError_t _e = (expr);                         \
    if (_e != cudaSuccess) return cuda_fail(_e, what); \
  } while (0)

#define RSLM_ARG(cond, msg)                                         \
  do {                                                              \
    if (!(cond)) return fail(RSLM_ERR_INVALID_ARG, std::string(msg)); \
  } while (0)

// Makes the index's device current for the duration of a call.
struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

cudaStream_t as_stream(void* s) { return reinterpret_cast<cudaStream_t>(s); }

template <typename T>
cudaError_t dev_alloc(rslm_index* ix, T** p, size_t count) {
  const size_t bytes = count * sizeof(T) > 0 ? count * sizeof(T) : 16;
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(p), bytes);
  if (e == cudaSuccess) ix->device_bytes += int64_t(bytes);
  return e;
}

void free_all(rslm_index* ix) {
  void* ptrs[] = {ix->centroids, ix->part_off, ix->part_n, ix->assign, ix->slot_of_row, ix->ids,
                  ix->codes1,    ix->scales1,  ix->codes2, ix->scales2, ix->d_err,   ix->ctiles, ix->d_counters,
                  ix->cmeta,     ix->crows,    ix->crot2,   ix->cgemm};
  for (void* p : ptrs)
    if (p) cudaFree(p);
}

// Probe stage shared by rslm_probe and rslm_search (Sec. 5.5.1 step 3): the
// fused tensor-core probe where it applies (padded D <= 128, nlist >= 32
// nprobe), otherwise the tensor-core score GEMM with a row selection.
rslm_status run_probe(const rslm_index* ix, const float* queries, int64_t nq, int nprobe,
                      int32_t* out_probes, float* out_cs, cudaStream_t s) {
  if (nq == 0) return RSLM_OK;
  if (probe_fused_supported(ix, nprobe)) {
    RSLM_CK(launch_probe_fused(ix, queries, nq, nprobe, out_probes, out_cs, s), "fused probe launch");
    return RSLM_OK;
  }
  RSLM_CK(launch_probe_gemm(ix, queries, nq, nprobe, out_probes, out_cs, s), "probe GEMM launch");
  return RSLM_OK;
}

rslm_status check_query_args(const rslm_index* ix, int64_t nq, int nprobe) {
  RSLM_ARG(ix, "index is NULL");
  RSLM_ARG(nq >= 0 && nq < (int64_t(1) << 31), "nq out of range [0, 2^31)");
  RSLM_ARG(nprobe >= 1 && nprobe <= ix->nlist && nprobe <= kMaxNprobe,
           "nprobe must be in [1, min(nlist, 4096)]");
  return RSLM_OK;
}

}  // namespace

rslm_status rslm::set_last_error(rslm_status st, const std::string& msg) { return fail(st, msg); }

cudaEvent_t rslm::prof_start(const rslm_index* ix, cudaStream_t s, const char* kernel) {
  if (!ix->profile) return nullptr;
  cudaEvent_t a = nullptr, b = nullptr;
  if (cudaEventCreate(&a) != cudaSuccess) return nullptr;
  if (cudaEventCreate(&b) != cudaSuccess) {
    cudaEventDestroy(a);
    return nullptr;
  }
  cudaEventRecord(a, s);
  std::lock_guard<std::mutex> lock(ix->prof_mu);
  ix->prof_events.emplace_back(a, b);
  ix->prof_kernel = kernel;
  return b;
}

void rslm::prof_stop(cudaEvent_t stop, cudaStream_t s) {
  if (stop) cudaEventRecord(stop, s);
}

namespace {
void prof_clear(const rslm_index* ix) {
  std::lock_guard<std::mutex> lock(ix->prof_mu);
  for (auto& e : ix->prof_events) {
    cudaEventDestroy(e.first);
    cudaEventDestroy(e.second);
  }
  ix->prof_events.clear();
}
}  // namespace

extern "C" {

rslm_status rslm_index_create(int32_t dim, int32_t nlist, const float* centroids, int32_t score_bits,
                              int32_t rescore_bits, uint32_t flags, void* stream,
                              rslm_index** out) {
  RSLM_ARG(out, "out is NULL");
  *out = nullptr;
  RSLM_ARG(dim >= 1 && dim <= kMaxDim, "dim must be in [1, 4096]");
  RSLM_ARG(nlist >= 1, "nlist must be >= 1");
  RSLM_ARG(score_bits >= 1 && score_bits <= 4, "score_bits must be 1, 2, 3 or 4");
  RSLM_ARG(rescore_bits == 0 || rescore_bits == 4, "rescore_bits must be 0 or 4");
  RSLM_ARG((flags & ~(RSLM_GLOBAL_SCALE | RSLM_LITE | RSLM_RESCORE_READING_A | RSLM_FULL_VECTOR)) == 0,
           "unknown flag bits");
  RSLM_ARG(!(flags & RSLM_RESCORE_READING_A) || rescore_bits > 0, "RSLM_RESCORE_READING_A needs rescoring codes");
  RSLM_ARG(!(flags & RSLM_LITE) || (score_bits == 4 && dim >= 64),
           "RSLM_LITE needs score_bits == 4 and dim >= 64");
  RSLM_ARG(centroids, "centroids is NULL");
  {
    CodecSpec probe_spec;
    make_codec_spec(score_bits, dim, true, &probe_spec);
    // The scan keeps a 16-entry float table per nibble position of a row in
    // shared memory: 2 * stride * 16 * 4 bytes must fit in a CTA's 227 KB.
    RSLM_ARG(size_t(probe_spec.stride) * 2 * 16 * 4 <= size_t(200) * 1024,
             "dim too large for score_bits (scan table exceeds shared memory; 4-bit: dim <= 3200)");
  }
  rslm_index* ix = new rslm_index();
  cudaGetDevice(&ix->device);
  {
    // Search calls take their scratch from the device's stream-ordered pool;
    // keep freed blocks cached in the pool across synchronizations instead
    // of returning them to the driver (this process only).
    cudaMemPool_t pool;
    if (cudaDeviceGetDefaultMemPool(&pool, ix->device) == cudaSuccess) {
      uint64_t keep = ~uint64_t(0);
      cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep);
    }
  }
  ix->D = dim;
  ix->nlist = nlist;
  ix->bits = score_bits;
  ix->rescore_bits = rescore_bits;
  ix->flags = flags;
  ix->rot1 = make_rot_spec(dim, score_bits);
  make_codec_spec(score_bits, dim, true, &ix->cs1);
  if (flags & RSLM_LITE) {
    CodecSpec k8;
    make_codec_spec(3, 0, true, &k8);
    ix->cs1.lite_h = (flags & RSLM_GLOBAL_SCALE) ? 32 : 16;
    for (int i = 0; i < 8; ++i) {
      ix->cs1.cb8d[i] = k8.cbd[i];
      ix->cs1.cb8f[i] = k8.cbf[i];
      if (i < 7) ix->cs1.thr8[i] = k8.thr[i];
    }
  }
  if (rescore_bits) {
    ix->rot2 = make_rot_spec(dim, rescore_bits);
    make_codec_spec(rescore_bits, dim, false, &ix->cs2);
  }
  cudaStream_t s = as_stream(stream);
  cudaError_t e = dev_alloc(ix, &ix->centroids, size_t(nlist) * dim);
  if (e == cudaSuccess) e = dev_alloc(ix, &ix->d_err, 1);
  if (e == cudaSuccess) e = dev_alloc(ix, &ix->d_counters, kNumCounters);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(ix->centroids, centroids, size_t(nlist) * dim * sizeof(float),
                        cudaMemcpyDeviceToDevice, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(ix->d_err, 0, sizeof(int), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(ix->d_counters, 0, kNumCounters * sizeof(unsigned long long), s);
  if (e == cudaSuccess) e = probe_prepare(ix, s);
  if (e == cudaSuccess && (flags & RSLM_RESCORE_READING_A) && !(flags & RSLM_FULL_VECTOR)) {
    // reading A scores <q, c> in the rescoring rotation: R2 c of every centroid
    e = dev_alloc(ix, &ix->crot2, size_t(nlist) * ix->cs2.Dp);
    if (e == cudaSuccess) e = launch_rotate_rows(ix->rot2, ix->centroids, nlist, ix->crot2, ix->cs2.Dp, s);
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    free_all(ix);
    delete ix;
    return cuda_fail(e, "rslm_index_create");
  }
  *out = ix;
  return RSLM_OK;
}

rslm_status rslm_index_describe(const rslm_index* ix, rslm_index_desc* d) {
  RSLM_ARG(ix && d, "NULL argument");
  std::memset(d, 0, sizeof(*d));
  d->dim = ix->D;
  d->nlist = ix->nlist;
  d->score_bits = ix->bits;
  d->rescore_bits = ix->rescore_bits;
  d->group = ix->cs1.g;
  d->padded_dim = ix->cs1.Dp;
  d->code_bytes = ix->cs1.code_bytes;
  d->rescore_group = ix->rescore_bits ? ix->cs2.g : 0;
  d->rescore_padded_dim = ix->rescore_bits ? ix->cs2.Dp : 0;
  d->rescore_code_bytes = ix->rescore_bits ? ix->cs2.code_bytes : 0;
  d->rotation_passes = ix->rot1.two_pass ? 2 : 1;
  d->rescore_rotation_passes = ix->rescore_bits ? (ix->rot2.two_pass ? 2 : 1) : 0;
  d->n_rows = ix->n_rows;
  d->n_slots = ix->n_slots;
  d->device_bytes = ix->device_bytes;
  d->flags = ix->flags;
  return RSLM_OK;
}

rslm_status rslm_index_reserve(rslm_index* ix, const int32_t* assignment, int64_t n, void* stream) {
  RSLM_ARG(ix, "index is NULL");
  if (ix->n_rows != 0 || ix->slot_of_row) return fail(RSLM_ERR_STATE, "index already reserved");
  RSLM_ARG(n >= 1 && n < (int64_t(1) << 31), "n must be in [1, 2^31)");
  RSLM_ARG(assignment, "assignment is NULL");
  DeviceGuard g(ix->device);
  cudaStream_t s = as_stream(stream);
  std::vector<int32_t> a(n);
  RSLM_CK(cudaMemcpyAsync(a.data(), assignment, size_t(n) * 4, cudaMemcpyDeviceToHost, s),
          "copy assignment");
  RSLM_CK(cudaStreamSynchronize(s), "reserve sync");
  std::vector<int64_t> cnt(ix->nlist, 0);
  for (int64_t i = 0; i < n; ++i) {
    if (a[i] < 0 || a[i] >= ix->nlist)
      return fail(RSLM_ERR_INVALID_ARG, "assignment[" + std::to_string(i) + "] = " +
                                            std::to_string(a[i]) + " outside [0, nlist)");
    cnt[a[i]]++;
  }
  std::vector<int64_t> off(ix->nlist + 1, 0);
  std::vector<int32_t> pn(ix->nlist);
  for (int p = 0; p < ix->nlist; ++p) {
    off[p + 1] = off[p] + (cnt[p] + kTile - 1) / kTile * kTile;
    pn[p] = int32_t(cnt[p]);
  }
  const int64_t n_slots = off[ix->nlist];
  RSLM_ARG(n_slots < (int64_t(1) << 31), "padded slot count exceeds 2^31");
  std::vector<int32_t> slot(n);
  std::vector<int64_t> next(off.begin(), off.end() - 1);
  for (int64_t i = 0; i < n; ++i) slot[i] = int32_t(next[a[i]]++);

  cudaError_t e = dev_alloc(ix, &ix->assign, n);
  if (e == cudaSuccess) e = dev_alloc(ix, &ix->slot_of_row, n);
  if (e == cudaSuccess) e = dev_alloc(ix, &ix->part_off, ix->nlist + 1);
  if (e == cudaSuccess) e = dev_alloc(ix, &ix->part_n, ix->nlist);
  if (e == cudaSuccess) e = dev_alloc(ix, &ix->ids, n_slots);
  if (e == cudaSuccess) e = dev_alloc(ix, &ix->codes1, size_t(n_slots) * ix->cs1.stride);
  if (e == cudaSuccess) e = dev_alloc(ix, &ix->scales1, n_slots);
  if (e == cudaSuccess && ix->rescore_bits) {
    e = dev_alloc(ix, &ix->codes2, size_t(n_slots) * ix->cs2.stride);
    if (e == cudaSuccess) e = dev_alloc(ix, &ix->scales2, n_slots);
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(ix->assign, a.data(), size_t(n) * 4, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(ix->slot_of_row, slot.data(), size_t(n) * 4, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(ix->part_off, off.data(), off.size() * 8, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(ix->part_n, pn.data(), pn.size() * 4, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(ix->ids, 0xff, size_t(n_slots) * 8, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(ix->codes1, 0, size_t(n_slots) * ix->cs1.stride, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(ix->scales1, 0, size_t(n_slots) * 4, s);
  if (e == cudaSuccess && ix->rescore_bits) {
    e = cudaMemsetAsync(ix->codes2, 0, size_t(n_slots) * ix->cs2.stride, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(ix->scales2, 0, size_t(n_slots) * 4, s);
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    void** arrs[] = {(void**)&ix->assign, (void**)&ix->slot_of_row, (void**)&ix->part_off,
                     (void**)&ix->part_n, (void**)&ix->ids,         (void**)&ix->codes1,
                     (void**)&ix->scales1, (void**)&ix->codes2,     (void**)&ix->scales2};
    for (void** p : arrs) {
      if (*p) cudaFree(*p);
      *p = nullptr;
    }
    ix->device_bytes = int64_t(ix->nlist) * ix->D * 4 + 16;
    return cuda_fail(e, "rslm_index_reserve");
  }
  ix->n_rows = n;
  ix->n_slots = n_slots;
  ix->max_part_n = *std::max_element(pn.begin(), pn.end());
  return RSLM_OK;
}

rslm_status rslm_encode_all(const float* vectors, const int32_t* assignment, int64_t n, int32_t dim,
                            int32_t nlist, const float* centroids, int32_t score_bits,
                            int32_t rescore_bits, uint32_t flags, void* stream, rslm_index** out) {
  RSLM_ARG(out, "out is NULL");
  *out = nullptr;
  RSLM_ARG(n == 0 || vectors, "vectors is NULL");
  rslm_index* ix = nullptr;
  rslm_status st = rslm_index_create(dim, nlist, centroids, score_bits, rescore_bits, flags, stream, &ix);
  if (st != RSLM_OK) return st;
  st = rslm_index_reserve(ix, assignment, n, stream);
  if (st == RSLM_OK) st = rslm_encode(ix, vectors, 0, n, stream);
  if (st != RSLM_OK) {
    const std::string msg = g_last_error;
    rslm_index_destroy(ix);
    return fail(st, msg);
  }
  *out = ix;
  return RSLM_OK;
}

rslm_status rslm_encode(rslm_index* ix, const float* vectors, int64_t row_begin, int64_t rows,
                        void* stream) {
  RSLM_ARG(ix, "index is NULL");
  if (!ix->slot_of_row) return fail(RSLM_ERR_STATE, "rslm_index_reserve has not been called");
  RSLM_ARG(row_begin >= 0 && rows >= 0 && row_begin <= ix->n_rows && rows <= ix->n_rows - row_begin,
           "rows [row_begin, row_begin + rows) outside the reserved rows");
  RSLM_ARG(rows == 0 || vectors, "vectors is NULL");
  DeviceGuard g(ix->device);
  RSLM_CK(launch_encode(ix, vectors, row_begin, rows, as_stream(stream)), "encode launch");
  return RSLM_OK;
}

rslm_status rslm_rotate_queries(const rslm_index* ix, int32_t which, const float* queries, int64_t nq,
                                float* out, void* stream) {
  RSLM_ARG(ix, "index is NULL");
  RSLM_ARG(which == 1 || (which == 2 && ix->rescore_bits), "which must be 1, or 2 with rescoring codes");
  RSLM_ARG(nq >= 0, "nq < 0");
  RSLM_ARG(nq == 0 || (queries && out), "NULL array");
  DeviceGuard g(ix->device);
  const RotSpec& r = which == 1 ? ix->rot1 : ix->rot2;
  const int Dp = which == 1 ? ix->cs1.Dp : ix->cs2.Dp;
  RSLM_CK(launch_rotate_rows(r, queries, nq, out, Dp, as_stream(stream)), "rotate launch");
  return RSLM_OK;
}

rslm_status rslm_probe(const rslm_index* ix, const float* queries, int64_t nq, int32_t nprobe,
                       int32_t* out_probes, float* out_cs, void* stream) {
  rslm_status st = check_query_args(ix, nq, nprobe);
  if (st != RSLM_OK) return st;
  RSLM_ARG(nq == 0 || (queries && out_probes && out_cs), "NULL array");
  DeviceGuard g(ix->device);
  return run_probe(ix, queries, nq, nprobe, out_probes, out_cs, as_stream(stream));
}

rslm_status rslm_scan(const rslm_index* ix, const float* qrot, int64_t nq, const int32_t* probes,
                      const float* cs, int32_t nprobe, int32_t k, int64_t* out_ids,
                      float* out_scores, void* stream) {
  rslm_status st = check_query_args(ix, nq, nprobe);
  if (st != RSLM_OK) return st;
  if (!ix->slot_of_row) return fail(RSLM_ERR_STATE, "rslm_index_reserve has not been called");
  RSLM_ARG(k >= 1 && k <= kMaxK, "k must be in [1, 256]");
  RSLM_ARG(nq == 0 || (qrot && probes && cs && out_ids && out_scores), "NULL array");
  DeviceGuard g(ix->device);
  RSLM_CK(launch_scan(ix, qrot, nq, probes, cs, nprobe, k, k, out_ids, out_scores, as_stream(stream)),
          "scan launch");
  return RSLM_OK;
}

rslm_status rslm_scan_batched(const rslm_index* ix, const float* qrot, int64_t nq,
                              const int32_t* probes, const float* cs, int32_t nprobe, int32_t k,
                              int64_t* out_ids, float* out_scores, void* stream) {
  rslm_status st = check_query_args(ix, nq, nprobe);
  if (st != RSLM_OK) return st;
  if (!ix->slot_of_row) return fail(RSLM_ERR_STATE, "rslm_index_reserve has not been called");
  RSLM_ARG(k >= 1 && k <= kMaxK, "k must be in [1, 256]");
  RSLM_ARG(nq == 0 || (qrot && probes && cs && out_ids && out_scores), "NULL array");
  DeviceGuard g(ix->device);
  RSLM_CK(launch_scan_batched(ix, qrot, nq, probes, cs, nprobe, k, out_ids, out_scores,
                              as_stream(stream)),
          "batched scan");
  return RSLM_OK;
}

rslm_status rslm_rescore(const rslm_index* ix, const float* qrot2, int64_t nq, const int64_t* cand_ids,
                         const float* cand_scores, int32_t k, int32_t k_final, int64_t* out_ids,
                         float* out_scores, void* stream) {
  RSLM_ARG(ix, "index is NULL");
  if (!ix->rescore_bits) return fail(RSLM_ERR_STATE, "index has no rescoring codes");
  if (!ix->slot_of_row) return fail(RSLM_ERR_STATE, "rslm_index_reserve has not been called");
  RSLM_ARG(nq >= 0 && nq < (int64_t(1) << 31), "nq out of range");
  RSLM_ARG(k >= 1 && k <= kMaxK, "k must be in [1, 256]");
  RSLM_ARG(k_final >= 1 && k_final <= k, "k_final must be in [1, k]");
  RSLM_ARG(nq == 0 || (qrot2 && cand_ids && cand_scores && out_ids && out_scores), "NULL array");
  DeviceGuard g(ix->device);
  RSLM_CK(launch_rescore(ix, qrot2, nq, cand_ids, cand_scores, k, k_final, out_ids, out_scores,
                         as_stream(stream)),
          "rescore launch");
  return RSLM_OK;
}

rslm_status rslm_search(const rslm_index* ix, const float* queries, int64_t nq, int32_t nprobe,
                        int32_t k, int32_t rescore, int32_t k_final, int64_t* out_ids,
                        float* out_scores, void* stream) {
  rslm_status st = check_query_args(ix, nq, nprobe);
  if (st != RSLM_OK) return st;
  if (!ix->slot_of_row) return fail(RSLM_ERR_STATE, "rslm_index_reserve has not been called");
  RSLM_ARG(k >= 1 && k <= kMaxK, "k must be in [1, 256]");
  RSLM_ARG(k_final >= 1 && k_final <= k, "k_final must be in [1, k]");
  RSLM_ARG(nq == 0 || (queries && out_ids && out_scores), "NULL array");
  if (rescore && !ix->rescore_bits) return fail(RSLM_ERR_STATE, "index has no rescoring codes");
  if (nq == 0) return RSLM_OK;
  DeviceGuard g(ix->device);
  cudaStream_t s = as_stream(stream);
  const bool rs = rescore != 0;
  int32_t* probes = nullptr;
  float *cs = nullptr, *q1 = nullptr, *q2 = nullptr, *s1s = nullptr;
  int64_t* s1i = nullptr;
  cudaError_t e = cudaMallocAsync(reinterpret_cast<void**>(&probes), size_t(nq) * nprobe * 4, s);
  if (e == cudaSuccess) e = cudaMallocAsync(reinterpret_cast<void**>(&cs), size_t(nq) * nprobe * 4, s);
  if (e == cudaSuccess)
    e = cudaMallocAsync(reinterpret_cast<void**>(&q1), size_t(nq) * ix->cs1.Dp * 4, s);
  if (e == cudaSuccess && rs) {
    e = cudaMallocAsync(reinterpret_cast<void**>(&q2), size_t(nq) * ix->cs2.Dp * 4, s);
    if (e == cudaSuccess) e = cudaMallocAsync(reinterpret_cast<void**>(&s1i), size_t(nq) * k * 8, s);
    if (e == cudaSuccess) e = cudaMallocAsync(reinterpret_cast<void**>(&s1s), size_t(nq) * k * 4, s);
  }
  if (e != cudaSuccess) st = cuda_fail(e, "cudaMallocAsync(search workspace)");
  if (st == RSLM_OK) st = run_probe(ix, queries, nq, nprobe, probes, cs, s);
  if (st == RSLM_OK) {
    e = launch_rotate_rows(ix->rot1, queries, nq, q1, ix->cs1.Dp, s);
    // Partition-major tensor-core scan once partitions are shared by enough
    // queries (on average at least kBatchMinQueries per probed list).
    const bool batched = nq * nprobe >= int64_t(kBatchMinQueries) * ix->nlist;
    if (e == cudaSuccess && batched && (rs || k_final == k))
      e = launch_scan_batched(ix, q1, nq, probes, cs, nprobe, k, rs ? s1i : out_ids,
                              rs ? s1s : out_scores, s);
    else if (e == cudaSuccess)
      e = launch_scan(ix, q1, nq, probes, cs, nprobe, k, rs ? k : k_final, rs ? s1i : out_ids,
                      rs ? s1s : out_scores, s);
    if (e == cudaSuccess && rs) e = launch_rotate_rows(ix->rot2, queries, nq, q2, ix->cs2.Dp, s);
    if (e == cudaSuccess && rs)
      e = launch_rescore(ix, q2, nq, s1i, s1s, k, k_final, out_ids, out_scores, s);
    if (e != cudaSuccess) st = cuda_fail(e, "search launch");
  }
  void* temps[] = {probes, cs, q1, q2, s1i, s1s};
  for (void* p : temps)
    if (p) cudaFreeAsync(p, s);
  return st;
}

rslm_status rslm_export_codes(const rslm_index* ix, int32_t which, int64_t row_begin, int64_t rows,
                              uint8_t* codes, uint16_t* local_scale, uint16_t* global_scale,
                              void* stream) {
  RSLM_ARG(ix, "index is NULL");
  RSLM_ARG(which == 1 || (which == 2 && ix->rescore_bits), "which must be 1, or 2 with rescoring codes");
  if (!ix->slot_of_row) return fail(RSLM_ERR_STATE, "rslm_index_reserve has not been called");
  RSLM_ARG(row_begin >= 0 && rows >= 0 && row_begin <= ix->n_rows && rows <= ix->n_rows - row_begin,
           "row range out of bounds");
  RSLM_ARG(rows == 0 || (codes && local_scale && global_scale), "NULL array");
  DeviceGuard g(ix->device);
  RSLM_CK(launch_export_import(ix, which, row_begin, rows, codes, local_scale, global_scale, false,
                               as_stream(stream)),
          "export launch");
  return RSLM_OK;
}

rslm_status rslm_decompress(const rslm_index* ix, int32_t which, int64_t row_begin, int64_t rows, float* out,
                            void* stream) {
  RSLM_ARG(ix, "index is NULL");
  RSLM_ARG(which == 1 || (which == 2 && ix->rescore_bits), "which must be 1, or 2 with rescoring codes");
  if (!ix->slot_of_row) return fail(RSLM_ERR_STATE, "rslm_index_reserve has not been called");
  RSLM_ARG(row_begin >= 0 && rows >= 0 && row_begin <= ix->n_rows && rows <= ix->n_rows - row_begin,
           "row range out of bounds");
  RSLM_ARG(rows == 0 || out, "NULL array");
  DeviceGuard g(ix->device);
  RSLM_CK(launch_decompress(ix, which, row_begin, rows, out, as_stream(stream)), "decompress launch");
  return RSLM_OK;
}

rslm_status rslm_import_codes(rslm_index* ix, int32_t which, int64_t row_begin, int64_t rows,
                              const uint8_t* codes, const uint16_t* local_scale,
                              const uint16_t* global_scale, void* stream) {
  RSLM_ARG(ix, "index is NULL");
  RSLM_ARG(which == 1 || (which == 2 && ix->rescore_bits), "which must be 1, or 2 with rescoring codes");
  if (!ix->slot_of_row) return fail(RSLM_ERR_STATE, "rslm_index_reserve has not been called");
  RSLM_ARG(row_begin >= 0 && rows >= 0 && row_begin <= ix->n_rows && rows <= ix->n_rows - row_begin,
           "row range out of bounds");
  RSLM_ARG(rows == 0 || (codes && local_scale && global_scale), "NULL array");
  DeviceGuard g(ix->device);
  RSLM_CK(launch_export_import(ix, which, row_begin, rows, const_cast<uint8_t*>(codes),
                               const_cast<uint16_t*>(local_scale), const_cast<uint16_t*>(global_scale),
                               true, as_stream(stream)),
          "import launch");
  return RSLM_OK;
}

rslm_status rslm_codebook(int32_t bits, float* out, int32_t* K_out, int32_t* g_out) {
  RSLM_ARG(out && K_out && g_out, "NULL argument");
  CodecSpec c;
  if (!make_codec_spec(bits, 0, true, &c)) return fail(RSLM_ERR_INVALID_ARG, "bits must be 1..4");
  for (int i = 0; i < c.K * c.g; ++i) out[i] = c.cbf[i];
  *K_out = c.K;
  *g_out = c.g;
  return RSLM_OK;
}

rslm_status rslm_rotation_tables(int8_t* s1, int32_t* perm) {
  RSLM_ARG(s1 && perm, "NULL argument");
  rotation_tables(s1, perm);
  return RSLM_OK;
}

rslm_status rslm_e_max(int32_t dim, double* out) {
  RSLM_ARG(out, "NULL argument");
  RSLM_ARG(dim >= 1 && dim <= kMaxDim, "dim must be in [1, 4096]");
  *out = e_max(dim);
  return RSLM_OK;
}

rslm_status rslm_sync(const rslm_index* ix, void* stream) {
  RSLM_ARG(ix, "index is NULL");
  DeviceGuard g(ix->device);
  RSLM_CK(cudaStreamSynchronize(as_stream(stream)), "stream synchronize");
  RSLM_CK(cudaGetLastError(), "pending CUDA error");
  int h = 0;
  RSLM_CK(cudaMemcpy(&h, ix->d_err, sizeof(int), cudaMemcpyDeviceToHost), "read device error flag");
  if (h != 0) {
    cudaMemset(ix->d_err, 0, sizeof(int));
    if (h == kErrTimeout)
      return fail(RSLM_ERR_TIMEOUT, "a bounded wait for the tensor-core pipeline expired");
    const char* what = h == kErrBadProbe ? "probe list holds a partition id outside [0, nlist)"
                       : h == kErrBadCandidate ? "candidate id outside [-1, n_rows)"
                       : h == kErrSmemLayout   ? "a scan kernel's shared-memory layout did not fit its launch"
                                               : "device-side check failed";
    return fail(RSLM_ERR_DEVICE, what);
  }
  return RSLM_OK;
}

const char* rslm_last_error(void) { return g_last_error.c_str(); }

rslm_status rslm_counters(const rslm_index* ix, int64_t* out, int32_t n) {
  RSLM_ARG(ix && out, "NULL argument");
  RSLM_ARG(n >= 1 && n <= kNumCounters, "n must be in [1, 4]");
  DeviceGuard g(ix->device);
  RSLM_CK(cudaDeviceSynchronize(), "device synchronize");
  unsigned long long h[kNumCounters] = {};
  RSLM_CK(cudaMemcpy(h, ix->d_counters, sizeof(h), cudaMemcpyDeviceToHost), "read counters");
  for (int i = 0; i < n; ++i) out[i] = int64_t(h[i]);
  return RSLM_OK;
}

rslm_status rslm_profile_enable(rslm_index* ix, int32_t on) {
  RSLM_ARG(ix, "index is NULL");
  DeviceGuard g(ix->device);
  prof_clear(ix);
  ix->profile = on ? 1 : 0;
  return RSLM_OK;
}

rslm_status rslm_profile_read(rslm_index* ix, double* total_ms, int64_t* launches, char* kernel,
                              int32_t kernel_len) {
  RSLM_ARG(ix && total_ms && launches, "NULL argument");
  DeviceGuard g(ix->device);
  double tot = 0.0;
  int64_t n = 0;
  std::string name;
  {
    std::lock_guard<std::mutex> lock(ix->prof_mu);
    for (auto& e : ix->prof_events) {
      RSLM_CK(cudaEventSynchronize(e.second), "profile event");
      float ms = 0.0f;
      RSLM_CK(cudaEventElapsedTime(&ms, e.first, e.second), "profile elapsed");
      tot += ms;
      ++n;
    }
    name = ix->prof_kernel;
  }
  prof_clear(ix);
  *total_ms = tot;
  *launches = n;
  if (kernel && kernel_len > 0) {
    std::strncpy(kernel, name.c_str(), size_t(kernel_len) - 1);
    kernel[kernel_len - 1] = 0;
  }
  return RSLM_OK;
}

void rslm_index_destroy(rslm_index* ix) {
  if (!ix) return;
  DeviceGuard g(ix->device);
  prof_clear(ix);
  free_all(ix);
  delete ix;
}

}  // extern "C"
