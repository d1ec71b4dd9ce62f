// launch.h -- host launchers of the librslm kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "rslm_internal.h"

namespace rslm {

cudaError_t launch_rotate_rows(const RotSpec& rot, const float* in, int64_t n, float* out, int Dp,
                               cudaStream_t s);
cudaError_t launch_encode(const rslm_index* ix, const float* x, int64_t row_begin, int64_t rows,
                          cudaStream_t s);
// Reconstructions of rows [row_begin, row_begin + rows) from stage `which`'s
// codes (codec.cu): [rows * D] float32.
cudaError_t launch_decompress(const rslm_index* ix, int which, int64_t row_begin, int64_t rows, float* out,
                              cudaStream_t s);
cudaError_t launch_export_import(const rslm_index* ix, int which, int64_t row_begin, int64_t rows,
                                 uint8_t* codes, uint16_t* lscale, uint16_t* gscale, bool import,
                                 cudaStream_t s);
// Top-kk of the first n entries of every row of S (row stride ld) by
// (value desc, column asc).  flags: optional device scratch of `rows` ints
// enabling the warp-per-row kernel (used when ld % 4 == 0 and S is 16-byte
// aligned).
cudaError_t launch_select_topn(const float* S, int64_t rows, int64_t ld, int n, int kk,
                               int32_t* out_idx, float* out_val, int* flags, cudaStream_t s);
cudaError_t launch_scan(const rslm_index* ix, const float* qrot, int64_t nq, const int32_t* probes,
                        const float* cs, int nprobe, int k, int out_k, int64_t* out_ids,
                        float* out_scores, cudaStream_t s);
// Single-query scan of the first `nprobe` entries of probe lists whose rows
// are `probe_stride` long; queries with only_if[q] == 0 are skipped.
cudaError_t launch_scan_strided(const rslm_index* ix, const float* qrot, int64_t nq,
                                const int32_t* probes, int probe_stride, const float* cs, int nprobe,
                                int k, int out_k, int64_t* out_ids, float* out_scores,
                                const int* only_if, cudaStream_t s);
// The same scan of the queries qlist[0 .. *qcount) (a device-side count of
// at most nq), by a fixed grid whose blocks stride over the list.
cudaError_t launch_scan_listed(const rslm_index* ix, const float* qrot, int64_t nq, const int32_t* probes,
                               int probe_stride, const float* cs, int nprobe, int k, int64_t* out_ids,
                               float* out_scores, const int* qlist, const int* qcount, cudaStream_t s);
// Partition-major scan on the tensor cores (batched.cu); output as launch_scan.
cudaError_t launch_scan_batched(const rslm_index* ix, const float* qrot, int64_t nq,
                                const int32_t* probes, const float* cs, int nprobe, int k,
                                int64_t* out_ids, float* out_scores, cudaStream_t s);
cudaError_t launch_rescore(const rslm_index* ix, const float* qrot2, int64_t nq,
                           const int64_t* cand_ids, const float* cand_scores, int k, int k_final,
                           int64_t* out_ids, float* out_scores, cudaStream_t s);

// Tensor-core probes (probe.cu).  probe_prepare builds the centroid
// operands (the GEMM's for every shape, the fused probe's for padded
// D <= 128); probe_fused_supported says whether launch_probe_fused can serve
// nprobe; launch_probe_gemm serves every shape (score matrix + selection).
cudaError_t probe_prepare(rslm_index* ix, cudaStream_t s);
bool probe_fused_supported(const rslm_index* ix, int nprobe);
cudaError_t launch_probe_fused(const rslm_index* ix, const float* queries, int64_t nq, int nprobe,
                               int32_t* out_probes, float* out_cs, cudaStream_t s);
cudaError_t launch_probe_gemm(const rslm_index* ix, const float* queries, int64_t nq, int nprobe,
                              int32_t* out_probes, float* out_cs, cudaStream_t s);

}  // namespace rslm
