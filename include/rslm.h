/*
 * rslm.h -- C ABI of the GB300 (sm_103a) RSLM residual-code IVF search library.
 *
 * RSLM ("Rotated Scaled Lloyd-Max", a family of 1-4 bit training-free vector
 * codecs) encodes the residual r = x - a of every database vector x against an
 * approximation a (an IVF centroid, Sec. 5.5.1 step 2; or a previous stage's
 * reconstruction, Sec. 5.2), and searches by routing a query to the nprobe
 * partitions with the largest <q, centroid>, scoring every vector of those
 * partitions from its codes, taking the top-k and optionally rescoring the
 * survivors from higher-bit codes (Sec. 5.5.1 step 3; Sec. 2.1).
 *
 * Conventions shared by every call
 * --------------------------------
 * - Array arguments are DEVICE pointers owned by the caller unless a comment
 *   says "host".  They must stay valid until the work queued on `stream` has
 *   completed.  Matrices are row-major and densely packed.
 * - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *   Argument checks run synchronously and return before anything is queued;
 *   kernels then run asynchronously on `stream`.
 * - Every call returns an rslm_status.  RSLM_OK = 0.  On failure the call has
 *   queued nothing (argument errors) or the index is left in its previous
 *   valid state; rslm_last_error() returns a message for the calling thread.
 * - Device-side checks (a partition id out of range in a probe list, a bad
 *   candidate id) set a sticky flag on the index instead of faulting; the
 *   next rslm_sync() on that index returns RSLM_ERR_DEVICE and clears it.
 * - An index may be searched concurrently from several host threads on
 *   different streams once it is fully encoded; building (reserve, encode,
 *   import) must not overlap any other call on the same index.
 * - Limits: 1 <= dim <= 4096; nlist >= 1; score_bits in {1, 2, 3, 4};
 *   rescore_bits in {0, 4}; n <= 2^31 - 1 rows; 1 <= nprobe <= min(nlist,
 *   4096); 1 <= k <= 256; 1 <= k_final <= k; with score_bits = 4, dim <=
 *   3200 (the scan keeps a per-query table in shared memory).  Violations return
 *   RSLM_ERR_INVALID_ARG.
 *
 * Outputs: ids are original row ids (int64), scores float32, each query's list
 * sorted by (score descending, id ascending).  When fewer candidates than
 * requested exist the tail is id -1, score -INFINITY.
 */
#ifndef RSLM_H_
#define RSLM_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  RSLM_OK = 0,
  RSLM_ERR_INVALID_ARG = 1,
  RSLM_ERR_OUT_OF_MEMORY = 2,
  RSLM_ERR_CUDA = 3,
  RSLM_ERR_TIMEOUT = 4,
  RSLM_ERR_STATE = 5,
  RSLM_ERR_DEVICE = 6,
  RSLM_ERR_INTERNAL = 7
} rslm_status;

/* Flag for rslm_index_create.  Set: store the global scale of Sec. 3.5.2
 * (s = ||x|| / ||a + r~||, "RelApproxGlobal", the default of the paper's
 * end-to-end study).  Clear: local scaling only (Sec. 3.5.1, "RelApprox"),
 * the global scale is then 1. */
#define RSLM_GLOBAL_SCALE 1u

/* Flag for rslm_index_create.  Set: the scoring codes are Rslm4Lite (Sec.
 * 3.4, Rslm4Lite paragraph; with RSLM_GLOBAL_SCALE, RelApproxGlobal-
 * Rslm4Lite, Sec. 3.5.2).  score_bits must be 4 and dim >= 64.  The first
 * 16 rotated coordinates (32 with RSLM_GLOBAL_SCALE) are quantized with the
 * K = 8 levels of the 3-bit codec; bit i of the UE7M9 local-scale code is
 * stored as the top bit of code i and, with RSLM_GLOBAL_SCALE, bit i of the
 * UE4M12 global-scale code as the top bit of code 16 + i (i = 0 .. 15), so a
 * row is exactly ceil(dim / 2) code bytes.  The single-query scan reads the
 * scales from those bits; the index also keeps the decoded scale pair per
 * row (the `local_scale` / `global_scale` of rslm_export_codes and
 * rslm_import_codes, which then move codes that include the scale bits). */
#define RSLM_LITE 2u

/* Flag for rslm_index_create.  Set: the rescoring codes quantize x - c with
 * c the partition centroid, the first stage's own approximation ("reading
 * A": an independent finer code of the same residual), and rescoring scores
 * are G2 (<q, c> + L2 <R2 q, u2^>).  Clear ("reading B", Sec. 5.2): they
 * quantize x - a2 with a2 the full first-stage reconstruction, scored
 * G2 (s1 + L2 <R2 q, u2^>).  Needs rescore_bits > 0. */
#define RSLM_RESCORE_READING_A 4u

/* Flag for rslm_index_create.  Set: full-vector quantization (Sec. 3.5,
 * first paragraph): the codes quantize x itself (approximation 0).  The
 * partitions only route the probe; scores are G L <R q, u^> (no <q, c>
 * term, so rslm_scan ignores its cs argument). */
#define RSLM_FULL_VECTOR 8u

typedef struct rslm_index rslm_index;

/* Shape of an index, filled by rslm_index_describe. */
typedef struct {
  int32_t dim;            /* D */
  int32_t nlist;          /* number of IVF partitions */
  int32_t score_bits;     /* b of the scoring codes */
  int32_t rescore_bits;   /* 0 or 4 */
  int32_t group;          /* g: coordinates per 4-bit code (4, 2, 1 for b = 1, 2, 4) */
  int32_t padded_dim;     /* D' = g * ceil(D / g): width of a rotated scoring query */
  int32_t code_bytes;     /* canonical scoring-code bytes per row: ceil(D' / g / 2)
                             (ceil(3 D / 8) for score_bits = 3) */
  int32_t rescore_group;
  int32_t rescore_padded_dim;
  int32_t rescore_code_bytes;
  int32_t rotation_passes;         /* 1 or 2 (Sec. 3.1.3) for the scoring codes */
  int32_t rescore_rotation_passes;
  int64_t n_rows;         /* rows reserved (0 before rslm_index_reserve) */
  int64_t n_slots;        /* rows + per-partition padding to 128-row tiles */
  int64_t device_bytes;   /* device memory held by the index */
  uint32_t flags;
} rslm_index_desc;

/* Create an empty index on the current CUDA device.
 * centroids: device [nlist * dim] float32, copied (the caller may free it
 *   afterwards).  They are the approximations a of the first stage (IVF
 *   centroids, Sec. 5.5.1).
 * score_bits: bits per dimension of the scoring codes: 1 (4-D codebook,
 *   K = 16), 2 (2-D, K = 16), 3 (1-D, K = 8: Rslm3, eight codes packed in
 *   3 bytes, code i at bits 3i .. 3i + 2 of the row's byte stream, least
 *   significant bit first; the tensor-core scan decodes two codes (6 bits)
 *   per table lookup) or 4 (1-D, K = 16) (Sec. 3.2, Table "Rslm Codec
 *   Specifications").
 * rescore_bits: 0 (no rescoring) or 4: bits of the rescoring codes, which
 *   quantize x - a2 with a2 the full first-stage reconstruction (Sec. 5.2).
 * flags: any of RSLM_GLOBAL_SCALE, RSLM_LITE, RSLM_RESCORE_READING_A,
 *   RSLM_FULL_VECTOR, or 0.
 * On success *out receives the index; release it with rslm_index_destroy. */
rslm_status rslm_index_create(int32_t dim, int32_t nlist, const float* centroids,
                              int32_t score_bits, int32_t rescore_bits, uint32_t flags,
                              void* stream, rslm_index** out);

/* Fill *desc (host pointer). */
rslm_status rslm_index_describe(const rslm_index* index, rslm_index_desc* desc);

/* Fix the partition of every row and allocate the code storage (the IVF
 * layout of Sec. 5.5.1 step 1).  assignment: device [n] int32 in [0, nlist).
 * Rows of a partition are stored contiguously in row-id order, each
 * partition padded to a multiple of 128 rows.  Synchronizes `stream`.
 * May be called once per index. */
rslm_status rslm_index_reserve(rslm_index* index, const int32_t* assignment, int64_t n,
                               void* stream);

/* Encode rows [row_begin, row_begin + rows) (Sec. 3.4 pipeline on the
 * residual of Sec. 3.5): rotate (Sec. 3.1.3), EVT scale (Sec. 3.2), nearest
 * Lloyd-Max codeword, local scale ||r|| / ||u^|| as UE7M9 (Sec. 3.3,
 * 3.3.1), global scale as UE4M12 (Sec. 3.5.2), pack; then the rescoring
 * codes when rescore_bits > 0.  vectors: device [rows * dim] float32 holding
 * exactly those rows.  Chunks may come in any order; each row once. */
rslm_status rslm_encode(rslm_index* index, const float* vectors, int64_t row_begin, int64_t rows,
                        void* stream);

/* One call from vectors to an encoded index (the encode half of the
 * problem statement of Sec. 5.5.1: residuals of the vectors against their
 * partitions' centroids, coded as in Sec. 3.4 / 3.5): rslm_index_create
 * with (dim, nlist, centroids, score_bits, rescore_bits, flags), then
 * rslm_index_reserve(assignment, n), then rslm_encode of all n rows.
 * vectors: device [n * dim] float32; assignment: device [n] int32 in
 * [0, nlist); centroids: device [nlist * dim] float32 (copied).  The same
 * limits and errors as those calls; on any failure nothing is returned in
 * *out and the partial index is released.  Synchronizes `stream` (as
 * rslm_index_reserve does); the encode itself is queued on it. */
rslm_status rslm_encode_all(const float* vectors, const int32_t* assignment, int64_t n, int32_t dim,
                            int32_t nlist, const float* centroids, int32_t score_bits,
                            int32_t rescore_bits, uint32_t flags, void* stream, rslm_index** out);

/* Rotate query rows with the rotation of the scoring codes (which = 1) or of
 * the rescoring codes (which = 2) (Sec. 3.1.3; done once per query, Sec. 5.4).
 * queries: device [nq * dim] float32.  out: device [nq * padded_dim] (or
 * rescore_padded_dim) float32; the padded tail is written as 0 (Sec. 3.2:
 * trailing query terms are zeroed). */
rslm_status rslm_rotate_queries(const rslm_index* index, int32_t which, const float* queries,
                                int64_t nq, float* out, void* stream);

/* Probe (Sec. 5.5.1 step 3): for every query the nprobe partitions with the
 * largest <q, centroid>, ties to the lower partition id, in that order.
 * out_probes: device [nq * nprobe] int32; out_cs: device [nq * nprobe]
 * float32, the matching <q, centroid> values. */
rslm_status rslm_probe(const rslm_index* index, const float* queries, int64_t nq, int32_t nprobe,
                       int32_t* out_probes, float* out_cs, void* stream);

/* rslm_probe that allocates no device memory.  The paper has no counterpart:
 * this exists for callers that cannot allocate on the query path -- programs
 * whose device memory is all owned by another allocator (a framework's
 * caching allocator, a fixed budget handed out up front) and latency-critical
 * serving loops that forbid cudaMalloc / cudaFree because those calls can
 * synchronize the device.  Same arguments and results as rslm_probe; the
 * <q, centroid> scores of a query chunk live in a fixed 16 MiB device array
 * inside the library (held by every GPU that loads it, until exit) and are
 * computed by the library's own kernel rather than cuBLAS.
 * - The first call made with an index on a given device looks up that
 *   array's address on the device (cudaGetSymbolAddress); make that first
 *   call before any stream capture.
 * - All calls on a device share the array.  Calls whose GPU work may overlap
 *   (other streams, unordered host threads) race on it: serialise them.
 * - nlist above 4,194,304 (one query's scores must fit) returns
 *   RSLM_ERR_INVALID_ARG; larger nq is processed in chunks. */
rslm_status rslm_probe_noalloc(const rslm_index* index, const float* queries, int64_t nq,
                               int32_t nprobe, int32_t* out_probes, float* out_cs, void* stream);

/* Scan (Sec. 5.5.1 step 3 with the scores of Sec. 3.5.1-3.5.2): every row j
 * of every probed partition p scores s_j = G_j (cs_p + L_j <R q, u^_j>),
 * and the top k per query are kept.
 * qrot: device [nq * padded_dim] float32 (rslm_rotate_queries, which = 1).
 * probes / cs: device [nq * nprobe] as produced by rslm_probe (any valid
 * partition ids; out-of-range ids set the device error flag and are skipped).
 * out_ids: device [nq * k] int64; out_scores: device [nq * k] float32. */
rslm_status rslm_scan(const rslm_index* index, const float* qrot, int64_t nq, const int32_t* probes,
                      const float* cs, int32_t nprobe, int32_t k, int64_t* out_ids,
                      float* out_scores, void* stream);

/* Same inputs, outputs and results as rslm_scan, computed partition-major for
 * batches whose queries share partitions ("batched processing throughput" is
 * the IVF advantage the paper names in Sec. 1.2): the probe lists are
 * inverted per partition, each 128-row tile of codes is decoded once and
 * multiplied with up to 128 of its queries on the tensor cores (fp16 codeword
 * components, which are exact; queries split into fp16 hi + lo parts; fp32
 * accumulation), and only candidates at or above a per-query lower bound of
 * the k-th score (from a first pass over each query's first probed
 * partition) are kept.  A query with more than 16 k + 1024 such candidates is
 * re-scanned by the rslm_scan kernel.  Scores agree with rslm_scan within
 * float32 rounding; temporary device memory comes from the stream-ordered
 * allocator.  rslm_search picks this path when nq * nprobe >= 16 * nlist. */
rslm_status rslm_scan_batched(const rslm_index* index, const float* qrot, int64_t nq,
                              const int32_t* probes, const float* cs, int32_t nprobe, int32_t k,
                              int64_t* out_ids, float* out_scores, void* stream);

/* Rescore (Sec. 2.1, Sec. 5.2): each candidate j with first-stage score
 * s1_j = <q, a2_j> gets s2_j = G2_j (s1_j + L2_j <R2 q, u2^_j>) from its
 * 4-bit rescoring codes; the top k_final per query are returned.
 * qrot2: device [nq * rescore_padded_dim] (rslm_rotate_queries, which = 2).
 * cand_ids / cand_scores: device [nq * k] (rslm_scan output; id -1 = none).
 * out_ids: device [nq * k_final] int64; out_scores: device [nq * k_final]. */
rslm_status rslm_rescore(const rslm_index* index, const float* qrot2, int64_t nq,
                         const int64_t* cand_ids, const float* cand_scores, int32_t k,
                         int32_t k_final, int64_t* out_ids, float* out_scores, void* stream);

/* The whole query path: probe, rotate, scan, and (when rescore is nonzero and
 * the index has rescoring codes) rescore.  queries: device [nq * dim].
 * out_ids / out_scores: device [nq * k_final] (k_final = k without
 * rescoring).  Temporary device memory comes from the stream-ordered
 * allocator (cudaMallocAsync) and is released on `stream`. */
rslm_status rslm_search(const rslm_index* index, const float* queries, int64_t nq, int32_t nprobe,
                        int32_t k, int32_t rescore, int32_t k_final, int64_t* out_ids,
                        float* out_scores, void* stream);

/* Canonical codes of rows [row_begin, row_begin + rows): which = 1 scoring,
 * 2 rescoring.  codes: device [rows * code_bytes] uint8, row-major by row id,
 * the code of group i in the low nibble of byte i/2 when i is even, the high
 * nibble when odd (3-bit codes: bits 3i .. 3i + 2 of the row's byte
 * stream).  Code values index the codebook in ascending order (1-D) or in
 * lexicographic codeword order (2-D, 4-D).  local_scale / global_scale:
 * device [rows] uint16 (UE7M9 / UE4M12 codes). */
rslm_status rslm_export_codes(const rslm_index* index, int32_t which, int64_t row_begin,
                              int64_t rows, uint8_t* codes, uint16_t* local_scale,
                              uint16_t* global_scale, void* stream);

/* Inverse of rslm_export_codes: store externally produced codes and scales
 * for rows [row_begin, row_begin + rows) (after rslm_index_reserve). */
rslm_status rslm_import_codes(rslm_index* index, int32_t which, int64_t row_begin, int64_t rows,
                              const uint8_t* codes, const uint16_t* local_scale,
                              const uint16_t* global_scale, void* stream);

/* Decompression (Sec. 4; the inverse of the codec): the reconstructions of
 * rows [row_begin, row_begin + rows) from the stored codes and scales of
 * stage `which` (1: scoring, 2: rescoring), computed in float64 and written
 * to out: device [rows * dim] float32, row-major.
 *   which = 1: Ghat (a + Lhat R^T uhat) with a = the row's centroid (0 for
 *     RSLM_FULL_VECTOR);
 *   which = 2: Ghat2 (a2 + Lhat2 R2^T uhat2) with a2 = the stage-1
 *     reconstruction, or the stage-1 approximation with
 *     RSLM_RESCORE_READING_A.
 * Errors: RSLM_ERR_INVALID_ARG (bad which, range, NULL out),
 * RSLM_ERR_STATE before rslm_index_reserve.  Asynchronous on `stream`. */
rslm_status rslm_decompress(const rslm_index* index, int32_t which, int64_t row_begin, int64_t rows,
                            float* out, void* stream);

/* Codebook of a bit rate (Sec. 3.2) as the library uses it: host out
 * [K * g] float32 values (binary16-exact), K = 16.  *K_out, *g_out: host.
 * Needs no GPU. */
rslm_status rslm_codebook(int32_t bits, float* out, int32_t* K_out, int32_t* g_out);

/* Static tables of the rotation (Sec. 3.1.2) as the library uses them.
 * s1: host [256] int8 (+1/-1); perm: host [128] int32.  Needs no GPU. */
rslm_status rslm_rotation_tables(int8_t* s1, int32_t* perm);

/* E_max(D), the expected maximum of D iid |N(0,1)| (Sec. 3.2).  Needs no GPU. */
rslm_status rslm_e_max(int32_t dim, double* out);

/* Measurement support (no counterpart in the paper).  While enabled, every
 * launch of the dominant scan kernel of rslm_scan / rslm_scan_batched /
 * rslm_search on this index is bracketed by CUDA events recorded on the
 * launching stream.  rslm_profile_enable(index, 1) starts recording (and
 * clears earlier records), 0 stops.  rslm_profile_read waits for the recorded
 * events, returns the summed kernel time in *total_ms and the number of
 * launches in *launches (host pointers), writes the kernel's name into
 * kernel[kernel_len] (host, may be NULL) and clears the records. */
rslm_status rslm_profile_enable(rslm_index* index, int32_t on);
rslm_status rslm_profile_read(rslm_index* index, double* total_ms, int64_t* launches, char* kernel,
                              int32_t kernel_len);

/* Wait for `stream`, then report and clear the index's sticky device error
 * flag (RSLM_ERR_DEVICE) or a pending CUDA error (RSLM_ERR_CUDA). */
rslm_status rslm_sync(const rslm_index* index, void* stream);

/* Event counters of the index since its creation (a diagnostic for tests
 * and benchmarks; not a paper quantity).  Waits for the device, then writes
 * the first n (1..4) counters into out (host int64):
 *   out[0] queries whose tensor-core (batched) scan kept fewer than k
 *          candidates although the first probed partition gave a finite
 *          threshold; they are answered by the exact single-query scan.
 *          The two passes compute a row's score by the same arithmetic, so
 *          a nonzero value means a fault of the batched path;
 *   out[1] queries whose batched candidate buffer overflowed (many scores at
 *          the threshold); also answered by the exact scan (expected, rare);
 *   out[2] queries whose fused-probe candidate list overflowed (many
 *          centroid scores tied at the bound); answered by the exact probe;
 *   out[3] rows whose exact score the tensor-core scan's hi-only mode
 *          recomputed after its bounded pass (the candidates whose upper
 *          bound reached the k-th largest lower bound; a cost figure).
 * RSLM_ERR_INVALID_ARG for a NULL argument or n outside [1, 4]. */
rslm_status rslm_counters(const rslm_index* index, int64_t* out, int32_t n);

/* Message of the last failing call on this thread ("" if none). */
const char* rslm_last_error(void);

/* Release the index and its device memory.  NULL is ignored. */
void rslm_index_destroy(rslm_index* index);

#ifdef __cplusplus
}
#endif

#endif /* RSLM_H_ */
