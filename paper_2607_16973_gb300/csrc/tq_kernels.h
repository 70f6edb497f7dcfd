// Host-side launchers of the CUDA kernels (internal to libtq.so).
#pragma once

#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>
#include <vector>

namespace tq {

struct FilterDev {
  int64_t n = 0;
  int block = 64;
  int64_t n_tenants = 0;  // T distinct tenant ids
  int words = 0;          // ceil(T / 32)
  uint32_t* tenants = nullptr;    // device [T] sorted distinct raw ids
  uint32_t* dense = nullptr;      // device [n] dense tenant index per vector
  uint32_t* block_bits = nullptr; // device [nblocks * words]
};

// Encode (Sec. II-B steps 1-5): fused rotation GEMM + quantise + pack + scale;
// with cal_mu/cal_a (nullable, device [d]) a TQ+ calibration.
cudaError_t launch_encode(const float* X, int64_t n, int d, const float* R, const float* centroids,
                          const float* boundaries, int bits, int scale_mode, const float* cal_mu,
                          const float* cal_a, uint8_t* codes, float* scale, cudaStream_t s);

// Tensor-core encode (the same result, the rotation in TF32 with a
// three-product split on tcgen05): d a multiple of 32 in [128, kMaxD].  The
// plan (encode_plan_bytes(d) bytes, 16-byte aligned) holds a status word and
// R split into TF32 parts; launch_encode_tc records a timed-out wait in it.
bool encode_tc_supported(int d);
size_t encode_plan_bytes(int d);
cudaError_t launch_encode_plan(const float* R, int d, void* plan, cudaStream_t s);
cudaError_t launch_encode_tc(const float* X, int64_t n, int d, const void* plan, const float* centroids,
                             const float* boundaries, int bits, int scale_mode, const float* cal_mu,
                             const float* cal_a, uint8_t* codes, float* scale, cudaStream_t s);

// Query rotation on the tensor cores for batches of kRotTcMinBatch or more
// (d as for the tensor-core encoder): q' = R q in TF32 with the three-product
// split, the contraction split over rotate_tc_splits(nq, d) CTAs whose
// partial products (part, rotate_tc_part_bytes bytes; none with one split,
// which writes `out` directly) are added in a fixed order.  Clears the
// status word and zeroes `n_counters` merge counters.
bool rotate_tc_applies(int64_t nq, int d);
int rotate_tc_splits(int64_t nq, int d);
size_t rotate_tc_part_bytes(int64_t nq, int d);
cudaError_t launch_rotate_tc(const float* Q, int64_t nq, int d, const float* R, float* out, float* part,
                             int* status, int* counters, int64_t n_counters, cudaStream_t s);

// TQ+ calibration (Sec. II-B): per-coordinate shift mu and scale a from n
// rows, into device [d] arrays; ws of calibrate_workspace(n, d) bytes.
size_t calibrate_workspace(int64_t n, int d);
cudaError_t launch_calibrate(const float* X, int64_t n, int d, const float* R, float* mu, float* a, void* ws,
                             cudaStream_t s);
// Queries of a TQ+ search: qrot *= a in place, bias[q] = sum_j qrot_j mu_j.
cudaError_t launch_calib_query(float* qrot, int64_t nq, int d, const float* mu, const float* a, float* bias,
                               cudaStream_t s);

// q' = R q for nq queries: out [nq * d] float32.  Also zeroes the status word
// and `n_counters` merge counters (each nullable) for the search it starts.
cudaError_t launch_rotate(const float* Q, int64_t nq, int d, const float* R, float* out, int* status,
                          int* counters, int64_t n_counters, cudaStream_t s);

// Per-query allow bitmaps over the dense tenant index: out [nq * words].
cudaError_t launch_allow_bits(const FilterDev& f, const int64_t* allow_off,
                              const uint32_t* allow_tenants, int64_t nq, uint32_t* out,
                              cudaStream_t s);

// Filter build: dense index per vector and per-block tenant bitmaps.
cudaError_t launch_filter_build(const uint32_t* tenant_ids, FilterDev& f, cudaStream_t s);
// Rows f.n .. f.n+n_new-1 (ids tenant_ids[0 .. n_new-1], every one already in
// f.tenants) into dense and block_bits, which must have room for them.
cudaError_t launch_filter_extend(const uint32_t* tenant_ids, int64_t n_new, const FilterDev& f, cudaStream_t s);
// The raw tenant id of each of f's n rows into raw [f.n].
cudaError_t launch_filter_raw_ids(const FilterDev& f, uint32_t* raw, cudaStream_t s);

// LUT scan: per-CTA top-k candidates [nq][grid_x][k] (score, id).  `del`
// (nullable) is the tombstone bitmap: rows whose bit is set are skipped.
// With a filter, `allow_bits` [nq * f->words] are the queries' allow bitmaps
// and `bmask` [nq * filter_mask_words(*f)] their block masks.  `fix` selects
// the fixed-point byte-pair table for 4-bit codes (else the exact fp32 one).
// `err` is the search status word the scan's bounded waits report to.  The
// last CTA of each query merges the CTA lists into out_ids/out_scores
// (written as ext[row] with an id map); `counters` [nq] must be zero (the
// query rotation zeroes them).  `bias` [nq] (nullable): a TQ+ search's
// per-query term, added to each raw score before the per-vector scale.
int scan_lut_grid_x(int64_t nq, int64_t n, int k, int bits, int d);
cudaError_t launch_scan_lut(const float* qrot, int64_t nq, int d, const float* centroids, int bits,
                            const uint8_t* codes, const float* scale, int64_t n, const uint32_t* del,
                            const FilterDev* f, const uint32_t* allow_bits, const uint32_t* bmask, bool fix,
                            int k, int grid_x, float* cand_s, int32_t* cand_i, int* err, int* counters,
                            const uint64_t* ext, int64_t* out_ids, float* out_scores, const float* bias,
                            cudaStream_t s, cudaEvent_t ev0, cudaEvent_t ev1);

// The 4-bit lookup scan with the rotated query folded into per-byte-position
// tables (k_scan_fold): bits 4, d >= 256 and a multiple of 32, k <= kFoldMaxK,
// codes 16-byte aligned, n below 2^31 less two passes.  Arguments and
// results as launch_scan_lut; grid_x from scan_fold_grid_x.
bool fold_supported(int bits, int d, int k, int64_t n);
int scan_fold_grid_x(int64_t nq, int64_t n);
cudaError_t launch_scan_fold(const float* qrot, int64_t nq, int d, const float* centroids, const uint8_t* codes,
                             const float* scale, int64_t n, const uint32_t* del, const FilterDev* f,
                             const uint32_t* allow_bits, const uint32_t* bmask, int k, int grid_x, float* cand_s,
                             int32_t* cand_i, int* err, int* counters, const uint64_t* ext, int64_t* out_ids,
                             float* out_scores, const float* bias, cudaStream_t s, cudaEvent_t ev0,
                             cudaEvent_t ev1);

// Per-query bitmap over the filter's blocks: bit b set when block b holds a
// tenant the query allows.  out [nq * filter_mask_words(f)].
int filter_mask_words(const FilterDev& f);
cudaError_t launch_block_mask(const FilterDev& f, const uint32_t* allow, int64_t nq, uint32_t* mask,
                              cudaStream_t s);

// Final merge of per-CTA candidates into sorted top-k; with `ext` (nullable)
// the rows are written as ext[row].
cudaError_t launch_merge(const float* cand_s, const int32_t* cand_i, int64_t nq, int per_query,
                         int k, const uint64_t* ext, int64_t* out_ids, float* out_scores, cudaStream_t s);

// Merge of S sources x m candidates per query ([S][nq][m]) with global int64
// ids (-1 = padding).
cudaError_t launch_merge_global(const float* cand_s, const int64_t* cand_i, int64_t S, int64_t nq, int64_t m,
                                int k, int64_t* out_ids, float* out_scores, cudaStream_t s);

// Tensor-core decode-GEMM scan (bits 2, 4, 8; k <= kMaxKMma).  With
// allow_bits [nq * words] (and the filter's dense tenant index) a vector whose
// tenant the query does not allow never enters its list.
bool mma_supported(int bits, int d, int k);
int scan_mma_grid_x(int64_t nq, int64_t n, int k, int bits);
size_t mma_qpack_bytes(int64_t nq, int d);
cudaError_t launch_scan_mma(const float* qrot, int64_t nq, int d, const float* centroids, int bits,
                            const uint8_t* codes, const float* scale, int64_t n, const uint32_t* del,
                            const uint32_t* dense, const uint32_t* allow_bits, int words, const float* bias,
                            int k, int grid_x, void* qpack, float* cand_s, int32_t* cand_i, int* err, cudaStream_t s,
                            cudaEvent_t ev0, cudaEvent_t ev1);

int device_sm_count();
cudaError_t set_max_dynamic_smem(const void* func, int bytes);

// cudaMalloc that fails while the calling thread's tq_debug_fail_allocs
// count is positive (testing hook for the out-of-memory paths).
cudaError_t dev_malloc(void** p, size_t bytes);

// One CTA that waits, with the scans' bounded wait, on an mbarrier nothing
// completes (testing hook for the timeout path).
cudaError_t launch_debug_wait(long long budget, int* status, cudaStream_t s);

}  // namespace tq

// Opaque handle of the C ABI (include/tq.h): the filter's device arrays and
// the device they live on.
struct tq_filter {
  tq::FilterDev f;
  int device = 0;
  int64_t cap = 0;                     // rows dense / block_bits have room for
  std::vector<uint32_t> tenants_host;  // host copy of f.tenants
};
