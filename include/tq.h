/*
 * tq.h - C ABI of the GB300 TurboQuant search library (libtq.so).
 *
 * The library implements the data-parallel hot path of TurboQuant as studied
 * in "TurboVec: A Case Study in Cost-Efficient Private Retrieval for
 * Enterprise RAG via Codebook-Oblivious Quantization" (arXiv 2607.16973):
 *
 *   Sec. II-B, steps 1-5: normalise (keep the norm), rotate by a fixed random
 *     orthogonal R, quantise every coordinate with a Lloyd-Max codebook derived
 *     from the analytic coordinate marginal (no corpus data), bit-pack, and
 *     score with a per-vector length-renormalisation scalar;
 *   Sec. III-A/III-B: flat (brute-force) top-k inner-product search with an
 *     allowlist of tenants passed to the scan; blocks with no allowed vector
 *     are skipped before scoring, disallowed vectors in scored blocks never
 *     enter the top-k;
 *   Sec. III-C: the add() / search() / search(allowlist) operations.
 *
 * Conventions shared by every call:
 *  - Sizes are element counts.  d must be a multiple of 32 with 32 <= d <= 8192;
 *    bits is 2, 3, 4 or 8.
 *  - "host" pointers are ordinary CPU memory; "device" pointers are CUDA device
 *    memory of the current device, owned by the caller, which must keep them
 *    alive until the work queued on `stream` has finished.  Device pointers
 *    must be 16-byte aligned.
 *  - Device calls are asynchronous and stream-ordered on `stream` (a
 *    cudaStream_t passed as void*; NULL is the legacy default stream).  They
 *    validate every argument before queueing any work.
 *  - Errors: every call returns a tq_status.  TQ_EINVAL for invalid arguments
 *    (nothing is queued), TQ_ECUDA when the CUDA runtime reports an error,
 *    TQ_ENOMEM when a library-owned allocation fails, TQ_EUNSUPPORTED for a
 *    valid request this build cannot serve.  tq_last_error() returns a
 *    thread-local message for the last non-OK status of the calling thread.
 *    No call aborts, prints or lets a C++ exception escape.
 *  - Packed codes: row i holds d*bits/8 bytes, a little-endian bit stream in
 *    which coordinate j occupies bits [bits*j, bits*j + bits).  At d = 1536,
 *    bits = 4 that is 768 bytes per vector (Sec. II-B step 4).
 */
#ifndef TQ_H
#define TQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum tq_status {
  TQ_OK = 0,
  TQ_EINVAL = 1,
  TQ_ENOMEM = 2,
  TQ_ECUDA = 3,
  TQ_ETIMEOUT = 4,
  TQ_EUNSUPPORTED = 5
} tq_status;

/* Coordinate marginal the codebook is fitted to (Sec. II-A: "Beta/Gaussian
 * marginals after random rotation"; Sec. II-B step 3). */
enum { TQ_MARGINAL_BETA = 0, TQ_MARGINAL_GAUSS = 1 };

/* Per-vector scoring scalar (Sec. II-B step 5, "length-renormalized scoring"):
 *  NORM      scale = ||x|| / ||c[code]||   (reconstruction keeps the length of x)
 *  NONE      scale = ||x||                 (no renormalisation)
 *  UNBIASED  scale = ||x|| / <y, c[code]>  (self inner product is exact)
 * A zero row gets scale 0 in every mode. */
enum { TQ_SCALE_NORM = 0, TQ_SCALE_NONE = 1, TQ_SCALE_UNBIASED = 2 };

/* Search kernels: AUTO picks by batch size; LUT forces the per-query lookup
 * scan, MMA forces the tensor-core decode-GEMM scan (used by tests).
 * LUT_FIXED is the lookup scan with, for 4-bit codes at d >= 512, a table of
 * 15-bit fixed-point centroid values (each centroid rounded to a step near
 * max|c| / 16383, chosen to make the largest rounding error small: about
 * 6e-7 for the d = 1536 codebook; the score error is that rounding error
 * weighted by the rotated query, about 2.5e-7 rms for unit queries).  It
 * moves half the shared-memory bytes of the exact fp32 table per code but
 * needs more instructions per code.  LUT_FOLD is the lookup scan for 4-bit
 * codes (d >= 256, k <= 32, n < 2^31 - 13312) with the rotated query folded
 * into one float32 table per packed-byte position, T_m[x] = q'_2m c[x & 15]
 * + q'_2m+1 c[x >> 4] (Sec. II-B step 5): one 4-byte lookup and one add per
 * packed byte, built 256 coordinates at a time; TQ_EUNSUPPORTED where it does
 * not apply.  AUTO does not pick it: the byte-pair scan is faster on GB300. */
enum { TQ_PATH_AUTO = 0, TQ_PATH_LUT = 1, TQ_PATH_MMA = 2, TQ_PATH_LUT_FIXED = 3, TQ_PATH_LUT_FOLD = 4 };

typedef struct tq_filter tq_filter; /* opaque, library-owned */

/* Thread-local, NUL-terminated message describing the calling thread's last
 * non-OK status; "" if none.  The pointer stays valid until the next call. */
const char* tq_last_error(void);

/* ABI version of this header (major * 100 + minor). */
int tq_version(void);

/*
 * tq_codebook - Lloyd-Max scalar quantiser of the rotated-coordinate marginal
 * (Sec. II-B step 3; Sec. II-A: derived analytically, no corpus-dependent
 * training).  Host-only, deterministic, takes no data.
 *   d          dimension (>= 8); selects the marginal f_d(x) proportional to
 *              (1 - x^2)^((d-3)/2) on [-1, 1] (BETA) or N(0, 1/d) (GAUSS)
 *   bits       1..8; L = 2^bits levels
 *   marginal   TQ_MARGINAL_BETA or TQ_MARGINAL_GAUSS
 *   centroids  host out [L], ascending, symmetric (c_i = -c_{L-1-i})
 *   boundaries host out [L-1], t_i = (c_i + c_{i+1}) / 2; coordinate y maps to
 *              code #{i : t_i < y}
 *   distortion host out, per-coordinate mean squared error (nullable)
 * Returns TQ_EINVAL on bad d/bits/marginal or a NULL required pointer.
 */
tq_status tq_codebook(int d, int bits, int marginal, float* centroids,
                      float* boundaries, double* distortion);

/*
 * tq_rotation - the "fixed random orthogonal matrix R" of Sec. II-B step 2.
 * Host-only.  R = Q diag(sign(diag(U))) where G = Q U is the QR factorisation
 * of a d x d standard Gaussian matrix filled row-major from splitmix64(seed)
 * through Box-Muller (pair p: a = out(2p), b = out(2p+1),
 * u1 = ((a>>11)+1) 2^-53, u2 = (b>>11) 2^-53, g = sqrt(-2 ln u1) (cos, sin)(2 pi u2)).
 *   d     dimension (>= 2, <= 8192)
 *   seed  generator seed
 *   R     host out [d*d] float32, row-major; the rotation is y = R x
 * Computed in float64 and rounded once.
 */
tq_status tq_rotation(int d, uint64_t seed, float* R);

/*
 * tq_encode - add(): encode n rows (Sec. II-B steps 1-5).
 * For each row x: n = ||x||; y = R x / n (y = 0 if n = 0); code_j =
 * #{i : boundaries[i] < y_j}; pack; scale per scale_mode.
 *   X           device [n*d] float32, row-major
 *   n           rows (>= 0; 0 is a no-op)
 *   R           device [d*d] float32 row-major (tq_rotation's layout)
 *   centroids   device [2^bits] float32, ascending
 *   boundaries  device [2^bits - 1] float32, ascending
 *   bits        2, 3, 4 or 8
 *   scale_mode  TQ_SCALE_*
 *   codes       device out [n * d*bits/8] uint8
 *   scale       device out [n] float32
 * y is computed in float32 (FFMA); a coordinate within ~1e-6 of a boundary may
 * land in either neighbouring cell.
 */
tq_status tq_encode(const float* X, int64_t n, int d, const float* R,
                    const float* centroids, const float* boundaries, int bits,
                    int scale_mode, uint8_t* codes, float* scale, void* stream);

/*
 * TQ+ calibration (Sec. II-B, "TQ+ calibration and data dependence"): the
 * paper fits per-coordinate shift and scale parameters from the first batch
 * of indexed vectors so that the coordinate quantiles match the canonical
 * marginal, keeping only first and second moments; it gives no formula.  This
 * library's reading: over the batch's non-zero rows, y = R x / ||x||;
 * mu_j = mean of y_j, sigma_j = its population standard deviation, a_j =
 * sigma_j sqrt(d) (the canonical marginal's spread is 1/sqrt(d)), a_j = 1
 * where sigma_j = 0 (mu = 0, a = 1 without a non-zero row).  Encoding then
 * quantises z_j = (y_j - mu_j) / a_j with the canonical codebook, and the
 * reconstruction is a_j c[code_j] + mu_j.
 *
 * tq_calibrate_workspace  bytes of device scratch tq_calibrate needs for n rows
 * tq_calibrate   X device [n*d] float32 (n >= 1), R as for tq_encode;
 *                mu, a device out [d] float32; deterministic (fixed summation
 *                order).
 * tq_encode_ex   tq_encode with a calibration (cal_mu, cal_a device [d], or
 *                both NULL for plain TurboQuant): codes of z, and the
 *                per-vector scalar (scale_mode) taken on the reconstruction.
 */
tq_status tq_calibrate_workspace(int64_t n, int d, size_t* bytes);
tq_status tq_calibrate(const float* X, int64_t n, int d, const float* R, float* mu, float* a,
                       void* workspace, size_t ws_bytes, void* stream);
tq_status tq_encode_ex(const float* X, int64_t n, int d, const float* R,
                       const float* centroids, const float* boundaries, int bits,
                       int scale_mode, const float* cal_mu, const float* cal_a,
                       uint8_t* codes, float* scale, void* stream);

/*
 * Tensor-core encode: tq_encode_ex with the rotation (Sec. II-B step 2) on the
 * tensor cores in TF32.  TF32 keeps 10 mantissa bits, so each operand is split
 * into two TF32 parts, v = v_hi + v_lo (v_hi = tf32(v), v_lo = tf32(v - v_hi)),
 * and y = x_hi.R_hi + x_hi.R_lo + x_lo.R_hi is accumulated in float32: a
 * relative error of a few 2^-22 per product, so, as with tq_encode, a
 * coordinate within ~1e-6 of a boundary may land in either neighbouring cell.
 *
 * tq_encode_plan_bytes  device bytes of a plan for dimension d; TQ_EUNSUPPORTED
 *                unless d is a multiple of 32 in [128, 8192]
 * tq_encode_plan R device [d*d] float32 (tq_rotation's layout); plan: caller-
 *                owned device memory, 16-byte aligned, of plan_bytes >=
 *                tq_encode_plan_bytes(d).  Writes a status word and R split
 *                into R_hi and R_lo.  The plan depends on R only: build it
 *                once per index, keep it while encoding.
 * tq_encode_planned  the arguments of tq_encode_ex with the plan in place of
 *                R (d must be the plan's); same results and argument rules.
 *                Its waits are bounded: one that gives up (which does not
 *                happen in normal operation) is recorded in the plan's status
 *                word, and that call's codes are invalid.
 * tq_encode_check  waits for `stream`, then returns TQ_ETIMEOUT if an encode
 *                with this plan gave up since the plan was built or last
 *                checked (clearing the record), else TQ_OK.
 */
tq_status tq_encode_plan_bytes(int d, size_t* bytes);
tq_status tq_encode_plan(const float* R, int d, void* plan, size_t plan_bytes, void* stream);
tq_status tq_encode_planned(const float* X, int64_t n, int d, const void* plan,
                            const float* centroids, const float* boundaries, int bits,
                            int scale_mode, const float* cal_mu, const float* cal_a,
                            uint8_t* codes, float* scale, void* stream);
tq_status tq_encode_check(const void* plan, void* stream);

/*
 * tq_filter_build - per-corpus tenant filter for search(allowlist=...)
 * (Sec. III-B: filtering at vector-block granularity).
 *   tenant_ids  device [n] uint32: the tenant of each vector
 *   n           vectors (>= 1)
 *   block       vectors per filter block: 32 or 64 (the paper uses 32)
 *   out         host out: a new library-owned handle; free with
 *               tq_filter_destroy
 * The handle holds the sorted distinct tenant ids (T of them), each vector's
 * dense tenant index and a T-bit tenant bitmap per block, all in device
 * memory.  Synchronises `stream` (the distinct ids are counted on the host).
 */
tq_status tq_filter_build(const uint32_t* tenant_ids, int64_t n, int block,
                          tq_filter** out, void* stream);

/*
 * tq_filter_append - online ingest for the filter (Sec. III-A: indexes take
 * new vectors without a rebuild): rows n .. n+n_new-1 of the corpus get the
 * tenants tenant_ids[0 .. n_new-1] (device uint32 [n_new]).  When every
 * tenant is already known the new rows' dense indices and block bits are
 * written in place (a block shared with earlier rows keeps their bits), the
 * arrays doubling when full; a tenant the filter has not seen changes the
 * sorted tenant list, so the filter is rebuilt from all rows.  Either way the
 * result equals tq_filter_build over all n+n_new rows.  Synchronises
 * `stream`; on failure the filter is unchanged.  The caller ensures no queued
 * search still uses the handle.
 */
tq_status tq_filter_append(tq_filter* filter, const uint32_t* tenant_ids, int64_t n_new,
                           void* stream);

/* Frees a handle from tq_filter_build (NULL is a no-op).  The caller ensures
 * no queued search still uses it. */
tq_status tq_filter_destroy(tq_filter* filter);

/* Reports a handle's vector count, block size and distinct tenant count
 * (each out pointer nullable). */
tq_status tq_filter_info(const tq_filter* filter, int64_t* n, int* block,
                         int64_t* n_tenants);

/*
 * tq_search_workspace - bytes of device scratch tq_search needs for these
 * sizes on the current device (query rotation, allow bitmaps, per-CTA top-k
 * candidates).  filter may be NULL (unfiltered).
 */
tq_status tq_search_workspace(int64_t nq, int64_t n, int d, int bits, int k,
                              const tq_filter* filter, size_t* bytes);

/*
 * tq_search - search() / search(allowlist=...): top-k inner product of each
 * query against the encoded corpus (Sec. II-B step 5, Sec. III-B).
 * score(q, i) = scale[i] * sum_j (R q)_j * centroids[code_ij]; the k best
 * allowed vectors per query by (score descending, id ascending).
 *   Q              device [nq*d] float32 queries (not quantised)
 *   nq             queries (>= 0; 0 is a no-op)
 *   R, centroids   as for tq_encode
 *   codes          device [n * d*bits/8] packed codes (tq_encode output)
 *   scale          device [n] float32, or NULL for scale 1
 *   n              corpus vectors (>= 1)
 *   filter         NULL (every vector allowed) or a handle built for these
 *                  n vectors
 *   allow_off      device [nq+1] int64 CSR offsets into allow_tenants
 *                  (required iff filter != NULL; allow_off[0] = 0, non-decreasing)
 *   allow_tenants  device uint32 tenant ids allowed per query; ids absent from
 *                  the corpus are ignored; an empty list allows nothing
 *   k              1..256
 *   out_ids        device out [nq*k] int64, -1 where fewer than k vectors are allowed
 *   out_scores     device out [nq*k] float32, -INFINITY where out_ids is -1
 *   workspace      device scratch of ws_bytes >= tq_search_workspace(...)
 * Kernels (TQ_PATH_AUTO): batches of 16 or more queries over 2-, 4- or 8-bit
 * codes with d a multiple of 64 and k <= 64 run the tensor-core scan (fp16
 * products, float32 accumulation), filtered or not; the rest run the lookup
 * scan (float32 sums).
 */
tq_status tq_search(const float* Q, int64_t nq, int d, const float* R,
                    const float* centroids, int bits, const uint8_t* codes,
                    const float* scale, int64_t n, const tq_filter* filter,
                    const int64_t* allow_off, const uint32_t* allow_tenants,
                    int k, int64_t* out_ids, float* out_scores, void* workspace,
                    size_t ws_bytes, void* stream);

/*
 * tq_search_ex - tq_search over an id-mapped index (Sec. III-A: external
 * uint64 ids, O(1) deletion) and/or a TQ+ index (Sec. II-B).  Same arguments
 * and results as tq_search, plus:
 *   deleted   device [ceil(n/32)] uint32 tombstone bitmap, or NULL: bit i % 32
 *             of word i / 32 set means row i is deleted and is never returned
 *             (like a vector whose tenant is not allowed)
 *   ext_ids   device [n] uint64 external id of each row, or NULL: results are
 *             written as ext_ids[row] (bit pattern in the int64 out_ids);
 *             the ranking tie-break stays on the row (insertion order), and
 *             -1 (all ones) still marks an empty slot, so it must not be used
 *             as an external id
 *   cal_mu, cal_a  device [d] float32 each, or both NULL: the TQ+
 *             calibration the codes were encoded with (tq_encode_ex); the
 *             scores are then those of the reconstruction a_j c[code_j] + mu_j
 * tq_search(...) is tq_search_ex(..., NULL, NULL, NULL, NULL, ...).  A
 * tq_idmap handle (below) keeps the first two arrays and the id -> row map.
 */
tq_status tq_search_ex(const float* Q, int64_t nq, int d, const float* R,
                       const float* centroids, int bits, const uint8_t* codes,
                       const float* scale, int64_t n, const tq_filter* filter,
                       const int64_t* allow_off, const uint32_t* allow_tenants,
                       const uint32_t* deleted, const uint64_t* ext_ids,
                       const float* cal_mu, const float* cal_a,
                       int k, int64_t* out_ids, float* out_scores, void* workspace,
                       size_t ws_bytes, void* stream);

/*
 * tq_search_host - tq_search_ex for queries and results in host memory: the
 * search() call of a serving process whose requests arrive in host memory.
 * Queues, on `stream`, the query transfer, the search and the result
 * transfer; returns without waiting (synchronise `stream` before reading the
 * results).  Page-locked host buffers are used in place: the kernels read the
 * queries (batches below 16, whose rotation runs on plain loads) and write
 * the results (when both result buffers are page-locked) over the host link,
 * with no copy operations; otherwise the queries and results are copied
 * through the device staging buffer (asynchronously when page-locked).
 *   Q_host       host [nq*d] float32 queries
 *   ids_host     host out [nq*k] int64;  scores_host  host out [nq*k] float32
 *   staging      device scratch of staging_bytes >= tq_search_host_staging()
 *                (the device copies of the queries and results, where used)
 *   the other arguments as for tq_search_ex (R, centroids, codes, scale,
 *   allow_off, allow_tenants, deleted, ext_ids, cal_mu, cal_a and workspace
 *   are device memory).
 * The host buffers must stay valid, and the queries unchanged, until the
 * search has run.
 */
tq_status tq_search_host_staging(int64_t nq, int d, int k, size_t* bytes);
tq_status tq_search_host(const float* Q_host, int64_t nq, int d, const float* R,
                         const float* centroids, int bits, const uint8_t* codes,
                         const float* scale, int64_t n, const tq_filter* filter,
                         const int64_t* allow_off, const uint32_t* allow_tenants,
                         const uint32_t* deleted, const uint64_t* ext_ids,
                         const float* cal_mu, const float* cal_a, int k,
                         int64_t* ids_host, float* scores_host, void* staging,
                         size_t staging_bytes, void* workspace, size_t ws_bytes,
                         void* stream);

/*
 * tq_idmap - the id map of an id-mapped index (Sec. III-A): external uint64
 * ids for rows 0, 1, 2, ... in insertion order, O(1) lookup and deletion.
 * Library-owned: a host hash map id -> row plus two device arrays sized for
 * `capacity` rows, the external ids [capacity] uint64 and the tombstone
 * bitmap [ceil(capacity/32)] uint32 (zero = live), which tq_idmap_device
 * returns for tq_search_ex.  Rows are never reused: a deleted row stays
 * tombstoned, and its id may be added again as a new row.  A handle is not
 * thread-safe: calls on one handle must be serialised by the caller and
 * queue their copies on one stream (or be synchronised between streams), and
 * a search that reads the device arrays must be ordered (same stream, or
 * synchronised) after the add or remove whose effect it should see.  Removal
 * is O(1) per id on the host plus one copy of the touched bitmap words.
 *
 * tq_idmap_create  capacity rows (1..2^31-1) on the current device; device
 *                  arrays zero-initialised (synchronously).  TQ_ENOMEM if the
 *                  allocation fails.
 * tq_idmap_destroy frees everything (NULL is a no-op); the caller makes sure
 *                  no queued work still reads the device arrays.
 * tq_idmap_add     appends n_new rows with the given external ids (host array,
 *                  copied before the call returns); *first_row receives the
 *                  first new row.  TQ_EINVAL, with nothing changed, if the
 *                  capacity would be exceeded, an id is -1, or an id is already
 *                  live (in the map or twice in the batch).
 * tq_idmap_remove  deletes the rows of the given external ids (host array):
 *                  each live id leaves the map and its row's tombstone bit is
 *                  set on the device (stream-ordered); ids that are not live
 *                  are ignored.  *n_removed (nullable) receives how many were.
 * tq_idmap_lookup  row of a live external id, or -1.
 * tq_idmap_info    rows used, capacity, live ids (any pointer may be NULL).
 * tq_idmap_device  the device arrays (valid until tq_idmap_destroy).
 * tq_idmap_export  host copies of the rows' external ids (host [rows] uint64)
 *                  and the tombstone bitmap (host [ceil(rows/32)] uint32), for
 *                  persistence; reads only host state.
 * tq_idmap_import  fills an empty map with n rows from such copies (host
 *                  arrays; the live ids must be distinct and not -1; no bit
 *                  past row n may be set); the device copies are queued on
 *                  `stream`.  TQ_EINVAL, with the map left empty, otherwise.
 */
typedef struct tq_idmap tq_idmap;
tq_status tq_idmap_create(int64_t capacity, tq_idmap** out);
tq_status tq_idmap_destroy(tq_idmap* m);
tq_status tq_idmap_add(tq_idmap* m, const uint64_t* ext_ids, int64_t n_new, int64_t* first_row,
                       void* stream);
tq_status tq_idmap_remove(tq_idmap* m, const uint64_t* ext_ids, int64_t n, int64_t* n_removed,
                          void* stream);
tq_status tq_idmap_lookup(const tq_idmap* m, uint64_t ext_id, int64_t* row);
tq_status tq_idmap_info(const tq_idmap* m, int64_t* rows, int64_t* capacity, int64_t* live);
tq_status tq_idmap_device(const tq_idmap* m, const uint32_t** deleted, const uint64_t** ext_ids);
tq_status tq_idmap_export(const tq_idmap* m, uint64_t* ext_ids, uint32_t* deleted);
tq_status tq_idmap_import(tq_idmap* m, const uint64_t* ext_ids, const uint32_t* deleted, int64_t n,
                          void* stream);

/*
 * tq_search_static - tq_search without a workspace, for callers that cannot
 * allocate device memory (for example a C host program or plugin that is
 * handed device pointers for its inputs and outputs but owns no allocator, or
 * a serving loop that must not call cudaMalloc, which can block, synchronise
 * the device or fail under memory pressure mid-request).  The paper has no
 * counterpart: it is an interface convenience of this library.
 * Same arguments and results as tq_search (always the lookup scan: the
 * byte-pair one, or the fixed-point table under TQ_PATH_LUT_FIXED; never the
 * query-folded one), minus workspace/ws_bytes.  Its scratch is one 8 MiB device array per GPU; the
 * call allocates nothing.  Sizes whose scratch (about nq*d*4 bytes of rotated
 * queries plus nq*k*8 bytes per scan CTA of candidates) exceeds 8 MiB return
 * TQ_EINVAL with the byte counts.  The first call on each device looks the
 * array's device address up (make it before any stream capture); under CUDA's
 * lazy module loading (the default) that first call is also the one that
 * reserves the array on the device, which then holds it until the process
 * exits, so make one warm-up call per device before serving (TQ_ENOMEM if the
 * device has no room for it).  All calls on a device share the array: calls
 * whose work overlaps on the GPU (two streams or two threads) race and must be
 * serialised by the caller.  The status for d > 2048 is TQ_EUNSUPPORTED, as
 * for tq_search.
 */
tq_status tq_search_static(const float* Q, int64_t nq, int d, const float* R,
                           const float* centroids, int bits, const uint8_t* codes,
                           const float* scale, int64_t n, const tq_filter* filter,
                           const int64_t* allow_off, const uint32_t* allow_tenants,
                           int k, int64_t* out_ids, float* out_scores, void* stream);

/*
 * tq_merge_topk - exact merge of per-shard top-k lists.  When the corpus is
 * split by contiguous row ranges (one shard per device, each searched with
 * tq_search), the k best of the whole corpus are the k best, by the same
 * (score descending, id ascending) order tq_search uses (Sec. III-B top-k),
 * of the union of every shard's k best with ids shifted to global rows.
 *   cand_ids     device [n_src*nq*m] int64 global ids, laid out [n_src][nq][m]
 *                (what an all-gather of every shard's [nq][m] result gives):
 *                candidate j of source s for query q is at (s*nq + q)*m + j;
 *                -1 marks an empty slot, which never displaces a real candidate
 *   cand_scores  device [n_src*nq*m] float32, same layout
 *   n_src        sources (1..4096)
 *   nq           queries (>= 0; 0 is a no-op)
 *   m            candidates per source and query (0..2^20)
 *   k            1..256
 *   out_ids      device out [nq*k] int64, -1 where fewer than k real candidates
 *   out_scores   device out [nq*k] float32, -INFINITY where out_ids is -1
 * Candidates are read-only; a (score, id) pair given twice is kept twice.
 */
tq_status tq_merge_topk(const int64_t* cand_ids, const float* cand_scores,
                        int64_t n_src, int64_t nq, int64_t m, int k,
                        int64_t* out_ids, float* out_scores, void* stream);

/*
 * tq_search_check - waits for `stream` and reports how the last tq_search that
 * used `workspace` ended on the GPU.  tq_search validates its arguments and
 * queues its kernels; the tensor-core scan's waits on its pipelines are
 * bounded (about 2 s of SM clock), and a wait that gives up stops the kernel
 * and records where in the workspace's status word instead of hanging.
 *   workspace  the device workspace passed to tq_search (16-byte aligned)
 * Returns TQ_OK, TQ_ETIMEOUT (the results of that search are invalid; the
 * context and the library stay usable) or TQ_ECUDA.  Every tq_search clears
 * the word before its kernels run.
 */
tq_status tq_search_check(const void* workspace, void* stream);

/* Testing hooks.  They exercise the failure paths without faulting the GPU.
 * tq_debug_fail_allocs(count): the calling thread's next `count` library-owned
 * device allocations (tq_filter_build) fail as out of memory (TQ_ENOMEM).
 * tq_debug_bounded_wait(budget_cycles, workspace, stream): queues one CTA that
 * waits, with the scans' bounded wait and a budget of budget_cycles SM cycles
 * (1 .. 4e9), on an mbarrier nothing completes; the wait gives up and records
 * its timeout in the workspace's status word, which tq_search_check reports. */
tq_status tq_debug_fail_allocs(int count);
tq_status tq_debug_bounded_wait(long long budget_cycles, void* workspace,
                                void* stream);

/* Selects the search kernels for later tq_search calls of the calling thread
 * (TQ_PATH_*).  AUTO is the default. */
tq_status tq_set_search_path(int path);

/* Records two caller-created CUDA events (cudaEvent_t passed as void*) on the
 * search stream immediately before and after the scan kernel of the calling
 * thread's later tq_search calls, for per-kernel timing.  NULL, NULL turns it
 * off. */
tq_status tq_profile_events(void* scan_start, void* scan_stop);

#ifdef __cplusplus
}
#endif

#endif /* TQ_H */
