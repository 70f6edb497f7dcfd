// C ABI entry points that queue device work: tq_encode, tq_filter_*,
// tq_search_workspace, tq_search / tq_search_ex.  Every argument is validated before any
// work is queued; CUDA errors come back as TQ_ECUDA with the runtime's text.
#include <cuda_runtime.h>

#include <algorithm>
#include <iterator>
#include <cstring>
#include <new>
#include <vector>

#include "tq_internal.h"
#include "tq_kernels.h"

namespace tq {
namespace {

tq_status cuda_fail(const char* where, cudaError_t e) {
  return fail(TQ_ECUDA, "%s: %s (%s)", where, cudaGetErrorString(e), cudaGetErrorName(e));
}

tq_status check_common(const char* fn, int d, int bits) {
  if (d < 32 || d > kMaxD || d % 32 != 0)
    return fail(TQ_EINVAL, "%s: d=%d must be a multiple of 32 in [32, %d]", fn, d, kMaxD);
  if (!valid_bits(bits)) return fail(TQ_EINVAL, "%s: bits=%d must be 2, 3, 4 or 8", fn, bits);
  return TQ_OK;
}

constexpr size_t kAlign = 256;
inline size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

struct SearchPlan {
  int grid_lut = 1, grid_mma = 0, grid_fold = 0;
  size_t off_status = 0, off_cnt = 0, off_bias = 0, off_rot = 0, off_part = 0, off_allow = 0, off_mask = 0,
         off_qpack = 0, off_cs = 0, off_ci = 0, total = 0;
  bool rot_tc = false;  // the query rotation runs on the tensor cores
};

// Workspace layout (both scan paths): status word | merge counters (one per
// query) | TQ+ query terms (one per query) | rotated queries | partial
// rotations (tensor-core rotation) | allow bitmaps | block masks | fp16 query
// tiles (tensor-core scan) | candidate scores | ids.
SearchPlan plan_search(int64_t nq, int64_t n, int d, int bits, int k, const tq_filter* filter) {
  SearchPlan p;
  p.grid_lut = scan_lut_grid_x(nq, n, k, bits, d);
  const bool mma = mma_supported(bits, d, k);
  p.grid_mma = mma ? scan_mma_grid_x(nq, n, k, bits) : 0;
  p.grid_fold = fold_supported(bits, d, k, n) ? scan_fold_grid_x(nq, n) : 0;
  const int per_query = std::max(std::max(p.grid_lut, p.grid_mma), p.grid_fold) * k;
  size_t off = 0;
  p.off_status = off;
  off = align_up(off + sizeof(int));
  p.off_cnt = off;
  off = align_up(off + (size_t)nq * sizeof(int));
  p.off_bias = off;
  off = align_up(off + (size_t)nq * sizeof(float));
  p.off_rot = off;
  off = align_up(off + (size_t)nq * d * sizeof(float));
  p.rot_tc = rotate_tc_applies(nq, d);
  p.off_part = off;
  if (p.rot_tc) off = align_up(off + rotate_tc_part_bytes(nq, d));
  p.off_allow = off;
  if (filter) off = align_up(off + (size_t)nq * filter->f.words * sizeof(uint32_t));
  p.off_mask = off;
  if (filter) off = align_up(off + (size_t)nq * filter_mask_words(filter->f) * sizeof(uint32_t));
  p.off_qpack = off;
  if (mma) off = align_up(off + mma_qpack_bytes(nq, d));
  p.off_cs = off;
  off = align_up(off + (size_t)nq * per_query * sizeof(float));
  p.off_ci = off;
  off = align_up(off + (size_t)nq * per_query * sizeof(int32_t));
  p.total = off;
  return p;
}

}  // namespace
}  // namespace tq

using tq::fail;

extern "C" tq_status tq_encode_ex(const float* X, int64_t n, int d, const float* R,
                                  const float* centroids, const float* boundaries, int bits,
                                  int scale_mode, const float* cal_mu, const float* cal_a, uint8_t* codes,
                                  float* scale, void* stream) {
  tq_status st = tq::check_common("tq_encode", d, bits);
  if (st != TQ_OK) return st;
  if (n < 0 || n > INT32_MAX) return fail(TQ_EINVAL, "tq_encode: n=%lld outside [0, 2^31-1]", (long long)n);
  if (scale_mode != TQ_SCALE_NORM && scale_mode != TQ_SCALE_NONE && scale_mode != TQ_SCALE_UNBIASED)
    return fail(TQ_EINVAL, "tq_encode: unknown scale_mode %d", scale_mode);
  if (n == 0) return tq::ok();
  if (!X || !R || !centroids || !boundaries || !codes || !scale)
    return fail(TQ_EINVAL, "tq_encode: NULL device pointer");
  if (!tq::aligned16(X) || !tq::aligned16(R) || !tq::aligned16(codes))
    return fail(TQ_EINVAL, "tq_encode: X, R and codes must be 16-byte aligned");
  if (((uintptr_t)scale & 3u) || ((uintptr_t)centroids & 3u) || ((uintptr_t)boundaries & 3u))
    return fail(TQ_EINVAL, "tq_encode: scale, centroids and boundaries must be 4-byte aligned");
  if ((cal_mu == nullptr) != (cal_a == nullptr))
    return fail(TQ_EINVAL, "tq_encode_ex: a TQ+ calibration needs both mu and a");
  if (((uintptr_t)cal_mu & 3u) || ((uintptr_t)cal_a & 3u))
    return fail(TQ_EINVAL, "tq_encode_ex: mu and a must be 4-byte aligned");
  cudaError_t e = tq::launch_encode(X, n, d, R, centroids, boundaries, bits, scale_mode, cal_mu, cal_a, codes,
                                    scale, (cudaStream_t)stream);
  if (e != cudaSuccess) return tq::cuda_fail("tq_encode", e);
  return tq::ok();
}

extern "C" tq_status tq_encode(const float* X, int64_t n, int d, const float* R, const float* centroids,
                               const float* boundaries, int bits, int scale_mode, uint8_t* codes, float* scale,
                               void* stream) {
  return tq_encode_ex(X, n, d, R, centroids, boundaries, bits, scale_mode, nullptr, nullptr, codes, scale, stream);
}

extern "C" tq_status tq_encode_plan_bytes(int d, size_t* bytes) {
  if (!bytes) return fail(TQ_EINVAL, "tq_encode_plan_bytes: NULL bytes");
  if (!tq::encode_tc_supported(d))
    return fail(TQ_EUNSUPPORTED, "tq_encode_plan_bytes: d=%d is not a multiple of 32 in [128, %d]", d, tq::kMaxD);
  *bytes = tq::encode_plan_bytes(d);
  return tq::ok();
}

extern "C" tq_status tq_encode_plan(const float* R, int d, void* plan, size_t plan_bytes, void* stream) {
  if (!tq::encode_tc_supported(d))
    return fail(TQ_EUNSUPPORTED, "tq_encode_plan: d=%d is not a multiple of 32 in [128, %d]", d, tq::kMaxD);
  if (!R || !plan) return fail(TQ_EINVAL, "tq_encode_plan: NULL device pointer");
  if (!tq::aligned16(R) || !tq::aligned16(plan)) return fail(TQ_EINVAL, "tq_encode_plan: R and plan must be 16-byte aligned");
  if (plan_bytes < tq::encode_plan_bytes(d))
    return fail(TQ_EINVAL, "tq_encode_plan: plan_bytes %zu < %zu", plan_bytes, tq::encode_plan_bytes(d));
  const cudaError_t e = tq::launch_encode_plan(R, d, plan, (cudaStream_t)stream);
  if (e != cudaSuccess) return tq::cuda_fail("tq_encode_plan", e);
  return tq::ok();
}

extern "C" tq_status tq_encode_planned(const float* X, int64_t n, int d, const void* plan,
                                       const float* centroids, const float* boundaries, int bits,
                                       int scale_mode, const float* cal_mu, const float* cal_a, uint8_t* codes,
                                       float* scale, void* stream) {
  tq_status st = tq::check_common("tq_encode_planned", d, bits);
  if (st != TQ_OK) return st;
  if (!tq::encode_tc_supported(d))
    return fail(TQ_EUNSUPPORTED, "tq_encode_planned: d=%d is not a multiple of 32 in [128, %d]", d, tq::kMaxD);
  if (n < 0 || n > INT32_MAX) return fail(TQ_EINVAL, "tq_encode_planned: n=%lld outside [0, 2^31-1]", (long long)n);
  if (scale_mode != TQ_SCALE_NORM && scale_mode != TQ_SCALE_NONE && scale_mode != TQ_SCALE_UNBIASED)
    return fail(TQ_EINVAL, "tq_encode_planned: unknown scale_mode %d", scale_mode);
  if (n == 0) return tq::ok();
  if (!X || !plan || !centroids || !boundaries || !codes || !scale)
    return fail(TQ_EINVAL, "tq_encode_planned: NULL device pointer");
  if (!tq::aligned16(X) || !tq::aligned16(plan) || !tq::aligned16(codes))
    return fail(TQ_EINVAL, "tq_encode_planned: X, plan and codes must be 16-byte aligned");
  if (((uintptr_t)scale & 3u) || ((uintptr_t)centroids & 3u) || ((uintptr_t)boundaries & 3u))
    return fail(TQ_EINVAL, "tq_encode_planned: scale, centroids and boundaries must be 4-byte aligned");
  if ((cal_mu == nullptr) != (cal_a == nullptr))
    return fail(TQ_EINVAL, "tq_encode_planned: a TQ+ calibration needs both mu and a");
  if (((uintptr_t)cal_mu & 3u) || ((uintptr_t)cal_a & 3u))
    return fail(TQ_EINVAL, "tq_encode_planned: mu and a must be 4-byte aligned");
  const cudaError_t e = tq::launch_encode_tc(X, n, d, plan, centroids, boundaries, bits, scale_mode, cal_mu, cal_a,
                                             codes, scale, (cudaStream_t)stream);
  if (e != cudaSuccess) return tq::cuda_fail("tq_encode_planned", e);
  return tq::ok();
}

extern "C" tq_status tq_encode_check(const void* plan, void* stream) {
  if (!plan) return fail(TQ_EINVAL, "tq_encode_check: NULL plan");
  if (!tq::aligned16(plan)) return fail(TQ_EINVAL, "tq_encode_check: plan must be 16-byte aligned");
  cudaStream_t s = (cudaStream_t)stream;
  int word = 0;
  cudaError_t e = cudaMemcpyAsync(&word, plan, sizeof(int), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e == cudaSuccess && word != 0) e = cudaMemsetAsync(const_cast<void*>(plan), 0, sizeof(int), s);
  if (e == cudaSuccess && word != 0) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return tq::cuda_fail("tq_encode_check", e);
  if (word == 0) return tq::ok();
  if (word / 1000 == TQ_ETIMEOUT)
    return fail(TQ_ETIMEOUT, "tq_encode_check: a bounded wait (site %d) gave up; those codes are invalid", word % 1000);
  return fail(TQ_ECUDA, "tq_encode_check: unexpected status word %d", word);
}

extern "C" tq_status tq_calibrate_workspace(int64_t n, int d, size_t* bytes) {
  if (!bytes) return fail(TQ_EINVAL, "tq_calibrate_workspace: NULL bytes");
  if (n < 1 || n > INT32_MAX) return fail(TQ_EINVAL, "tq_calibrate_workspace: n=%lld outside [1, 2^31-1]", (long long)n);
  if (d < 32 || d > tq::kMaxD || d % 32 != 0)
    return fail(TQ_EINVAL, "tq_calibrate_workspace: d=%d must be a multiple of 32 in [32, %d]", d, tq::kMaxD);
  *bytes = tq::calibrate_workspace(n, d);
  return tq::ok();
}

extern "C" tq_status tq_calibrate(const float* X, int64_t n, int d, const float* R, float* mu, float* a,
                                  void* workspace, size_t ws_bytes, void* stream) {
  size_t need = 0;
  tq_status st = tq_calibrate_workspace(n, d, &need);
  if (st != TQ_OK) return st;
  if (!X || !R || !mu || !a || !workspace) return fail(TQ_EINVAL, "tq_calibrate: NULL device pointer");
  if (!tq::aligned16(X) || !tq::aligned16(R) || !tq::aligned16(workspace))
    return fail(TQ_EINVAL, "tq_calibrate: X, R and workspace must be 16-byte aligned");
  if (((uintptr_t)mu & 3u) || ((uintptr_t)a & 3u)) return fail(TQ_EINVAL, "tq_calibrate: misaligned mu or a");
  if (ws_bytes < need) return fail(TQ_EINVAL, "tq_calibrate: workspace of %zu bytes, %zu needed", ws_bytes, need);
  const cudaError_t e = tq::launch_calibrate(X, n, d, R, mu, a, workspace, (cudaStream_t)stream);
  if (e != cudaSuccess) return tq::cuda_fail("tq_calibrate", e);
  return tq::ok();
}

extern "C" tq_status tq_filter_build(const uint32_t* tenant_ids, int64_t n, int block,
                                     tq_filter** out, void* stream) {
  if (!out) return fail(TQ_EINVAL, "tq_filter_build: NULL out");
  *out = nullptr;
  if (n < 1 || n > INT32_MAX) return fail(TQ_EINVAL, "tq_filter_build: n=%lld outside [1, 2^31-1]", (long long)n);
  if (block != 32 && block != 64) return fail(TQ_EINVAL, "tq_filter_build: block=%d must be 32 or 64", block);
  if (!tenant_ids) return fail(TQ_EINVAL, "tq_filter_build: NULL tenant_ids");
  cudaStream_t s = (cudaStream_t)stream;
  tq_filter* h = nullptr;
  try {
    std::vector<uint32_t> ids((size_t)n);
    cudaError_t e = cudaMemcpyAsync(ids.data(), tenant_ids, (size_t)n * sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return tq::cuda_fail("tq_filter_build: reading tenant ids", e);
    std::sort(ids.begin(), ids.end());
    ids.erase(std::unique(ids.begin(), ids.end()), ids.end());
    h = new tq_filter();
    cudaGetDevice(&h->device);
    h->cap = n;
    tq::FilterDev& f = h->f;
    f.n = n;
    f.block = block;
    f.n_tenants = (int64_t)ids.size();
    f.words = (int)((f.n_tenants + 31) / 32);
    const int64_t nblocks = (n + block - 1) / block;
    e = tq::dev_malloc(reinterpret_cast<void**>(&f.tenants), ids.size() * sizeof(uint32_t));
    if (e == cudaSuccess) e = tq::dev_malloc(reinterpret_cast<void**>(&f.dense), (size_t)n * sizeof(uint32_t));
    if (e == cudaSuccess)
      e = tq::dev_malloc(reinterpret_cast<void**>(&f.block_bits), (size_t)nblocks * f.words * sizeof(uint32_t));
    if (e != cudaSuccess) {
      tq_filter_destroy(h);
      cudaGetLastError();
      return fail(TQ_ENOMEM, "tq_filter_build: device allocation failed: %s", cudaGetErrorString(e));
    }
    e = cudaMemcpyAsync(f.tenants, ids.data(), ids.size() * sizeof(uint32_t), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = tq::launch_filter_build(tenant_ids, f, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);  // `ids` is freed on return
    if (e != cudaSuccess) {
      tq_filter_destroy(h);
      return tq::cuda_fail("tq_filter_build", e);
    }
    h->tenants_host = std::move(ids);
    *out = h;
    return tq::ok();
  } catch (const std::bad_alloc&) {
    if (h) tq_filter_destroy(h);
    return fail(TQ_ENOMEM, "tq_filter_build: out of host memory");
  }
}

// Appends rows to a filter.  Rows whose tenants the filter already knows are
// added in place: their dense indices and block bits are written, and the
// arrays grow (doubling) when they are full.  A new tenant changes the sorted
// tenant list and with it every dense index and the bitmap width, so then the
// filter is rebuilt from all rows' raw ids.  The old arrays stay in place
// until the new ones are complete, so a failure leaves the filter unchanged.
extern "C" tq_status tq_filter_append(tq_filter* h, const uint32_t* tenant_ids, int64_t n_new, void* stream) {
  if (!h) return fail(TQ_EINVAL, "tq_filter_append: NULL filter");
  if (n_new < 0 || n_new > INT32_MAX - h->f.n)
    return fail(TQ_EINVAL, "tq_filter_append: %lld rows + %lld new outside [0, 2^31-1]", (long long)h->f.n,
                (long long)n_new);
  if (n_new == 0) return tq::ok();
  if (!tenant_ids) return fail(TQ_EINVAL, "tq_filter_append: NULL tenant_ids");
  cudaStream_t s = (cudaStream_t)stream;
  tq::FilterDev& f = h->f;
  const int64_t n_total = f.n + n_new;
  uint32_t *dense = nullptr, *bits = nullptr, *tenants = nullptr, *raw = nullptr;
  auto release = [&] {
    cudaFree(dense);
    cudaFree(bits);
    cudaFree(tenants);
    cudaFree(raw);
  };
  try {
    std::vector<uint32_t> ids((size_t)n_new);
    cudaError_t e = cudaMemcpyAsync(ids.data(), tenant_ids, (size_t)n_new * sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return tq::cuda_fail("tq_filter_append: reading tenant ids", e);
    std::sort(ids.begin(), ids.end());
    ids.erase(std::unique(ids.begin(), ids.end()), ids.end());
    std::vector<uint32_t> merged;
    std::set_union(h->tenants_host.begin(), h->tenants_host.end(), ids.begin(), ids.end(),
                   std::back_inserter(merged));
    const bool same_tenants = merged.size() == h->tenants_host.size();
    const int64_t cap = n_total <= h->cap ? h->cap : std::min<int64_t>(INT32_MAX, std::max(n_total, 2 * h->cap));
    const int words = same_tenants ? f.words : (int)((merged.size() + 31) / 32);
    const int64_t cap_blocks = (cap + f.block - 1) / f.block;
    if (same_tenants && cap == h->cap) {  // room left: write the new rows in place
      e = tq::launch_filter_extend(tenant_ids, n_new, f, s);
      if (e == cudaSuccess) e = cudaStreamSynchronize(s);
      if (e != cudaSuccess) return tq::cuda_fail("tq_filter_append", e);
      f.n = n_total;
      return tq::ok();
    }
    e = tq::dev_malloc(reinterpret_cast<void**>(&dense), (size_t)cap * sizeof(uint32_t));
    if (e == cudaSuccess) e = tq::dev_malloc(reinterpret_cast<void**>(&bits), (size_t)cap_blocks * words * 4);
    if (e == cudaSuccess && !same_tenants)
      e = tq::dev_malloc(reinterpret_cast<void**>(&tenants), merged.size() * sizeof(uint32_t));
    if (e == cudaSuccess && !same_tenants)
      e = tq::dev_malloc(reinterpret_cast<void**>(&raw), (size_t)n_total * sizeof(uint32_t));
    if (e != cudaSuccess) {
      release();
      cudaGetLastError();
      return fail(TQ_ENOMEM, "tq_filter_append: device allocation failed: %s", cudaGetErrorString(e));
    }
    e = cudaMemsetAsync(bits, 0, (size_t)cap_blocks * words * 4, s);
    tq::FilterDev g = f;  // the grown (or rebuilt) filter
    g.dense = dense;
    g.block_bits = bits;
    if (same_tenants) {  // grow: copy the old rows' arrays, then add the new rows
      const int64_t old_blocks = (f.n + f.block - 1) / f.block;
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(dense, f.dense, (size_t)f.n * sizeof(uint32_t), cudaMemcpyDeviceToDevice, s);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(bits, f.block_bits, (size_t)old_blocks * words * 4, cudaMemcpyDeviceToDevice, s);
      if (e == cudaSuccess) e = tq::launch_filter_extend(tenant_ids, n_new, g, s);
    } else {  // rebuild from every row's raw id
      g.tenants = tenants;
      g.n_tenants = (int64_t)merged.size();
      g.words = words;
      g.n = n_total;
      if (e == cudaSuccess) e = tq::launch_filter_raw_ids(f, raw, s);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(raw + f.n, tenant_ids, (size_t)n_new * sizeof(uint32_t), cudaMemcpyDeviceToDevice, s);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(tenants, merged.data(), merged.size() * sizeof(uint32_t), cudaMemcpyHostToDevice, s);
      if (e == cudaSuccess) e = tq::launch_filter_build(raw, g, s);
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);  // `merged` is freed on return
    if (e != cudaSuccess) {
      cudaStreamSynchronize(s);
      release();
      return tq::cuda_fail("tq_filter_append", e);
    }
    cudaFree(raw);
    cudaFree(f.dense);
    cudaFree(f.block_bits);
    if (!same_tenants) {
      cudaFree(f.tenants);
      h->tenants_host = std::move(merged);
    }
    g.n = n_total;
    f = g;
    h->cap = cap;
    return tq::ok();
  } catch (const std::bad_alloc&) {
    cudaStreamSynchronize(s);
    release();
    return fail(TQ_ENOMEM, "tq_filter_append: out of host memory");
  }
}

extern "C" tq_status tq_filter_destroy(tq_filter* filter) {
  if (!filter) return tq::ok();
  cudaFree(filter->f.tenants);
  cudaFree(filter->f.dense);
  cudaFree(filter->f.block_bits);
  delete filter;
  return tq::ok();
}

extern "C" tq_status tq_filter_info(const tq_filter* filter, int64_t* n, int* block, int64_t* n_tenants) {
  if (!filter) return fail(TQ_EINVAL, "tq_filter_info: NULL filter");
  if (n) *n = filter->f.n;
  if (block) *block = filter->f.block;
  if (n_tenants) *n_tenants = filter->f.n_tenants;
  return tq::ok();
}

namespace {
tq_status check_search(int64_t nq, int64_t n, int d, int bits, int k) {
  tq_status st = tq::check_common("tq_search", d, bits);
  if (st != TQ_OK) return st;
  if (nq < 0 || nq > (1 << 24)) return fail(TQ_EINVAL, "tq_search: nq=%lld outside [0, 2^24]", (long long)nq);
  if (n < 1 || n > INT32_MAX - 1) return fail(TQ_EINVAL, "tq_search: n=%lld outside [1, 2^31-2]", (long long)n);
  if (k < 1 || k > tq::kMaxK) return fail(TQ_EINVAL, "tq_search: k=%d outside [1, %d]", k, tq::kMaxK);
  if (d > 2048) return fail(TQ_EUNSUPPORTED, "tq_search: d=%d > 2048 is not supported by this build", d);
  return TQ_OK;
}
}  // namespace

extern "C" tq_status tq_search_workspace(int64_t nq, int64_t n, int d, int bits, int k,
                                         const tq_filter* filter, size_t* bytes) {
  if (!bytes) return fail(TQ_EINVAL, "tq_search_workspace: NULL bytes");
  tq_status st = check_search(nq, n, d, bits, k);
  if (st != TQ_OK) return st;
  *bytes = tq::plan_search(nq, n, d, bits, k, filter).total;
  return tq::ok();
}

extern "C" tq_status tq_search_ex(const float* Q, int64_t nq, int d, const float* R,
                                  const float* centroids, int bits, const uint8_t* codes,
                                  const float* scale, int64_t n, const tq_filter* filter,
                                  const int64_t* allow_off, const uint32_t* allow_tenants,
                                  const uint32_t* deleted, const uint64_t* ext_ids, const float* cal_mu,
                                  const float* cal_a, int k, int64_t* out_ids, float* out_scores, void* workspace,
                                  size_t ws_bytes, void* stream) {
  tq_status st = check_search(nq, n, d, bits, k);
  if (st != TQ_OK) return st;
  if (nq == 0) return tq::ok();
  if (!Q || !R || !centroids || !codes || !out_ids || !out_scores || !workspace)
    return fail(TQ_EINVAL, "tq_search: NULL device pointer");
  if (!tq::aligned16(Q) || !tq::aligned16(R) || !tq::aligned16(codes) || !tq::aligned16(workspace))
    return fail(TQ_EINVAL, "tq_search: Q, R, codes and workspace must be 16-byte aligned");
  if (((uintptr_t)centroids & 3u) || ((uintptr_t)scale & 3u) || ((uintptr_t)out_scores & 3u) ||
      ((uintptr_t)out_ids & 7u) || ((uintptr_t)deleted & 3u) || ((uintptr_t)ext_ids & 7u))
    return fail(TQ_EINVAL, "tq_search: misaligned centroids/scale/out/deleted/ext_ids pointers");
  if (filter) {
    if (filter->f.n != n)
      return fail(TQ_EINVAL, "tq_search: filter built for n=%lld, search has n=%lld",
                  (long long)filter->f.n, (long long)n);
    if (!allow_off || !allow_tenants)
      return fail(TQ_EINVAL, "tq_search: a filter needs allow_off and allow_tenants");
    if (((uintptr_t)allow_off & 7u) || ((uintptr_t)allow_tenants & 3u))
      return fail(TQ_EINVAL, "tq_search: misaligned allowlist pointers");
  }
  if ((cal_mu == nullptr) != (cal_a == nullptr))
    return fail(TQ_EINVAL, "tq_search_ex: a TQ+ calibration needs both mu and a");
  if (((uintptr_t)cal_mu & 3u) || ((uintptr_t)cal_a & 3u))
    return fail(TQ_EINVAL, "tq_search_ex: mu and a must be 4-byte aligned");
  const int path = tq::search_path();
  const bool can_mma = tq::mma_supported(bits, d, k);
  if (path == TQ_PATH_MMA && !can_mma)
    return fail(TQ_EUNSUPPORTED, "tq_search: the tensor-core scan needs bits 2/4/8, d %% 64 == 0 and k <= %d",
                tq::kMaxKMma);
  const bool use_mma = can_mma && (path == TQ_PATH_MMA || (path == TQ_PATH_AUTO && nq >= tq::kMmaMinBatch));
  const bool can_fold = tq::fold_supported(bits, d, k, n);
  if (path == TQ_PATH_LUT_FOLD && !can_fold)
    return fail(TQ_EUNSUPPORTED,
                "tq_search: the query-folded scan needs bits 4, d >= 256, k <= %d and n < 2^31 - 13312",
                tq::kFoldMaxK);
  // AUTO keeps the byte-pair scan: on GB300 it is the faster of the two (218
  // against 228 us per query at 999,000 x 1536)
  const bool use_fold = !use_mma && can_fold && path == TQ_PATH_LUT_FOLD;
  const tq::SearchPlan p = tq::plan_search(nq, n, d, bits, k, filter);
  if (ws_bytes < p.total)
    return fail(TQ_EINVAL, "tq_search: workspace of %zu bytes, %zu needed", ws_bytes, p.total);
  cudaStream_t s = (cudaStream_t)stream;
  char* ws = static_cast<char*>(workspace);
  int* status = reinterpret_cast<int*>(ws + p.off_status);
  int* counters = reinterpret_cast<int*>(ws + p.off_cnt);
  float* qrot = reinterpret_cast<float*>(ws + p.off_rot);
  uint32_t* allow = filter ? reinterpret_cast<uint32_t*>(ws + p.off_allow) : nullptr;
  uint32_t* bmask = filter ? reinterpret_cast<uint32_t*>(ws + p.off_mask) : nullptr;
  float* cs = reinterpret_cast<float*>(ws + p.off_cs);
  int32_t* ci = reinterpret_cast<int32_t*>(ws + p.off_ci);
  float* bias = cal_mu ? reinterpret_cast<float*>(ws + p.off_bias) : nullptr;
  // the rotation also clears the status word and zeroes the merge counters
  cudaError_t e = p.rot_tc ? tq::launch_rotate_tc(Q, nq, d, R, qrot, reinterpret_cast<float*>(ws + p.off_part),
                                                  status, counters, nq, s)
                           : tq::launch_rotate(Q, nq, d, R, qrot, status, counters, nq, s);
  if (e == cudaSuccess && cal_mu) e = tq::launch_calib_query(qrot, nq, d, cal_mu, cal_a, bias, s);
  if (use_mma) {
    if (e == cudaSuccess && filter) e = tq::launch_allow_bits(filter->f, allow_off, allow_tenants, nq, allow, s);
    if (e == cudaSuccess)
      e = tq::launch_scan_mma(qrot, nq, d, centroids, bits, codes, scale, n, deleted,
                              filter ? filter->f.dense : nullptr, allow, filter ? filter->f.words : 0, bias, k,
                              p.grid_mma, ws + p.off_qpack, cs, ci, status, s, (cudaEvent_t)tq::profile_start(),
                              (cudaEvent_t)tq::profile_stop());
    if (e == cudaSuccess) e = tq::launch_merge(cs, ci, nq, p.grid_mma * k, k, ext_ids, out_ids, out_scores, s);
  } else {
    if (e == cudaSuccess && filter) e = tq::launch_allow_bits(filter->f, allow_off, allow_tenants, nq, allow, s);
    if (e == cudaSuccess && filter) e = tq::launch_block_mask(filter->f, allow, nq, bmask, s);
    if (e == cudaSuccess && use_fold)
      e = tq::launch_scan_fold(qrot, nq, d, centroids, codes, scale, n, deleted, filter ? &filter->f : nullptr,
                               allow, bmask, k, p.grid_fold, cs, ci, status, counters, ext_ids, out_ids,
                               out_scores, bias, s, (cudaEvent_t)tq::profile_start(),
                               (cudaEvent_t)tq::profile_stop());
    else if (e == cudaSuccess)
      e = tq::launch_scan_lut(qrot, nq, d, centroids, bits, codes, scale, n, deleted,
                              filter ? &filter->f : nullptr, allow, bmask,
                              path == TQ_PATH_LUT_FIXED && d >= tq::kFixMinD,
                              k, p.grid_lut, cs, ci, status, counters, ext_ids, out_ids, out_scores, bias, s,
                              (cudaEvent_t)tq::profile_start(), (cudaEvent_t)tq::profile_stop());
  }
  if (e != cudaSuccess) return tq::cuda_fail("tq_search", e);
  return tq::ok();
}

extern "C" tq_status tq_search(const float* Q, int64_t nq, int d, const float* R,
                               const float* centroids, int bits, const uint8_t* codes,
                               const float* scale, int64_t n, const tq_filter* filter,
                               const int64_t* allow_off, const uint32_t* allow_tenants, int k,
                               int64_t* out_ids, float* out_scores, void* workspace,
                               size_t ws_bytes, void* stream) {
  return tq_search_ex(Q, nq, d, R, centroids, bits, codes, scale, n, filter, allow_off, allow_tenants, nullptr,
                      nullptr, nullptr, nullptr, k, out_ids, out_scores, workspace, ws_bytes, stream);
}

namespace {
// staging layout of tq_search_host: queries | ids | scores
struct HostStaging {
  size_t off_ids, off_scores, total;
};
HostStaging host_staging(int64_t nq, int d, int k) {
  HostStaging h;
  h.off_ids = tq::align_up((size_t)nq * d * sizeof(float));
  h.off_scores = h.off_ids + tq::align_up((size_t)nq * k * sizeof(int64_t));
  h.total = h.off_scores + tq::align_up((size_t)nq * k * sizeof(float));
  return h;
}
}  // namespace

extern "C" tq_status tq_search_host_staging(int64_t nq, int d, int k, size_t* bytes) {
  if (!bytes) return fail(TQ_EINVAL, "tq_search_host_staging: NULL bytes");
  if (nq < 0 || nq > (1 << 24) || d < 1 || d > tq::kMaxD || k < 1 || k > tq::kMaxK)
    return fail(TQ_EINVAL, "tq_search_host_staging: nq=%lld d=%d k=%d out of range", (long long)nq, d, k);
  *bytes = host_staging(nq, d, k).total;
  return tq::ok();
}

namespace {
// The device address of page-locked, mapped host memory (every page-locked
// allocation is mapped under unified addressing), or nullptr for pageable
// memory, which the kernels cannot reach.
void* mapped_host(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();  // not sticky
    return nullptr;
  }
  return a.type == cudaMemoryTypeHost ? a.devicePointer : nullptr;
}
}  // namespace

extern "C" tq_status tq_search_host(const float* Q_host, int64_t nq, int d, const float* R,
                                    const float* centroids, int bits, const uint8_t* codes,
                                    const float* scale, int64_t n, const tq_filter* filter,
                                    const int64_t* allow_off, const uint32_t* allow_tenants,
                                    const uint32_t* deleted, const uint64_t* ext_ids, const float* cal_mu,
                                    const float* cal_a, int k, int64_t* ids_host, float* scores_host, void* staging,
                                    size_t staging_bytes, void* workspace, size_t ws_bytes, void* stream) {
  tq_status st = check_search(nq, n, d, bits, k);
  if (st != TQ_OK) return st;
  if (nq == 0) return tq::ok();
  if (!Q_host || !ids_host || !scores_host || !staging)
    return fail(TQ_EINVAL, "tq_search_host: NULL query, result or staging pointer");
  if (!tq::aligned16(staging)) return fail(TQ_EINVAL, "tq_search_host: staging must be 16-byte aligned");
  const HostStaging h = host_staging(nq, d, k);
  if (staging_bytes < h.total)
    return fail(TQ_EINVAL, "tq_search_host: staging of %zu bytes, %zu needed", staging_bytes, h.total);
  char* stg = static_cast<char*>(staging);
  cudaStream_t s = (cudaStream_t)stream;
  // Page-locked buffers are used in place: the query rotation reads the
  // queries over the host link (when it runs on plain loads: batches the
  // tensor-core rotation, fed by TMA from device memory, does not take), and
  // the merge writes the results there; otherwise they go through `staging`.
  const float* q_dev = tq::rotate_tc_applies(nq, d) ? nullptr : static_cast<const float*>(mapped_host(Q_host));
  int64_t* ids_dev = static_cast<int64_t*>(mapped_host(ids_host));
  float* scores_dev = static_cast<float*>(mapped_host(scores_host));
  const bool out_in_place = ids_dev && scores_dev;
  cudaError_t e = cudaSuccess;
  if (!q_dev) {
    float* q_stg = reinterpret_cast<float*>(stg);
    e = cudaMemcpyAsync(q_stg, Q_host, (size_t)nq * d * sizeof(float), cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return tq::cuda_fail("tq_search_host: query copy", e);
    q_dev = q_stg;
  }
  if (!out_in_place) {
    ids_dev = reinterpret_cast<int64_t*>(stg + h.off_ids);
    scores_dev = reinterpret_cast<float*>(stg + h.off_scores);
  }
  st = tq_search_ex(q_dev, nq, d, R, centroids, bits, codes, scale, n, filter, allow_off, allow_tenants, deleted,
                    ext_ids, cal_mu, cal_a, k, ids_dev, scores_dev, workspace, ws_bytes, stream);
  if (st != TQ_OK) return st;
  if (!out_in_place) {
    e = cudaMemcpyAsync(ids_host, ids_dev, (size_t)nq * k * sizeof(int64_t), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(scores_host, scores_dev, (size_t)nq * k * sizeof(float), cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) return tq::cuda_fail("tq_search_host: result copy", e);
  }
  return tq::ok();
}

extern "C" tq_status tq_merge_topk(const int64_t* cand_ids, const float* cand_scores, int64_t n_src, int64_t nq,
                                   int64_t m, int k, int64_t* out_ids, float* out_scores, void* stream) {
  if (nq < 0 || nq > (1 << 24)) return fail(TQ_EINVAL, "tq_merge_topk: nq=%lld outside [0, 2^24]", (long long)nq);
  if (n_src < 1 || n_src > 4096) return fail(TQ_EINVAL, "tq_merge_topk: n_src=%lld outside [1, 4096]", (long long)n_src);
  if (m < 0 || m > (1 << 20)) return fail(TQ_EINVAL, "tq_merge_topk: m=%lld outside [0, 2^20]", (long long)m);
  if (k < 1 || k > tq::kMaxK) return fail(TQ_EINVAL, "tq_merge_topk: k=%d outside [1, %d]", k, tq::kMaxK);
  if (nq == 0) return tq::ok();
  if (!out_ids || !out_scores || (m > 0 && (!cand_ids || !cand_scores)))
    return fail(TQ_EINVAL, "tq_merge_topk: NULL device pointer");
  if (((uintptr_t)cand_ids & 7u) || ((uintptr_t)out_ids & 7u) || ((uintptr_t)cand_scores & 3u) ||
      ((uintptr_t)out_scores & 3u))
    return fail(TQ_EINVAL, "tq_merge_topk: misaligned pointers");
  const cudaError_t e =
      tq::launch_merge_global(cand_scores, cand_ids, n_src, nq, m, k, out_ids, out_scores, (cudaStream_t)stream);
  if (e != cudaSuccess) return tq::cuda_fail("tq_merge_topk", e);
  return tq::ok();
}

extern "C" tq_status tq_search_check(const void* workspace, void* stream) {
  if (!workspace) return fail(TQ_EINVAL, "tq_search_check: NULL workspace");
  if (!tq::aligned16(workspace)) return fail(TQ_EINVAL, "tq_search_check: workspace must be 16-byte aligned");
  cudaStream_t s = (cudaStream_t)stream;
  int word = 0;
  cudaError_t e = cudaMemcpyAsync(&word, workspace, sizeof(int), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return tq::cuda_fail("tq_search_check", e);
  if (word == 0) return tq::ok();
  if (word / 1000 == TQ_ETIMEOUT)
    return fail(TQ_ETIMEOUT, "tq_search_check: a bounded wait (site %d) gave up; the results are invalid",
                word % 1000);
  return fail(TQ_ECUDA, "tq_search_check: unexpected status word %d", word);
}

extern "C" tq_status tq_debug_bounded_wait(long long budget_cycles, void* workspace, void* stream) {
  if (!workspace || !tq::aligned16(workspace))
    return fail(TQ_EINVAL, "tq_debug_bounded_wait: NULL or misaligned workspace");
  if (budget_cycles < 1 || budget_cycles > tq::kWaitCyclesMax)
    return fail(TQ_EINVAL, "tq_debug_bounded_wait: budget %lld outside [1, %lld]", budget_cycles,
                tq::kWaitCyclesMax);
  const cudaError_t e = tq::launch_debug_wait(budget_cycles, static_cast<int*>(workspace), (cudaStream_t)stream);
  if (e != cudaSuccess) return tq::cuda_fail("tq_debug_bounded_wait", e);
  return tq::ok();
}
