// tq_search_static: the lookup-scan search for callers that cannot allocate
// device memory.
//
// Some callers have no way to hand the library a workspace: a plain C host
// program or plugin that only receives device pointers for its inputs and
// outputs from someone else, or a latency-critical serving loop that must
// not call cudaMalloc/cudaFree (an allocation can block, synchronise the
// device or fail under memory pressure in the middle of a request).  For them
// this entry point keeps its scratch (status word, merge counters, rotated
// queries, allow bitmaps, block masks, per-CTA top-k candidates) in one
// file-scope device array of kStaticScratchBytes.  It
// allocates nothing and calls no allocating routine.
//
// The array's name in host code is only a host-side stand-in, never a device
// address, so the device address is looked up with cudaGetSymbolAddress, once
// per device, with that device current: the first call on a device does this
// set-up (make that first call before any stream capture).  With CUDA's lazy
// module loading (the default) that lookup is also what loads the array's
// module on the device, so the first call on each device is the one that
// reserves the 8 MiB, which the device then holds until the process exits: a
// server makes one warm-up call per device before it starts serving.  If the
// device has no room for the array, that first call returns TQ_ENOMEM.
//
// Every call on a device shares the one array and the array keeps the last
// call's contents; nothing in it needs to start at zero because each kernel
// writes every word it later reads.  Calls whose work overlaps on the GPU (two streams, or two
// host threads) race on the array: serialise them.
#include <cuda_runtime.h>

#include <mutex>

#include "tq_internal.h"
#include "tq_kernels.h"

namespace tq {
namespace {

constexpr size_t kStaticScratchBytes = 8u << 20;  // 8 MiB per device
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

std::mutex g_static_mu;
void* g_static_ptr[kMaxDevices] = {};

inline size_t up256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace
}  // namespace tq

extern "C" tq_status tq_search_static(const float* Q, int64_t nq, int d, const float* R,
                                      const float* centroids, int bits, const uint8_t* codes,
                                      const float* scale, int64_t n, const tq_filter* filter,
                                      const int64_t* allow_off, const uint32_t* allow_tenants, int k,
                                      int64_t* out_ids, float* out_scores, void* stream) {
  using tq::fail;
  // the same checks, in the same order, as tq_search: the two report the same
  // status for the same arguments
  if (d < 32 || d > tq::kMaxD || d % 32 != 0)
    return fail(TQ_EINVAL, "tq_search_static: d=%d must be a multiple of 32 in [32, %d]", d, tq::kMaxD);
  if (!tq::valid_bits(bits)) return fail(TQ_EINVAL, "tq_search_static: bits=%d must be 2, 3, 4 or 8", bits);
  if (nq < 0 || nq > (1 << 24)) return fail(TQ_EINVAL, "tq_search_static: nq=%lld outside [0, 2^24]", (long long)nq);
  if (n < 1 || n > INT32_MAX - 1) return fail(TQ_EINVAL, "tq_search_static: n=%lld outside [1, 2^31-2]", (long long)n);
  if (k < 1 || k > tq::kMaxK) return fail(TQ_EINVAL, "tq_search_static: k=%d outside [1, %d]", k, tq::kMaxK);
  if (d > 2048) return fail(TQ_EUNSUPPORTED, "tq_search_static: d=%d > 2048 is not supported by this build", d);
  if (nq == 0) return tq::ok();
  if (!Q || !R || !centroids || !codes || !out_ids || !out_scores)
    return fail(TQ_EINVAL, "tq_search_static: NULL device pointer");
  if (!tq::aligned16(Q) || !tq::aligned16(R) || !tq::aligned16(codes))
    return fail(TQ_EINVAL, "tq_search_static: Q, R and codes must be 16-byte aligned");
  if (((uintptr_t)centroids & 3u) || ((uintptr_t)scale & 3u) || ((uintptr_t)out_scores & 3u) ||
      ((uintptr_t)out_ids & 7u))
    return fail(TQ_EINVAL, "tq_search_static: misaligned centroids/scale/out pointers");
  const tq::FilterDev* f = nullptr;
  if (filter) {
    if (filter->f.n != n)
      return fail(TQ_EINVAL, "tq_search_static: filter built for n=%lld, search has n=%lld",
                  (long long)filter->f.n, (long long)n);
    if (!allow_off || !allow_tenants)
      return fail(TQ_EINVAL, "tq_search_static: a filter needs allow_off and allow_tenants");
    if (((uintptr_t)allow_off & 7u) || ((uintptr_t)allow_tenants & 3u))
      return fail(TQ_EINVAL, "tq_search_static: misaligned allowlist pointers");
    f = &filter->f;
  }

  // scratch plan: status word | merge counters | rotated queries | allow bitmaps | block masks |
  // candidate scores | ids
  const int gx = tq::scan_lut_grid_x(nq, n, k, bits, d);
  const size_t head = 256 + tq::up256((size_t)nq * sizeof(int));
  const size_t rot = tq::up256((size_t)nq * d * sizeof(float));
  const size_t allow = f ? tq::up256((size_t)nq * f->words * sizeof(uint32_t)) : 0;
  const size_t mask = f ? tq::up256((size_t)nq * tq::filter_mask_words(*f) * sizeof(uint32_t)) : 0;
  const size_t cs = tq::up256((size_t)nq * gx * k * sizeof(float));
  const size_t ci = tq::up256((size_t)nq * gx * k * sizeof(int32_t));
  const size_t need = head + rot + allow + mask + cs + ci;
  if (need > tq::kStaticScratchBytes)
    return fail(TQ_EINVAL,
                "tq_search_static: these sizes need %zu bytes of scratch but the static scratch holds %zu "
                "(reduce nq or k, or use tq_search with a workspace)",
                need, tq::kStaticScratchBytes);

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(TQ_ECUDA, "tq_search_static: cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= tq::kMaxDevices) return fail(TQ_EUNSUPPORTED, "tq_search_static: device %d", dev);
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(tq::g_static_mu);
    if (!tq::g_static_ptr[dev]) {
      e = cudaGetSymbolAddress(&tq::g_static_ptr[dev], tq::g_static_scratch);
      if (e != cudaSuccess) {
        tq::g_static_ptr[dev] = nullptr;
        if (e == cudaErrorMemoryAllocation) {
          cudaGetLastError();  // not sticky: clear it so later calls start clean
          return fail(TQ_ENOMEM, "tq_search_static: no device memory for the %zu-byte static scratch: %s",
                      tq::kStaticScratchBytes, cudaGetErrorString(e));
        }
        return fail(TQ_ECUDA, "tq_search_static: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
      }
    }
    scratch = tq::g_static_ptr[dev];
  }

  cudaStream_t s = (cudaStream_t)stream;
  int* status = static_cast<int*>(scratch);  // the scans' bounded waits report here
  int* counters = reinterpret_cast<int*>(static_cast<char*>(scratch) + 256);
  char* base = static_cast<char*>(scratch) + head;
  float* qrot = reinterpret_cast<float*>(base);
  uint32_t* allow_bits = f ? reinterpret_cast<uint32_t*>(base + rot) : nullptr;
  uint32_t* bmask = f ? reinterpret_cast<uint32_t*>(base + rot + allow) : nullptr;
  float* cand_s = reinterpret_cast<float*>(base + rot + allow + mask);
  int32_t* cand_i = reinterpret_cast<int32_t*>(base + rot + allow + mask + cs);
  e = tq::launch_rotate(Q, nq, d, R, qrot, status, counters, nq, s);
  if (e == cudaSuccess && f) e = tq::launch_allow_bits(*f, allow_off, allow_tenants, nq, allow_bits, s);
  if (e == cudaSuccess && f) e = tq::launch_block_mask(*f, allow_bits, nq, bmask, s);
  if (e == cudaSuccess)
    e = tq::launch_scan_lut(qrot, nq, d, centroids, bits, codes, scale, n, nullptr, f, allow_bits, bmask,
                            tq::search_path() == TQ_PATH_LUT_FIXED && d >= tq::kFixMinD, k, gx, cand_s, cand_i,
                            status, counters, nullptr, out_ids, out_scores, nullptr, s, nullptr, nullptr);
  if (e != cudaSuccess) return fail(TQ_ECUDA, "tq_search_static: %s", cudaGetErrorString(e));
  return tq::ok();
}
