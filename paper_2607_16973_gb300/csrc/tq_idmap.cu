// tq_idmap: the id map of an id-mapped index (Sec. III-A: external uint64
// ids, O(1) deletion).  Host side: a hash map external id -> row and a host
// copy of the tombstone bitmap; device side: the external id of every row and
// the tombstone bitmap, which the scans read (a deleted row never enters a
// top-k list; the merge writes rows as external ids).  Rows are appended in
// order and never reused.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <new>
#include <unordered_map>
#include <vector>

#include "tq_internal.h"
#include "tq_kernels.h"

struct tq_idmap {
  int device = 0;
  int64_t capacity = 0, rows = 0;
  std::unordered_map<uint64_t, int64_t> live;  // external id -> row, live rows only
  std::vector<uint32_t> dead;                  // host copy of the tombstone bitmap
  std::vector<uint64_t> ext;                   // host copy of the external ids, [rows]
  uint64_t* d_ext = nullptr;                   // [capacity]
  uint32_t* d_dead = nullptr;                  // [ceil(capacity / 32)]
};

namespace {

constexpr uint64_t kEmptyId = ~0ull;  // the -1 of an empty result slot

using tq::fail;

tq_status cuda_fail(const char* where, cudaError_t e) {
  return fail(TQ_ECUDA, "%s: %s (%s)", where, cudaGetErrorString(e), cudaGetErrorName(e));
}

}  // namespace

extern "C" tq_status tq_idmap_create(int64_t capacity, tq_idmap** out) {
  if (!out) return fail(TQ_EINVAL, "tq_idmap_create: NULL out");
  *out = nullptr;
  if (capacity < 1 || capacity > INT32_MAX)
    return fail(TQ_EINVAL, "tq_idmap_create: capacity=%lld outside [1, 2^31-1]", (long long)capacity);
  tq_idmap* m = nullptr;
  try {
    m = new tq_idmap();
    cudaGetDevice(&m->device);
    m->capacity = capacity;
    const size_t words = (size_t)((capacity + 31) / 32);
    m->dead.assign(words, 0u);
    cudaError_t e = tq::dev_malloc(reinterpret_cast<void**>(&m->d_ext), (size_t)capacity * sizeof(uint64_t));
    if (e == cudaSuccess) e = tq::dev_malloc(reinterpret_cast<void**>(&m->d_dead), words * sizeof(uint32_t));
    if (e != cudaSuccess) {
      tq_idmap_destroy(m);
      cudaGetLastError();
      return fail(TQ_ENOMEM, "tq_idmap_create: device allocation failed: %s", cudaGetErrorString(e));
    }
    e = cudaMemset(m->d_ext, 0, (size_t)capacity * sizeof(uint64_t));
    if (e == cudaSuccess) e = cudaMemset(m->d_dead, 0, words * sizeof(uint32_t));
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
      tq_idmap_destroy(m);
      return cuda_fail("tq_idmap_create", e);
    }
    *out = m;
    return tq::ok();
  } catch (const std::bad_alloc&) {
    if (m) tq_idmap_destroy(m);
    return fail(TQ_ENOMEM, "tq_idmap_create: out of host memory");
  }
}

extern "C" tq_status tq_idmap_destroy(tq_idmap* m) {
  if (!m) return tq::ok();
  cudaFree(m->d_ext);
  cudaFree(m->d_dead);
  delete m;
  return tq::ok();
}

extern "C" tq_status tq_idmap_add(tq_idmap* m, const uint64_t* ext_ids, int64_t n_new, int64_t* first_row,
                                  void* stream) {
  if (!m) return fail(TQ_EINVAL, "tq_idmap_add: NULL map");
  if (n_new < 0) return fail(TQ_EINVAL, "tq_idmap_add: n_new=%lld < 0", (long long)n_new);
  if (n_new > 0 && !ext_ids) return fail(TQ_EINVAL, "tq_idmap_add: NULL ext_ids");
  if (n_new > m->capacity - m->rows)
    return fail(TQ_EINVAL, "tq_idmap_add: %lld rows + %lld new exceed the capacity %lld", (long long)m->rows,
                (long long)n_new, (long long)m->capacity);
  if (first_row) *first_row = m->rows;
  if (n_new == 0) return tq::ok();
  try {
    // insert id by id; on a conflict undo this batch's inserts, so nothing changes
    for (int64_t i = 0; i < n_new; ++i) {
      const uint64_t id = ext_ids[i];
      const bool bad = id == kEmptyId;
      if (bad || !m->live.emplace(id, m->rows + i).second) {
        for (int64_t j = 0; j < i; ++j) m->live.erase(ext_ids[j]);
        return fail(TQ_EINVAL, bad ? "tq_idmap_add: id %llu (-1) marks empty result slots"
                                   : "tq_idmap_add: id %llu is already live",
                    (unsigned long long)id);
      }
    }
    // the host copy is pageable: cudaMemcpyAsync has read it when it returns,
    // so the caller's array (pinned or not) is free as soon as this call returns
    m->ext.insert(m->ext.end(), ext_ids, ext_ids + n_new);
  } catch (const std::bad_alloc&) {
    for (int64_t j = 0; j < n_new; ++j) {
      auto it = m->live.find(ext_ids[j]);
      if (it != m->live.end() && it->second >= m->rows) m->live.erase(it);
    }
    return fail(TQ_ENOMEM, "tq_idmap_add: out of host memory");
  }
  const cudaError_t e = cudaMemcpyAsync(m->d_ext + m->rows, m->ext.data() + m->rows, (size_t)n_new * sizeof(uint64_t),
                                        cudaMemcpyHostToDevice, (cudaStream_t)stream);
  if (e != cudaSuccess) {
    for (int64_t j = 0; j < n_new; ++j) m->live.erase(ext_ids[j]);
    m->ext.resize((size_t)m->rows);
    return cuda_fail("tq_idmap_add", e);
  }
  m->rows += n_new;
  return tq::ok();
}

extern "C" tq_status tq_idmap_remove(tq_idmap* m, const uint64_t* ext_ids, int64_t n, int64_t* n_removed,
                                     void* stream) {
  if (n_removed) *n_removed = 0;
  if (!m) return fail(TQ_EINVAL, "tq_idmap_remove: NULL map");
  if (n < 0) return fail(TQ_EINVAL, "tq_idmap_remove: n=%lld < 0", (long long)n);
  if (n > 0 && !ext_ids) return fail(TQ_EINVAL, "tq_idmap_remove: NULL ext_ids");
  int64_t removed = 0, wlo = INT64_MAX, whi = -1;
  for (int64_t i = 0; i < n; ++i) {
    auto it = m->live.find(ext_ids[i]);
    if (it == m->live.end()) continue;
    const int64_t row = it->second;
    m->live.erase(it);
    m->dead[(size_t)(row >> 5)] |= 1u << (row & 31);
    wlo = row >> 5 < wlo ? row >> 5 : wlo;
    whi = row >> 5 > whi ? row >> 5 : whi;
    ++removed;
  }
  if (n_removed) *n_removed = removed;
  if (removed == 0) return tq::ok();
  // the touched words, from the pageable host copy (read before the call returns)
  const cudaError_t e = cudaMemcpyAsync(m->d_dead + wlo, m->dead.data() + wlo, (size_t)(whi - wlo + 1) * 4,
                                        cudaMemcpyHostToDevice, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail("tq_idmap_remove", e);
  return tq::ok();
}

extern "C" tq_status tq_idmap_lookup(const tq_idmap* m, uint64_t ext_id, int64_t* row) {
  if (!m || !row) return fail(TQ_EINVAL, "tq_idmap_lookup: NULL map or row");
  auto it = m->live.find(ext_id);
  *row = it == m->live.end() ? -1 : it->second;
  return tq::ok();
}

extern "C" tq_status tq_idmap_info(const tq_idmap* m, int64_t* rows, int64_t* capacity, int64_t* live) {
  if (!m) return fail(TQ_EINVAL, "tq_idmap_info: NULL map");
  if (rows) *rows = m->rows;
  if (capacity) *capacity = m->capacity;
  if (live) *live = (int64_t)m->live.size();
  return tq::ok();
}

extern "C" tq_status tq_idmap_device(const tq_idmap* m, const uint32_t** deleted, const uint64_t** ext_ids) {
  if (!m) return fail(TQ_EINVAL, "tq_idmap_device: NULL map");
  if (deleted) *deleted = m->d_dead;
  if (ext_ids) *ext_ids = m->d_ext;
  return tq::ok();
}

extern "C" tq_status tq_idmap_export(const tq_idmap* m, uint64_t* ext_ids, uint32_t* deleted) {
  if (!m) return fail(TQ_EINVAL, "tq_idmap_export: NULL map");
  if (m->rows > 0 && (!ext_ids || !deleted)) return fail(TQ_EINVAL, "tq_idmap_export: NULL output array");
  std::copy(m->ext.begin(), m->ext.begin() + m->rows, ext_ids);
  std::copy(m->dead.begin(), m->dead.begin() + (m->rows + 31) / 32, deleted);
  return tq::ok();
}

extern "C" tq_status tq_idmap_import(tq_idmap* m, const uint64_t* ext_ids, const uint32_t* deleted, int64_t n,
                                     void* stream) {
  if (!m) return fail(TQ_EINVAL, "tq_idmap_import: NULL map");
  if (m->rows != 0) return fail(TQ_EINVAL, "tq_idmap_import: the map already holds %lld rows", (long long)m->rows);
  if (n < 0 || n > m->capacity)
    return fail(TQ_EINVAL, "tq_idmap_import: n=%lld outside [0, capacity %lld]", (long long)n,
                (long long)m->capacity);
  if (n == 0) return tq::ok();
  if (!ext_ids || !deleted) return fail(TQ_EINVAL, "tq_idmap_import: NULL ext_ids or deleted");
  const size_t words = (size_t)((n + 31) / 32);
  if (n % 32 != 0 && (deleted[words - 1] >> (n % 32)) != 0u)
    return fail(TQ_EINVAL, "tq_idmap_import: tombstone bits set past row %lld", (long long)n);
  try {
    for (int64_t r = 0; r < n; ++r) {
      if ((deleted[r >> 5] >> (r & 31)) & 1u) continue;
      const uint64_t id = ext_ids[r];
      if (id == kEmptyId || !m->live.emplace(id, r).second) {
        m->live.clear();
        return fail(TQ_EINVAL, "tq_idmap_import: live id %llu at row %lld is -1 or repeated",
                    (unsigned long long)id, (long long)r);
      }
    }
    m->ext.assign(ext_ids, ext_ids + n);
    std::copy(deleted, deleted + words, m->dead.begin());
  } catch (const std::bad_alloc&) {
    m->live.clear();
    m->ext.clear();
    return fail(TQ_ENOMEM, "tq_idmap_import: out of host memory");
  }
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = cudaMemcpyAsync(m->d_ext, m->ext.data(), (size_t)n * sizeof(uint64_t), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(m->d_dead, m->dead.data(), words * 4, cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) {
    m->live.clear();
    m->ext.clear();
    std::fill(m->dead.begin(), m->dead.end(), 0u);
    return cuda_fail("tq_idmap_import", e);
  }
  m->rows = n;
  return tq::ok();
}
