// Top-k helpers shared by the lookup scans: per-warp sorted lists, the
// merge of per-CTA lists into a query's result (Sec. II-B step 5: the k best
// inner products, ties by the lower id), and programmatic-launch waits.
// Each translation unit gets its own copies (internal linkage).
#pragma once

#include <cuda_runtime.h>

#include <climits>
#include <cmath>
#include <cstdint>

#include "tq_internal.h"

namespace tq {
namespace {

constexpr unsigned FULL = 0xffffffffu;

// Bit v % 32 of word v / 32 of the tombstone bitmap marks row v deleted.  It
// is read only for a vector that would enter a list, so a scan with few
// candidates per step pays almost nothing for it.
__device__ __forceinline__ bool tombstoned(const uint32_t* __restrict__ del, int v) {
  return del && ((__ldg(del + (v >> 5)) >> (v & 31)) & 1u);
}
// Programmatic dependent launch: a kernel launched with the
// programmatic-serialization attribute may start while the kernel before it
// in the stream still runs; it must wait here before reading anything that
// kernel (or any earlier one) wrote.  Without the attribute both are no-ops
// in effect.  The kernel before it lets it start early with launch_dependents.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename I>
__device__ __forceinline__ bool better(float s1, I i1, float s2, I i2) {
  return s1 > s2 || (s1 == s2 && i1 < i2);
}

// Bitonic sort of P (a power of two) (score, id) pairs in shared memory, best
// first.  All threads of the block take part.
template <typename I>
__device__ void block_sort(float* s, I* id, int P) {
  for (int size = 2; size <= P; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int t = threadIdx.x; t < P / 2; t += blockDim.x) {
        const int i = 2 * t - (t & (stride - 1));
        const int j = i + stride;
        const float si = s[i], sj = s[j];
        const I ii = id[i], ij = id[j];
        const bool best_first = (i & size) == 0;
        const bool swap = best_first ? better(sj, ij, si, ii) : better(si, ii, sj, ij);
        if (swap) {
          s[i] = sj;
          s[j] = si;
          id[i] = ij;
          id[j] = ii;
        }
      }
      __syncthreads();
    }
  }
}

// Inserts (s, id) into a warp's sorted list of `cnt` entries (capacity k).
// The caller has checked that it beats the k-th entry (or cnt < k).
__device__ __forceinline__ void warp_insert(float* ws, int* wi, int k, int cnt, float s, int id) {
  const int lane = threadIdx.x & 31;
  int pos = 0;
  for (int base = 0; base < cnt; base += 32) {
    const int i = base + lane;
    const bool b = i < cnt && better(ws[i], wi[i], s, id);
    pos += __popc(__ballot_sync(FULL, b));
  }
  const int last = min(cnt, k - 1);  // entries [pos, last) move down one slot
  for (int base = ((max(last, 1) - 1) >> 5) << 5; base >= 0; base -= 32) {
    if (base + 32 <= pos) break;
    const int i = base + lane;
    const bool mv = i >= pos && i < last;
    float sv = 0.f;
    int iv = 0;
    if (mv) {
      sv = ws[i];
      iv = wi[i];
    }
    __syncwarp();
    if (mv) {
      ws[i + 1] = sv;
      wi[i + 1] = iv;
    }
    __syncwarp();
  }
  if (lane == 0) {
    ws[pos] = s;
    wi[pos] = id;
  }
  __syncwarp();
}
// Sorts one (score, id) pair per lane across the warp, best first (lane 0
// the best): a bitonic network of shuffles.
__device__ __forceinline__ void warp_sort32(float& sv, int& iv) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1)
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const float os = __shfl_xor_sync(FULL, sv, stride);
      const int oi = __shfl_xor_sync(FULL, iv, stride);
      // the lower lane of a pair keeps the better entry in a best-first run
      const bool keep_better = ((lane & stride) == 0) == ((lane & size) == 0);
      if (keep_better ? better(os, oi, sv, iv) : better(sv, iv, os, oi)) {
        sv = os;
        iv = oi;
      }
    }
}

// merge_lists_block for k <= 32 and at most 16 candidates per thread: every
// candidate comes to shared memory in one round trip of loads, both bounds
// (see merge_lists_block) are taken there, and the survivors go to a 32-entry
// buffer that one warp sorts.  Returns false (nothing written) when more than
// 32 candidates survive, for the general path to redo the merge.
__device__ bool merge_lists_small(const float* cs, const int* ci, int nlists, int k, const uint64_t* __restrict__ ext,
                                  int64_t* out_ids, float* out_scores, float* ss, int* si) {
  __shared__ float sv_s[32];
  __shared__ int sv_i[32];
  __shared__ float bs_s[2];
  __shared__ int bs_i[2];
  __shared__ int nsv;
  const int total = nlists * k;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  {
    float va[16];
    int vb[16];
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      const int c = tid + u * (int)blockDim.x;
      va[u] = c < total ? __ldcg(cs + c) : 0.f;
      vb[u] = c < total ? __ldcg(ci + c) : 0;
    }
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      const int c = tid + u * (int)blockDim.x;
      if (c < total) {
        ss[c] = va[u];
        si[c] = vb[u];
      }
    }
  }
  if (tid == 0) nsv = 0;
  __syncthreads();
  if (warp < 2) {  // warp 0: T, the best k-th entry of a list; warp 1: the k-th best of the lanes' best heads
    float bs = -INFINITY;
    int bi = INT_MAX;
    for (int l = lane; l < nlists; l += 32) {
      const int c = l * k + (warp == 0 ? k - 1 : 0);
      if (better(ss[c], si[c], bs, bi)) {
        bs = ss[c];
        bi = si[c];
      }
    }
    warp_sort32(bs, bi);
    const int pick = warp == 0 ? 0 : k - 1;
    if (lane == pick) {
      bs_s[warp] = bs;
      bs_i[warp] = bi;
    }
  }
  __syncthreads();
  float ts = bs_s[0];
  int ti = bs_i[0];
  if (better(bs_s[1], bs_i[1], ts, ti)) {
    ts = bs_s[1];
    ti = bs_i[1];
  }
  for (int c = tid; c < total; c += blockDim.x)
    if (si[c] != INT_MAX && !better(ts, ti, ss[c], si[c])) {
      const int p = atomicAdd(&nsv, 1);
      if (p < 32) {
        sv_s[p] = ss[c];
        sv_i[p] = si[c];
      }
    }
  __syncthreads();
  const int n_sv = nsv;
  if (n_sv > 32) return false;  // every thread sees the same count
  if (warp == 0) {
    float sv = lane < n_sv ? sv_s[lane] : -INFINITY;
    int iv = lane < n_sv ? sv_i[lane] : INT_MAX;
    warp_sort32(sv, iv);
    if (lane < k) {
      const bool empty = iv == INT_MAX;
      out_ids[lane] = empty ? -1 : ext ? (int64_t)__ldg(ext + iv) : (int64_t)iv;
      out_scores[lane] = empty ? -INFINITY : sv;
    }
  }
  return true;
}

// Merge of per-CTA candidate lists that are each sorted best first and hold
// exactly k entries (padding (-inf, INT_MAX) at the end).  The k-th entry T of
// any one list is beaten or matched by that list's k entries, so the global
// k-th best is at least as good as the best such T and worse candidates are
// skipped at once.  Each warp keeps a sorted top-k of its share of the rest
// (ballot, then one warp-wide insertion per candidate that still beats the
// warp's k-th); warp 0 then folds the sorted warp lists into the result,
// leaving each list at its first entry that no longer qualifies.  With an
// id map the result rows are written as their external ids.  Every thread of
// the block calls it; cs/ci hold one query's lists [nlists][k] (read through
// L2: in the scans' tail other CTAs of the same grid wrote them); ws/wi are
// shared scratch of (blockDim.x / 32) * k entries; out_* point at the query's
// k results.
//
// The candidates at least as good as that bound are few (about k to a few
// times k): they are gathered into `scratch` (shared, scratch_bytes) and
// sorted by the whole block, the result being the first k.  Only when they
// do not fit does each warp insert its share into a sorted list of k.
__device__ void merge_lists_block(const float* cs, const int* ci, int nlists, int k, const uint64_t* __restrict__ ext,
                                  int64_t* out_ids, float* out_scores, float* ws, int* wi, unsigned char* scratch,
                                  size_t scratch_bytes) {
  __shared__ float red_s[32];
  __shared__ int red_i[32];
  __shared__ int nsurv;
  const int nwarps = blockDim.x >> 5;
  const int total = nlists * k;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int cap = (int)min((size_t)8192, scratch_bytes / 8);
  float* ss = reinterpret_cast<float*>(scratch);
  int* si = reinterpret_cast<int*>(ss + cap);
  if (k <= 32 && nwarps >= 2 && total <= min(cap, 16 * (int)blockDim.x) && nlists >= k)
    if (merge_lists_small(cs, ci, nlists, k, ext, out_ids, out_scores, ss, si)) return;
  // Two bounds on the global k-th best, the better one kept: T, the best
  // k-th entry of any list (that list's k entries are at least as good), and
  // the k-th best list head (the heads are k distinct candidates).  T is tight
  // when the best entries crowd into a few lists, the head bound when they are
  // spread over many.  The heads go to the scratch, loaded with the k-th
  // entries in the same round trip.
  const bool heads = nlists >= k && nlists <= min(cap, 512);
  __shared__ float hb_s;
  __shared__ int hb_i;
  if (tid == 0) {
    nsurv = 0;
    hb_s = -INFINITY;  // no head bound (too few lists, or too many for one warp's registers)
    hb_i = INT_MAX;
  }
  float ts = -INFINITY;
  int ti = INT_MAX;
  for (int l = tid; l < nlists; l += blockDim.x) {
    const float a = __ldcg(cs + (size_t)l * k + k - 1);
    const int b = __ldcg(ci + (size_t)l * k + k - 1);
    if (heads) {
      ss[l] = __ldcg(cs + (size_t)l * k);
      si[l] = __ldcg(ci + (size_t)l * k);
    }
    if (better(a, b, ts, ti)) {
      ts = a;
      ti = b;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float a = __shfl_xor_sync(FULL, ts, o);
    const int b = __shfl_xor_sync(FULL, ti, o);
    if (better(a, b, ts, ti)) {
      ts = a;
      ti = b;
    }
  }
  if (lane == 0) {
    red_s[warp] = ts;
    red_i[warp] = ti;
  }
  __syncthreads();
  if (heads && warp == 0) {
    if (k <= 32) {
      // the k-th best of the lanes' best heads (k distinct heads, so a valid
      // bound; with ~10 heads a lane it is close to the k-th best head): one
      // compare per head, then a shuffle sort of the 32 lane maxima
      float bs = -INFINITY;
      int bi = INT_MAX;
      for (int l = lane; l < nlists; l += 32)
        if (better(ss[l], si[l], bs, bi)) {
          bs = ss[l];
          bi = si[l];
        }
      warp_sort32(bs, bi);
      if (lane == k - 1) {
        hb_s = bs;
        hb_i = bi;
      }
    } else {
      // the k-th best head score exactly: the heads' order-preserving integer
      // keys sit in registers and the key is found bit by bit from the top
      // (the largest v with at least k keys >= v is the k-th largest key)
      uint32_t key[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int l = lane + 32 * j;
        uint32_t u = 0;  // below every score's key
        if (l < nlists) {
          const uint32_t b = __float_as_uint(ss[l]);
          u = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
        }
        key[j] = u;
      }
      uint32_t v = 0;
      for (int bit = 31; bit >= 0; --bit) {
        const uint32_t cand = v | (1u << bit);
        int c = 0;
#pragma unroll
        for (int j = 0; j < 16; ++j) c += key[j] >= cand ? 1 : 0;
        if (__reduce_add_sync(FULL, c) >= k) v = cand;
      }
      if (lane == 0) {  // every candidate with that score or better passes: the id is the worst one
        hb_s = __uint_as_float((v & 0x80000000u) ? (v & 0x7FFFFFFFu) : ~v);
        hb_i = INT_MAX;
      }
    }
  }
  ts = red_s[0];
  ti = red_i[0];
  for (int w = 1; w < nwarps; ++w)
    if (better(red_s[w], red_i[w], ts, ti)) {
      ts = red_s[w];
      ti = red_i[w];
    }
  __syncthreads();  // the head bound is written; the gather below reuses the scratch
  if (better(hb_s, hb_i, ts, ti)) {
    ts = hb_s;
    ti = hb_i;
  }
  // 2. gather the candidates at least as good as the bound (eight loads per thread in flight)
  for (int c0 = tid; c0 < total; c0 += 8 * blockDim.x) {
    float va[8];
    int vb[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int c = c0 + u * blockDim.x;
      va[u] = c < total ? __ldcg(cs + c) : -INFINITY;
      vb[u] = c < total ? __ldcg(ci + c) : INT_MAX;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      if (vb[u] != INT_MAX && !better(ts, ti, va[u], vb[u])) {
        const int p = atomicAdd(&nsurv, 1);
        if (p < cap) {
          ss[p] = va[u];
          si[p] = vb[u];
        }
      }
    }
  }
  __syncthreads();
  const int nsv = nsurv;
  if (nsv <= 32 && k <= 32) {  // 3a. few of them (the usual case): one warp sorts them with shuffles
    if (warp == 0) {
      float sv = lane < nsv ? ss[lane] : -INFINITY;
      int iv = lane < nsv ? si[lane] : INT_MAX;
      warp_sort32(sv, iv);
      if (lane < k) {
        const bool empty = iv == INT_MAX;
        out_ids[lane] = empty ? -1 : ext ? (int64_t)__ldg(ext + iv) : (int64_t)iv;
        out_scores[lane] = empty ? -INFINITY : sv;
      }
    }
    return;
  }
  int P = 1;
  while (P < nsv || P < k) P <<= 1;
  if (P <= cap) {  // 3. sort them (the order is total: the result does not depend on the gathering order)
    for (int i = nsv + tid; i < P; i += blockDim.x) {
      ss[i] = -INFINITY;
      si[i] = INT_MAX;
    }
    __syncthreads();
    block_sort(ss, si, P);
    for (int i = tid; i < k; i += blockDim.x) {
      const bool empty = si[i] == INT_MAX;
      out_ids[i] = empty ? -1 : ext ? (int64_t)__ldg(ext + si[i]) : (int64_t)si[i];
      out_scores[i] = empty ? -INFINITY : ss[i];
    }
    return;
  }
  // too many to sort in the scratch: each warp inserts its share into a list of k
  auto rs = [&](int c) { return __ldcg(cs + c); };
  auto ri = [&](int c) { return __ldcg(ci + c); };
  for (int i = lane; i < k; i += 32) {
    ws[warp * k + i] = -INFINITY;
    wi[warp * k + i] = INT_MAX;
  }
  __syncthreads();
  // 2. per-warp sorted top-k of the candidates at least as good as T
  float* ls = ws + warp * k;
  int* li = wi + warp * k;
  int cnt = 0;
  float th_s = -INFINITY;
  int th_i = INT_MAX;
  for (int c0 = warp * 32; c0 < total; c0 += blockDim.x) {
    const int c = c0 + lane;
    float a = -INFINITY;
    int b = INT_MAX;
    if (c < total) {
      a = rs(c);
      b = ri(c);
    }
    const bool cand = b != INT_MAX && !better(ts, ti, a, b) && better(a, b, th_s, th_i);
    unsigned m = __ballot_sync(FULL, cand);
    while (m) {
      const int src = __ffs(m) - 1;
      m &= m - 1;
      const float sv = __shfl_sync(FULL, a, src);
      const int iv = __shfl_sync(FULL, b, src);
      if (better(sv, iv, th_s, th_i)) {
        warp_insert(ls, li, k, cnt, sv, iv);
        cnt = min(cnt + 1, k);
        if (cnt == k) {
          th_s = ls[k - 1];
          th_i = li[k - 1];
        }
      }
    }
  }
  __syncthreads();
  // 3. warp 0 folds the other warps' sorted lists into its own
  if (warp == 0) {
    for (int w = 1; w < nwarps; ++w) {
      for (int i = 0; i < k; ++i) {
        const float sv = ws[w * k + i];
        const int iv = wi[w * k + i];
        if (iv == INT_MAX || !better(sv, iv, th_s, th_i)) break;  // sorted: the rest are worse
        warp_insert(ls, li, k, cnt, sv, iv);
        cnt = min(cnt + 1, k);
        if (cnt == k) {
          th_s = ls[k - 1];
          th_i = li[k - 1];
        }
      }
    }
    for (int i = lane; i < k; i += 32) {
      const bool empty = li[i] == INT_MAX;
      out_ids[i] = empty ? -1 : ext ? (int64_t)__ldg(ext + li[i]) : (int64_t)li[i];
      out_scores[i] = empty ? -INFINITY : ls[i];
    }
  }
}

// Publishes a scan CTA's sorted list of k (already in cand_*) and, in the
// last CTA of the query to finish (an arrival counter per query, zeroed by
// the query rotation that starts every search), merges all of the query's
// lists into its results: no separate merge launch.  ls/li: the CTA's list
// scratch (at least blockDim.x / 32 * k entries).
__device__ __forceinline__ void merge_if_last(const float* cand_s, const int* cand_i, int k, int* counters,
                                              const uint64_t* ext, int64_t* out_ids, float* out_scores, float* ls,
                                              int* li, unsigned char* scratch, size_t scratch_bytes) {
  __shared__ int last;
  const int q = blockIdx.y;
  __syncthreads();  // the CTA's list is written ...
  if (threadIdx.x == 0) {
    // one acquire-release arrival: releases this CTA's list (through the
    // barrier) and, for the last CTA, acquires every other CTA's
    int prev;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(prev) : "l"(counters + q) : "memory");
    last = prev == (int)gridDim.x - 1;
  }
  __syncthreads();
  if (!last) return;
  const size_t base = (size_t)q * gridDim.x * k;
  merge_lists_block(cand_s + base, cand_i + base, gridDim.x, k, ext, out_ids + (size_t)q * k,
                    out_scores + (size_t)q * k, ls, li, scratch, scratch_bytes);
}

// The CTA's top-k from its warps' sorted lists (warp w's k entries at w*k,
// padded with (-inf, INT_MAX)), written to out.  With k <= 32, warp 0 merges
// them: a list head per lane, k rounds of a warp argmax, the winning lane's
// list advancing; otherwise the block sorts all P entries.
__device__ __forceinline__ void cta_lists_out(float* ls, int* li, int nw, int k, int P, float* out_s, int* out_i) {
  const int tid = threadIdx.x, lane = tid & 31;
  if (k <= 32 && nw <= 32) {
    if (tid < 32) {
      int pos = 0;
      for (int r = 0; r < k; ++r) {
        float bs = -INFINITY;
        int bi = INT_MAX;
        if (lane < nw && pos < k) {
          bs = ls[lane * k + pos];
          bi = li[lane * k + pos];
        }
        int bl = lane;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          const float os = __shfl_xor_sync(FULL, bs, o);
          const int oi = __shfl_xor_sync(FULL, bi, o);
          const int ol = __shfl_xor_sync(FULL, bl, o);
          // identical (padding) entries: the lowest lane wins, so every lane agrees
          if (better(os, oi, bs, bi) || (os == bs && oi == bi && ol < bl)) {
            bs = os;
            bi = oi;
            bl = ol;
          }
        }
        if (lane == 0) {
          out_s[r] = bs;
          out_i[r] = bi;
        }
        if (lane == bl) ++pos;
      }
    }
    return;
  }
  block_sort(ls, li, P);
  for (int i = tid; i < k; i += blockDim.x) {
    out_s[i] = ls[i];
    out_i[i] = li[i];
  }
}

}  // namespace
}  // namespace tq
