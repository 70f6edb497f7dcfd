// Search-side kernels: the lookup scan with fused top-k (Sec. II-B step 5,
// Sec. III-B), per-query allow bitmaps, the filter build and the final merge.
//
// Lookup scan layout.  One warp scores 8 consecutive vectors per step.  Each
// packed row is cut into chunks of 16 codes (2*bits bytes); lane l owns chunks
// l, l+32, l+64, ... of every row, so each load instruction of a warp reads a
// contiguous run of one row and every lane always handles the same
// coordinates.  Lane l keeps the rotated query's values for its coordinates
// in registers and looks the centroid of each code up in a table replicated
// across the 32 shared-memory banks (entry (code, lane) lives in bank lane), so
// the lookups of a warp never conflict.  score = scale * sum_j q'_j c[code_j].
//
// Top-k: each warp keeps a sorted list of its k best (score desc, id asc) in
// shared memory, entered only when a score beats the list's k-th entry; a
// disallowed vector never enters (Sec. III-B: dropped at heap insert), and
// neither does a deleted one (its bit set in the caller's tombstone bitmap,
// the O(1) deletion of the id-mapped index of Sec. III-A).  Blocks
// of `block` vectors whose tenant bitmap shares no bit with the query's allow
// bitmap are skipped before any code byte is read (Sec. III-B).
#include <cuda_runtime.h>

#include <climits>
#include <limits>
#include <cmath>
#include <cstdint>

#include "tq_internal.h"
#include "tq_kernels.h"

namespace tq {
namespace {

constexpr unsigned FULL = 0xffffffffu;

// Bit v % 32 of word v / 32 of the tombstone bitmap marks row v deleted.  It
// is read only for a vector that would enter a list, so a scan with few
// candidates per step pays almost nothing for it.
__device__ __forceinline__ bool tombstoned(const uint32_t* __restrict__ del, int v) {
  return del && ((__ldg(del + (v >> 5)) >> (v & 31)) & 1u);
}
constexpr int SCAN_NT = 256;
constexpr int SCAN_WARPS = SCAN_NT / 32;
constexpr int MERGE_P = 2048;

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

// Shifts x so that the bit at position p lands at bit 7 (p is a compile-time
// constant after unrolling).
__device__ __forceinline__ uint32_t to_bit7(uint32_t x, int p) { return p >= 7 ? x >> (p - 7) : x << (7 - p); }

// 16 codes of `BITS` bits starting at a chunk boundary.  off(t, lane4) is the
// byte offset of code t's entry for this lane in the bank-replicated centroid
// table (entry (c, lane) at (c * 32 + lane) * 4): one shift and one
// three-input logic op per code.
template <int BITS>
struct Chunk;

template <>
struct Chunk<4> {
  uint32_t w0, w1;
  __device__ __forceinline__ void load(const uint8_t* p) {
    const uint2 v = __ldcs(reinterpret_cast<const uint2*>(p));
    w0 = v.x;
    w1 = v.y;
  }
  __device__ __forceinline__ void zero() { w0 = w1 = 0; }
  __device__ __forceinline__ uint32_t off(int t, uint32_t lane4) const {
    return (to_bit7(t < 8 ? w0 : w1, 4 * (t & 7)) & 0x780u) | lane4;
  }
};

template <>
struct Chunk<2> {
  uint32_t w;
  __device__ __forceinline__ void load(const uint8_t* p) { w = __ldcs(reinterpret_cast<const unsigned int*>(p)); }
  __device__ __forceinline__ void zero() { w = 0; }
  __device__ __forceinline__ uint32_t off(int t, uint32_t lane4) const { return (to_bit7(w, 2 * t) & 0x180u) | lane4; }
};

template <>
struct Chunk<8> {
  uint4 w;
  __device__ __forceinline__ void load(const uint8_t* p) { w = __ldcs(reinterpret_cast<const uint4*>(p)); }
  __device__ __forceinline__ void zero() { w = make_uint4(0, 0, 0, 0); }
  __device__ __forceinline__ uint32_t off(int t, uint32_t lane4) const {
    const uint32_t x = t < 4 ? w.x : t < 8 ? w.y : t < 12 ? w.z : w.w;
    return (to_bit7(x, 8 * (t & 3)) & 0x7F80u) | lane4;
  }
};

template <>
struct Chunk<3> {
  uint64_t v;  // 48 bits
  __device__ __forceinline__ void load(const uint8_t* p) {
    const unsigned short* h = reinterpret_cast<const unsigned short*>(p);
    v = (uint64_t)__ldcs(h) | ((uint64_t)__ldcs(h + 1) << 16) | ((uint64_t)__ldcs(h + 2) << 32);
  }
  __device__ __forceinline__ void zero() { v = 0; }
  __device__ __forceinline__ uint32_t off(int t, uint32_t lane4) const {
    const int p = 3 * t;
    const uint32_t x = (uint32_t)(p >= 7 ? v >> (p - 7) : v << (7 - p));
    return (x & 0x380u) | lane4;
  }
};

// Byte-pair lookups for 4-bit codes.  A packed byte x holds two codes, so one
// 8-byte load of T[x] = (c[x & 15], c[x >> 4]) fetches both centroids and one
// paired FMA adds q'_{2m} c[x & 15] and q'_{2m+1} c[x >> 4] into a float2
// accumulator: per two codes one byte permute (the byte moved to bits 8..15
// next to lane * 8, which is the entry's address), one shared load and one
// FMA instruction.  T is replicated per lane, entry (x, lane) at
// (x * 32 + lane) * 8 bytes, so a warp's 32 loads hit 32 different 8-byte
// bank pairs in two wavefronts whatever the bytes are.
constexpr int PAIR_TAB_BYTES = 256 * 32 * 8;

__device__ __forceinline__ void pair_table_init(float2* ptab, const float* __restrict__ centroids, int tid, int nt) {
  for (int i = tid; i < 256 * 32; i += nt) {
    const int x = i >> 5;
    ptab[i] = make_float2(__ldg(centroids + (x & 15)), __ldg(centroids + (x >> 4)));
  }
}

// This lane's part of one vector's score: its S chunks of 16 codes against
// the matching (q'_{2m}, q'_{2m+1}) pairs.  Both 4-bit scans use exactly this
// order of operations, so filtered and unfiltered scores agree bit for bit.
template <int S>
__device__ __forceinline__ float pair_dot(const Chunk<4> (&ch)[S], const float2 (&q2)[S][8], const char* tab,
                                          uint32_t lane8) {
  float2 acc = make_float2(0.f, 0.f);
#pragma unroll
  for (int s = 0; s < S; ++s) {
#pragma unroll
    for (int b = 0; b < 8; ++b) {
      const uint32_t w = b < 4 ? ch[s].w0 : ch[s].w1;
      const uint32_t addr = __byte_perm(w, lane8, 0x5504u | ((uint32_t)(b & 3) << 4));
      acc = __ffma2_rn(q2[s][b], *reinterpret_cast<const float2*>(tab + addr), acc);
    }
  }
  return acc.x + acc.y;
}

template <int S>
__device__ __forceinline__ void load_q2(float2 (&q2)[S][8], const float* qq, int nchunks, int lane) {
#pragma unroll
  for (int s = 0; s < S; ++s) {
    const int chunk = lane + 32 * s;
#pragma unroll
    for (int m = 0; m < 8; ++m)
      q2[s][m] = chunk < nchunks ? make_float2(qq[chunk * 16 + 2 * m], qq[chunk * 16 + 2 * m + 1])
                                 : make_float2(0.f, 0.f);
  }
}

// Sums p[0..7] across the warp: afterwards lanes 4i..4i+3 hold the total of
// p[i] (a transposed butterfly: 4 + 2 + 1 + 1 + 1 shuffles for 8 values).
__device__ __forceinline__ float warp_sum8(float (&p)[8]) {
  const int lane = threadIdx.x & 31;
  const bool h16 = lane & 16, h8 = lane & 8, h4 = lane & 4;
  float a[4], b[2];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float send = h16 ? p[i] : p[i + 4];
    const float keep = h16 ? p[i + 4] : p[i];
    a[i] = keep + __shfl_xor_sync(FULL, send, 16);
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const float send = h8 ? a[i] : a[i + 2];
    const float keep = h8 ? a[i + 2] : a[i];
    b[i] = keep + __shfl_xor_sync(FULL, send, 8);
  }
  float c = (h4 ? b[1] : b[0]) + __shfl_xor_sync(FULL, h4 ? b[0] : b[1], 4);
  c += __shfl_xor_sync(FULL, c, 2);
  c += __shfl_xor_sync(FULL, c, 1);
  return c;
}

// Each warp scores 8 consecutive vectors per step: all their code loads (and
// their scales and tenants) are issued before any arithmetic, so a warp keeps
// 8 x d*bits/8 bytes in flight.
template <int BITS, int S>
__global__ void __launch_bounds__(SCAN_NT, 2)
k_scan_lut(const float* __restrict__ qrot, int d, const float* __restrict__ centroids,
           const uint8_t* __restrict__ codes, const float* __restrict__ scale, int n,
           const uint32_t* __restrict__ del,
           const uint32_t* __restrict__ dense, const uint32_t* __restrict__ block_bits, int words,
           int fblock, const uint32_t* __restrict__ allow_bits, int k, int P,
           float* __restrict__ cand_s, int* __restrict__ cand_i) {
  constexpr int L = 1 << BITS;
  constexpr int CB = 2 * BITS;
  constexpr int V = 8;  // vectors per warp step; a CTA step covers 64
  // 4-bit codes use the byte-pair table (pair_dot), other widths the
  // per-code table [L][32] with entry (c, lane) in bank lane
  constexpr int TAB_BYTES = BITS == 4 ? PAIR_TAB_BYTES : L * 32 * 4;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  float* ctab = reinterpret_cast<float*>(smem_raw);
  float* ls = reinterpret_cast<float*>(smem_raw + TAB_BYTES);  // [P] scores; warp w's list at [w*k, w*k+k)
  int* li = reinterpret_cast<int*>(ls + P);                     // [P] ids
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int q = blockIdx.y;
  if constexpr (BITS == 4) pair_table_init(reinterpret_cast<float2*>(smem_raw), centroids, tid, SCAN_NT);
  else
    for (int i = tid; i < L * 32; i += SCAN_NT) ctab[i] = __ldg(centroids + (i >> 5));
  for (int i = tid; i < P; i += SCAN_NT) {
    ls[i] = -INFINITY;
    li[i] = INT_MAX;
  }
  const int nchunks = d >> 4;
  const float* qq = qrot + (size_t)q * d;
  float qr[BITS == 4 ? 1 : S][16];
  float2 q2[BITS == 4 ? S : 1][8];
  if constexpr (BITS == 4) {
    load_q2(q2, qq, nchunks, lane);
  } else {
#pragma unroll
    for (int s = 0; s < S; ++s) {
      const int chunk = lane + 32 * s;
#pragma unroll
      for (int t = 0; t < 16; ++t) qr[s][t] = chunk < nchunks ? qq[chunk * 16 + t] : 0.f;
    }
  }
  __syncthreads();

  const int64_t row_bytes = (int64_t)d * BITS / 8;
  const uint32_t* ab = allow_bits ? allow_bits + (size_t)q * words : nullptr;
  float* wl_s = ls + warp * k;
  int* wl_i = li + warp * k;
  int cnt = 0;
  float th_s = -INFINITY;
  int th_i = INT_MAX;
  const int nsteps = (n + SCAN_WARPS * V - 1) / (SCAN_WARPS * V);
  const int my = (lane >> 2) & 7;  // the vector whose total this lane ends up holding
  const uint32_t lane4 = (uint32_t)lane * 4u;
  for (int st = blockIdx.x; st < nsteps; st += gridDim.x) {
    const int v0 = st * (SCAN_WARPS * V) + warp * V;
    if (v0 >= n) continue;
    if (ab) {  // the warp's 8 vectors lie in one filter block (block is 32 or 64)
      const int fb = v0 / fblock;
      uint32_t any = 0;
      for (int w = lane; w < words; w += 32) any |= __ldg(block_bits + (size_t)fb * words + w) & __ldg(ab + w);
      if (!__any_sync(FULL, any != 0u)) continue;  // no allowed vector: skip before reading codes
    }
    const int vm = v0 + my;
    float sc_my = 0.f;
    uint32_t ten_my = 0;
    if ((lane & 3) == 0 && vm < n) {
      sc_my = scale ? __ldg(scale + vm) : 1.0f;
      if (ab) ten_my = __ldg(dense + vm);
    }
    Chunk<BITS> ch[V][S];
#pragma unroll
    for (int i = 0; i < V; ++i) {
      const uint8_t* row = codes + (size_t)(v0 + i) * row_bytes;
#pragma unroll
      for (int s = 0; s < S; ++s) {
        const int chunk = lane + 32 * s;
        if (v0 + i < n && chunk < nchunks) ch[i][s].load(row + chunk * CB);
        else ch[i][s].zero();
      }
    }
    // keep every load above in flight before the first lookup below
    asm volatile("" ::: "memory");
    float p[V];
    const char* tab = reinterpret_cast<const char*>(ctab);
#pragma unroll
    for (int i = 0; i < V; ++i) {
      if constexpr (BITS == 4) {
        p[i] = pair_dot<S>(ch[i], q2, tab, lane4 * 2u);
      } else {
        float acc = 0.f;
#pragma unroll
        for (int s = 0; s < S; ++s)
#pragma unroll
          for (int t = 0; t < 16; ++t)
            acc = fmaf(qr[s][t], *reinterpret_cast<const float*>(tab + ch[i][s].off(t, lane4)), acc);
        p[i] = acc;
      }
    }
    const float total = warp_sum8(p);
    float score = -INFINITY;
    bool cand = false;
    if ((lane & 3) == 0 && vm < n) {
      score = total * sc_my;
      const bool allowed = !ab || ((__ldg(ab + (ten_my >> 5)) >> (ten_my & 31)) & 1u);
      cand = allowed && better(score, vm, th_s, th_i) && !tombstoned(del, vm);
    }
    unsigned m = __ballot_sync(FULL, cand);
    while (m) {  // in vector order; re-checked against the moving threshold
      const int src = __ffs(m) - 1;
      m &= m - 1;
      const float s = __shfl_sync(FULL, score, src);
      const int vv = v0 + ((src >> 2) & 7);
      if (better(s, vv, th_s, th_i)) {
        warp_insert(wl_s, wl_i, k, cnt, s, vv);
        cnt = min(cnt + 1, k);
        if (cnt == k) {
          th_s = wl_s[k - 1];
          th_i = wl_i[k - 1];
        }
      }
    }
  }
  __syncthreads();
  block_sort(ls, li, P);
  for (int i = tid; i < k; i += SCAN_NT) {
    const size_t o = ((size_t)q * gridDim.x + blockIdx.x) * k + i;
    cand_s[o] = ls[i];
    cand_i[o] = li[i];
  }
}

// Sums p[0..3] across the warp: afterwards lanes 8i..8i+7 hold the total of
// p[i] (2 + 1 + 1 + 1 + 1 shuffles for 4 values).
__device__ __forceinline__ float warp_sum4(float (&p)[4]) {
  const int lane = threadIdx.x & 31;
  const bool h16 = lane & 16, h8 = lane & 8;
  float a[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const float send = h16 ? p[i] : p[i + 2];
    const float keep = h16 ? p[i + 2] : p[i];
    a[i] = keep + __shfl_xor_sync(FULL, send, 16);
  }
  float c = (h8 ? a[1] : a[0]) + __shfl_xor_sync(FULL, h8 ? a[0] : a[1], 8);
  c += __shfl_xor_sync(FULL, c, 4);
  c += __shfl_xor_sync(FULL, c, 2);
  c += __shfl_xor_sync(FULL, c, 1);
  return c;
}

// Unfiltered lookup scan with a register double buffer: each warp scores 4
// consecutive vectors per step and issues the next step's code loads before
// it starts on the current ones, so every warp always has loads in flight.
template <int BITS, int S>
__global__ void __launch_bounds__(SCAN_NT, 2)
k_scan_lut_stream(const float* __restrict__ qrot, int d, const float* __restrict__ centroids,
                  const uint8_t* __restrict__ codes, const float* __restrict__ scale, int n,
                  const uint32_t* __restrict__ del, int k, int P,
                  float* __restrict__ cand_s, int* __restrict__ cand_i) {
  constexpr int L = 1 << BITS;
  constexpr int CB = 2 * BITS;
  constexpr int V = 4;  // vectors per warp step; a CTA step covers 32
  extern __shared__ __align__(16) unsigned char smem_raw[];
  float* ctab = reinterpret_cast<float*>(smem_raw);  // [L][32], entry (c, lane) in bank lane
  float* ls = ctab + L * 32;                          // [P] scores; warp w's list at [w*k, w*k+k)
  int* li = reinterpret_cast<int*>(ls + P);           // [P] ids
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int q = blockIdx.y;
  for (int i = tid; i < L * 32; i += SCAN_NT) ctab[i] = __ldg(centroids + (i >> 5));
  for (int i = tid; i < P; i += SCAN_NT) {
    ls[i] = -INFINITY;
    li[i] = INT_MAX;
  }
  const int nchunks = d >> 4;
  const float* qq = qrot + (size_t)q * d;
  float qr[S][16];
#pragma unroll
  for (int s = 0; s < S; ++s) {
    const int chunk = lane + 32 * s;
#pragma unroll
    for (int t = 0; t < 16; ++t) qr[s][t] = chunk < nchunks ? qq[chunk * 16 + t] : 0.f;
  }
  __syncthreads();

  const int64_t row_bytes = (int64_t)d * BITS / 8;
  float* wl_s = ls + warp * k;
  int* wl_i = li + warp * k;
  int cnt = 0;
  float th_s = -INFINITY;
  int th_i = INT_MAX;
  const int nsteps = (n + SCAN_WARPS * V - 1) / (SCAN_WARPS * V);
  const int my = (lane >> 3) & 3;  // the vector whose total this lane ends up holding
  const uint32_t lane4 = (uint32_t)lane * 4u;
  const char* tab = reinterpret_cast<const char*>(ctab);

  Chunk<BITS> cur[V][S], nxt[V][S];
  float sc_cur = 0.f, sc_nxt = 0.f;
  auto load_step = [&](int st, Chunk<BITS> (&buf)[V][S], float& sc) {
    const int v0 = st * (SCAN_WARPS * V) + warp * V;
#pragma unroll
    for (int i = 0; i < V; ++i) {
      const uint8_t* row = codes + (size_t)(v0 + i) * row_bytes;
#pragma unroll
      for (int s = 0; s < S; ++s) {
        const int chunk = lane + 32 * s;
        if (st < nsteps && v0 + i < n && chunk < nchunks) buf[i][s].load(row + chunk * CB);
        else buf[i][s].zero();
      }
    }
    const int vm = v0 + my;
    sc = 0.f;
    if (st < nsteps && (lane & 7) == 0 && vm < n) sc = scale ? __ldg(scale + vm) : 1.0f;
  };
  int st = blockIdx.x;
  load_step(st, cur, sc_cur);
  for (; st < nsteps; st += gridDim.x) {
    load_step(st + gridDim.x, nxt, sc_nxt);   // next step's loads go out first
    asm volatile("" ::: "memory");
    const int v0 = st * (SCAN_WARPS * V) + warp * V;
    float p[V];
#pragma unroll
    for (int i = 0; i < V; ++i) {
      float acc = 0.f;
#pragma unroll
      for (int s = 0; s < S; ++s)
#pragma unroll
        for (int t = 0; t < 16; ++t)
          acc = fmaf(qr[s][t], *reinterpret_cast<const float*>(tab + cur[i][s].off(t, lane4)), acc);
      p[i] = acc;
    }
    const float total = warp_sum4(p);
    const int vm = v0 + my;
    float score = -INFINITY;
    bool cand = false;
    if ((lane & 7) == 0 && vm < n) {
      score = total * sc_cur;
      cand = better(score, vm, th_s, th_i) && !tombstoned(del, vm);
    }
    unsigned m = __ballot_sync(FULL, cand);
    while (m) {  // in vector order; re-checked against the moving threshold
      const int src = __ffs(m) - 1;
      m &= m - 1;
      const float sv = __shfl_sync(FULL, score, src);
      const int vv = v0 + ((src >> 3) & 3);
      if (better(sv, vv, th_s, th_i)) {
        warp_insert(wl_s, wl_i, k, cnt, sv, vv);
        cnt = min(cnt + 1, k);
        if (cnt == k) {
          th_s = wl_s[k - 1];
          th_i = wl_i[k - 1];
        }
      }
    }
#pragma unroll
    for (int i = 0; i < V; ++i)
#pragma unroll
      for (int s = 0; s < S; ++s) cur[i][s] = nxt[i][s];
    sc_cur = sc_nxt;
  }
  __syncthreads();
  block_sort(ls, li, P);
  for (int i = tid; i < k; i += SCAN_NT) {
    const size_t o = ((size_t)q * gridDim.x + blockIdx.x) * k + i;
    cand_s[o] = ls[i];
    cand_i[o] = li[i];
  }
}

// Unfiltered 4-bit scan with byte-pair lookups (pair_dot); otherwise as
// k_scan_lut_stream: 4 vectors per warp step, next step's loads in flight.
template <int S>
__global__ void __launch_bounds__(SCAN_NT, 2)
k_scan_pair_stream(const float* __restrict__ qrot, int d, const float* __restrict__ centroids,
                   const uint8_t* __restrict__ codes, const float* __restrict__ scale, int n,
                   const uint32_t* __restrict__ del, int k, int P,
                   float* __restrict__ cand_s, int* __restrict__ cand_i) {
  constexpr int V = 4;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  float2* ptab = reinterpret_cast<float2*>(smem_raw);  // [256][32]
  float* ls = reinterpret_cast<float*>(smem_raw + PAIR_TAB_BYTES);
  int* li = reinterpret_cast<int*>(ls + P);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int q = blockIdx.y;
  pair_table_init(ptab, centroids, tid, SCAN_NT);
  for (int i = tid; i < P; i += SCAN_NT) {
    ls[i] = -INFINITY;
    li[i] = INT_MAX;
  }
  const int nchunks = d >> 4;
  float2 q2[S][8];  // (q'_{2m}, q'_{2m+1}) of the 16 coordinates of chunk lane + 32 s
  load_q2(q2, qrot + (size_t)q * d, nchunks, lane);
  __syncthreads();

  const int64_t row_bytes = (int64_t)d / 2;
  float* wl_s = ls + warp * k;
  int* wl_i = li + warp * k;
  int cnt = 0;
  float th_s = -INFINITY;
  int th_i = INT_MAX;
  const int nsteps = (n + SCAN_WARPS * V - 1) / (SCAN_WARPS * V);
  const int my = (lane >> 3) & 3;
  const uint32_t lane8 = (uint32_t)lane * 8u;
  const char* tab = reinterpret_cast<const char*>(ptab);

  Chunk<4> cur[V][S], nxt[V][S];
  float sc_cur = 0.f, sc_nxt = 0.f;
  auto load_step = [&](int st, Chunk<4> (&buf)[V][S], float& sc) {
    const int v0 = st * (SCAN_WARPS * V) + warp * V;
#pragma unroll
    for (int i = 0; i < V; ++i) {
      const uint8_t* row = codes + (size_t)(v0 + i) * row_bytes;
#pragma unroll
      for (int s = 0; s < S; ++s) {
        const int chunk = lane + 32 * s;
        if (st < nsteps && v0 + i < n && chunk < nchunks) buf[i][s].load(row + chunk * 8);
        else buf[i][s].zero();
      }
    }
    const int vm = v0 + my;
    sc = 0.f;
    if (st < nsteps && (lane & 7) == 0 && vm < n) sc = scale ? __ldg(scale + vm) : 1.0f;
  };
  int st = blockIdx.x;
  load_step(st, cur, sc_cur);
  for (; st < nsteps; st += gridDim.x) {
    load_step(st + gridDim.x, nxt, sc_nxt);
    asm volatile("" ::: "memory");
    const int v0 = st * (SCAN_WARPS * V) + warp * V;
    float p[V];
#pragma unroll
    for (int i = 0; i < V; ++i) p[i] = pair_dot<S>(cur[i], q2, tab, lane8);
    const float total = warp_sum4(p);
    const int vm = v0 + my;
    float score = -INFINITY;
    bool cand = false;
    if ((lane & 7) == 0 && vm < n) {
      score = total * sc_cur;
      cand = better(score, vm, th_s, th_i) && !tombstoned(del, vm);
    }
    unsigned m = __ballot_sync(FULL, cand);
    while (m) {
      const int src = __ffs(m) - 1;
      m &= m - 1;
      const float sv = __shfl_sync(FULL, score, src);
      const int vv = v0 + ((src >> 3) & 3);
      if (better(sv, vv, th_s, th_i)) {
        warp_insert(wl_s, wl_i, k, cnt, sv, vv);
        cnt = min(cnt + 1, k);
        if (cnt == k) {
          th_s = wl_s[k - 1];
          th_i = wl_i[k - 1];
        }
      }
    }
#pragma unroll
    for (int i = 0; i < V; ++i)
#pragma unroll
      for (int s = 0; s < S; ++s) cur[i][s] = nxt[i][s];
    sc_cur = sc_nxt;
  }
  __syncthreads();
  block_sort(ls, li, P);
  for (int i = tid; i < k; i += SCAN_NT) {
    const size_t o = ((size_t)q * gridDim.x + blockIdx.x) * k + i;
    cand_s[o] = ls[i];
    cand_i[o] = li[i];
  }
}

// Merges the candidates of each query into its sorted top-k, P - k at a time.
// Candidates come from S sources laid out [S][nq][m]: candidate j of source
// src for query q is cand_*[(src * nq + q) * m + j].  Candidates whose id is
// `pad` never beat a real one and come out as (-1, -INFINITY).
template <typename I>
__global__ void __launch_bounds__(1024)
k_merge(const float* __restrict__ cand_s, const I* __restrict__ cand_i, int64_t S, int64_t nq, int64_t m, int k,
        int P, I pad, int64_t* __restrict__ out_ids, float* __restrict__ out_scores) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  I* id = reinterpret_cast<I*>(smem_raw);
  float* s = reinterpret_cast<float*>(id + P);
  const int64_t q = blockIdx.x;
  const int64_t total = S * m;
  constexpr I kWorst = std::numeric_limits<I>::max();
  for (int i = threadIdx.x; i < k; i += blockDim.x) {
    s[i] = -INFINITY;
    id[i] = kWorst;
  }
  const int chunk = P - k;
  for (int64_t c0 = 0; c0 < total; c0 += chunk) {
    for (int i = threadIdx.x; i < chunk; i += blockDim.x) {
      const int64_t c = c0 + i;
      float sv = -INFINITY;
      I v = kWorst;
      if (c < total) {
        const int64_t src = c / m, j = c - src * m;
        const int64_t o = (src * nq + q) * m + j;
        if (cand_i[o] != pad) {
          v = cand_i[o];
          sv = cand_s[o];
        }
      }
      s[k + i] = sv;
      id[k + i] = v;
    }
    __syncthreads();
    block_sort(s, id, P);
  }
  for (int i = threadIdx.x; i < k; i += blockDim.x) {
    const bool empty = id[i] == kWorst;
    out_ids[q * k + i] = empty ? -1 : (int64_t)id[i];
    out_scores[q * k + i] = empty ? -INFINITY : s[i];
  }
}

// Merge of per-CTA candidate lists that are each sorted best first and hold
// exactly k entries (padding (-inf, INT_MAX) at the end).  The k-th entry T of
// any one list is beaten or matched by that list's k entries, so the global
// k-th best is at least as good as the best such T and worse candidates are
// skipped at once.  Each warp keeps a sorted top-k of its share of the rest
// (ballot, then one warp-wide insertion per candidate that still beats the
// warp's k-th); warp 0 then folds the sorted warp lists into the result,
// leaving each list at its first entry that no longer qualifies.  With an
// id map the result rows are written as their external ids.
__global__ void __launch_bounds__(1024)
k_merge_lists(const float* __restrict__ cand_s, const int* __restrict__ cand_i, int nlists, int k,
              const uint64_t* __restrict__ ext, int64_t* __restrict__ out_ids, float* __restrict__ out_scores) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int nwarps = blockDim.x >> 5;
  float* ws = reinterpret_cast<float*>(smem_raw);  // [nwarps][k]
  int* wi = reinterpret_cast<int*>(ws + nwarps * k);
  __shared__ float red_s[32];
  __shared__ int red_i[32];
  const int64_t q = blockIdx.x;
  const int total = nlists * k;
  const float* cs = cand_s + q * total;
  const int* ci = cand_i + q * total;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // 1. T = best k-th entry over the lists
  float ts = -INFINITY;
  int ti = INT_MAX;
  for (int l = tid; l < nlists; l += blockDim.x) {
    const float a = cs[l * k + k - 1];
    const int b = ci[l * k + k - 1];
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
  for (int i = lane; i < k; i += 32) {
    ws[warp * k + i] = -INFINITY;
    wi[warp * k + i] = INT_MAX;
  }
  __syncthreads();
  ts = red_s[0];
  ti = red_i[0];
  for (int w = 1; w < nwarps; ++w)
    if (better(red_s[w], red_i[w], ts, ti)) {
      ts = red_s[w];
      ti = red_i[w];
    }
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
      a = cs[c];
      b = ci[c];
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
      out_ids[q * k + i] = empty ? -1 : ext ? (int64_t)__ldg(ext + li[i]) : (int64_t)li[i];
      out_scores[q * k + i] = empty ? -INFINITY : ls[i];
    }
  }
}

__device__ __forceinline__ int64_t find_tenant(const uint32_t* __restrict__ tenants, int64_t T, uint32_t x) {
  int64_t lo = 0, hi = T;
  while (lo < hi) {
    const int64_t mid = (lo + hi) >> 1;
    if (__ldg(tenants + mid) < x) lo = mid + 1; else hi = mid;
  }
  return (lo < T && __ldg(tenants + lo) == x) ? lo : -1;
}

__global__ void k_allow_bits(const uint32_t* __restrict__ tenants, int64_t T, int words,
                             const int64_t* __restrict__ off, const uint32_t* __restrict__ ids,
                             uint32_t* __restrict__ out) {
  const int64_t q = blockIdx.x;
  uint32_t* o = out + q * words;
  for (int w = threadIdx.x; w < words; w += blockDim.x) o[w] = 0u;
  __syncthreads();
  const int64_t a = off[q], b = off[q + 1];
  for (int64_t j = a + threadIdx.x; j < b; j += blockDim.x) {
    const int64_t pos = find_tenant(tenants, T, ids[j]);
    if (pos >= 0) atomicOr(o + (pos >> 5), 1u << (pos & 31));
  }
}

// Rows v0 .. v0+n-1 get their dense tenant index and set their bit in their
// block's bitmap (bits already set by earlier rows of a shared block stay).
__global__ void k_filter_build(const uint32_t* __restrict__ tenant_ids, int64_t n, int64_t v0,
                               const uint32_t* __restrict__ tenants, int64_t T, int words, int block,
                               uint32_t* __restrict__ dense, uint32_t* __restrict__ block_bits) {
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < n; v += (int64_t)gridDim.x * blockDim.x) {
    const int64_t pos = find_tenant(tenants, T, tenant_ids[v]);  // always found: tenants holds every id
    const uint32_t p = (uint32_t)(pos < 0 ? 0 : pos);
    const int64_t r = v0 + v;
    dense[r] = p;
    atomicOr(block_bits + (r / block) * words + (p >> 5), 1u << (p & 31));
  }
}

// raw[v] = tenants[dense[v]]: the tenant ids of rows 0 .. n-1 back from a filter.
__global__ void k_filter_raw_ids(const uint32_t* __restrict__ dense, const uint32_t* __restrict__ tenants, int64_t n,
                                 uint32_t* __restrict__ raw) {
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < n; v += (int64_t)gridDim.x * blockDim.x)
    raw[v] = __ldg(tenants + __ldg(dense + v));
}

int next_pow2(int x) {
  int p = 1;
  while (p < x) p <<= 1;
  return p;
}

template <int BITS, int S>
cudaError_t scan_lut_typed(dim3 grid, size_t smem, cudaStream_t s, const float* qrot, int d,
                           const float* centroids, const uint8_t* codes, const float* scale, int n,
                           const uint32_t* del, const uint32_t* dense, const uint32_t* block_bits, int words, int fblock,
                           const uint32_t* allow, int k, int P, float* cs, int* ci) {
  cudaError_t e;
  if (BITS == 4 && !allow) {
    const size_t psmem = (size_t)PAIR_TAB_BYTES + (size_t)P * (sizeof(float) + sizeof(int));
    e = set_max_dynamic_smem(reinterpret_cast<const void*>(k_scan_pair_stream<S>), (int)psmem);
    if (e != cudaSuccess) return e;
    k_scan_pair_stream<S><<<grid, SCAN_NT, psmem, s>>>(qrot, d, centroids, codes, scale, n, del, k, P, cs, ci);
    return cudaGetLastError();
  }
  if (!allow) {
    e = set_max_dynamic_smem(reinterpret_cast<const void*>(k_scan_lut_stream<BITS, S>), (int)smem);
    if (e != cudaSuccess) return e;
    k_scan_lut_stream<BITS, S><<<grid, SCAN_NT, smem, s>>>(qrot, d, centroids, codes, scale, n, del, k, P, cs, ci);
    return cudaGetLastError();
  }
  const size_t fsmem = BITS == 4 ? (size_t)PAIR_TAB_BYTES + (size_t)P * (sizeof(float) + sizeof(int)) : smem;
  e = set_max_dynamic_smem(reinterpret_cast<const void*>(k_scan_lut<BITS, S>), (int)fsmem);
  if (e != cudaSuccess) return e;
  k_scan_lut<BITS, S><<<grid, SCAN_NT, fsmem, s>>>(qrot, d, centroids, codes, scale, n, del, dense, block_bits,
                                                   words, fblock, allow, k, P, cs, ci);
  return cudaGetLastError();
}

template <int BITS>
cudaError_t scan_lut_bits(int S, dim3 grid, size_t smem, cudaStream_t s, const float* qrot, int d,
                          const float* centroids, const uint8_t* codes, const float* scale, int n,
                          const uint32_t* del, const uint32_t* dense, const uint32_t* block_bits, int words, int fblock,
                          const uint32_t* allow, int k, int P, float* cs, int* ci) {
  switch (S) {
    case 1: return scan_lut_typed<BITS, 1>(grid, smem, s, qrot, d, centroids, codes, scale, n, del, dense, block_bits, words, fblock, allow, k, P, cs, ci);
    case 2: return scan_lut_typed<BITS, 2>(grid, smem, s, qrot, d, centroids, codes, scale, n, del, dense, block_bits, words, fblock, allow, k, P, cs, ci);
    case 3: return scan_lut_typed<BITS, 3>(grid, smem, s, qrot, d, centroids, codes, scale, n, del, dense, block_bits, words, fblock, allow, k, P, cs, ci);
    case 4: return scan_lut_typed<BITS, 4>(grid, smem, s, qrot, d, centroids, codes, scale, n, del, dense, block_bits, words, fblock, allow, k, P, cs, ci);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

int scan_lut_grid_x(int64_t nq, int64_t n, int k, int bits, int d) {
  (void)k;
  (void)bits;
  (void)d;
  // one resident wave (two CTAs per SM) for a single query
  const int64_t target = (int64_t)device_sm_count() * 2;
  int64_t gx = (target + nq - 1) / (nq > 0 ? nq : 1);
  const int64_t blocks = (n + 31) / 32;
  if (gx > blocks) gx = blocks;
  if (gx < 1) gx = 1;
  return (int)gx;
}

cudaError_t launch_scan_lut(const float* qrot, int64_t nq, int d, const float* centroids, int bits,
                            const uint8_t* codes, const float* scale, int64_t n, const uint32_t* del,
                            const FilterDev* f, const uint32_t* allow_bits, int k, int grid_x, float* cand_s,
                            int32_t* cand_i, cudaStream_t s, cudaEvent_t ev0, cudaEvent_t ev1) {
  if (nq == 0) return cudaSuccess;
  const int S = (d + 511) / 512;
  const int P = next_pow2(SCAN_WARPS * k);
  const size_t smem = (size_t)(1 << bits) * 32 * sizeof(float) + (size_t)P * (sizeof(float) + sizeof(int));
  const dim3 grid((unsigned)grid_x, (unsigned)nq);
  const uint32_t* dense = f ? f->dense : nullptr;
  const uint32_t* bb = f ? f->block_bits : nullptr;
  const int words = f ? f->words : 0;
  const int fblock = f ? f->block : 64;
  cudaError_t e;
  if (ev0 && (e = cudaEventRecord(ev0, s)) != cudaSuccess) return e;
  switch (bits) {
    case 2: e = scan_lut_bits<2>(S, grid, smem, s, qrot, d, centroids, codes, scale, (int)n, del, dense, bb, words, fblock, allow_bits, k, P, cand_s, cand_i); break;
    case 3: e = scan_lut_bits<3>(S, grid, smem, s, qrot, d, centroids, codes, scale, (int)n, del, dense, bb, words, fblock, allow_bits, k, P, cand_s, cand_i); break;
    case 4: e = scan_lut_bits<4>(S, grid, smem, s, qrot, d, centroids, codes, scale, (int)n, del, dense, bb, words, fblock, allow_bits, k, P, cand_s, cand_i); break;
    case 8: e = scan_lut_bits<8>(S, grid, smem, s, qrot, d, centroids, codes, scale, (int)n, del, dense, bb, words, fblock, allow_bits, k, P, cand_s, cand_i); break;
    default: e = cudaErrorInvalidValue;
  }
  if (e != cudaSuccess) return e;
  if (ev1 && (e = cudaEventRecord(ev1, s)) != cudaSuccess) return e;
  return cudaSuccess;
}

cudaError_t launch_merge(const float* cand_s, const int32_t* cand_i, int64_t nq, int per_query,
                         int k, const uint64_t* ext, int64_t* out_ids, float* out_scores, cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  // per_query = grid_x * k: one sorted list of k per scan CTA
  // up to 32 warps, fewer for long lists (each warp keeps k entries in shared memory)
  const int nlists = per_query / k;
  int warps = std::max(1, std::min(32, (nlists + 31) / 32));
  while (warps > 1 && (size_t)warps * k * 8 > 48 * 1024) warps >>= 1;
  const size_t smem = (size_t)warps * k * (sizeof(float) + sizeof(int32_t));
  k_merge_lists<<<(unsigned)nq, 32 * warps, smem, s>>>(cand_s, cand_i, nlists, k, ext, out_ids, out_scores);
  return cudaGetLastError();
}

cudaError_t launch_merge_global(const float* cand_s, const int64_t* cand_i, int64_t S, int64_t nq, int64_t m,
                                int k, int64_t* out_ids, float* out_scores, cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  const int64_t total = S * m;
  int P = next_pow2((int)std::min<int64_t>(total + k, MERGE_P));
  P = std::max(P, next_pow2(std::max(2 * k, 64)));  // at least k new candidates per pass
  const size_t smem = (size_t)P * (sizeof(float) + sizeof(int64_t));
  k_merge<int64_t><<<(unsigned)nq, 1024, smem, s>>>(cand_s, cand_i, S, nq, m, k, P, (int64_t)-1, out_ids,
                                                     out_scores);
  return cudaGetLastError();
}

cudaError_t launch_allow_bits(const FilterDev& f, const int64_t* allow_off,
                              const uint32_t* allow_tenants, int64_t nq, uint32_t* out,
                              cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  k_allow_bits<<<(unsigned)nq, 128, 0, s>>>(f.tenants, f.n_tenants, f.words, allow_off, allow_tenants, out);
  return cudaGetLastError();
}

cudaError_t launch_filter_build(const uint32_t* tenant_ids, FilterDev& f, cudaStream_t s) {
  const int64_t nblocks = (f.n + f.block - 1) / f.block;
  cudaError_t e = cudaMemsetAsync(f.block_bits, 0, (size_t)nblocks * f.words * sizeof(uint32_t), s);
  if (e != cudaSuccess) return e;
  const int grid = (int)std::min<int64_t>((f.n + 255) / 256, (int64_t)device_sm_count() * 8);
  k_filter_build<<<grid, 256, 0, s>>>(tenant_ids, f.n, 0, f.tenants, f.n_tenants, f.words, f.block, f.dense,
                                      f.block_bits);
  return cudaGetLastError();
}

cudaError_t launch_filter_extend(const uint32_t* tenant_ids, int64_t n_new, const FilterDev& f, cudaStream_t s) {
  if (n_new == 0) return cudaSuccess;
  const int grid = (int)std::min<int64_t>((n_new + 255) / 256, (int64_t)device_sm_count() * 8);
  k_filter_build<<<grid, 256, 0, s>>>(tenant_ids, n_new, f.n, f.tenants, f.n_tenants, f.words, f.block, f.dense,
                                      f.block_bits);
  return cudaGetLastError();
}

cudaError_t launch_filter_raw_ids(const FilterDev& f, uint32_t* raw, cudaStream_t s) {
  if (f.n == 0) return cudaSuccess;
  const int grid = (int)std::min<int64_t>((f.n + 255) / 256, (int64_t)device_sm_count() * 8);
  k_filter_raw_ids<<<grid, 256, 0, s>>>(f.dense, f.tenants, f.n, raw);
  return cudaGetLastError();
}

}  // namespace tq
