// Search-side kernels: the lookup scan with fused top-k (Sec. II-B step 5,
// Sec. III-B), per-query allow bitmaps, the filter build and the final merge.
//
// Lookup scan layout.  One warp scores 4 consecutive vectors per step.  Each
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
// bitmap are skipped before any code byte is read (Sec. III-B): a small kernel
// turns the two bitmaps into one bit per block and query first.
#include <cuda_runtime.h>

#include <climits>
#include <limits>
#include <cmath>
#include <cstdint>

#include "tq_internal.h"
#include "tq_kernels.h"
#include "tq_wait.cuh"
#include "tq_topk.cuh"

namespace tq {
namespace {


constexpr int SCAN_NT = 256;
constexpr int SCAN_WARPS = SCAN_NT / 32;
constexpr int MERGE_P = 2048;

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

// Fixed-point byte-pair table for 4-bit codes.  The exact table above moves
// 8 bytes through shared memory per packed byte (two fp32 centroids), which
// bounds the scan by the shared-memory datapath (128 B per cycle per SM).
// Here each centroid is a signed 15-bit integer c_v = rint(centroid_v / step)
// and the entry (x, lane) = c[x & 15] | c[x >> 4] << 16 is 4 bytes: one
// wavefront per warp lookup instead of two.  The entry feeds 2-way integer
// dot products (dp2a: two 16-bit halves times two bytes, added to a 32-bit
// accumulator) without any conversion: each lane quantises its 48 rotated
// query coordinates to 24-bit integers q_j = rint(q'_j / s) (s = the lane's
// largest |q'_j| / (2^23 - 1)), split into bytes q_j = 2^16 h_j + 2^8 m_j + l_j
// (h signed), and per packed byte makes three dp2a's, one per byte plane of
// the coordinate pair.  Per lane and vector, 2^16 A_h + 2^8 A_m + A_l is the
// exact integer sum_j q_j c_j, and s * step times it the lane's part of the
// score.  The rounding of the centroids to the step is the only error beyond
// float32 (about 2^-16 of the largest centroid per centroid): the step is the
// one, among FIX_CANDIDATES values in [d0, 1.25 d0) (d0 = max|c| / 16383),
// whose largest rounding error over the 16 centroids is least, chosen the
// same way by every CTA.
constexpr int FIX_CANDIDATES = 2048;

// Fills the fixed-point table (uint32 entry (x, lane) at index x * 64 + lane;
// the other half of each 256-byte row is unused) and returns the step.  All
// threads of the CTA call it; `red` is shared scratch of 2 * 32 words.
__device__ float fix_table_init(uint32_t* tab, const float* __restrict__ centroids, float* red, int tid, int nt) {
  float c[16];
  float m = 0.f;
#pragma unroll
  for (int v = 0; v < 16; ++v) {
    c[v] = __ldg(centroids + v);
    m = fmaxf(m, fabsf(c[v]));
  }
  const float d0 = m > 0.f ? m / 16383.0f * (1.0f + 0x1p-20f) : 1.0f;
  float best_e = INFINITY;
  int best_i = 0;
  for (int i = tid; i < FIX_CANDIDATES; i += nt) {
    const float st = d0 * (1.0f + (float)i * (0.25f / FIX_CANDIDATES));
    const float inv = 1.0f / st;
    float e = 0.f;
#pragma unroll
    for (int v = 0; v < 16; ++v) {
      const float r = c[v] * inv;
      e = fmaxf(e, fabsf(r - rintf(r)));
    }
    e *= st;
    if (e < best_e) {  // candidates are visited in increasing i: ties keep the smaller
      best_e = e;
      best_i = i;
    }
  }
  const int lane = tid & 31, warp = tid >> 5;
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float oe = __shfl_xor_sync(FULL, best_e, o);
    const int oi = __shfl_xor_sync(FULL, best_i, o);
    if (oe < best_e || (oe == best_e && oi < best_i)) {
      best_e = oe;
      best_i = oi;
    }
  }
  if (lane == 0) {
    red[warp] = best_e;
    reinterpret_cast<int*>(red)[32 + warp] = best_i;
  }
  __syncthreads();
  best_e = red[0];
  best_i = reinterpret_cast<int*>(red)[32];
  for (int w = 1; w < nt / 32; ++w) {
    const float oe = red[w];
    const int oi = reinterpret_cast<int*>(red)[32 + w];
    if (oe < best_e || (oe == best_e && oi < best_i)) {
      best_e = oe;
      best_i = oi;
    }
  }
  const float step = d0 * (1.0f + (float)best_i * (0.25f / FIX_CANDIDATES));
  __shared__ uint32_t su[16];
  if (tid < 16) su[tid] = (uint32_t)min(16383, max(-16383, (int)rintf(c[tid] / step))) & 0xFFFFu;
  __syncthreads();
  for (int i = tid; i < 256 * 32; i += nt) {
    const int x = i >> 5;
    tab[x * 64 + (i & 31)] = su[x & 15] | (su[x >> 4] << 16);
  }
  return step;
}

// Quantises this lane's query pairs (q'_{2m}, q'_{2m+1}) to 24-bit integers
// and replaces each pair, in place, by its byte planes: .x = (l_e, l_o, m_e,
// m_o) and .y = (h_e, h_o, 0, 0) as bit patterns.  Returns s * step, the
// factor of the lane's integer sums.
template <int S>
__device__ __forceinline__ float fix_query_bytes(float2 (&q2)[S][8], float step) {
  float mx = 0.f;
#pragma unroll
  for (int s = 0; s < S; ++s)
#pragma unroll
    for (int m = 0; m < 8; ++m) mx = fmaxf(mx, fmaxf(fabsf(q2[s][m].x), fabsf(q2[s][m].y)));
  const float sq = mx > 0.f ? mx / 8388607.0f : 1.0f;
  const float inv = 1.0f / sq;
#pragma unroll
  for (int s = 0; s < S; ++s)
#pragma unroll
    for (int m = 0; m < 8; ++m) {
      const int e = min(8388607, max(-8388607, __float2int_rn(q2[s][m].x * inv)));
      const int o = min(8388607, max(-8388607, __float2int_rn(q2[s][m].y * inv)));
      const uint32_t lo = (uint32_t)(e & 0xFF) | ((uint32_t)(o & 0xFF) << 8) | ((uint32_t)((e >> 8) & 0xFF) << 16) |
                          ((uint32_t)((o >> 8) & 0xFF) << 24);
      const uint32_t hi = (uint32_t)((e >> 16) & 0xFF) | ((uint32_t)((o >> 16) & 0xFF) << 8);
      q2[s][m] = make_float2(__uint_as_float(lo), __uint_as_float(hi));
    }
  return sq * step;
}

__device__ __forceinline__ int dp2a_lo_su(uint32_t a, uint32_t b, int c) {  // a: two s16, b: bytes 0-1 unsigned
  int d;
  asm("dp2a.lo.s32.u32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}
__device__ __forceinline__ int dp2a_hi_su(uint32_t a, uint32_t b, int c) {  // bytes 2-3 unsigned
  int d;
  asm("dp2a.hi.s32.u32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}
__device__ __forceinline__ int dp2a_lo_ss(uint32_t a, uint32_t b, int c) {  // bytes 0-1 signed
  int d;
  asm("dp2a.lo.s32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// This lane's part of one vector's score with the fixed-point table: the
// exact integer sum, scaled by `f` (fix_query_bytes).
template <int S>
__device__ __forceinline__ float pair16_dot(const Chunk<4> (&ch)[S], const float2 (&q2)[S][8], const char* tab,
                                            uint32_t lane4, float f) {
  int al = 0, am = 0, ah = 0;
#pragma unroll
  for (int s = 0; s < S; ++s) {
#pragma unroll
    for (int b = 0; b < 8; ++b) {
      const uint32_t w = b < 4 ? ch[s].w0 : ch[s].w1;
      const uint32_t addr = __byte_perm(w, lane4, 0x5504u | ((uint32_t)(b & 3) << 4));
      const uint32_t e = *reinterpret_cast<const uint32_t*>(tab + addr);
      const uint32_t p0 = __float_as_uint(q2[s][b].x), p1 = __float_as_uint(q2[s][b].y);
      al = dp2a_lo_su(e, p0, al);
      am = dp2a_hi_su(e, p0, am);
      ah = dp2a_lo_ss(e, p1, ah);
    }
  }
  const long long t = ((long long)ah << 16) + ((long long)am << 8) + (long long)al;
  return (float)t * f;
}

// The lookup scan.  Each warp scores 4 consecutive vectors per step (a CTA
// step covers 32) and issues the next step's code loads before it starts on
// the current ones (register double buffer), so every warp always has loads
// in flight.  4-bit codes use a byte-pair table (FIX: the fixed-point one,
// else the exact fp32 one), other widths a per-code fp32 table replicated in
// the 32 banks.  With FILT, `bmask` holds one bit per filter block of the
// query: steps whose block has no allowed tenant are passed over before any
// of their code bytes is read (Sec. III-B), and in the others a vector whose
// tenant the query does not allow never enters the top-k.  Filtered and
// unfiltered scans share every operation on the scores, so filtering by every
// tenant reproduces the unfiltered result bit for bit.
template <int BITS, int S, bool FILT, bool FIX>
__global__ void __launch_bounds__(SCAN_NT, 2)
k_scan_stream(const float* __restrict__ qrot, int d, const float* __restrict__ centroids,
              const uint8_t* __restrict__ codes, const float* __restrict__ scale, int n,
              const uint32_t* __restrict__ del, const uint32_t* __restrict__ dense,
              const uint32_t* __restrict__ allow_bits, int words, const uint32_t* __restrict__ bmask,
              int mask_words, int fblock, int k, int P, float* __restrict__ cand_s, int* __restrict__ cand_i,
              int* __restrict__ counters, const uint64_t* __restrict__ ext, int64_t* __restrict__ out_ids,
              float* __restrict__ out_scores, const float* __restrict__ bias) {
  constexpr int L = 1 << BITS;
  constexpr int CB = 2 * BITS;   // bytes of a 16-code chunk
  constexpr int V = 4;           // vectors per warp step; a CTA step covers 32
  constexpr bool PAIR = BITS == 4;
  constexpr int TAB_BYTES = PAIR ? PAIR_TAB_BYTES : L * 32 * 4;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  float* ls = reinterpret_cast<float*>(smem_raw + TAB_BYTES);  // [P] scores; warp w's list at [w*k, w*k+k)
  int* li = reinterpret_cast<int*>(ls + P);                     // [P] ids
  __shared__ float red[64];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int q = blockIdx.y;
  float qs = 1.0f;  // the fixed-point table's step
  if constexpr (PAIR && FIX) {
    qs = fix_table_init(reinterpret_cast<uint32_t*>(smem_raw), centroids, red, tid, SCAN_NT);
  } else if constexpr (PAIR) {
    pair_table_init(reinterpret_cast<float2*>(smem_raw), centroids, tid, SCAN_NT);
  } else {
    float* ctab = reinterpret_cast<float*>(smem_raw);
    for (int i = tid; i < L * 32; i += SCAN_NT) ctab[i] = __ldg(centroids + (i >> 5));
  }
  for (int i = tid; i < P; i += SCAN_NT) {
    ls[i] = -INFINITY;
    li[i] = INT_MAX;
  }
  griddep_wait();  // the rotated queries (and allow bitmaps, block masks) are written
  const float bq = bias ? bias[q] : 0.f;  // a TQ+ index's per-query term (else 0)
  const int nchunks = d >> 4;
  const float* qq = qrot + (size_t)q * d;
  float qr[PAIR ? 1 : S][16];
  float2 q2[PAIR ? S : 1][8];
  float qf = 0.f;  // fixed-point table: the factor of the lanes' integer sums
  if constexpr (PAIR) {
    load_q2(q2, qq, nchunks, lane);
    if constexpr (FIX) qf = fix_query_bytes<S>(q2, qs);
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
  const uint32_t* ab = FILT ? allow_bits + (size_t)q * words : nullptr;
  const uint32_t* bm = FILT ? bmask + (size_t)q * mask_words : nullptr;
  float* wl_s = ls + warp * k;
  int* wl_i = li + warp * k;
  int cnt = 0;
  float th_s = -INFINITY;
  int th_i = INT_MAX;
  const int nsteps = (n + SCAN_WARPS * V - 1) / (SCAN_WARPS * V);
  const int my = (lane >> 3) & 3;  // the vector whose total this lane ends up holding
  const uint32_t lane4 = (uint32_t)lane * 4u;
  const char* tab = reinterpret_cast<const char*>(smem_raw);
  // the CTA's next step at or after st whose filter block holds an allowed
  // tenant (every thread takes the same decisions)
  auto active = [&](int st) {
    if constexpr (FILT) {
      while (st < nsteps) {
        const int fb = st * (SCAN_WARPS * V) / fblock;
        if ((__ldg(bm + (fb >> 5)) >> (fb & 31)) & 1u) break;
        st += gridDim.x;
      }
    }
    return st;
  };

  Chunk<BITS> cur[V][S], nxt[V][S];
  float sc_cur = 0.f, sc_nxt = 0.f;
  uint32_t tn_cur = 0, tn_nxt = 0;
  auto load_step = [&](int st, Chunk<BITS> (&buf)[V][S], float& sc, uint32_t& tn) {
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
    tn = 0;
    if (st < nsteps && (lane & 7) == 0 && vm < n) {
      sc = scale ? __ldg(scale + vm) : 1.0f;
      if (FILT) tn = __ldg(dense + vm);
    }
  };
  int st = active(blockIdx.x);
  load_step(st, cur, sc_cur, tn_cur);
  while (st < nsteps) {
    const int st_next = active(st + gridDim.x);
    load_step(st_next, nxt, sc_nxt, tn_nxt);  // next step's loads go out first
    asm volatile("" ::: "memory");
    const int v0 = st * (SCAN_WARPS * V) + warp * V;
    float p[V];
#pragma unroll
    for (int i = 0; i < V; ++i) {
      if constexpr (PAIR && FIX) {
        p[i] = pair16_dot<S>(cur[i], q2, tab, lane4, qf);
      } else if constexpr (PAIR) {
        p[i] = pair_dot<S>(cur[i], q2, tab, lane4 * 2u);
      } else {
        float acc = 0.f;
#pragma unroll
        for (int s = 0; s < S; ++s)
#pragma unroll
          for (int t = 0; t < 16; ++t)
            acc = fmaf(qr[s][t], *reinterpret_cast<const float*>(tab + cur[i][s].off(t, lane4)), acc);
        p[i] = acc;
      }
    }
    const float total = warp_sum4(p);
    const int vm = v0 + my;
    float score = -INFINITY;
    bool cand = false;
    if ((lane & 7) == 0 && vm < n) {
      score = (total + bq) * sc_cur;
      const bool allowed = !FILT || ((__ldg(ab + (tn_cur >> 5)) >> (tn_cur & 31)) & 1u);
      cand = allowed && better(score, vm, th_s, th_i) && !tombstoned(del, vm);
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
    tn_cur = tn_nxt;
    st = st_next;
  }
  __syncthreads();
  {
    const size_t o = ((size_t)q * gridDim.x + blockIdx.x) * k;
    cta_lists_out(ls, li, SCAN_WARPS, k, P, cand_s + o, cand_i + o);
  }
  // the lookup table is dead by now: its bytes are the merge's scratch
  merge_if_last(cand_s, cand_i, k, counters, ext, out_ids, out_scores, ls, li, smem_raw, TAB_BYTES);
}

// ---------------------------------------------------------------------------
// The lookup scan fed by bulk copies.  k_scan_stream keeps the next step's
// codes in registers, so the bytes a warp has in flight are bounded by its
// registers (about 48 KB per SM), too few to cover HBM latency at full rate.
// Here each of the CTA's RING_WARPS warps streams its own sequence of 4-vector
// steps through a private ring of `ns` shared-memory slots: lane 0 queues a
// 1-D bulk copy (cp.async.bulk, completion counted on the slot's mbarrier)
// for the step `ns` places ahead as soon as a slot's codes are in registers,
// so ns slots per warp (about 144 KB per SM) are always on their way.  The
// scoring is k_scan_stream's, operation for operation.  A step that is not
// whole (the corpus tail) is read with plain loads.  Waits are bounded: a
// wait that gives up raises the CTA's abort flag and records its site in the
// status word; every warp then stops, waits (bounded) for its own copies still
// in flight, and the CTA ends.
constexpr int RING_WARPS = 16;
constexpr int RING_NT = RING_WARPS * 32;
constexpr int RING_MAX_NS = 4;

__device__ __forceinline__ uint32_t sh_u32(const void* p) { return static_cast<uint32_t>(__cvta_generic_to_shared(p)); }

__device__ __forceinline__ void ring_mbar_init(uint64_t* bar) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(sh_u32(bar)));
}

__device__ __forceinline__ void ring_copy(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(sh_u32(bar)), "r"(bytes) : "memory");
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(sh_u32(dst)), "l"(src), "r"(bytes), "r"(sh_u32(bar))
               : "memory");
}

__device__ __forceinline__ bool ring_wait_drain(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  for (uint32_t i = 0;; ++i) {
    if (mbar_try_wait_parity(bar, parity)) return true;
    if ((i & 63) == 63 && clock64() - t0 > kWaitCycles) return false;
  }
}

// Reads 16-code chunk `chunk` of a row held in shared memory.
template <int BITS>
__device__ __forceinline__ void chunk_from_smem(Chunk<BITS>& c, const unsigned char* p);
template <>
__device__ __forceinline__ void chunk_from_smem<4>(Chunk<4>& c, const unsigned char* p) {
  const uint2 v = *reinterpret_cast<const uint2*>(p);
  c.w0 = v.x;
  c.w1 = v.y;
}
template <>
__device__ __forceinline__ void chunk_from_smem<2>(Chunk<2>& c, const unsigned char* p) {
  c.w = *reinterpret_cast<const uint32_t*>(p);
}
template <>
__device__ __forceinline__ void chunk_from_smem<8>(Chunk<8>& c, const unsigned char* p) {
  c.w = *reinterpret_cast<const uint4*>(p);
}
template <>
__device__ __forceinline__ void chunk_from_smem<3>(Chunk<3>& c, const unsigned char* p) {
  const unsigned short* h = reinterpret_cast<const unsigned short*>(p);
  c.v = (uint64_t)h[0] | ((uint64_t)h[1] << 16) | ((uint64_t)h[2] << 32);
}

template <int BITS, int S, bool FILT, bool FIX>
__global__ void __launch_bounds__(RING_NT, 1)
k_scan_ring(const float* __restrict__ qrot, int d, const float* __restrict__ centroids,
            const uint8_t* __restrict__ codes, const float* __restrict__ scale, int n,
            const uint32_t* __restrict__ del, const uint32_t* __restrict__ dense,
            const uint32_t* __restrict__ allow_bits, int words, const uint32_t* __restrict__ bmask, int mask_words,
            int fblock, int k, int P, int ns, float* __restrict__ cand_s, int* __restrict__ cand_i,
            int* __restrict__ err, int* __restrict__ counters, const uint64_t* __restrict__ ext,
            int64_t* __restrict__ out_ids, float* __restrict__ out_scores, const float* __restrict__ bias) {
  constexpr int L = 1 << BITS;
  constexpr int CB = 2 * BITS;
  constexpr int V = 4;
  constexpr bool PAIR = BITS == 4;
  constexpr int TAB_BYTES = PAIR ? PAIR_TAB_BYTES : L * 32 * 4;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int rb = d * BITS / 8;
  const int slot_bytes = V * rb;  // a multiple of 16 for d % 32 == 0
  unsigned char* ring = smem_raw + TAB_BYTES;
  float* ls = reinterpret_cast<float*>(ring + (size_t)RING_WARPS * ns * slot_bytes);
  int* li = reinterpret_cast<int*>(ls + P);
  uint64_t* bars = reinterpret_cast<uint64_t*>(li + P + (P & 1));  // 8-byte aligned
  __shared__ float red[64];
  __shared__ int stepq[RING_WARPS][RING_MAX_NS];
  __shared__ volatile int abort_flag;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int q = blockIdx.y;
  const int nsteps = (n + V - 1) / V;  // warp steps of 4 vectors
  const int wstride = gridDim.x * RING_WARPS;
  uint64_t* wbar = bars + warp * RING_MAX_NS;
  unsigned char* wring = ring + (size_t)warp * ns * slot_bytes;
  const uint32_t* bm = FILT ? bmask + (size_t)q * mask_words : nullptr;
  // this warp's next step at or after `ws` whose filter block holds an allowed tenant
  auto active = [&](int ws) {
    if constexpr (FILT) {
      while (ws < nsteps) {
        const int fb = ws * V / fblock;
        if ((__ldg(bm + (fb >> 5)) >> (fb & 31)) & 1u) break;
        ws += wstride;
      }
    }
    return ws;
  };
  uint32_t pend = 0;  // slots with a copy in flight (lane 0's view, shared by shuffle)
  auto issue = [&](int ws, int s) {
    __syncwarp();  // every lane has read the slot's previous codes
    if (lane == 0) {
      stepq[warp][s] = ws;
      if (ws < nsteps && (ws + 1) * V <= n) {
        ring_copy(wring + s * slot_bytes, codes + (size_t)ws * slot_bytes, (uint32_t)slot_bytes, wbar + s);
        pend |= 1u << s;
      }
    }
    __syncwarp();
  };
  if (tid == 0) abort_flag = 0;
  if (lane == 0) {
    for (int s = 0; s < ns; ++s) ring_mbar_init(wbar + s);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();
  if constexpr (FILT) griddep_wait();  // the block masks steer the first copies
  // the first ns steps go out before the table is built
  int next_ws = active(blockIdx.x * RING_WARPS + warp);
  for (int s = 0; s < ns; ++s) {
    issue(next_ws, s);
    next_ws = active(next_ws + wstride);
  }
  float qs = 1.0f;  // the fixed-point table's step
  if constexpr (PAIR && FIX) {
    qs = fix_table_init(reinterpret_cast<uint32_t*>(smem_raw), centroids, red, tid, RING_NT);
  } else if constexpr (PAIR) {
    pair_table_init(reinterpret_cast<float2*>(smem_raw), centroids, tid, RING_NT);
  } else {
    float* ctab = reinterpret_cast<float*>(smem_raw);
    for (int i = tid; i < L * 32; i += RING_NT) ctab[i] = __ldg(centroids + (i >> 5));
  }
  for (int i = tid; i < P; i += RING_NT) {
    ls[i] = -INFINITY;
    li[i] = INT_MAX;
  }
  if constexpr (!FILT) griddep_wait();  // the rotated queries are written
  const float bq = bias ? bias[q] : 0.f;  // a TQ+ index's per-query term (else 0)
  const int nchunks = d >> 4;
  const float* qq = qrot + (size_t)q * d;
  float qr[PAIR ? 1 : S][16];
  float2 q2[PAIR ? S : 1][8];
  float qf = 0.f;  // fixed-point table: the factor of the lanes' integer sums
  if constexpr (PAIR) {
    load_q2(q2, qq, nchunks, lane);
    if constexpr (FIX) qf = fix_query_bytes<S>(q2, qs);
  } else {
#pragma unroll
    for (int s = 0; s < S; ++s) {
      const int chunk = lane + 32 * s;
#pragma unroll
      for (int t = 0; t < 16; ++t) qr[s][t] = chunk < nchunks ? qq[chunk * 16 + t] : 0.f;
    }
  }
  __syncthreads();

  const uint32_t* ab = FILT ? allow_bits + (size_t)q * words : nullptr;
  float* wl_s = ls + warp * k;
  int* wl_i = li + warp * k;
  int cnt = 0;
  float th_s = -INFINITY;
  int th_i = INT_MAX;
  const int my = (lane >> 3) & 3;
  const uint32_t lane4 = (uint32_t)lane * 4u;
  const char* tab = reinterpret_cast<const char*>(smem_raw);
  uint32_t par = 0;  // phase parity of each slot's next completion
  for (int it = 0;; ++it) {
    const int s = it % ns;
    const int ws = stepq[warp][s];
    if (ws >= nsteps) break;
    if (abort_flag) break;
    const int v0 = ws * V;
    Chunk<BITS> cur[V][S];
    if (v0 + V <= n) {  // whole step: its codes came by bulk copy
      bool ok = true;
      if (lane == 0) ok = bounded_wait(wbar + s, (par >> s) & 1u, &abort_flag, err, 20, kWaitCycles);
      ok = __shfl_sync(FULL, ok ? 1 : 0, 0) != 0;
      if (!ok) break;
      par ^= 1u << s;
      pend &= ~(1u << s);
      __syncwarp();
      const unsigned char* src = wring + s * slot_bytes;
#pragma unroll
      for (int i = 0; i < V; ++i)
#pragma unroll
        for (int c = 0; c < S; ++c) {
          const int chunk = lane + 32 * c;
          if (chunk < nchunks) chunk_from_smem<BITS>(cur[i][c], src + i * rb + chunk * CB);
          else cur[i][c].zero();
        }
    } else {
#pragma unroll
      for (int i = 0; i < V; ++i)
#pragma unroll
        for (int c = 0; c < S; ++c) {
          const int chunk = lane + 32 * c;
          if (v0 + i < n && chunk < nchunks) cur[i][c].load(codes + (size_t)(v0 + i) * rb + chunk * CB);
          else cur[i][c].zero();
        }
    }
    const int vm = v0 + my;
    float sc = 0.f;
    uint32_t tn = 0;
    if ((lane & 7) == 0 && vm < n) {
      sc = scale ? __ldg(scale + vm) : 1.0f;
      if (FILT) tn = __ldg(dense + vm);
    }
    // the slot's codes are in registers: queue the step ns places ahead
    issue(next_ws, s);
    next_ws = active(next_ws + wstride);
    float p[V];
#pragma unroll
    for (int i = 0; i < V; ++i) {
      if constexpr (PAIR && FIX) {
        p[i] = pair16_dot<S>(cur[i], q2, tab, lane4, qf);
      } else if constexpr (PAIR) {
        p[i] = pair_dot<S>(cur[i], q2, tab, lane4 * 2u);
      } else {
        float acc = 0.f;
#pragma unroll
        for (int c = 0; c < S; ++c)
#pragma unroll
          for (int t = 0; t < 16; ++t)
            acc = fmaf(qr[c][t], *reinterpret_cast<const float*>(tab + cur[i][c].off(t, lane4)), acc);
        p[i] = acc;
      }
    }
    const float total = warp_sum4(p);
    float score = -INFINITY;
    bool cand = false;
    if ((lane & 7) == 0 && vm < n) {
      score = (total + bq) * sc;
      const bool allowed = !FILT || ((__ldg(ab + (tn >> 5)) >> (tn & 31)) & 1u);
      cand = allowed && better(score, vm, th_s, th_i) && !tombstoned(del, vm);
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
  }
  // never leave with copies in flight (only after an abort can there be any)
  if (lane == 0)
    for (int s = 0; s < ns; ++s)
      if ((pend >> s) & 1u) ring_wait_drain(wbar + s, (par >> s) & 1u);
  __syncthreads();
  {
    const size_t o = ((size_t)q * gridDim.x + blockIdx.x) * k;
    cta_lists_out(ls, li, RING_WARPS, k, P, cand_s + o, cand_i + o);
  }
  // the lookup table is dead by now: its bytes are the merge's scratch
  merge_if_last(cand_s, cand_i, k, counters, ext, out_ids, out_scores, ls, li, smem_raw, TAB_BYTES);
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

// Merge of every scan CTA's list, one block per query (the tensor-core scan's
// lists; the lookup scans merge in their own last CTA).
__global__ void __launch_bounds__(1024)
k_merge_lists(const float* __restrict__ cand_s, const int* __restrict__ cand_i, int nlists, int k,
              const uint64_t* __restrict__ ext, int64_t* __restrict__ out_ids, float* __restrict__ out_scores,
              size_t scratch_bytes) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  float* ws = reinterpret_cast<float*>(smem_raw);  // [nwarps][k]
  int* wi = reinterpret_cast<int*>(ws + (blockDim.x >> 5) * k);
  unsigned char* scratch = reinterpret_cast<unsigned char*>(wi + (blockDim.x >> 5) * k);
  const int64_t q = blockIdx.x;
  merge_lists_block(cand_s + q * nlists * k, cand_i + q * nlists * k, nlists, k, ext, out_ids + q * k,
                    out_scores + q * k, ws, wi, scratch, scratch_bytes);
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

// Bit b of query q's block mask: filter block b holds a tenant the query
// allows (its tenant bitmap shares a bit with the query's allow bitmap).  A
// warp owns one mask word (32 blocks): lane w reads word w of each block's
// bitmap, all 32 blocks' loads in flight at once.
__global__ void __launch_bounds__(256)
k_block_mask(const uint32_t* __restrict__ block_bits, int64_t nblocks, int words, const uint32_t* __restrict__ allow,
             int mask_words, uint32_t* __restrict__ mask) {
  const int64_t q = blockIdx.y;
  const int lane = threadIdx.x & 31;
  griddep_launch_dependents();
  const int64_t mw = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (mw >= mask_words) return;  // whole warps
  const uint32_t* a = allow + q * words;
  uint32_t bits = 0;
  for (int w0 = 0; w0 < words; w0 += 32) {
    const int w = w0 + lane;
    const uint32_t aw = w < words ? __ldg(a + w) : 0u;
    uint32_t x[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const int64_t b = mw * 32 + j;
      x[j] = (w < words && b < nblocks) ? (__ldg(block_bits + b * words + w) & aw) : 0u;
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) bits |= (__any_sync(FULL, x[j] != 0u) ? 1u : 0u) << j;
  }
  if (lane == 0) mask[q * mask_words + mw] = bits;
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

struct ScanArgs {
  const float* qrot;
  int d;
  const float* centroids;
  const uint8_t* codes;
  const float* scale;
  int n;
  const uint32_t* del;
  const uint32_t* dense;
  const uint32_t* allow;
  int words;
  const uint32_t* bmask;
  int mask_words;
  int fblock;
  int k, P;
  float* cs;
  int* ci;
  int* err;
  int* counters;
  const uint64_t* ext;
  int64_t* out_ids;
  float* out_scores;
  bool pdl;
  const float* bias;
};

// Launches `kernel`, with programmatic stream serialization when `pdl` (the
// kernel then overlaps the tail of the one before it and waits for it with
// griddep_wait before reading its results).
template <typename... Params, typename... Args>
cudaError_t launch_maybe_pdl(bool pdl, void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem,
                             cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// Dynamic shared memory of the ring scan with `ns` slots per warp.
constexpr size_t kRingSmemMax = 232448 - 2048;  // 227 KB less the static arrays
size_t ring_smem(int bits, int d, int P, int ns) {
  const size_t tab = bits == 4 ? (size_t)PAIR_TAB_BYTES : (size_t)(1 << bits) * 32 * sizeof(float);
  return tab + (size_t)RING_WARPS * ns * 4 * (d * bits / 8) + (size_t)P * (sizeof(float) + sizeof(int)) +
         (size_t)RING_WARPS * RING_MAX_NS * sizeof(uint64_t);
}

// Slots per warp of the ring scan (as many as fit, at most RING_MAX_NS), or 0
// for the register-fed k_scan_stream.  Measured on GB300 (999,000 x 1536,
// batch 1): the ring reads 3-bit codes 23% faster (1.69 vs 1.37 TB/s), but for
// 2- and 4-bit codes the scan is bound by the shared-memory datapath the
// lookups use, and the ring's copies add to that traffic (4-bit 2.83 vs 3.55
// TB/s, 2-bit 1.18 vs 1.28), so only 3-bit codes take it.
int ring_slots(int bits, int d, int k) {
  if (bits != 3) return 0;
  const int P = next_pow2(RING_WARPS * k);
  for (int ns = RING_MAX_NS; ns >= 2; --ns)
    if (ring_smem(bits, d, P, ns) <= kRingSmemMax) return ns;
  return 0;
}

template <int BITS, int S, bool FILT, bool FIX>
cudaError_t scan_typed(dim3 grid, size_t smem, cudaStream_t s, const ScanArgs& a) {
  const int ns = BITS == 3 ? ring_slots(BITS, a.d, a.k) : 0;
  if constexpr (BITS == 3) if (ns >= 2) {
    const int P = next_pow2(RING_WARPS * a.k);
    const size_t rsmem = ring_smem(BITS, a.d, P, ns);
    const void* fn = reinterpret_cast<const void*>(k_scan_ring<BITS, S, FILT, FIX>);
    const cudaError_t e = set_max_dynamic_smem(fn, (int)rsmem);
    if (e != cudaSuccess) return e;
    return launch_maybe_pdl(a.pdl, k_scan_ring<BITS, S, FILT, FIX>, grid, dim3(RING_NT), rsmem, s, a.qrot, a.d,
                            a.centroids, a.codes, a.scale, a.n, a.del, a.dense, a.allow, a.words, a.bmask,
                            a.mask_words, a.fblock, a.k, P, ns, a.cs, a.ci, a.err, a.counters, a.ext, a.out_ids,
                            a.out_scores, a.bias);
  }
  const void* fn = reinterpret_cast<const void*>(k_scan_stream<BITS, S, FILT, FIX>);
  const cudaError_t e = set_max_dynamic_smem(fn, (int)smem);
  if (e != cudaSuccess) return e;
  return launch_maybe_pdl(a.pdl, k_scan_stream<BITS, S, FILT, FIX>, grid, dim3(SCAN_NT), smem, s, a.qrot, a.d,
                          a.centroids, a.codes, a.scale, a.n, a.del, a.dense, a.allow, a.words, a.bmask,
                          a.mask_words, a.fblock, a.k, a.P, a.cs, a.ci, a.counters, a.ext, a.out_ids, a.out_scores,
                          a.bias);
}

template <int BITS, int S>
cudaError_t scan_variant(bool filt, bool fix, dim3 grid, size_t smem, cudaStream_t s, const ScanArgs& a) {
  if constexpr (BITS == 4) {
    if (fix)
      return filt ? scan_typed<BITS, S, true, true>(grid, smem, s, a) : scan_typed<BITS, S, false, true>(grid, smem, s, a);
  } else {
    (void)fix;
  }
  return filt ? scan_typed<BITS, S, true, false>(grid, smem, s, a) : scan_typed<BITS, S, false, false>(grid, smem, s, a);
}

template <int BITS>
cudaError_t scan_bits(int S, bool filt, bool fix, dim3 grid, size_t smem, cudaStream_t s, const ScanArgs& a) {
  switch (S) {
    case 1: return scan_variant<BITS, 1>(filt, fix, grid, smem, s, a);
    case 2: return scan_variant<BITS, 2>(filt, fix, grid, smem, s, a);
    case 3: return scan_variant<BITS, 3>(filt, fix, grid, smem, s, a);
    case 4: return scan_variant<BITS, 4>(filt, fix, grid, smem, s, a);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

int scan_lut_grid_x(int64_t nq, int64_t n, int k, int bits, int d) {
  // one resident wave for a single query: one ring-scan CTA per SM, or two
  // register-fed CTAs
  const int64_t target = (int64_t)device_sm_count() * (ring_slots(bits, d, k) >= 2 ? 1 : 2);
  int64_t gx = (target + nq - 1) / (nq > 0 ? nq : 1);
  const int64_t blocks = (n + 31) / 32;
  if (gx > blocks) gx = blocks;
  if (gx < 1) gx = 1;
  return (int)gx;
}

int filter_mask_words(const FilterDev& f) {
  const int64_t nblocks = (f.n + f.block - 1) / f.block;
  return (int)((nblocks + 31) / 32);
}

cudaError_t launch_scan_lut(const float* qrot, int64_t nq, int d, const float* centroids, int bits,
                            const uint8_t* codes, const float* scale, int64_t n, const uint32_t* del,
                            const FilterDev* f, const uint32_t* allow_bits, const uint32_t* bmask, bool fix,
                            int k, int grid_x, float* cand_s, int32_t* cand_i, int* err, int* counters,
                            const uint64_t* ext, int64_t* out_ids, float* out_scores, const float* bias,
                            cudaStream_t s, cudaEvent_t ev0, cudaEvent_t ev1) {
  if (nq == 0) return cudaSuccess;
  const int S = (d + 511) / 512;
  const int P = next_pow2(SCAN_WARPS * k);
  const size_t tab = bits == 4 ? (size_t)PAIR_TAB_BYTES : (size_t)(1 << bits) * 32 * sizeof(float);
  const size_t smem = tab + (size_t)P * (sizeof(float) + sizeof(int));
  const dim3 grid((unsigned)grid_x, (unsigned)nq);
  ScanArgs a{qrot, d, centroids, codes, scale, (int)n, del,
             f ? f->dense : nullptr, allow_bits, f ? f->words : 0, bmask, f ? filter_mask_words(*f) : 0,
             f ? f->block : 64, k, P, cand_s, cand_i, err, counters, ext, out_ids, out_scores,
             // overlap with the kernel before (not on the legacy default stream, and not
             // between profiling events, which would serialise the two anyway)
             s != nullptr && ev0 == nullptr, bias};
  const bool filt = f != nullptr;
  cudaError_t e;
  if (ev0 && (e = cudaEventRecord(ev0, s)) != cudaSuccess) return e;
  switch (bits) {
    case 2: e = scan_bits<2>(S, filt, fix, grid, smem, s, a); break;
    case 3: e = scan_bits<3>(S, filt, fix, grid, smem, s, a); break;
    case 4: e = scan_bits<4>(S, filt, fix, grid, smem, s, a); break;
    case 8: e = scan_bits<8>(S, filt, fix, grid, smem, s, a); break;
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
  while (warps > 1 && (size_t)warps * k * 8 > 24 * 1024) warps >>= 1;
  // scratch for gathering and sorting the candidates that pass the bound
  const size_t want = (size_t)next_pow2(std::max(nlists * k, 2)) * 8;
  // (dynamic plus the kernel's few static bytes stay under the default 48 KB)
  const size_t scratch = std::min<size_t>(want, 40 * 1024 - (size_t)warps * k * 8);
  const size_t smem = (size_t)warps * k * (sizeof(float) + sizeof(int32_t)) + scratch;
  k_merge_lists<<<(unsigned)nq, 32 * warps, smem, s>>>(cand_s, cand_i, nlists, k, ext, out_ids, out_scores,
                                                       scratch);
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

cudaError_t launch_block_mask(const FilterDev& f, const uint32_t* allow, int64_t nq, uint32_t* mask,
                              cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  const int mw = filter_mask_words(f);
  const dim3 grid((unsigned)((mw + 7) / 8), (unsigned)nq);
  k_block_mask<<<grid, 256, 0, s>>>(f.block_bits, (f.n + f.block - 1) / f.block, f.words, allow, mw, mask);
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
