// The 4-bit lookup scan with the rotated query folded into its table (Sec.
// II-B step 5: score(v) = scale_v * <q', c[codes_v]>, top-k by Sec. III-B).
//
// Packed byte m of a row holds codes 2m (low nibble) and 2m+1 (high nibble),
// so <q', c[codes_v]> = sum_m T_m[x_{v,m}] with
//     T_m[x] = q'_{2m} c[x & 15] + q'_{2m+1} c[x >> 4].
// Per packed byte that is one 4-byte table read and one add, where the
// query-independent byte-pair table of k_scan_stream reads 8 bytes (two
// centroids) and multiplies by q' itself: half the shared-memory traffic per
// code byte, which is what bounds those scans.  The tables of all d/2 byte
// positions take d/2 KB (768 KB at d = 1536), more than an SM holds, so a CTA
// works through its rows one slice of 128 byte positions (256 coordinates) at
// a time: it builds the slice's 128 KB of tables, scores that slice of each
// of its rows, adds the partial sums into per-row accumulators in shared
// memory, and goes on to the next slice.  After the last slice the
// accumulators hold the rows' full sums; the per-vector scale, the TQ+ term,
// the filter, the tombstones and the per-warp top-k lists follow as in the
// other lookup scans, and the last CTA of each query merges the CTA lists.
//
// Bank layout.  A sub-tile is 16 rows x one 128-byte slice (one TMA box,
// 2 KB); lanes l and l + 16 share row l % 16, lane l reading words
// w = (j + l) % 32 for steps j = 0..15, so the lanes of a step read 32
// different words, one per bank, and the two lanes of a row cover its 32
// words.  The tables of word w's four byte positions 4w + t live in bank w:
// entry x of position 4w + t sits at byte (t >> 1) * 65536 + x * 256 +
// (t & 1) * 128 + 4w.  One byte permute places byte t of the word at bits
// 8..15 next to 4w, which is that offset less a compile-time constant, so a
// step's 32 table reads never conflict either.  One shuffle adds the two
// halves of each row.
//
// Streaming: each of the 16 warps owns two 2 KB stages and scores sub-tiles
// t = warp, warp + 16, ... of each slice.  Its lane 0 queues the TMA load of
// the sub-tile two places ahead as soon as a stage's words are read, and an
// L2 prefetch of the one FOLD_PF places beyond that.  Every mbarrier wait is
// bounded: one that gives up raises the CTA's abort flag and records its
// site in the search status word; the warps then skip the remaining
// sub-tiles (still meeting every barrier of the slice loop), wait (bounded)
// for their own loads in flight, and the CTA ends.
//
// Measured on GB300 (999,000 x 1536, batch 1, whole search): 228 us against
// 218 us for the byte-pair scan.  Half the shared-memory bytes per code byte
// do not pay here: beside the 128 KB of tables only 64 KB of stages and 16
// warps fit in an SM, and the scan is bound by latency and issue rather than
// by the shared-memory datapath (8 warps: 233 us; one 4 KB stage per warp:
// 266 us; 8-row sub-tiles: 430 us).  The search's AUTO path therefore keeps
// the byte-pair scan; this one is TQ_PATH_LUT_FOLD.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cudaTypedefs.h>

#include <climits>
#include <cmath>
#include <cstdint>

#include "tq_internal.h"
#include "tq_kernels.h"
#include "tq_tc.cuh"
#include "tq_topk.cuh"

namespace tq {
namespace {

#ifndef TQ_FOLD_CW
#define TQ_FOLD_CW 16
#endif
#ifndef TQ_FOLD_ACC
#define TQ_FOLD_ACC 4
#endif
constexpr int FOLD_CW = TQ_FOLD_CW;                 // warps
constexpr int FOLD_NT = FOLD_CW * 32;
constexpr int FOLD_ACC = TQ_FOLD_ACC;               // partial-sum chains per lane (2 or 4)
constexpr int FOLD_SLICE = 128;                     // packed bytes per slice (32 words)
#ifndef TQ_FOLD_G
#define TQ_FOLD_G 2
#endif
#ifndef TQ_FOLD_PF
#define TQ_FOLD_PF 8
#endif
constexpr int FOLD_G = TQ_FOLD_G;                   // lanes per row
constexpr int FOLD_SUB = 32 / FOLD_G;               // rows per sub-tile
constexpr int FOLD_STEPS = 32 / FOLD_G;             // words of a row per lane
constexpr int FOLD_STAGE = FOLD_SUB * FOLD_SLICE;   // one TMA box
constexpr int FOLD_NS = 65536 / FOLD_CW / FOLD_STAGE;  // stages per warp (64 KB in all)
constexpr int FOLD_XQ = FOLD_NT / 64;               // table build: thread groups per high nibble set
static_assert(FOLD_NS >= 1 && FOLD_XQ >= 1 && 16 % FOLD_XQ == 0, "warps and stages");
constexpr int FOLD_TAB = FOLD_SLICE * 256 * 4;      // 128 KB of tables
constexpr int FOLD_ROWS = 6656;                     // rows per pass (accumulators)
constexpr int FOLD_OFF_STAGE = FOLD_TAB;
constexpr int FOLD_OFF_ACC = FOLD_OFF_STAGE + FOLD_CW * FOLD_NS * FOLD_STAGE;
constexpr int FOLD_OFF_LIST = FOLD_OFF_ACC + FOLD_ROWS * 4;
constexpr int FOLD_NBARS = FOLD_CW * FOLD_NS;
constexpr int FOLD_PF = TQ_FOLD_PF;                 // sub-tiles per warp prefetched into L2 ahead
static_assert(FOLD_G == 1 || FOLD_G == 2 || FOLD_G == 4 || FOLD_G == 8, "lanes per row");
static_assert(FOLD_ROWS % 32 == 0, "passes hold whole 32-row groups");

// A warp's position in its sub-tile sequence: pass (first row p0), slice, sub-tile.
struct FoldCursor {
  int p0, s, t;
};

__device__ __forceinline__ void l2_prefetch_2d(const CUtensorMap* map, int x, int y) {
  asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];"
               ::"l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y)
               : "memory");
}

// One sub-tile's partial sums: lane l takes row l % FOLD_SUB of stage ST and
// its FOLD_STEPS words (j + l) % 32, j < FOLD_STEPS, against the slice's
// tables; the FOLD_G lanes of a row then add their parts (lanes l < FOLD_SUB
// hold the row sums).  ta[j] = 4 * ((j + l) % 32), ca[j] its byte offset in
// the warp's stage 0.
template <int ST>
__device__ __forceinline__ float fold_sub(const unsigned char* sm, const uint32_t (&ta)[FOLD_STEPS],
                                          const uint32_t (&ca)[FOLD_STEPS]) {
  float a[FOLD_ACC];
#pragma unroll
  for (int i = 0; i < FOLD_ACC; ++i) a[i] = 0.f;
#pragma unroll
  for (int j = 0; j < FOLD_STEPS; ++j) {
    const uint32_t w = *reinterpret_cast<const uint32_t*>(sm + ca[j] + ST * FOLD_STAGE);
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const uint32_t off = __byte_perm(w, ta[j], 0x7604u | ((uint32_t)t << 4));
      const float v = *reinterpret_cast<const float*>(sm + off + (t >> 1) * 65536 + (t & 1) * 128);
      a[t % FOLD_ACC] += v;
    }
  }
  float v = FOLD_ACC == 4 ? (a[0] + a[2]) + (a[1] + a[3]) : a[0] + a[FOLD_ACC - 1];
#pragma unroll
  for (int o = FOLD_SUB; o < 32; o <<= 1) v += __shfl_xor_sync(FULL, v, o);
  return v;
}

template <int ST = 0>
__device__ __forceinline__ float fold_sub_at(int st, const unsigned char* sm, const uint32_t (&ta)[FOLD_STEPS],
                                             const uint32_t (&ca)[FOLD_STEPS]) {
  if constexpr (ST + 1 < FOLD_NS) {
    if (st != ST) return fold_sub_at<ST + 1>(st, sm, ta, ca);
  }
  return fold_sub<ST>(sm, ta, ca);
}

template <bool FILT>
__global__ void __launch_bounds__(FOLD_NT, 1)
k_scan_fold(const __grid_constant__ CUtensorMap tmap, const float* __restrict__ qrot, int d,
            const float* __restrict__ centroids, const float* __restrict__ scale, int n, int rows_per_cta,
            const uint32_t* __restrict__ del, const uint32_t* __restrict__ dense,
            const uint32_t* __restrict__ allow_bits, int words, const uint32_t* __restrict__ bmask,
            int mask_words, int fblock, int k, int P, float* __restrict__ cand_s, int* __restrict__ cand_i,
            int* __restrict__ err, int* __restrict__ counters, const uint64_t* __restrict__ ext,
            int64_t* __restrict__ out_ids, float* __restrict__ out_scores, const float* __restrict__ bias) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  __shared__ volatile int abort_flag;
  float* acc = reinterpret_cast<float*>(smem_raw + FOLD_OFF_ACC);
  float* ls = reinterpret_cast<float*>(smem_raw + FOLD_OFF_LIST);
  int* li = reinterpret_cast<int*>(ls + P);
  uint64_t* full = reinterpret_cast<uint64_t*>(li + P);  // P is even: 8-byte aligned
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int q = blockIdx.y;
  const int rb = d >> 1;
  const int nslices = (rb + FOLD_SLICE - 1) / FOLD_SLICE;
  const int row0 = (int)min((int64_t)blockIdx.x * rows_per_cta, (int64_t)n);
  const int row1 = (int)min((int64_t)row0 + rows_per_cta, (int64_t)n);
  const uint32_t* bm = FILT ? bmask + (size_t)q * mask_words : nullptr;
  // a sub-tile (FOLD_SUB rows from a multiple of FOLD_SUB) and a 32-row group
  // (from a multiple of 32) each lie in one filter block of 32 or 64 rows
  auto tile_on = [&](int r) -> bool {
    if constexpr (FILT) {
      const int fb = r / fblock;
      return (__ldg(bm + (fb >> 5)) >> (fb & 31)) & 1u;
    } else {
      (void)r;
      return true;
    }
  };
  auto ntiles_of = [&](int p0) { return (min(FOLD_ROWS, row1 - p0) + FOLD_SUB - 1) / FOLD_SUB; };
  // this warp's sub-tiles in the order it scores them: pass, slice, sub-tile
  // t = warp + FOLD_CW i; advances `c` to the next one (false past the last)
  auto next_tile = [&](FoldCursor& c) -> bool {
    for (;;) {
      if (c.p0 >= row1) return false;
      c.t = c.t < 0 ? warp : c.t + FOLD_CW;
      if (c.t >= ntiles_of(c.p0)) {
        c.t = -1;
        if (++c.s >= nslices) {
          c.s = 0;
          c.p0 += FOLD_ROWS;
        }
        continue;
      }
      if (tile_on(c.p0 + c.t * FOLD_SUB)) return true;
    }
  };
  uint64_t* wfull = full + warp * FOLD_NS;
  unsigned char* wstage = smem_raw + FOLD_OFF_STAGE + warp * FOLD_NS * FOLD_STAGE;
  if (lane == 0) {
    for (int b = 0; b < FOLD_NS; ++b) mbar_init(wfull + b, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (tid == 0) abort_flag = 0;
  for (int i = tid; i < P; i += FOLD_NT) {
    ls[i] = -INFINITY;
    li[i] = INT_MAX;
  }
  __syncwarp();
  // lane 0 of each warp streams the warp's own sub-tiles: the next FOLD_NS into
  // its stages, and FOLD_PF further ones into L2 ahead of them; the codes are
  // the caller's, so (unfiltered) this starts while the rotation may still run
  FoldCursor ic{row0, 0, -1}, pc{row0, 0, -1};
  uint32_t issued = 0;
  bool pmore = true;
  if (lane == 0) {
    if constexpr (FILT) griddep_wait();  // the block masks steer the loads
    for (int b = 0; b < FOLD_NS && next_tile(ic); ++b) {
      mbar_arrive_expect_tx(wfull + b, FOLD_STAGE);
      tma_load_2d(wstage + b * FOLD_STAGE, &tmap, ic.s * FOLD_SLICE, ic.p0 + ic.t * FOLD_SUB, wfull + b);
      ++issued;
    }
    pc = ic;
    for (int i = 0; i < FOLD_PF && pmore; ++i)
      if ((pmore = next_tile(pc))) l2_prefetch_2d(&tmap, pc.s * FOLD_SLICE, pc.p0 + pc.t * FOLD_SUB);
  }
  float cen[16];
#pragma unroll
  for (int u = 0; u < 16; ++u) cen[u] = __ldg(centroids + u);
  uint32_t ta[FOLD_STEPS], ca[FOLD_STEPS];
#pragma unroll
  for (int j = 0; j < FOLD_STEPS; ++j) {
    ta[j] = (uint32_t)((j + lane) & 31) * 4u;
    ca[j] = (uint32_t)(FOLD_OFF_STAGE + warp * FOLD_NS * FOLD_STAGE + (lane % FOLD_SUB) * FOLD_SLICE) + ta[j];
  }
  // this thread's share of each table build: word bw, byte positions
  // 4 bw + btlo (+ 2), entries x = 16 (bxq + FOLD_XQ m) + u
  const int bw = tid & 31, btlo = (tid >> 5) & 1, bxq = tid >> 6;
  unsigned char* bdst = smem_raw + bxq * 4096 + btlo * 128 + bw * 4;
  float chi[16 / FOLD_XQ];  // centroids of the high nibbles this thread's entries take
#pragma unroll
  for (int m = 0; m < 16 / FOLD_XQ; ++m) chi[m] = __ldg(centroids + bxq + FOLD_XQ * m);
  griddep_wait();  // the rotated queries (and TQ+ terms) are written
  const float bq = bias ? bias[q] : 0.f;
  const float* qq = qrot + (size_t)q * d;
  const uint32_t* ab = FILT ? allow_bits + (size_t)q * words : nullptr;
  float* wl_s = ls + warp * k;
  int* wl_i = li + warp * k;
  int cnt = 0;
  float th_s = -INFINITY;
  int th_i = INT_MAX;
  uint32_t used = 0;  // tiles this warp has scored
  for (int p0 = row0; p0 < row1; p0 += FOLD_ROWS) {
    const int prow = min(FOLD_ROWS, row1 - p0);
    const int ntiles = ntiles_of(p0);
    for (int s = 0; s < nslices; ++s) {
      __syncthreads();  // every warp is done with the previous slice's tables
#pragma unroll
      for (int th = 0; th < 2; ++th) {
        const int pos = s * FOLD_SLICE + bw * 4 + btlo + 2 * th;  // packed byte position
        const float qa = pos < rb ? __ldg(qq + 2 * pos) : 0.f;
        const float qb = pos < rb ? __ldg(qq + 2 * pos + 1) : 0.f;
        float A[16];
#pragma unroll
        for (int u = 0; u < 16; ++u) A[u] = qa * cen[u];
#pragma unroll
        for (int m = 0; m < 16 / FOLD_XQ; ++m) {
          const float B = qb * chi[m];
#pragma unroll
          for (int u = 0; u < 16; ++u)
            *reinterpret_cast<float*>(bdst + th * 65536 + m * (FOLD_XQ * 4096) + u * 256) = A[u] + B;
        }
      }
      __syncthreads();
      for (int t = warp; t < ntiles; t += FOLD_CW) {
        if (!tile_on(p0 + t * FOLD_SUB)) continue;
        const uint32_t c = used++;
        const int st = (int)(c % FOLD_NS);
        if (!warp_wait(wfull + st, (c / FOLD_NS) & 1u, &abort_flag, err, 41)) continue;
        const float part = fold_sub_at(st, smem_raw, ta, ca);
        __syncwarp();  // every lane has read its words of the stage
        if (lane == 0 && !abort_flag && next_tile(ic)) {
          // the stage is free: the sub-tile FOLD_NS ahead goes into it
          fence_proxy_async();
          mbar_arrive_expect_tx(wfull + st, FOLD_STAGE);
          tma_load_2d(wstage + st * FOLD_STAGE, &tmap, ic.s * FOLD_SLICE, ic.p0 + ic.t * FOLD_SUB, wfull + st);
          ++issued;
          if (pmore && (pmore = next_tile(pc))) l2_prefetch_2d(&tmap, pc.s * FOLD_SLICE, pc.p0 + pc.t * FOLD_SUB);
        }
        const int lr = t * FOLD_SUB + lane;
        if (lane < FOLD_SUB && lr < prow) acc[lr] = s == 0 ? part : acc[lr] + part;
      }
    }
    __syncthreads();  // every row's sum is in acc
    // the pass's rows are scored: candidates into the warp's sorted list, 32
    // rows (one per lane) at a time
    const int ngroups = (prow + 31) / 32;
    for (int t = warp; t < ngroups; t += FOLD_CW) {
      if (!tile_on(p0 + t * 32)) continue;
      const int lr = t * 32 + lane;
      const int v = p0 + lr;
      float score = -INFINITY;
      bool cand = false;
      if (lr < prow) {
        const float sc = scale ? __ldg(scale + v) : 1.0f;
        score = (acc[lr] + bq) * sc;
        bool allowed = true;
        if constexpr (FILT) {
          const uint32_t tn = __ldg(dense + v);
          allowed = (__ldg(ab + (tn >> 5)) >> (tn & 31)) & 1u;
        }
        cand = allowed && better(score, v, th_s, th_i) && !tombstoned(del, v);
      }
      unsigned m = __ballot_sync(FULL, cand);
      while (m) {
        const int src = __ffs(m) - 1;
        m &= m - 1;
        const float sv = __shfl_sync(FULL, score, src);
        const int vv = p0 + t * 32 + src;
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
  }
  // never leave with loads in flight: the last load of each stage has landed
  // (at once, unless a wait gave up)
  if (lane == 0)
    for (int b = 0; b < FOLD_NS; ++b) {
      const uint32_t uses = issued > (uint32_t)b ? (issued - b + FOLD_NS - 1) / FOLD_NS : 0;
      if (uses) mbar_wait_drain(wfull + b, (uses - 1) & 1u);
    }
  __syncthreads();
  {
    const size_t o = ((size_t)q * gridDim.x + blockIdx.x) * k;
    cta_lists_out(ls, li, FOLD_CW, k, P, cand_s + o, cand_i + o);
  }
  // the tables are dead by now: their bytes are the merge's scratch
  merge_if_last(cand_s, cand_i, k, counters, ext, out_ids, out_scores, ls, li, smem_raw, FOLD_TAB);
}

int fold_list_p(int k) {
  int p = 1;
  while (p < FOLD_CW * k) p <<= 1;  // the warp lists (and the merge's per-warp scratch)
  return p;
}

}  // namespace

bool fold_supported(int bits, int d, int k, int64_t n) {
  // rows are int32 in the kernel; a pass start p0 + FOLD_ROWS must not overflow
  return bits == 4 && d >= 2 * FOLD_SLICE && d % 32 == 0 && k >= 1 && k <= kFoldMaxK &&
         n <= (int64_t)INT32_MAX - 2 * FOLD_ROWS;
}

int scan_fold_grid_x(int64_t nq, int64_t n) {
  const int64_t tiles = (n + 31) / 32;
  int64_t gx = device_sm_count() / (nq > 0 ? nq : 1);
  if (gx > tiles) gx = tiles;
  if (gx < 1) gx = 1;
  const int64_t per = (tiles + gx - 1) / gx;  // tiles per CTA
  return (int)((tiles + per - 1) / per);
}

cudaError_t launch_scan_fold(const float* qrot, int64_t nq, int d, const float* centroids, const uint8_t* codes,
                             const float* scale, int64_t n, const uint32_t* del, const FilterDev* f,
                             const uint32_t* allow_bits, const uint32_t* bmask, int k, int grid_x, float* cand_s,
                             int32_t* cand_i, int* err, int* counters, const uint64_t* ext, int64_t* out_ids,
                             float* out_scores, const float* bias, cudaStream_t s, cudaEvent_t ev0,
                             cudaEvent_t ev1) {
  if (nq == 0) return cudaSuccess;
  if (!fold_supported(4, d, k, n) || n < 1 || grid_x < 1) return cudaErrorInvalidValue;
  PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
  if (!enc) return cudaErrorNotSupported;
  CUtensorMap map;
  const cuuint64_t gdim[2] = {(cuuint64_t)row_bytes(d, 4), (cuuint64_t)n};
  const cuuint64_t gstride[1] = {(cuuint64_t)row_bytes(d, 4)};
  const cuuint32_t box[2] = {(cuuint32_t)FOLD_SLICE, (cuuint32_t)FOLD_SUB};
  const cuuint32_t estride[2] = {1, 1};
  const CUresult r = enc(&map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(codes), gdim, gstride, box,
                         estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  const int64_t tiles = (n + 31) / 32;  // CTAs own whole 32-row groups
  const int64_t per = (tiles + grid_x - 1) / grid_x;
  const int rows_per_cta = (int)(per * 32);
  const int P = fold_list_p(k);
  const size_t smem = (size_t)FOLD_OFF_LIST + (size_t)P * (sizeof(float) + sizeof(int)) +
                      (size_t)FOLD_NBARS * sizeof(uint64_t);
  const bool filt = f != nullptr;
  const void* fn = filt ? reinterpret_cast<const void*>(k_scan_fold<true>)
                        : reinterpret_cast<const void*>(k_scan_fold<false>);
  cudaError_t e = set_max_dynamic_smem(fn, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid_x, (unsigned)nq);
  cfg.blockDim = dim3(FOLD_NT);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  // overlap with the rotation (not on the legacy default stream, and not
  // between profiling events, which would serialise the two anyway)
  cfg.numAttrs = (s != nullptr && ev0 == nullptr) ? 1 : 0;
  if (ev0 && (e = cudaEventRecord(ev0, s)) != cudaSuccess) return e;
  const uint32_t* dn = filt ? f->dense : nullptr;
  const int words = filt ? f->words : 0, mw = filt ? filter_mask_words(*f) : 0, fb = filt ? f->block : 64;
  e = filt ? cudaLaunchKernelEx(&cfg, k_scan_fold<true>, map, qrot, d, centroids, scale, (int)n, rows_per_cta,
                                del, dn, allow_bits, words, bmask, mw, fb, k, P, cand_s, cand_i, err, counters,
                                ext, out_ids, out_scores, bias)
           : cudaLaunchKernelEx(&cfg, k_scan_fold<false>, map, qrot, d, centroids, scale, (int)n, rows_per_cta,
                                del, dn, allow_bits, words, bmask, mw, fb, k, P, cand_s, cand_i, err, counters,
                                ext, out_ids, out_scores, bias);
  if (e != cudaSuccess) return e;
  if (ev1 && (e = cudaEventRecord(ev1, s)) != cudaSuccess) return e;
  return cudaSuccess;
}

}  // namespace tq
