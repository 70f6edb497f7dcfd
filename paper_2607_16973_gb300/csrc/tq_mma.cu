// Tensor-core scan for query batches (Sec. II-B step 5 as a GEMM):
//   S[q, v] = scale_v * sum_j q'_j c[code_vj]
// with the rotated queries on the MMA's M dimension (128 per tile) and corpus
// vectors on N (256 per tile), fp16 operands and fp32 accumulation in tensor
// memory (TMEM).  A CTA owns QT (1 or 2) query tiles and a strided set of
// vector tiles.  With one query tile TMEM holds two accumulator sets, so the
// epilogue of one vector tile overlaps the MMAs of the next; with two, the
// next tile's MMAs wait for the epilogue.  Roles (warp-specialised, 23 warps):
//   warps 0-7, 19-22  decoders, in groups of four warps that take turns on
//               K-blocks (with one query tile, warps 12-15 are a fourth
//               group): expand one K-block (64 coordinates) of packed codes,
//               brought to shared memory by TMA, into fp16 centroid values
//               laid out as the K-major, 128-byte-swizzled B operand;
//   warps 8-15  epilogue: read the 128 x 256 fp32 accumulators from TMEM (one
//               query per thread; warps 8-11 the first query tile, 12-15 the
//               second), apply the per-vector scale and keep each query's
//               top-k in a thread-private sorted list (rows marked in the
//               optional tombstone bitmap never enter it);
//   warp 16     code producer: TMA of the code tiles; allocates TMEM;
//   warp 17     MMA issuer: one thread issues tcgen05.mma (M=128, N=256,
//               K=16) and commits completion to mbarriers;
//   warp 18     query producer: 1-D bulk copies of pre-swizzled fp16 query
//               blocks.
// Every wait is bounded: on
// timeout the CTA raises `abort`, writes an error code to the status word and
// exits after draining what it has in flight.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>

#include <climits>
#include <cmath>
#include <cstdint>
#include <mutex>

#include "tq_internal.h"
#include "tq_kernels.h"
#include "tq_wait.cuh"
#include "tq_tc.cuh"

namespace tq {
namespace {

constexpr int MMA_M = 128;            // queries per tile
constexpr int MMA_N = 256;            // vectors per tile
constexpr int KB = 64;                // coordinates per K-block (128 B of fp16)
constexpr int MAX_CST = 8;  // raw code tiles in flight (HBM latency)
constexpr int RAW_ROW_MAX = 128;  // bytes of each row one code tile carries (one 128-B line)
constexpr int MAX_AST = 4;  // query blocks in flight (L2-resident)
constexpr int EPI_WARP0 = 8;
// Decoders work in groups of four warps that take turns on K-blocks (group g
// takes it = g, g + G, ...).  Warps 0-3, 4-7 and 19-22 are groups; with one
// query tile the epilogue needs only warps 8-11, so warps 12-15 are a fourth.
template <int QT>
__host__ __device__ constexpr int dec_groups() { return QT == 1 ? 4 : 3; }
// The plan runs ng <= dec_groups groups (as shared memory allows) and one
// decoded fp16 stage per group: a group decodes its K-blocks in order, so it
// is never more than one phase ahead on its stage's barriers (a shared stage
// would let a group two phases ahead pass a parity wait early).
// Decoder group of a warp, or -1.
template <int QT>
__device__ __forceinline__ int dec_group(int warp) {
  if (warp < 8) return warp >> 2;
  if (warp >= 19) return 2;
  if (QT == 1 && warp >= 12 && warp < 16) return 3;
  return -1;
}
template <int QT>
__host__ __device__ constexpr int epi_warps() { return QT == 1 ? 4 : 8; }
constexpr int CODE_WARP = 16, MMA_WARP = 17, QUERY_WARP = 18;
constexpr int NTHREADS = 23 * 32;  // warps 19-22: one more decoder group
constexpr uint32_t kMaxDynSmem = 232448;  // 227 KB per block on sm_100-class GPUs
constexpr int A_BYTES = MMA_M * KB * 2;   // 16 KB
// Vectors per tile.  (Tiles of 128 with two query tiles would leave room for
// two accumulator sets, but M128 N128 MMAs ran at about two thirds of the
// per-flop rate of N256 ones on this GPU, more than the overlap gains.)
template <int QT>
__host__ __device__ constexpr int tile_n() { return MMA_N; }
template <int QT>
__host__ __device__ constexpr int b_bytes() { return tile_n<QT>() * KB * 2; }
template <int N>
__host__ __device__ constexpr uint32_t idesc() {
  return (1u << 4) | (0u << 7) | (0u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(MMA_M >> 4) << 24);
}

template <int N>
__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}"
      ::"r"(d_tmem), "l"(a), "l"(b), "r"(idesc<N>()), "r"(accumulate));
}

__device__ __forceinline__ bool better(float s1, int i1, float s2, int i2) {
  return s1 > s2 || (s1 == s2 && i1 < i2);
}

struct MmaSmem {
  uint32_t a, b, raw, tab, scale, dense, lists_s, lists_i, bars, total;
};

template <int BITS>
__host__ __device__ constexpr int raw_bytes_per_row() { return KB * BITS / 8; }

// 4-bit codes decode in registers (no table); 2- and 8-bit use a table
// replicated in all 32 banks (entry e of lane l at e*32 + l).
template <int BITS>
__host__ __device__ constexpr int tab_bytes() {
  return BITS == 4 ? 0 : BITS == 2 ? 16 * 32 * 4 : BITS == 3 ? 64 * 32 * 4 : 256 * 32 * 2;
}

// K-blocks per code tile for rows of up to rr bytes per tile.  A TMA box's
// inner extent is a multiple of 16 bytes: 3-bit K-blocks are 24 bytes, so
// their tiles carry 4 (96 bytes) or 2 (48 bytes).
__host__ __device__ inline int tile_sub(int bits, int rr) {
  if (bits == 3) return rr >= 96 ? 4 : 2;
  return rr / (KB * bits / 8);
}

// Shared-memory plan for QT query tiles per CTA, `cst` raw code stages and
// `ast` query stages.
template <int BITS, int QT>
__host__ __device__ inline MmaSmem mma_smem_layout(int k, int cst, int ast, int rr, int ng) {
  MmaSmem L{};
  uint32_t off = 0;
  L.a = off;
  off += (uint32_t)ast * QT * A_BYTES;
  L.b = off;
  off += (uint32_t)ng * b_bytes<QT>();
  L.raw = off;
  off += (uint32_t)cst * tile_n<QT>() * rr;
  L.tab = off;
  off += tab_bytes<BITS>();
  L.scale = off;
  off += tile_n<QT>() * 4;
  L.dense = off;  // tenant index of each vector of the tile (filtered searches)
  off += tile_n<QT>() * 4;
  L.lists_s = off;
  off += (uint32_t)QT * k * MMA_M * 4;
  L.lists_i = off;
  off += (uint32_t)QT * k * MMA_M * 4;
  off = (off + 15) & ~15u;
  L.bars = off;
  off += 48 * 8;
  L.total = off + 1024;  // slack to align the base to 1024 bytes
  // at most one CTA per SM: each allocates all 512 TMEM columns
  if (L.total < 116u * 1024u) L.total = 116u * 1024u;
  return L;
}

struct MmaPlan {
  int qt = 1, cst = 2, ast = 2, rr = RAW_ROW_MAX;  // rr: bytes of each row per code tile
  int ng = 2;                                      // decoder groups = decoded stages
  uint32_t smem = 0;
};

// Decoder groups that may run with code tiles of `sub` K-blocks in `cst`
// stages.  Waits on a code stage use the phase parity, so a group must never
// be two phases ahead on a stage: true when every group uses every tile
// (sub >= g) or when each stage is always shared by the same groups
// (cst * sub a multiple of g).
int active_groups(int ng, int sub, int cst) {
  int g = ng;
  while (g > 2 && !(sub >= g || (cst * sub) % g == 0)) --g;
  if (!(sub >= g || (cst * sub) % g == 0)) g = 1;
  return g;
}

constexpr int MIN_PREFETCH_KB = 6;  // K-blocks of codes in flight (HBM latency)

// Picks query tiles per CTA, decoder groups and ring depths that fit in shared
// memory: prefer two query tiles per decoded code tile, then as many decoder
// groups as the role layout has (all of them able to run), with at least
// MIN_PREFETCH_KB K-blocks of codes in flight, then deeper rings.
template <int BITS>
MmaPlan mma_plan(int64_t nq, int k) {
  MmaPlan best;
  // first pass as above; the second relaxes the prefetch floor and allows
  // fewer groups (large k at 8 bits needs the room for its lists)
  for (int pass = 0; pass < 2; ++pass) {
    const int min_pf = pass == 0 ? MIN_PREFETCH_KB : 2;
    for (int qt = (nq > MMA_M ? 2 : 1); qt >= 1; --qt) {
      const int gmax = qt == 2 ? dec_groups<2>() : dec_groups<1>();
      for (int ng = gmax; ng >= 2; --ng) {
        for (int rr = RAW_ROW_MAX; rr >= 64; rr >>= 1) {
          const int sub = tile_sub(BITS, rr);  // for d a multiple of 256
          for (int ast = 3; ast >= 2; --ast) {
            for (int cst = MAX_CST; cst >= 2; --cst) {
              if (cst * sub < min_pf || active_groups(ng, sub, cst) != ng) continue;
              const uint32_t need = qt == 2 ? mma_smem_layout<BITS, 2>(k, cst, ast, rr, ng).total
                                            : mma_smem_layout<BITS, 1>(k, cst, ast, rr, ng).total;
              if (need <= kMaxDynSmem) {
                best.qt = qt;
                best.cst = cst;
                best.ast = ast;
                best.rr = rr;
                best.ng = ng;
                best.smem = need;
                return best;
              }
            }
          }
        }
      }
    }
  }
  best.smem = 0;  // does not fit
  return best;
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
  return d;
}

// Eight 4-bit codes (nibble i of w is code i) -> eight fp16 centroids, in
// registers.  tl[j] / th[j] hold the low / high bytes of the fp16 centroids
// 4j .. 4j+3.  A byte permute picks table bytes by the code's low 3 bits from
// entries 0-7 and 8-15; the sign-replicate selector mode turns each code's
// bit 3 into a 0x00/0xFF byte mask that chooses between the two.
__device__ __forceinline__ uint4 decode8_4bit(uint32_t w, const uint32_t (&tl)[4], const uint32_t (&th)[4]) {
  const uint32_t sel = w & 0x77777777u;
  const uint32_t w4 = w << 4;
  uint32_t o[4];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const uint32_t sh = h ? sel >> 16 : sel;
    const uint32_t m = prmt(w4, w, h ? 0xFBEAu : 0xD9C8u);  // byte i = 0xFF iff code 4h+i >= 8
    const uint32_t lo = (prmt(tl[0], tl[1], sh) & ~m) | (prmt(tl[2], tl[3], sh) & m);
    const uint32_t hi = (prmt(th[0], th[1], sh) & ~m) | (prmt(th[2], th[3], sh) & m);
    o[2 * h] = prmt(lo, hi, 0x5140u);
    o[2 * h + 1] = prmt(lo, hi, 0x7362u);
  }
  return make_uint4(o[0], o[1], o[2], o[3]);
}

template <int BITS, int QT>
__global__ void __launch_bounds__(NTHREADS, 1)
k_scan_mma(const __grid_constant__ CUtensorMap codes_map, const __half* __restrict__ qpack,
           const float* __restrict__ centroids, const float* __restrict__ scale,
           const uint32_t* __restrict__ del, const uint32_t* __restrict__ dense,
           const uint32_t* __restrict__ allow_bits, int words, const float* __restrict__ bias, int n, int nq,
           int d, int k, int cst, int ast, int rr, int sub, int ng, int gact, float* __restrict__ cand_s,
           int* __restrict__ cand_i, int* __restrict__ err) {
  constexpr int RAWB = raw_bytes_per_row<BITS>();
  // A code tile carries `sub` consecutive K-blocks of 256 rows: rows of
  // sub*RAWB bytes (128 B, one full line, when d allows), stored with the
  // 128-B swizzle in that case so the decoders' reads do not conflict.
  const int rrow = sub * RAWB;
  const bool swz = rrow == 128;
  constexpr int NT = tile_n<QT>();       // vectors per tile
  constexpr int B_BYTES = b_bytes<QT>();
  constexpr int NSETS = 2 / QT;          // accumulator sets in TMEM (QT x NSETS x NT = 512 columns)
  // gact <= ng decoder groups run (the launcher picks gact so that no group
  // can get two phases ahead on a code stage); group g uses decoded stage g
  const int G = gact, BST = gact;
  constexpr int EPI_WARPS = epi_warps<QT>(), EPI_THREADS = EPI_WARPS * 32;
  extern __shared__ unsigned char smem_dyn[];
  // pointer arithmetic on the shared array (not an integer round trip) keeps
  // every access below a shared-memory access
  unsigned char* base = smem_dyn + ((1024u - (smem_u32(smem_dyn) & 1023u)) & 1023u);
  const MmaSmem L = mma_smem_layout<BITS, QT>(k, cst, ast, rr, ng);
  unsigned char* sA = base + L.a;
  unsigned char* sB = base + L.b;
  unsigned char* sRaw = base + L.raw;
  float* sScale = reinterpret_cast<float*>(base + L.scale);
  uint32_t* sDense = reinterpret_cast<uint32_t*>(base + L.dense);
  float* lst_s = reinterpret_cast<float*>(base + L.lists_s);
  int* lst_i = reinterpret_cast<int*>(base + L.lists_i);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + L.bars);
  uint64_t* cfull = bars;                      // [MAX_CST] code tile landed
  uint64_t* cempty = bars + 8;                 // [MAX_CST] code tile decoded (stage free)
  uint64_t* afull = bars + 16;                 // [MAX_AST] query block(s) landed
  uint64_t* aempty = bars + 20;                // [MAX_AST] MMAs done with the query block(s)
  uint64_t* dec = bars + 24;                   // [BST <= 4] decoded B tile written
  uint64_t* bempty = bars + 28;                // [BST] MMAs done with the decoded tile
  uint64_t* acc_full = bars + 32;              // [NSETS] accumulators complete
  uint64_t* acc_empty = bars + 34;             // [NSETS] accumulators read out
  uint64_t* fin = bars + 36;                   // all MMAs of this CTA complete
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 37);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 38);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int qt0 = blockIdx.y * QT;                     // first query tile of this CTA
  const int nqt = (nq + MMA_M - 1) / MMA_M;
  const int qts = min(QT, nqt - qt0);                  // query tiles present (1..QT)
  const int kblocks = d / KB;
  const int ntiles = (n + NT - 1) / NT;
  const int my_tiles = blockIdx.x < ntiles ? (ntiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;

  if (BITS == 2) {
    uint32_t* tab = reinterpret_cast<uint32_t*>(base + L.tab);
    for (int i = tid; i < 16 * 32; i += NTHREADS) {
      const int e = i >> 5;
      const __half2 h = __floats2half2_rn(centroids[e & 3], centroids[e >> 2]);
      tab[i] = *reinterpret_cast<const uint32_t*>(&h);
    }
  } else if (BITS == 3) {  // entry e = two consecutive 3-bit codes (e & 7, e >> 3), in bank `lane`
    uint32_t* tab = reinterpret_cast<uint32_t*>(base + L.tab);
    for (int i = tid; i < 64 * 32; i += NTHREADS) {
      const int e = i >> 5;
      const __half2 h = __floats2half2_rn(centroids[e & 7], centroids[e >> 3]);
      tab[i] = *reinterpret_cast<const uint32_t*>(&h);
    }
  } else if (BITS == 8) {
    __half* tab = reinterpret_cast<__half*>(base + L.tab);
    for (int i = tid; i < 256 * 32; i += NTHREADS) tab[i] = __float2half_rn(centroids[i >> 5]);
  }
  if (tid == 0) {
    for (int s = 0; s < MAX_CST; ++s) {
      mbar_init(cfull + s, 1);
      // one arrival per decoder warp that uses the tile: a tile of `sub`
      // consecutive K-blocks is used by min(sub, G) groups
      mbar_init(cempty + s, 4 * min(sub, G));
    }
    for (int s = 0; s < MAX_AST; ++s) {
      mbar_init(afull + s, 1);
      mbar_init(aempty + s, 1);
    }
    for (int s = 0; s < BST; ++s) {
      mbar_init(dec + s, 4);  // the four warps of one decoder group
      mbar_init(bempty + s, 1);
    }
    for (int b = 0; b < NSETS; ++b) {
      mbar_init(acc_full + b, 1);
      mbar_init(acc_empty + b, EPI_WARPS);  // one arrival per epilogue warp
    }
    mbar_init(fin, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == CODE_WARP) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(smem_u32(tmem_slot)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int total_it = my_tiles * kblocks;

  if (warp == CODE_WARP) {
    // ------------------------------------------------- code tiles (TMA, HBM)
    if (lane == 0) {
      int issued = 0;
      const int total_loads = total_it / sub;
      for (int ld = 0; ld < total_loads; ++ld) {
        const int s = ld % cst, use = ld / cst;
        if (use > 0 && !mbar_wait(cempty + s, (use - 1) & 1, abort_flag, err, 1)) break;
        const int it = ld * sub;
        const int t = blockIdx.x + (it / kblocks) * gridDim.x;
        const int kb = it % kblocks;
        mbar_arrive_expect_tx(cfull + s, NT * rrow);
        tma_load_2d(sRaw + s * NT * rr, &codes_map, kb * RAWB, t * NT, cfull + s);
        issued = ld + 1;
      }
      // never leave with copies in flight: wait (bounded) for the last one of each stage
      for (int s = 0; s < cst && s < issued; ++s) mbar_wait_drain(cfull + s, ((issued - 1 - s) / cst) & 1);
    }
  } else if (warp == QUERY_WARP) {
    // ------------------------------------------ query blocks (bulk copy, L2)
    if (lane == 0) {
      int issued = 0;
      for (int it = 0; it < total_it; ++it) {
        const int s = it % ast, use = it / ast;
        if (use > 0 && !mbar_wait(aempty + s, (use - 1) & 1, abort_flag, err, 6)) break;
        const int kb = it % kblocks;
        mbar_arrive_expect_tx(afull + s, qts * A_BYTES);
        for (int j = 0; j < qts; ++j)
          bulk_load(sA + (s * QT + j) * A_BYTES, qpack + ((size_t)(qt0 + j) * kblocks + kb) * (A_BYTES / 2),
                    A_BYTES, afull + s);
        issued = it + 1;
      }
      for (int s = 0; s < ast && s < issued; ++s) mbar_wait_drain(afull + s, ((issued - 1 - s) / ast) & 1);
    }
  } else if (warp == MMA_WARP) {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      int bs = 0, bpar = 0, as = 0, apar = 0, kb = 0, tile_i = 0, set = 0, spar = 0;
      for (int it = 0; it < total_it; ++it) {
        if (kb == 0 && tile_i >= NSETS && !mbar_wait(acc_empty + set, spar ^ 1, abort_flag, err, 2)) break;
        if (!mbar_wait(dec + bs, bpar, abort_flag, err, 3)) break;
        if (!mbar_wait(afull + as, apar, abort_flag, err, 7)) break;
        tc_fence_after();
        const uint32_t b0 = smem_u32(sB + bs * B_BYTES);
        for (int j = 0; j < qts; ++j) {
          const uint32_t a0 = smem_u32(sA + (as * QT + j) * A_BYTES);
          const uint32_t dt = tmem + (uint32_t)((set * QT + j) * NT);
#pragma unroll
          for (int kk = 0; kk < KB / 16; ++kk)
            mma_f16<NT>(dt, sw128_desc(a0 + kk * 32), sw128_desc(b0 + kk * 32), (kb | kk) != 0);
        }
        mma_commit(bempty + bs);
        mma_commit(aempty + as);
        if (kb == kblocks - 1) mma_commit(acc_full + set);
        if (++bs == BST) {
          bs = 0;
          bpar ^= 1;
        }
        if (++as == ast) {
          as = 0;
          apar ^= 1;
        }
        if (++kb == kblocks) {
          kb = 0;
          ++tile_i;
          if (++set == NSETS) {
            set = 0;
            spar ^= 1;
          }
        }
      }
      mma_commit(fin);
      mbar_wait_drain(fin, 0);
    }
  } else if (dec_group<QT>(warp) >= 0) {
    // ---------------------------------------------------------- decoders
    constexpr int PARTS = RAWB / 16;                 // 16-byte parts per row per K-block
    constexpr int CODES = 16 * 8 / BITS;             // codes per part
    constexpr int CHUNKS = CODES / 8;                // 16-byte fp16 chunks per part
    uint32_t tl[4] = {0, 0, 0, 0}, th[4] = {0, 0, 0, 0};
    if (BITS == 4) {
#pragma unroll
      for (int e = 0; e < 16; ++e) {
        const __half h = __float2half_rn(centroids[e]);
        const uint32_t bitsv = (uint32_t)__half_as_ushort(h);
        tl[e >> 2] |= (bitsv & 0xFFu) << (8 * (e & 3));
        th[e >> 2] |= (bitsv >> 8) << (8 * (e & 3));
      }
    }
    // G groups of four warps take turns on K-blocks (group g: it = g, g + G,
    // ...), so one group's fence and barrier round trip overlap the others'
    // decoding.  K-block it goes to decoded stage it % BST = the group's own.
    const int grp = dec_group<QT>(warp);
    const int gtid = (warp & 3) * 32 + lane;
    for (int it = grp < G ? grp : total_it; it < total_it; it += G) {  // groups >= gact stay idle
      const int ld = it / sub, sb = it % sub;           // code tile and its K-block
      const int cs = ld % cst, bs = it % BST;
      if (!warp_wait(cfull + cs, (ld / cst) & 1, abort_flag, err, 4)) break;
      if (it >= BST && !warp_wait(bempty + bs, ((it / BST) - 1) & 1, abort_flag, err, 8)) break;
      const unsigned char* raw = sRaw + cs * NT * rr;
      unsigned char* bdst = sB + bs * B_BYTES;
      if constexpr (BITS == 3) {
        // 3-bit codes: 3 bytes hold 8 codes (a little-endian 24-bit field);
        // each pair of codes is one lookup of two fp16 centroids
        const uint32_t* tab = reinterpret_cast<const uint32_t*>(base + L.tab);
        for (int item = gtid; item < NT * 8; item += 128) {
          const int r = item >> 3, g = item & 7;
          const unsigned char* src = raw + r * rrow + sb * RAWB + 3 * g;
          const uint32_t x = (uint32_t)src[0] | ((uint32_t)src[1] << 8) | ((uint32_t)src[2] << 16);
          uint32_t o[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) o[j] = tab[(((x >> (6 * j)) & 63u) << 5) | lane];
          *reinterpret_cast<uint4*>(bdst + sw128_offset(r, g)) = make_uint4(o[0], o[1], o[2], o[3]);
        }
      } else
      for (int item = gtid; item < NT * PARTS; item += 128) {
        const int r = item / PARTS, p = item % PARTS;
        const int chunk = sb * PARTS + p;  // 16-byte chunk of the row in this code tile
        const uint4 w4 = *reinterpret_cast<const uint4*>(
            raw + r * rrow + ((swz ? (chunk ^ (r & 7)) : chunk) << 4));
        const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
        for (int c = 0; c < CHUNKS; ++c) {
          uint4 out;
          if (BITS == 4) {          // chunk c: bytes 4c..4c+3, 8 codes
            out = decode8_4bit(w[c], tl, th);
          } else if (BITS == 2) {   // chunk c: bytes 2c, 2c+1, 8 codes
            const uint32_t* tab = reinterpret_cast<const uint32_t*>(base + L.tab);
            const uint32_t x = w[c >> 1] >> (16 * (c & 1));
            uint32_t o[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) o[j] = tab[(((x >> (4 * j)) & 0xFu) << 5) | lane];
            out = make_uint4(o[0], o[1], o[2], o[3]);
          } else {                  // chunk c: bytes 8c..8c+7, 8 codes
            const unsigned short* tab = reinterpret_cast<const unsigned short*>(base + L.tab);
            uint32_t o[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const uint32_t x = w[2 * c + (j >> 1)] >> (16 * (j & 1));
              o[j] = (uint32_t)tab[((x & 0xFFu) << 5) | lane] | ((uint32_t)tab[(((x >> 8) & 0xFFu) << 5) | lane] << 16);
            }
            out = make_uint4(o[0], o[1], o[2], o[3]);
          }
          *reinterpret_cast<uint4*>(bdst + sw128_offset(r, p * CHUNKS + c)) = out;
        }
      }
      fence_proxy_async();  // make this thread's writes visible to the tensor core
      __syncwarp();
      if (lane == 0) {
        if (sb + G >= sub) mbar_arrive(cempty + cs);  // this group's last K-block of the code tile
        mbar_arrive(dec + bs);
      }
    }
  } else {
    // ---------------------------------------------------------- epilogue
    // Eight warps: warp 8 + g reads TMEM lanes 32 (g % 4) .. + 31 (a warp may
    // only touch the lane quarter warp % 4) of query tile g / 4, so with two
    // query tiles per CTA both tiles are read out at once.
    const int g = warp - EPI_WARP0;
    const int e = g & 3;
    const int jsel = g >> 2;                 // this warp's query tile within the CTA
    const int row = e * 32 + lane;           // query row within that tile
    const int etid = g * 32 + lane;
    const bool mine = jsel < qts;            // warps 12-15 idle with one query tile
    const int q = (qt0 + jsel) * MMA_M + row;
    // a filtered search: this query's allow bitmap over the dense tenant index
    const uint32_t* ab = allow_bits && q < nq ? allow_bits + (size_t)q * words : nullptr;
    const float bq = bias && q < nq ? bias[q] : 0.f;  // a TQ+ index's per-query term (else 0)
    float* ls = lst_s + jsel * k * MMA_M;
    int* li = lst_i + jsel * k * MMA_M;
    if (mine) {
      for (int i = 0; i < k; ++i) {
        ls[i * MMA_M + row] = -INFINITY;
        li[i * MMA_M + row] = INT_MAX;
      }
    }
    float th_s = -INFINITY;
    int th_i = INT_MAX;
    float ps0 = 0.f, ps1 = 0.f, ps2 = 0.f, ps3 = 0.f;  // parked candidates of the current tile
    int pi0 = 0, pi1 = 0, pi2 = 0, pi3 = 0, npark = 0;
    // Inserts (sc, v) into this thread's sorted list if it beats entry
    // k-1: walk up while the entry above is worse, shifting it down; the
    // new entry k-1 is the first one shifted, or (sc, v) if nothing moves.
    auto insert = [&](float sc, int v) {
      if (!better(sc, v, th_s, th_i)) return;
      float nts = sc;
      int nti = v;
      int pos = k - 1;
      while (pos > 0) {
        const float as = ls[(pos - 1) * MMA_M + row];
        const int ai = li[(pos - 1) * MMA_M + row];
        if (!better(sc, v, as, ai)) break;
        ls[pos * MMA_M + row] = as;
        li[pos * MMA_M + row] = ai;
        if (pos == k - 1) {
          nts = as;
          nti = ai;
        }
        --pos;
      }
      ls[pos * MMA_M + row] = sc;
      li[pos * MMA_M + row] = v;
      th_s = nts;
      th_i = nti;
    };
    for (int tile_i = 0; tile_i < my_tiles; ++tile_i) {
      const int t = blockIdx.x + tile_i * gridDim.x;
      const int v0 = t * NT;
      const int set = tile_i % NSETS;
      // scales of this tile's vectors (the previous tile's readers are done:
      // they passed the named barrier below)
      for (int j = etid; j < NT; j += EPI_THREADS) {
        const int v = v0 + j;
        sScale[j] = v < n ? (scale ? scale[v] : 1.0f) : 0.0f;
        if (allow_bits) sDense[j] = v < n ? __ldg(dense + v) : 0u;
      }
      asm volatile("bar.sync 1, %0;" ::"n"(EPI_THREADS) : "memory");
      // all epilogue warps take the same decision, so none is left at bar.sync
      const int ok = warp_wait(acc_full + set, (tile_i / NSETS) & 1, abort_flag, err, 5) ? 1 : 0;
      int all_ok;
      asm volatile(
          "{\n .reg .pred p, q;\n setp.ne.s32 p, %1, 0;\n bar.red.and.pred q, 1, %2, p;\n"
          " selp.s32 %0, 1, 0, q;\n}"
          : "=r"(all_ok)
          : "r"(ok), "n"(EPI_THREADS)
          : "memory");
      if (!all_ok) break;
      tc_fence_after();
      if (mine) {
        const uint32_t tb = tmem + ((uint32_t)(32 * e) << 16) + (uint32_t)((set * QT + jsel) * NT);
        // one 16-column chunk: scale, flag the scores that may enter the list
        // (branch-free); flagged ones (rare after the first tiles) are parked
        // in registers and inserted after the accumulator is released, so the
        // insertions overlap the next tile's MMAs; a full park inserts at once
        auto chunk = [&](uint32_t (&r)[16], int c0) {
          if (q >= nq) return;
          const int valid = min(16, n - (v0 + c0));
          uint32_t m = 0;
#pragma unroll
          for (int jj = 0; jj < 16; jj += 4) {
            const float4 s4 = *reinterpret_cast<const float4*>(sScale + c0 + jj);
            const float2 x = __fmul2_rn(make_float2(__uint_as_float(r[jj]) + bq, __uint_as_float(r[jj + 1]) + bq),
                                        make_float2(s4.x, s4.y));
            const float2 y = __fmul2_rn(make_float2(__uint_as_float(r[jj + 2]) + bq,
                                                    __uint_as_float(r[jj + 3]) + bq),
                                        make_float2(s4.z, s4.w));
            r[jj] = __float_as_uint(x.x);
            r[jj + 1] = __float_as_uint(x.y);
            r[jj + 2] = __float_as_uint(y.x);
            r[jj + 3] = __float_as_uint(y.y);
            m |= (x.x >= th_s ? 1u : 0u) << jj;
            m |= (x.y >= th_s ? 1u : 0u) << (jj + 1);
            m |= (y.x >= th_s ? 1u : 0u) << (jj + 2);
            m |= (y.y >= th_s ? 1u : 0u) << (jj + 3);
          }
          if (valid < 16) m &= valid > 0 ? (1u << valid) - 1u : 0u;
          while (m) {
            const int jj = __ffs(m) - 1;
            m &= m - 1;
            float sc = 0.f;
#pragma unroll
            for (int t = 0; t < 16; ++t) sc = t == jj ? __uint_as_float(r[t]) : sc;
            const int v = v0 + c0 + jj;
            if (!better(sc, v, th_s, th_i)) continue;
            if (del && ((__ldg(del + (v >> 5)) >> (v & 31)) & 1u)) continue;  // deleted row
            if (ab) {  // tenant not allowed: never enters the list (Sec. III-B)
              const uint32_t t = sDense[c0 + jj];
              if (!((__ldg(ab + (t >> 5)) >> (t & 31)) & 1u)) continue;
            }
            if (npark < 4) {
              ps0 = npark == 0 ? sc : ps0;
              pi0 = npark == 0 ? v : pi0;
              ps1 = npark == 1 ? sc : ps1;
              pi1 = npark == 1 ? v : pi1;
              ps2 = npark == 2 ? sc : ps2;
              pi2 = npark == 2 ? v : pi2;
              ps3 = npark == 3 ? sc : ps3;
              pi3 = npark == 3 ? v : pi3;
              ++npark;
            } else {
              insert(sc, v);
            }
          }
        };
        // two chunks in flight: the next chunk's TMEM load overlaps this one's work
        uint32_t ra[16], rb[16];
        tmem_ld16_issue(tb, ra);
        tmem_wait16(ra);
#pragma unroll 1
        for (int c0 = 0; c0 < NT; c0 += 32) {
          tmem_ld16_issue(tb + (uint32_t)(c0 + 16), rb);
          chunk(ra, c0);
          tmem_wait16(rb);
          if (c0 + 32 < NT) tmem_ld16_issue(tb + (uint32_t)(c0 + 32), ra);
          chunk(rb, c0 + 16);
          if (c0 + 32 < NT) tmem_wait16(ra);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty + set);
      // the accumulator is free: insert the parked candidates while the next
      // tile's MMAs run
      if (npark > 0) insert(ps0, pi0);
      if (npark > 1) insert(ps1, pi1);
      if (npark > 2) insert(ps2, pi2);
      if (npark > 3) insert(ps3, pi3);
      npark = 0;
      asm volatile("bar.sync 1, %0;" ::"n"(EPI_THREADS) : "memory");
    }
    if (mine && q < nq) {
      for (int i = 0; i < k; ++i) {
        const size_t o = ((size_t)q * gridDim.x + blockIdx.x) * k + i;
        cand_s[o] = ls[i * MMA_M + row];
        cand_i[o] = li[i * MMA_M + row];
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == CODE_WARP) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
}

// Rotated queries (float32 [nq, d]) -> fp16 A blocks [qtile][kblock][128 x 64],
// K-major with the 128-byte swizzle, rows past nq zero.
__global__ void k_pack_queries(const float* __restrict__ qrot, int nq, int d, __half* __restrict__ out) {
  const int kblocks = d / KB;
  const int qt = blockIdx.y, kb = blockIdx.x;
  unsigned char* dst = reinterpret_cast<unsigned char*>(out) + ((size_t)qt * kblocks + kb) * A_BYTES;
  for (int i = threadIdx.x; i < MMA_M * (KB / 8); i += blockDim.x) {
    const int r = i / (KB / 8), c = i % (KB / 8);
    const int q = qt * MMA_M + r;
    uint32_t o[4] = {0, 0, 0, 0};
    if (q < nq) {
      const float* src = qrot + (size_t)q * d + kb * KB + c * 8;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const __half2 h = __floats2half2_rn(src[2 * j], src[2 * j + 1]);
        o[j] = *reinterpret_cast<const uint32_t*>(&h);
      }
    }
    *reinterpret_cast<uint4*>(dst + sw128_offset(r, c)) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

template <int BITS, int QT>
cudaError_t launch_typed(const MmaPlan& P, const CUtensorMap& map, const __half* qpack, const float* centroids,
                         const float* scale, const uint32_t* del, const uint32_t* dense, const uint32_t* allow,
                         int words, const float* bias, int n, int nq, int d, int k, int sub, int grid_x, float* cs,
                         int* ci, int* err, cudaStream_t s) {
  const int gact = active_groups(P.ng, sub, P.cst);
  cudaError_t e = set_max_dynamic_smem(reinterpret_cast<const void*>(k_scan_mma<BITS, QT>), (int)P.smem);
  if (e != cudaSuccess) return e;
  const int nqt = (nq + MMA_M - 1) / MMA_M;
  const dim3 grid((unsigned)grid_x, (unsigned)((nqt + QT - 1) / QT));
  k_scan_mma<BITS, QT><<<grid, NTHREADS, P.smem, s>>>(map, qpack, centroids, scale, del, dense, allow, words, bias,
                                                         n, nq, d, k, P.cst, P.ast, P.rr, sub, P.ng, gact, cs, ci,
                                                         err);
  return cudaGetLastError();
}

MmaPlan plan_for(int bits, int64_t nq, int k) {
  return bits == 2 ? mma_plan<2>(nq, k) : bits == 3 ? mma_plan<3>(nq, k) : bits == 4 ? mma_plan<4>(nq, k)
                                                                           : mma_plan<8>(nq, k);
}

}  // namespace

bool mma_supported(int bits, int d, int k) {
  // 3-bit code tiles carry an even number of K-blocks: d a multiple of 128
  return (bits == 2 || bits == 3 || bits == 4 || bits == 8) && d % (bits == 3 ? 2 * KB : KB) == 0 && k >= 1 &&
         k <= kMaxKMma && plan_for(bits, 1, k).smem != 0;
}

int scan_mma_grid_x(int64_t nq, int64_t n, int k, int bits) {
  const int64_t qtiles = (nq + MMA_M - 1) / MMA_M;
  const int qt = plan_for(bits, nq, k).qt;
  const int64_t groups = (qtiles + qt - 1) / qt;
  const int64_t ntiles = (n + MMA_N - 1) / MMA_N;
  int64_t gx = ((int64_t)device_sm_count() + groups - 1) / groups;
  if (gx > ntiles) gx = ntiles;
  if (gx < 1) gx = 1;
  return (int)gx;
}

size_t mma_qpack_bytes(int64_t nq, int d) {
  return (size_t)((nq + MMA_M - 1) / MMA_M) * (d / KB) * A_BYTES;
}

cudaError_t launch_scan_mma(const float* qrot, int64_t nq, int d, const float* centroids, int bits,
                            const uint8_t* codes, const float* scale, int64_t n, const uint32_t* del,
                            const uint32_t* dense, const uint32_t* allow_bits, int words, const float* bias,
                            int k, int grid_x, void* qpack, float* cand_s, int32_t* cand_i, int* err, cudaStream_t s,
                            cudaEvent_t ev0, cudaEvent_t ev1) {
  if (nq == 0) return cudaSuccess;
  PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
  if (!enc) return cudaErrorNotSupported;
  const int rawb = KB * bits / 8;
  const MmaPlan P = plan_for(bits, nq, k);
  if (P.smem == 0) return cudaErrorInvalidValue;
  // K-blocks per code tile: up to P.rr bytes of each row, dividing the row's K-blocks
  const int kblocks = d / KB;
  int sub = tile_sub(bits, P.rr);
  while (sub > (bits == 3 ? 2 : 1) && kblocks % sub != 0) sub >>= 1;
  if (kblocks % sub != 0 || (sub * rawb) % 16 != 0) return cudaErrorInvalidValue;
  CUtensorMap map;
  const cuuint64_t gdim[2] = {(cuuint64_t)row_bytes(d, bits), (cuuint64_t)n};
  const cuuint64_t gstride[1] = {(cuuint64_t)row_bytes(d, bits)};
  const cuuint32_t box[2] = {(cuuint32_t)(sub * rawb), (cuuint32_t)MMA_N};
  const cuuint32_t estride[2] = {1, 1};
  CUresult r = enc(&map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(codes), gdim, gstride, box,
                   estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   sub * rawb == RAW_ROW_MAX ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  const dim3 pgrid((unsigned)(d / KB), (unsigned)((nq + MMA_M - 1) / MMA_M));
  k_pack_queries<<<pgrid, 256, 0, s>>>(qrot, (int)nq, d, static_cast<__half*>(qpack));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (ev0 && (e = cudaEventRecord(ev0, s)) != cudaSuccess) return e;
  const __half* qp = static_cast<const __half*>(qpack);
#define TQ_MMA_CASE(B)                                                                                \
  case B:                                                                                             \
    e = P.qt == 2 ? launch_typed<B, 2>(P, map, qp, centroids, scale, del, dense, allow_bits, words, bias, \
                                       (int)n, (int)nq, d, k, sub, grid_x, cand_s, cand_i, err, s)        \
                  : launch_typed<B, 1>(P, map, qp, centroids, scale, del, dense, allow_bits, words, bias, \
                                       (int)n, (int)nq, d, k, sub, grid_x, cand_s, cand_i, err, s);       \
    break;
  switch (bits) {
    TQ_MMA_CASE(2)
    TQ_MMA_CASE(3)
    TQ_MMA_CASE(4)
    TQ_MMA_CASE(8)
    default: return cudaErrorInvalidValue;
  }
#undef TQ_MMA_CASE
  if (e != cudaSuccess) return e;
  if (ev1 && (e = cudaEventRecord(ev1, s)) != cudaSuccess) return e;
  return cudaSuccess;
}

}  // namespace tq
