// Tensor-core scan for query batches (Sec. II-B step 5 as a GEMM):
//   S[q, v] = scale_v * sum_j q'_j c[code_vj]
// with the rotated queries on the MMA's M dimension (128 per tile) and corpus
// vectors on N (256 per MMA), fp16 operands and fp32 accumulation in tensor
// memory (TMEM).  One CTA owns one query tile and a strided set of 256-vector
// tiles.  Roles (warp-specialised, 10 warps):
//   warps 0-3  decoders: expand one K-block (64 coordinates) of packed codes,
//              brought to shared memory by TMA, into fp16 centroid values laid
//              out as the K-major, 128-byte-swizzled B operand;
//   warps 4-7  epilogue: read the 128 x 256 fp32 accumulator from TMEM (one
//              query per thread), apply the per-vector scale and keep each
//              query's top-k in a thread-private sorted list;
//   warp 8     producer: TMA of the code tile and a 1-D bulk copy of the
//              pre-swizzled fp16 query block, one mbarrier per stage;
//              allocates TMEM;
//   warp 9     MMA issuer: one thread issues tcgen05.mma (M=128, N=256, K=16)
//              and commits completion to mbarriers.
// TMEM holds two 256-column accumulators so the epilogue of one vector tile
// overlaps the MMAs of the next.  Every wait is bounded: on timeout the CTA
// raises `abort`, writes an error code to a flag in the workspace and exits.
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

namespace tq {
namespace {

constexpr int MMA_M = 128;            // queries per tile
constexpr int MMA_N = 256;            // vectors per tile
constexpr int KB = 64;                // coordinates per K-block (128 B of fp16)
constexpr int STAGES = 2;
constexpr int NTHREADS = 320;
constexpr int A_BYTES = MMA_M * KB * 2;   // 16 KB
constexpr int B_BYTES = MMA_N * KB * 2;   // 32 KB
constexpr long long WAIT_CYCLES = 4000000000LL;  // ~2 s at 2 GHz

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase with the given parity; false on timeout or abort.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          int* err, int where) {
  const long long t0 = clock64();
  for (uint32_t i = 0;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63) == 63) {
      if (*abort_flag) return false;
      if (clock64() - t0 > WAIT_CYCLES) {
        *abort_flag = 1;
        atomicExch(err, TQ_ETIMEOUT * 1000 + where);
        return false;
      }
    }
  }
}

// Bounded wait that ignores `abort` (used to drain work already in flight).
__device__ __forceinline__ bool mbar_wait_drain(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  for (uint32_t i = 0;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63) == 63 && clock64() - t0 > WAIT_CYCLES) return false;
  }
}

__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
      ::"r"(smem_u32(dst)), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row
// atoms of 1024 bytes (stride byte offset), sm_100 descriptor version 1.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;             // leading byte offset (unused with 128-B swizzle)
  d |= (uint64_t)(1024 >> 4) << 32;   // stride byte offset: next 8-row atom
  d |= (uint64_t)1 << 46;             // descriptor version
  d |= (uint64_t)2 << 61;             // swizzle mode: 128 B
  return d;
}

// Instruction descriptor, kind::f16: D f32, A and B f16, both K-major, M x N.
constexpr uint32_t IDESC = (1u << 4) | (0u << 7) | (0u << 10) | ((uint32_t)(MMA_N >> 3) << 17) |
                           ((uint32_t)(MMA_M >> 4) << 24);

__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}"
      ::"r"(d_tmem), "l"(a), "l"(b), "r"(IDESC), "r"(accumulate));
}

__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
               ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ bool better(float s1, int i1, float s2, int i2) {
  return s1 > s2 || (s1 == s2 && i1 < i2);
}

// Byte offset of 16-byte chunk c of row r in a K-major, 128-B swizzled tile.
__device__ __forceinline__ uint32_t sw128_offset(int r, int c) {
  return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4));
}

struct MmaSmem {
  uint32_t a, b, raw, tab, scale, lists_s, lists_i, bars, total;
};

template <int BITS>
__host__ __device__ constexpr int raw_bytes_per_row() { return KB * BITS / 8; }

template <int BITS>
__host__ __device__ constexpr int tab_bytes() {
  return BITS == 4 ? 256 * 32 * 4 : BITS == 2 ? 16 * 32 * 4 : 256 * 32 * 2;
}

template <int BITS>
__host__ __device__ inline MmaSmem mma_smem_layout(int k) {
  MmaSmem L{};
  uint32_t off = 0;
  L.a = off;
  off += STAGES * A_BYTES;
  L.b = off;
  off += STAGES * B_BYTES;
  L.raw = off;
  off += STAGES * MMA_N * raw_bytes_per_row<BITS>();
  L.tab = off;
  off += tab_bytes<BITS>();
  L.scale = off;
  off += MMA_N * 4;
  L.lists_s = off;
  off += (uint32_t)k * MMA_M * 4;
  L.lists_i = off;
  off += (uint32_t)k * MMA_M * 4;
  off = (off + 15) & ~15u;
  L.bars = off;
  off += 16 * 8;
  L.total = off + 1024;  // slack to align the base to 1024 bytes
  // at most one CTA per SM: each allocates all 512 TMEM columns
  if (L.total < 116u * 1024u) L.total = 116u * 1024u;
  return L;
}

template <int BITS>
__global__ void __launch_bounds__(NTHREADS, 1)
k_scan_mma(const __grid_constant__ CUtensorMap codes_map, const __half* __restrict__ qpack,
           const float* __restrict__ centroids, const float* __restrict__ scale, int n, int nq, int d,
           int k, float* __restrict__ cand_s, int* __restrict__ cand_i, int* __restrict__ err) {
  constexpr int RAWB = raw_bytes_per_row<BITS>();
  extern __shared__ unsigned char smem_dyn[];
  unsigned char* base = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_dyn) + 1023) & ~(uintptr_t)1023);
  const MmaSmem L = mma_smem_layout<BITS>(k);
  unsigned char* sA = base + L.a;
  unsigned char* sB = base + L.b;
  unsigned char* sRaw = base + L.raw;
  float* sScale = reinterpret_cast<float*>(base + L.scale);
  float* lst_s = reinterpret_cast<float*>(base + L.lists_s);
  int* lst_i = reinterpret_cast<int*>(base + L.lists_i);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + L.bars);
  uint64_t* full = bars;                 // [STAGES] TMA bytes landed
  uint64_t* empty = bars + 2;            // [STAGES] MMAs done reading the stage
  uint64_t* dec = bars + 4;              // [STAGES] decoded B written
  uint64_t* acc_full = bars + 6;         // [2] accumulator complete
  uint64_t* acc_empty = bars + 8;        // [2] accumulator read out
  uint64_t* fin = bars + 10;             // all MMAs of this CTA complete
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 11);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 12);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int qt = blockIdx.y;
  const int kblocks = d / KB;
  const int ntiles = (n + MMA_N - 1) / MMA_N;
  const int my_tiles = blockIdx.x < ntiles ? (ntiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;

  // decode table, replicated in all 32 banks: entry e for lane l at e*32 + l
  if (BITS == 4) {
    uint32_t* tab = reinterpret_cast<uint32_t*>(base + L.tab);
    for (int i = tid; i < 256 * 32; i += NTHREADS) {
      const int e = i >> 5;
      const __half2 h = __floats2half2_rn(centroids[e & 15], centroids[e >> 4]);
      tab[i] = *reinterpret_cast<const uint32_t*>(&h);
    }
  } else if (BITS == 2) {
    uint32_t* tab = reinterpret_cast<uint32_t*>(base + L.tab);
    for (int i = tid; i < 16 * 32; i += NTHREADS) {
      const int e = i >> 5;
      const __half2 h = __floats2half2_rn(centroids[e & 3], centroids[e >> 2]);
      tab[i] = *reinterpret_cast<const uint32_t*>(&h);
    }
  } else {
    __half* tab = reinterpret_cast<__half*>(base + L.tab);
    for (int i = tid; i < 256 * 32; i += NTHREADS) tab[i] = __float2half_rn(centroids[i >> 5]);
  }
  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
      mbar_init(dec + s, 128);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full + b, 1);
      mbar_init(acc_empty + b, 128);
    }
    mbar_init(fin, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 8) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(smem_u32(tmem_slot)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int total_it = my_tiles * kblocks;

  if (warp == 8) {
    // ---------------------------------------------------------- producer
    if (lane == 0) {
      int issued = 0;
      for (int it = 0; it < total_it; ++it) {
        const int s = it % STAGES;
        const int use = it / STAGES;
        if (use > 0 && !mbar_wait(empty + s, (use - 1) & 1, abort_flag, err, 1)) break;
        const int t = blockIdx.x + (it / kblocks) * gridDim.x;
        const int kb = it % kblocks;
        mbar_arrive_expect_tx(full + s, A_BYTES + MMA_N * RAWB);
        tma_load_2d(sRaw + s * MMA_N * RAWB, &codes_map, kb * RAWB, t * MMA_N, full + s);
        bulk_load(sA + s * A_BYTES, qpack + ((size_t)qt * kblocks + kb) * (A_BYTES / 2), A_BYTES, full + s);
        issued = it + 1;
      }
      // never leave with copies in flight: wait (bounded) for the last one of each stage
      for (int s = 0; s < STAGES && s < issued; ++s) {
        const int last_use = (issued - 1 - s) / STAGES;
        mbar_wait_drain(full + s, last_use & 1);
      }
    }
  } else if (warp == 9) {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      for (int it = 0; it < total_it; ++it) {
        const int s = it % STAGES;
        const int tile_i = it / kblocks;
        const int kb = it % kblocks;
        const int buf = tile_i & 1;
        if (kb == 0 && tile_i >= 2 && !mbar_wait(acc_empty + buf, ((tile_i >> 1) - 1) & 1, abort_flag, err, 2))
          break;
        if (!mbar_wait(dec + s, (it / STAGES) & 1, abort_flag, err, 3)) break;
        tc_fence_after();
        const uint32_t a0 = smem_u32(sA + s * A_BYTES);
        const uint32_t b0 = smem_u32(sB + s * B_BYTES);
#pragma unroll
        for (int kk = 0; kk < KB / 16; ++kk)
          mma_f16(tmem + buf * MMA_N, sw128_desc(a0 + kk * 32), sw128_desc(b0 + kk * 32), (kb | kk) != 0);
        mma_commit(empty + s);
        if (kb == kblocks - 1) mma_commit(acc_full + buf);
      }
      mma_commit(fin);
      mbar_wait_drain(fin, 0);
    }
  } else if (warp < 4) {
    // ---------------------------------------------------------- decoders
    constexpr int PARTS = RAWB / 16;                 // 16-byte parts per row per K-block
    constexpr int CODES = 16 * 8 / BITS;             // codes per part
    constexpr int CHUNKS = CODES / 8;                // 16-byte fp16 chunks per part
    for (int it = 0; it < total_it; ++it) {
      const int s = it % STAGES;
      if (!mbar_wait(full + s, (it / STAGES) & 1, abort_flag, err, 4)) break;
      const unsigned char* raw = sRaw + s * MMA_N * RAWB;
      unsigned char* bdst = sB + s * B_BYTES;
      for (int item = tid; item < MMA_N * PARTS; item += 128) {
        const int r = item / PARTS, p = item % PARTS;
        const uint4 w4 = *reinterpret_cast<const uint4*>(raw + r * RAWB + p * 16);
        const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
        for (int c = 0; c < CHUNKS; ++c) {
          uint32_t o[4];
          if (BITS == 4) {          // chunk c: bytes 4c..4c+3, 8 codes
            const uint32_t* tab = reinterpret_cast<const uint32_t*>(base + L.tab);
#pragma unroll
            for (int j = 0; j < 4; ++j) o[j] = tab[(((w[c] >> (8 * j)) & 0xFFu) << 5) | lane];
          } else if (BITS == 2) {   // chunk c: bytes 2c, 2c+1, 8 codes
            const uint32_t* tab = reinterpret_cast<const uint32_t*>(base + L.tab);
            const uint32_t x = w[c >> 1] >> (16 * (c & 1));
#pragma unroll
            for (int j = 0; j < 4; ++j) o[j] = tab[(((x >> (4 * j)) & 0xFu) << 5) | lane];
          } else {                  // chunk c: bytes 8c..8c+7, 8 codes
            const unsigned short* tab = reinterpret_cast<const unsigned short*>(base + L.tab);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const uint32_t x = w[2 * c + (j >> 1)] >> (16 * (j & 1));
              o[j] = (uint32_t)tab[((x & 0xFFu) << 5) | lane] | ((uint32_t)tab[(((x >> 8) & 0xFFu) << 5) | lane] << 16);
            }
          }
          *reinterpret_cast<uint4*>(bdst + sw128_offset(r, p * CHUNKS + c)) = make_uint4(o[0], o[1], o[2], o[3]);
        }
      }
      fence_proxy_async();
      mbar_arrive(dec + s);
    }
  } else {
    // ---------------------------------------------------------- epilogue
    const int e = warp - 4;                 // TMEM lanes 32e .. 32e+31
    const int row = tid - 128;              // query row within the tile
    const int q = qt * MMA_M + row;
    for (int i = 0; i < k; ++i) {
      lst_s[i * MMA_M + row] = -INFINITY;
      lst_i[i * MMA_M + row] = INT_MAX;
    }
    float th_s = -INFINITY;
    int th_i = INT_MAX;
    for (int tile_i = 0; tile_i < my_tiles; ++tile_i) {
      const int t = blockIdx.x + tile_i * gridDim.x;
      const int v0 = t * MMA_N;
      const int buf = tile_i & 1;
      // scales of this tile's vectors (the previous tile's readers are done:
      // they passed the named barrier below)
      for (int j = row; j < MMA_N; j += 128) {
        const int v = v0 + j;
        sScale[j] = v < n ? (scale ? scale[v] : 1.0f) : 0.0f;
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");
      // all four epilogue warps take the same decision, so none is left at bar.sync
      const int ok = mbar_wait(acc_full + buf, (tile_i >> 1) & 1, abort_flag, err, 5) ? 1 : 0;
      int all_ok;
      asm volatile(
          "{\n .reg .pred p, q;\n setp.ne.s32 p, %1, 0;\n bar.red.and.pred q, 1, 128, p;\n"
          " selp.s32 %0, 1, 0, q;\n}"
          : "=r"(all_ok)
          : "r"(ok)
          : "memory");
      if (!all_ok) break;
      tc_fence_after();
      for (int c0 = 0; c0 < MMA_N; c0 += 32) {
        uint32_t r[32];
        tmem_ld32(tmem + ((uint32_t)(32 * e) << 16) + buf * MMA_N + c0, r);
        if (q < nq) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int v = v0 + c0 + j;
            const float sc = __uint_as_float(r[j]) * sScale[c0 + j];
            if (v < n && better(sc, v, th_s, th_i)) {
              int pos = k - 1;
              while (pos > 0 && better(sc, v, lst_s[(pos - 1) * MMA_M + row], lst_i[(pos - 1) * MMA_M + row])) {
                lst_s[pos * MMA_M + row] = lst_s[(pos - 1) * MMA_M + row];
                lst_i[pos * MMA_M + row] = lst_i[(pos - 1) * MMA_M + row];
                --pos;
              }
              lst_s[pos * MMA_M + row] = sc;
              lst_i[pos * MMA_M + row] = v;
              th_s = lst_s[(k - 1) * MMA_M + row];
              th_i = lst_i[(k - 1) * MMA_M + row];
            }
          }
        }
      }
      tc_fence_before();
      mbar_arrive(acc_empty + buf);
      asm volatile("bar.sync 1, 128;" ::: "memory");
    }
    if (q < nq) {
      for (int i = 0; i < k; ++i) {
        const size_t o = ((size_t)q * gridDim.x + blockIdx.x) * k + i;
        cand_s[o] = lst_s[i * MMA_M + row];
        cand_i[o] = lst_i[i * MMA_M + row];
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 8) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
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

PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

template <int BITS>
cudaError_t launch_typed(const CUtensorMap& map, const __half* qpack, const float* centroids,
                         const float* scale, int n, int nq, int d, int k, int grid_x, float* cs, int* ci,
                         int* err, cudaStream_t s) {
  const MmaSmem L = mma_smem_layout<BITS>(k);
  cudaError_t e = cudaFuncSetAttribute(k_scan_mma<BITS>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)L.total);
  if (e != cudaSuccess) return e;
  const dim3 grid((unsigned)grid_x, (unsigned)((nq + MMA_M - 1) / MMA_M));
  k_scan_mma<BITS><<<grid, NTHREADS, L.total, s>>>(map, qpack, centroids, scale, n, nq, d, k, cs, ci, err);
  return cudaGetLastError();
}

}  // namespace

bool mma_supported(int bits, int d, int k) {
  return (bits == 2 || bits == 4 || bits == 8) && d % KB == 0 && k <= kMaxKMma;
}

int scan_mma_grid_x(int64_t nq, int64_t n) {
  const int64_t qtiles = (nq + MMA_M - 1) / MMA_M;
  const int64_t ntiles = (n + MMA_N - 1) / MMA_N;
  int64_t gx = ((int64_t)device_sm_count() + qtiles - 1) / qtiles;
  if (gx > ntiles) gx = ntiles;
  if (gx < 1) gx = 1;
  return (int)gx;
}

size_t mma_qpack_bytes(int64_t nq, int d) {
  return (size_t)((nq + MMA_M - 1) / MMA_M) * (d / KB) * A_BYTES;
}

cudaError_t launch_scan_mma(const float* qrot, int64_t nq, int d, const float* centroids, int bits,
                            const uint8_t* codes, const float* scale, int64_t n, int k, int grid_x,
                            void* qpack, float* cand_s, int32_t* cand_i, int* err, cudaStream_t s,
                            cudaEvent_t ev0, cudaEvent_t ev1) {
  if (nq == 0) return cudaSuccess;
  PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
  if (!enc) return cudaErrorNotSupported;
  const int rawb = KB * bits / 8;
  CUtensorMap map;
  const cuuint64_t gdim[2] = {(cuuint64_t)row_bytes(d, bits), (cuuint64_t)n};
  const cuuint64_t gstride[1] = {(cuuint64_t)row_bytes(d, bits)};
  const cuuint32_t box[2] = {(cuuint32_t)rawb, (cuuint32_t)MMA_N};
  const cuuint32_t estride[2] = {1, 1};
  CUresult r = enc(&map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(codes), gdim, gstride, box,
                   estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  const dim3 pgrid((unsigned)(d / KB), (unsigned)((nq + MMA_M - 1) / MMA_M));
  k_pack_queries<<<pgrid, 256, 0, s>>>(qrot, (int)nq, d, static_cast<__half*>(qpack));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (ev0 && (e = cudaEventRecord(ev0, s)) != cudaSuccess) return e;
  const __half* qp = static_cast<const __half*>(qpack);
  switch (bits) {
    case 2: e = launch_typed<2>(map, qp, centroids, scale, (int)n, (int)nq, d, k, grid_x, cand_s, cand_i, err, s); break;
    case 4: e = launch_typed<4>(map, qp, centroids, scale, (int)n, (int)nq, d, k, grid_x, cand_s, cand_i, err, s); break;
    case 8: e = launch_typed<8>(map, qp, centroids, scale, (int)n, (int)nq, d, k, grid_x, cand_s, cand_i, err, s); break;
    default: return cudaErrorInvalidValue;
  }
  if (e != cudaSuccess) return e;
  if (ev1 && (e = cudaEventRecord(ev1, s)) != cudaSuccess) return e;
  return cudaSuccess;
}

}  // namespace tq
