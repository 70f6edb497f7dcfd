// Tensor-core encode (Sec. II-B steps 1-5): the rotation Y = X R^T runs on
// tcgen05 in TF32 with a three-product split, followed by the same
// quantise / pack / per-vector-scale epilogue as the FFMA encoder.
//
// Precision.  TF32 keeps 10 explicit mantissa bits, so one TF32 product would
// move y by about 1e-5 (the width of a codebook cell's neighbourhood that the
// parity window allows).  Each operand is therefore split into two TF32 parts,
// v = v_hi + v_lo with v_hi = tf32(v), v_lo = tf32(v - v_hi), and
//   x . r  ~  x_hi . r_hi + x_hi . r_lo + x_lo . r_hi,
// which leaves a relative error of a few 2^-22 per product (the dropped
// x_lo . r_lo term and the rounding of the low parts), the same order as an
// fp32 FFMA dot product.  R is split once into a caller-owned plan
// (tq_encode_plan); X is split as its tiles arrive.
//
// Work.  A CTA owns panels of 128 rows of X (the MMA's M) and walks the d
// output coordinates in chunks of 256 (N), each chunk a full contraction over
// K = d in K-blocks of 16 coordinates (64-byte rows of fp32 with the 64-byte
// swizzle: five 40 KB shared-memory stages of the raw X tile and the R_hi and
// R_lo tiles).  The split X tile goes to tensor memory and is the MMAs' A
// operand there, so the tensor cores read only the R tiles from shared
// memory; TMEM holds one 128 x 256 fp32 accumulator and the five stages' x_hi
// and x_lo (32 columns each).  Chunks walk the K-blocks alternately forwards
// and backwards, so a chunk starts on the X tiles the previous one read last
// (still in L2).  Roles (14 warps):
//   warps 0-3   converters: thread t owns row t of each X tile, splits it into
//               x_hi and x_lo and stores both to its TMEM lane (tcgen05.st),
//               and sums x^2 over the first chunk's K-blocks (the row norm,
//               step 1);
//   warp 4      producer: TMA of the X tile and the R_hi / R_lo tiles;
//   warp 5      MMA issuer: allocates TMEM; one thread issues the three
//               tcgen05.mma products per K-step (M=128, N=256, K=8; A in
//               TMEM, B in shared memory);
//   warps 6-13  epilogue: warp w reads TMEM lanes 32 (w % 4) .. + 31 (one row
//               per thread), columns 0-127 (warps 6-9) or 128-255 (10-13) of
//               the chunk: y = acc / ||x|| (step 2), the code by boundary
//               search (step 3), packed straight to HBM (step 4), and the
//               per-row sums that give the scalar (step 5).
// Every wait is bounded: on timeout the CTA raises its abort flag, records
// TQ_ETIMEOUT * 1000 + site in the plan's status word, drains the copies and
// MMAs it has in flight and returns.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>

#include "tq_internal.h"
#include "tq_kernels.h"
#include "tq_tc.cuh"

namespace tq {
namespace {

constexpr int EM = 128;                     // rows of X per panel (MMA M)
constexpr int EN = 256;                     // output coordinates per chunk (MMA N)
constexpr int EK = 16;                      // coordinates per K-block (64 B of fp32)
constexpr int NSTAGE = 4;                   // K-block stages in flight
constexpr int X_BYTES = EM * EK * 4;        // 8 KB: an X tile (x_hi after the split)
constexpr int R_BYTES = EN * EK * 4;        // 16 KB: an R_hi or R_lo tile
constexpr int STAGE_BYTES = 2 * X_BYTES + 2 * R_BYTES;  // x_hi, x_lo, r_hi, r_lo (the rotation kernel)
// The encoder keeps the split X tile in tensor memory: a stage in shared
// memory is the raw X tile and the R_hi, R_lo tiles.
constexpr int ENC_NSTAGE = 5;
constexpr int ENC_STAGE_BYTES = X_BYTES + 2 * R_BYTES;  // 40 KB
constexpr uint32_t TM_A = EN;              // TMEM column of the first stage's x_hi (the accumulator is 0 .. EN-1)
constexpr uint32_t TM_A_STAGE = 2 * EK;    // columns per stage: x_hi, then x_lo
constexpr int CONV_WARPS = 4, PROD_WARP = 4, MMA_WARP = 5, EPI_WARP0 = 6, EPI_WARPS = 8;
constexpr int ENC_THREADS = (EPI_WARP0 + EPI_WARPS) * 32;  // 448
constexpr int EPI_THREADS = EPI_WARPS * 32;
constexpr uint32_t kEncDynSmemMax = 232448;  // 227 KB per block
// Plan layout: a 256-byte header whose first int is the status word, then
// R_hi (d x d fp32, row-major) and R_lo (d x d), i.e. one [2d x d] matrix.
constexpr size_t kPlanHeader = 256;

// Offsets in the 1024-byte-aligned dynamic shared memory.
struct EncSmem {
  // stage s at s * ENC_STAGE_BYTES: x, r_hi, r_lo tiles
  // boundaries and centroids: with codes of up to 4 bits one copy per bank
  // ([entry][32]), so the epilogue's data-dependent lookups never conflict
  static constexpr uint32_t bnd = ENC_NSTAGE * ENC_STAGE_BYTES;  // [512] floats
  static constexpr uint32_t cen = bnd + 512 * 4;         // [512] floats
  static constexpr uint32_t nrm = cen + 512 * 4;         // [2][128] row norms by panel parity
  static constexpr uint32_t inv = nrm + 2 * EM * 4;      // [2][128] 1 / norm
  static constexpr uint32_t part = inv + 2 * EM * 4;     // [2][2][128] double: sum c^2, sum y c of the column-128..255 warps
  static constexpr uint32_t bars = part + 4 * EM * 8;    // mbarriers
  static constexpr uint32_t nbars = 28;
  static constexpr uint32_t misc = bars + nbars * 8;     // TMEM address, abort flag
  static constexpr uint32_t total = misc + 16;
};
constexpr uint32_t kEncSmem = EncSmem::total + 1024;  // slack for the 1024-byte alignment
static_assert(kEncSmem <= kEncDynSmemMax, "encoder shared memory");

// Instruction descriptor, kind::tf32: D f32, A and B TF32, both K-major, M x N.
__host__ __device__ constexpr uint32_t idesc_tf32() {
  return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(EN >> 3) << 17) | ((uint32_t)(EM >> 4) << 24);
}

__device__ __forceinline__ void mma_tf32(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}"
      ::"r"(d_tmem), "l"(a), "l"(b), "r"(idesc_tf32()), "r"(accumulate));
}

// The same with A in tensor memory (M lanes, K columns of 32-bit values).
__device__ __forceinline__ void mma_tf32_ta(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::tf32 [%0], [%1], %2, %3, p;\n}"
      ::"r"(d_tmem), "r"(a_tmem), "l"(b), "r"(idesc_tf32()), "r"(accumulate));
}

// Stores 16 consecutive TMEM columns of this thread's lane.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};"
      ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

// v rounded to the nearest TF32 value (10 explicit mantissa bits; ties away
// from zero): add half of the 13 dropped bits' range, then clear them.  The
// carry of a full mantissa moves into the exponent, which is the correct
// rounding up to the next binade.
__device__ __forceinline__ float tf32_round(float v) {
  return __uint_as_float((__float_as_uint(v) + 0x1000u) & 0xFFFFE000u);
}

// Plan: R_hi = tf32(R), R_lo = tf32(R - R_hi) (the difference is exact in
// fp32), and a cleared status word.
__global__ void k_encode_plan(const float* __restrict__ R, int d, unsigned char* __restrict__ plan) {
  float* hi = reinterpret_cast<float*>(plan + kPlanHeader);
  float* lo = hi + (size_t)d * d;
  const size_t total = (size_t)d * d;
  if (blockIdx.x == 0 && threadIdx.x < kPlanHeader / 4) reinterpret_cast<int*>(plan)[threadIdx.x] = 0;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (size_t)gridDim.x * blockDim.x) {
    const float r = R[i];
    const float h = tf32_round(r);
    hi[i] = h;
    lo[i] = tf32_round(r - h);
  }
}

template <int BITS, bool CAL>
__global__ void __launch_bounds__(ENC_THREADS, 1)
k_encode_tc(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap rmap, int n, int d,
            const float* __restrict__ centroids, const float* __restrict__ boundaries, int scale_mode,
            const float* __restrict__ cal_mu, const float* __restrict__ cal_a, uint8_t* __restrict__ codes,
            float* __restrict__ scale, int* __restrict__ err) {
  constexpr int L = 1 << BITS;
  constexpr int REP = BITS <= 4 ? 32 : 1;  // copies of each table entry (one per bank)
  extern __shared__ unsigned char smem_dyn[];
  unsigned char* base = smem_dyn + ((1024u - (smem_u32(smem_dyn) & 1023u)) & 1023u);
  float* sBnd = reinterpret_cast<float*>(base + EncSmem::bnd);
  float* sCen = reinterpret_cast<float*>(base + EncSmem::cen);
  float* sNrm = reinterpret_cast<float*>(base + EncSmem::nrm);
  float* sInv = reinterpret_cast<float*>(base + EncSmem::inv);
  double* sPart = reinterpret_cast<double*>(base + EncSmem::part);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + EncSmem::bars);
  uint64_t* full = bars;             // [ENC_NSTAGE] X and R tiles landed
  uint64_t* conv = bars + 5;         // [ENC_NSTAGE] X tile split into tensor memory
  uint64_t* empty = bars + 10;       // [ENC_NSTAGE] MMAs done with the stage
  uint64_t* acc_full = bars + 15;    // the accumulator complete
  uint64_t* acc_empty = bars + 16;   // the accumulator read out
  uint64_t* norm_ready = bars + 18;  // [2] row norms of a panel written (by panel parity)
  uint64_t* norm_free = bars + 20;   // [2] row norms of a panel read
  uint64_t* part_ready = bars + 22;  // [2] column-128..255 sums of a panel written
  uint64_t* fin = bars + 24;         // every MMA of this CTA complete
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(base + EncSmem::misc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(base + EncSmem::misc + 4);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int KB = d / EK;                  // K-blocks per contraction
  const int C = (d + EN - 1) / EN;        // chunks per panel (the last one may be partial)
  const int panels = (n + EM - 1) / EM;
  const int my_panels = (int)blockIdx.x < panels ? (panels - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
  const long long total_it = (long long)my_panels * C * KB;

  for (int i = tid; i < 512; i += ENC_THREADS) {
    const int e = i / REP;
    sCen[i] = e < L ? centroids[e] : 0.f;
    sBnd[i] = e < L - 1 ? boundaries[e] : INFINITY;
  }
  if (tid == 0) {
    for (int s = 0; s < ENC_NSTAGE; ++s) {
      mbar_init(full + s, 1);
      mbar_init(conv + s, CONV_WARPS);
      mbar_init(empty + s, 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, EPI_WARPS);
    for (int b = 0; b < 2; ++b) {
      mbar_init(norm_ready + b, CONV_WARPS * 32);  // every converter thread, after its row
      mbar_init(norm_free + b, EPI_WARPS);
      mbar_init(part_ready + b, EPI_THREADS / 2);  // every column-128..255 thread, after its row
    }
    mbar_init(fin, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == MMA_WARP) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(smem_u32(tmem_slot)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == PROD_WARP) {
    // ------------------------------------------------ X, R_hi, R_lo tiles (TMA)
    if (lane == 0) {
      long long issued = 0;
      for (long long it = 0; it < total_it; ++it) {
        const int s = (int)(it % ENC_NSTAGE);
        const long long use = it / ENC_NSTAGE;
        if (use > 0 && !mbar_wait(empty + s, (uint32_t)((use - 1) & 1), abort_flag, err, 41)) break;
        const int kb = (int)(it % KB);
        const long long cs = it / KB;
        const int c = (int)(cs % C), i = (int)(cs / C);
        const int panel = (int)blockIdx.x + i * (int)gridDim.x;
        const int kc = (c & 1) ? KB - 1 - kb : kb;  // snake order over the K-blocks
        unsigned char* st = base + s * ENC_STAGE_BYTES;
        mbar_arrive_expect_tx(full + s, X_BYTES + 2 * R_BYTES);
        tma_load_2d(st, &xmap, kc * EK, panel * EM, full + s);
        // rows c*256 .. of R_hi, then of R_lo (rows d .. 2d-1 of the plan); in a
        // partial last chunk the rows past d are R_lo rows or zero fill, and the
        // epilogue never reads their columns
        tma_load_2d(st + X_BYTES, &rmap, kc * EK, c * EN, full + s);
        tma_load_2d(st + X_BYTES + R_BYTES, &rmap, kc * EK, d + c * EN, full + s);
        issued = it + 1;
      }
      // never leave with copies in flight: wait (bounded) for the last one of each stage
      for (int s = 0; s < ENC_NSTAGE && s < issued; ++s)
        mbar_wait_drain(full + s, (uint32_t)(((issued - 1 - s) / ENC_NSTAGE) & 1));
    }
  } else if (warp == MMA_WARP) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      for (long long it = 0; it < total_it; ++it) {
        const int s = (int)(it % ENC_NSTAGE);
        const long long use = it / ENC_NSTAGE;
        const int kb = (int)(it % KB);
        const long long cs = it / KB;
        if (kb == 0 && cs >= 1 && !mbar_wait(acc_empty, (uint32_t)((cs - 1) & 1), abort_flag, err, 42)) break;
        if (!mbar_wait(conv + s, (uint32_t)(use & 1), abort_flag, err, 43)) break;
        tc_fence_after();
        const uint32_t rh = smem_u32(base + s * ENC_STAGE_BYTES) + X_BYTES, rl = rh + R_BYTES;
        const uint32_t ah = tmem + TM_A + (uint32_t)s * TM_A_STAGE, al = ah + EK;
#pragma unroll
        for (int kk = 0; kk < EK / 8; ++kk) {  // K = 8 TF32 values: 32 bytes of each R row, 8 TMEM columns of x
          const uint32_t o = (uint32_t)kk * 32u, oa = (uint32_t)kk * 8u;
          mma_tf32_ta(tmem, ah + oa, sw64_desc(rh + o), (kb | kk) != 0);
          mma_tf32_ta(tmem, ah + oa, sw64_desc(rl + o), 1u);
          mma_tf32_ta(tmem, al + oa, sw64_desc(rh + o), 1u);
        }
        mma_commit(empty + s);
        if (kb == KB - 1) mma_commit(acc_full);
      }
      mma_commit(fin);
      mbar_wait_drain(fin, 0);
    }
  } else if (warp < CONV_WARPS) {
    // ------------------------------------------------------------- converters
    // Thread t owns row t; reading the 16-byte parts in logical order through
    // the 64-byte swizzle (part q of row t sits at part q ^ ((t >> 1) & 3))
    // keeps a warp's accesses free of bank conflicts.  The row's
    // sum of squares takes a fixed order: four float partials per K-block,
    // paired, then added in double across K-blocks (a plain float running
    // sum over d terms would lose ~sqrt(d) ulps).
    const int t = tid;
    double ss = 0.0;
    for (long long it = 0; it < total_it; ++it) {
      const int s = (int)(it % ENC_NSTAGE);
      const long long use = it / ENC_NSTAGE;
      const int kb = (int)(it % KB);
      const long long cs = it / KB;
      const int c = (int)(cs % C), i = (int)(cs / C);
      if (!warp_wait(full + s, (uint32_t)(use & 1), abort_flag, err, 44)) break;
      const unsigned char* xt = base + s * ENC_STAGE_BYTES;
      float p0 = 0.f, p1 = 0.f, p2 = 0.f, p3 = 0.f;
      uint32_t hv[EK], lv[EK];  // row t's x_hi and x_lo, in K order
#pragma unroll
      for (int q = 0; q < EK / 4; ++q) {
        const uint32_t off = (uint32_t)t * 64u + ((uint32_t)(q ^ ((t >> 1) & 3)) << 4);
        const float4 v = *reinterpret_cast<const float4*>(xt + off);
        p0 = fmaf(v.x, v.x, p0);
        p1 = fmaf(v.y, v.y, p1);
        p2 = fmaf(v.z, v.z, p2);
        p3 = fmaf(v.w, v.w, p3);
        const float vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const float hi = tf32_round(vv[u]);
          hv[4 * q + u] = __float_as_uint(hi);
          lv[4 * q + u] = __float_as_uint(tf32_round(vv[u] - hi));
        }
      }
      // lane quarter = this warp (warps 0-3), column = K index
      const uint32_t ta = tmem + ((uint32_t)(warp * 32) << 16) + TM_A + (uint32_t)s * TM_A_STAGE;
      tmem_st16(ta, hv);
      tmem_st16(ta + EK, lv);
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(conv + s);
      if (c == 0) ss += (double)((p0 + p1) + (p2 + p3));
      if (c == 0 && kb == KB - 1) {  // the panel's norms (step 1), double-buffered by panel parity
        const int pp = i & 1;
        if (i >= 2 && !warp_wait(norm_free + pp, (uint32_t)(((i >> 1) - 1) & 1), abort_flag, err, 45)) break;
        const float nr = (float)sqrt(ss);
        sNrm[pp * EM + t] = nr;
        sInv[pp * EM + t] = nr > 0.f ? 1.0f / nr : 0.f;
        mbar_arrive(norm_ready + pp);
        ss = 0.0;
      }
    }
  } else if (warp >= EPI_WARP0) {
    // --------------------------------------------------------------- epilogue
    const int quarter = warp & 3;            // TMEM lane quarter this warp may read
    const int h = (warp - EPI_WARP0) >> 2;   // column half of the chunk
    const int row = quarter * 32 + lane;
    const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(h * (EN / 2));
    const int64_t rbytes = (int64_t)d * BITS / 8;
    const int rl = lane & (REP - 1);  // this lane's copy of the tables
    float inv = 0.f, nr = 0.f;
    double c2 = 0.0, yc = 0.0;  // the row's sums over this thread's columns (float per 16, then double)
    int64_t grow = 0;
    // 16 consecutive accumulator columns (coordinates j0 .. j0+15) of this row
    auto group = [&](const uint32_t (&r)[16], int j0) {
      if (j0 >= d) return;  // columns of a partial last chunk (d is a multiple of 32)
      uint64_t packed = 0;  // 2-, 3- and 4-bit codes, little-endian bit stream
      uint32_t p8[4] = {0, 0, 0, 0};
      float g2 = 0.f, gy = 0.f;
#pragma unroll
      for (int t = 0; t < 16; ++t) {
        const float y = __uint_as_float(r[t]) * inv;
        float z = y, mu = 0.f, a = 1.f;
        if constexpr (CAL) {
          mu = __ldg(cal_mu + j0 + t);
          a = __ldg(cal_a + j0 + t);
          z = (y - mu) * (1.0f / a);
        }
        int code = 0;
#pragma unroll
        for (int step = L / 2; step >= 1; step >>= 1)
          if (z > sBnd[(code + step - 1) * REP + rl]) code += step;
        const float cc = sCen[code * REP + rl];
        const float cv = CAL ? fmaf(a, cc, mu) : cc;
        g2 = fmaf(cv, cv, g2);
        gy = fmaf(y, cv, gy);
        if constexpr (BITS == 8) p8[t >> 2] |= (uint32_t)code << (8 * (t & 3));
        else packed |= (uint64_t)code << (BITS * t);
      }
      c2 += (double)g2;
      yc += (double)gy;
      if (grow >= n) return;
      uint8_t* dst = codes + grow * rbytes + (int64_t)j0 * BITS / 8;
      if constexpr (BITS == 8) {
        *reinterpret_cast<uint4*>(dst) = make_uint4(p8[0], p8[1], p8[2], p8[3]);
      } else if constexpr (BITS == 4) {
        *reinterpret_cast<uint2*>(dst) = make_uint2((uint32_t)packed, (uint32_t)(packed >> 32));
      } else if constexpr (BITS == 2) {
        *reinterpret_cast<uint32_t*>(dst) = (uint32_t)packed;
      } else {  // 48 bits at an even byte offset (j0 / 16 * 6)
        uint16_t* d16 = reinterpret_cast<uint16_t*>(dst);
        d16[0] = (uint16_t)packed;
        d16[1] = (uint16_t)(packed >> 16);
        d16[2] = (uint16_t)(packed >> 32);
      }
    };
    const long long nchunks = (long long)my_panels * C;
    for (long long cs = 0; cs < nchunks; ++cs) {
      const int c = (int)(cs % C), i = (int)(cs / C);
      const int pp = i & 1;
      if (c == 0) {
        if (!warp_wait(norm_ready + pp, (uint32_t)((i >> 1) & 1), abort_flag, err, 46)) break;
        inv = sInv[pp * EM + row];
        nr = sNrm[pp * EM + row];
        __syncwarp();
        if (lane == 0) mbar_arrive(norm_free + pp);
        c2 = 0.0;
        yc = 0.0;
        grow = (int64_t)((int)blockIdx.x + i * (int)gridDim.x) * EM + row;
      }
      if (!warp_wait(acc_full, (uint32_t)(cs & 1), abort_flag, err, 47)) break;
      tc_fence_after();
      const uint32_t ta = tl;
      const int jb = c * EN + h * (EN / 2);
      uint32_t ra[16], rb[16];
      tmem_ld16_issue(ta, ra);
      tmem_wait16(ra);
#pragma unroll 1
      for (int g = 0; g < EN / 2; g += 32) {
        tmem_ld16_issue(ta + (uint32_t)(g + 16), rb);
        group(ra, jb + g);
        tmem_wait16(rb);
        if (g + 32 < EN / 2) tmem_ld16_issue(ta + (uint32_t)(g + 32), ra);
        group(rb, jb + g + 16);
        if (g + 32 < EN / 2) tmem_wait16(ra);
      }
      tc_fence_before();
      bool ok = true;
      if (c == C - 1) {
        // the panel's scalar (step 5): the column-128..255 threads hand their
        // sums to the column-0..127 threads of the same row, which hold the
        // accumulator set until they have read them (so the next panel's
        // sums cannot overwrite them first)
        double* pc = sPart + (2 * pp) * EM;      // sum c^2 by row
        double* py = sPart + (2 * pp + 1) * EM;  // sum y c by row
        if (h == 1) {
          pc[row] = c2;
          py[row] = yc;
          mbar_arrive(part_ready + pp);
        } else {
          ok = warp_wait(part_ready + pp, (uint32_t)((i >> 1) & 1), abort_flag, err, 48);
          if (ok && grow < n) {
            const float tc2 = (float)(c2 + pc[row]);
            const float tyc = (float)(yc + py[row]);
            float sv = 0.f;
            if (nr > 0.f) {
              if (scale_mode == TQ_SCALE_NONE) {
                sv = nr;
              } else if (scale_mode == TQ_SCALE_NORM) {
                const float cn = sqrtf(tc2);
                sv = cn > 0.f ? nr / cn : 0.f;
              } else {
                sv = tyc != 0.f ? nr / tyc : 0.f;
              }
            }
            scale[grow] = sv;
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty);
      if (!ok) break;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == MMA_WARP) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
}

// Query rotation on the tensor cores (Sec. II-B step 2 for a batch of
// queries): part[s] = Q R^T over split s of the K-blocks, with the same
// three-product TF32 split; the search is given R itself, so R's tiles are
// split in shared memory as they arrive, like Q's.  CTA (c, p, s) computes
// output coordinates c*256 .., query rows p*128 .., K-blocks
// [s*KB/S, (s+1)*KB/S); k_rotate_reduce adds the S partial products in a
// fixed order.  Roles (10 warps): warps 0-3 split the Q tile (row t) and the
// R tile (rows t, t+128); warp 4 issues the copies; warp 5 the MMAs (one
// 128 x 256 accumulator); warps 6-9 store the accumulator (lane quarter
// w % 4, all 256 columns).
constexpr int ROT_EPI0 = 6;
constexpr int ROT_THREADS = (ROT_EPI0 + 4) * 32;
constexpr uint32_t kRotBars = NSTAGE * STAGE_BYTES;
constexpr uint32_t kRotSmem = kRotBars + 16 * 8 + 16 + 1024;
static_assert(kRotSmem <= kEncDynSmemMax, "rotation shared memory");

__global__ void __launch_bounds__(ROT_THREADS, 1)
k_rotate_tc(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap rmap, int nq, int d,
            int S, float* __restrict__ part, int* __restrict__ err) {
  extern __shared__ unsigned char smem_dyn[];
  unsigned char* base = smem_dyn + ((1024u - (smem_u32(smem_dyn) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + kRotBars);
  uint64_t* full = bars;          // [NSTAGE] Q and R tiles landed
  uint64_t* conv = bars + 4;      // [NSTAGE] both tiles split
  uint64_t* empty = bars + 8;     // [NSTAGE] MMAs done with the stage
  uint64_t* acc_full = bars + 12;
  uint64_t* fin = bars + 13;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 16);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 16) + 1;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c = blockIdx.x, p = blockIdx.y, sp = blockIdx.z;
  const int KB = d / EK;
  const int kb0 = (int)((long long)sp * KB / S), nk = (int)((long long)(sp + 1) * KB / S) - kb0;
  if (tid == 0) {
    // a new search: clear the status word (any wait that gives up records
    // itself there, seconds after every CTA has started)
    if (c == 0 && p == 0 && sp == 0) *err = 0;
    for (int i = 0; i < NSTAGE; ++i) {
      mbar_init(full + i, 1);
      mbar_init(conv + i, CONV_WARPS);
      mbar_init(empty + i, 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(fin, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == MMA_WARP) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 256;" ::"r"(smem_u32(tmem_slot)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == PROD_WARP) {
    if (lane == 0) {
      int issued = 0;
      for (int it = 0; it < nk; ++it) {
        const int s = it % NSTAGE, use = it / NSTAGE;
        if (use > 0 && !mbar_wait(empty + s, (uint32_t)((use - 1) & 1), abort_flag, err, 51)) break;
        unsigned char* st = base + s * STAGE_BYTES;
        mbar_arrive_expect_tx(full + s, X_BYTES + R_BYTES);
        tma_load_2d(st, &qmap, (kb0 + it) * EK, p * EM, full + s);
        tma_load_2d(st + 2 * X_BYTES, &rmap, (kb0 + it) * EK, c * EN, full + s);
        issued = it + 1;
      }
      for (int s = 0; s < NSTAGE && s < issued; ++s)
        mbar_wait_drain(full + s, (uint32_t)(((issued - 1 - s) / NSTAGE) & 1));
    }
  } else if (warp == MMA_WARP) {
    if (lane == 0) {
      for (int it = 0; it < nk; ++it) {
        const int s = it % NSTAGE, use = it / NSTAGE;
        if (!mbar_wait(conv + s, (uint32_t)(use & 1), abort_flag, err, 52)) break;
        tc_fence_after();
        const uint32_t xh = smem_u32(base + s * STAGE_BYTES);
        const uint32_t xl = xh + X_BYTES, rh = xh + 2 * X_BYTES, rl = rh + R_BYTES;
#pragma unroll
        for (int kk = 0; kk < EK / 8; ++kk) {
          const uint32_t o = (uint32_t)kk * 32u;
          mma_tf32(tmem, sw64_desc(xh + o), sw64_desc(rh + o), (it | kk) != 0);
          mma_tf32(tmem, sw64_desc(xh + o), sw64_desc(rl + o), 1u);
          mma_tf32(tmem, sw64_desc(xl + o), sw64_desc(rh + o), 1u);
        }
        mma_commit(empty + s);
        if (it == nk - 1) mma_commit(acc_full);
      }
      mma_commit(fin);
      mbar_wait_drain(fin, 0);
    }
  } else if (warp < CONV_WARPS) {
    // thread t splits row t of the Q tile and rows t, t + 128 of the R tile
    const int t = tid;
    auto split_row = [&](unsigned char* hi, unsigned char* lo, int r) {
#pragma unroll
      for (int q = 0; q < EK / 4; ++q) {
        const uint32_t off = (uint32_t)r * 64u + ((uint32_t)(q ^ ((r >> 1) & 3)) << 4);
        const float4 v = *reinterpret_cast<const float4*>(hi + off);
        const float4 h = make_float4(tf32_round(v.x), tf32_round(v.y), tf32_round(v.z), tf32_round(v.w));
        *reinterpret_cast<float4*>(hi + off) = h;
        *reinterpret_cast<float4*>(lo + off) = make_float4(tf32_round(v.x - h.x), tf32_round(v.y - h.y),
                                                           tf32_round(v.z - h.z), tf32_round(v.w - h.w));
      }
    };
    for (int it = 0; it < nk; ++it) {
      const int s = it % NSTAGE, use = it / NSTAGE;
      if (!warp_wait(full + s, (uint32_t)(use & 1), abort_flag, err, 53)) break;
      unsigned char* st = base + s * STAGE_BYTES;
      split_row(st, st + X_BYTES, t);
      split_row(st + 2 * X_BYTES, st + 2 * X_BYTES + R_BYTES, t);
      split_row(st + 2 * X_BYTES, st + 2 * X_BYTES + R_BYTES, t + EM);
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) mbar_arrive(conv + s);
    }
  } else if (warp >= ROT_EPI0) {
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const int64_t q = (int64_t)p * EM + row;
    if (nk > 0 && warp_wait(acc_full, 0, abort_flag, err, 54)) {
      tc_fence_after();
      float* dst = part + ((int64_t)sp * nq + q) * d;
      const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16);
#pragma unroll 1
      for (int g = 0; g < EN / 16; ++g) {
        uint32_t r[16];
        tmem_ld16_issue(tl + (uint32_t)(g * 16), r);
        tmem_wait16(r);
        const int j0 = c * EN + g * 16;
        if (q < nq && j0 < d) {
          float4* o = reinterpret_cast<float4*>(dst + j0);
#pragma unroll
          for (int u = 0; u < 4; ++u)
            o[u] = make_float4(__uint_as_float(r[4 * u]), __uint_as_float(r[4 * u + 1]),
                               __uint_as_float(r[4 * u + 2]), __uint_as_float(r[4 * u + 3]));
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == MMA_WARP) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 256;" ::"r"(tmem));
}

// out = sum of the S partial products in split order; also zeroes the
// search's merge counters, and lets the scan launched after it (as a
// programmatic dependent) start its prologue.
__global__ void __launch_bounds__(256)
k_rotate_reduce(const float4* __restrict__ part, int S, int64_t n4, float4* __restrict__ out, int* counters,
                int64_t n_counters) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t i0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (counters)
    for (int64_t i = i0; i < n_counters; i += stride) counters[i] = 0;
  for (int64_t i = i0; i < n4; i += stride) {
    float4 a = __ldcs(part + i);
    for (int s = 1; s < S; ++s) {
      const float4 b = __ldcs(part + (int64_t)s * n4 + i);
      a.x += b.x;
      a.y += b.y;
      a.z += b.z;
      a.w += b.w;
    }
    out[i] = a;
  }
}

}  // namespace

bool encode_tc_supported(int d) { return d >= 128 && d <= kMaxD && d % EK == 0; }

size_t encode_plan_bytes(int d) { return kPlanHeader + (size_t)2 * d * d * sizeof(float); }

cudaError_t launch_encode_plan(const float* R, int d, void* plan, cudaStream_t s) {
  const size_t total = (size_t)d * d;
  const int grid = (int)std::min<size_t>((total + 255) / 256, (size_t)device_sm_count() * 8);
  k_encode_plan<<<grid, 256, 0, s>>>(R, d, static_cast<unsigned char*>(plan));
  return cudaGetLastError();
}

cudaError_t launch_encode_tc(const float* X, int64_t n, int d, const void* plan, const float* centroids,
                             const float* boundaries, int bits, int scale_mode, const float* cal_mu,
                             const float* cal_a, uint8_t* codes, float* scale, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  if (!encode_tc_supported(d)) return cudaErrorInvalidValue;
  PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
  if (!enc) return cudaErrorNotSupported;
  const unsigned char* pl = static_cast<const unsigned char*>(plan);
  CUtensorMap xmap, rmap;
  const cuuint32_t estride[2] = {1, 1};
  {
    const cuuint64_t gdim[2] = {(cuuint64_t)d, (cuuint64_t)n};
    const cuuint64_t gstride[1] = {(cuuint64_t)d * sizeof(float)};
    const cuuint32_t box[2] = {(cuuint32_t)EK, (cuuint32_t)EM};
    const CUresult r = enc(&xmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(X), gdim, gstride, box,
                           estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  }
  {
    const cuuint64_t gdim[2] = {(cuuint64_t)d, (cuuint64_t)2 * d};
    const cuuint64_t gstride[1] = {(cuuint64_t)d * sizeof(float)};
    const cuuint32_t box[2] = {(cuuint32_t)EK, (cuuint32_t)EN};
    const CUresult r = enc(&rmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<unsigned char*>(pl + kPlanHeader),
                           gdim, gstride, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
  }
  int* err = reinterpret_cast<int*>(const_cast<unsigned char*>(pl));
  const int64_t panels = (n + EM - 1) / EM;
  const int grid = (int)std::min<int64_t>(panels, (int64_t)device_sm_count());
  const bool cal = cal_mu != nullptr;
  cudaError_t e = cudaSuccess;
#define TQ_ENC_TC_CASE(B)                                                                                     \
  case B: {                                                                                                   \
    const void* fn = cal ? reinterpret_cast<const void*>(k_encode_tc<B, true>)                                \
                         : reinterpret_cast<const void*>(k_encode_tc<B, false>);                              \
    if ((e = set_max_dynamic_smem(fn, (int)kEncSmem)) != cudaSuccess) return e;                               \
    if (cal)                                                                                                  \
      k_encode_tc<B, true><<<grid, ENC_THREADS, kEncSmem, s>>>(xmap, rmap, (int)n, d, centroids, boundaries,  \
                                                               scale_mode, cal_mu, cal_a, codes, scale, err); \
    else                                                                                                      \
      k_encode_tc<B, false><<<grid, ENC_THREADS, kEncSmem, s>>>(xmap, rmap, (int)n, d, centroids, boundaries, \
                                                                scale_mode, nullptr, nullptr, codes, scale,   \
                                                                err);                                         \
    break;                                                                                                    \
  }
  switch (bits) {
    TQ_ENC_TC_CASE(2)
    TQ_ENC_TC_CASE(3)
    TQ_ENC_TC_CASE(4)
    TQ_ENC_TC_CASE(8)
    default: return cudaErrorInvalidValue;
  }
#undef TQ_ENC_TC_CASE
  return cudaGetLastError();
}

int rotate_tc_splits(int64_t nq, int d) {
  const int KB = d / EK;
  const int64_t items = ((nq + EM - 1) / EM) * ((d + EN - 1) / EN);
  int64_t sp = (int64_t)device_sm_count() / std::max<int64_t>(items, 1);
  sp = std::min<int64_t>(sp, std::max(1, KB / 8));  // at least 8 K-blocks per split
  return (int)std::max<int64_t>(sp, 1);
}

// (query tiles go on the grid's y dimension: at most 65535 of them)
bool rotate_tc_applies(int64_t nq, int d) {
  return nq >= kRotTcMinBatch && nq <= (int64_t)65535 * EM && encode_tc_supported(d);
}

// One split writes the rotated queries directly: no partial products.
size_t rotate_tc_part_bytes(int64_t nq, int d) {
  if (!rotate_tc_applies(nq, d)) return 0;
  const int S = rotate_tc_splits(nq, d);
  return S > 1 ? (size_t)S * nq * d * sizeof(float) : 0;
}

cudaError_t launch_rotate_tc(const float* Q, int64_t nq, int d, const float* R, float* out, float* part,
                             int* status, int* counters, int64_t n_counters, cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  if (!rotate_tc_applies(nq, d) || nq > INT32_MAX) return cudaErrorInvalidValue;
  PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
  if (!enc) return cudaErrorNotSupported;
  CUtensorMap qmap, rmap;
  const cuuint32_t estride[2] = {1, 1};
  const cuuint64_t gstride[1] = {(cuuint64_t)d * sizeof(float)};
  {
    const cuuint64_t gdim[2] = {(cuuint64_t)d, (cuuint64_t)nq};
    const cuuint32_t box[2] = {(cuuint32_t)EK, (cuuint32_t)EM};
    if (enc(&qmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(Q), gdim, gstride, box, estride,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  {
    const cuuint64_t gdim[2] = {(cuuint64_t)d, (cuuint64_t)d};
    const cuuint32_t box[2] = {(cuuint32_t)EK, (cuuint32_t)EN};
    if (enc(&rmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(R), gdim, gstride, box, estride,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  const int S = rotate_tc_splits(nq, d);
  cudaError_t e = set_max_dynamic_smem(reinterpret_cast<const void*>(k_rotate_tc), (int)kRotSmem);
  if (e != cudaSuccess) return e;
  const dim3 grid((unsigned)((d + EN - 1) / EN), (unsigned)((nq + EM - 1) / EM), (unsigned)S);
  k_rotate_tc<<<grid, ROT_THREADS, kRotSmem, s>>>(qmap, rmap, (int)nq, d, S, S > 1 ? part : out, status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (S == 1)  // the products are the rotated queries; only the merge counters remain
    return counters && n_counters > 0 ? cudaMemsetAsync(counters, 0, (size_t)n_counters * sizeof(int), s)
                                      : cudaSuccess;
  const int64_t n4 = nq * d / 4;
  const int blocks = (int)std::min<int64_t>((n4 + 255) / 256, (int64_t)device_sm_count() * 8);
  k_rotate_reduce<<<std::max(blocks, 1), 256, 0, s>>>(reinterpret_cast<const float4*>(part), S, n4,
                                                       reinterpret_cast<float4*>(out), counters, n_counters);
  return cudaGetLastError();
}

}  // namespace tq
