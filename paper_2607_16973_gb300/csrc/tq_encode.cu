// Encode (Sec. II-B steps 1-5) and query rotation (Sec. II-B step 2).
//
// The rotation y = R x is an FFMA SGEMM Y = X R^T (X row-major n x d, R
// row-major d x d, both K-contiguous).  Each CTA owns a panel of 128 rows and
// walks every 128-column tile of Y itself, so the per-row reductions the
// scale needs (sum c^2, sum y c) are accumulated in shared memory in a fixed
// order: results are deterministic and no scratch memory is used.  The
// epilogue of every tile divides by the row norm, searches the boundaries,
// and packs the codes straight to HBM (little-endian bit stream per row).
#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>
#include <mutex>

#include "tq_internal.h"
#include "tq_kernels.h"

namespace tq {
namespace {

constexpr int BM = 128, BN = 128, BK = 8, PAD = 4, NT = 256;

struct GemmSmem {
  float A[2][BK][BM + PAD];
  float B[2][BK][BN + PAD];
};

// Loads one BK-slice of an operand tile: 128 rows x 8 k as 256 float4.
__device__ __forceinline__ float4 load_slice(const float* __restrict__ M, int64_t row0,
                                             int64_t rows_valid, int d, int k0) {
  const int t = threadIdx.x;
  const int64_t r = row0 + (t >> 1);
  if (r < rows_valid)
    return __ldg(reinterpret_cast<const float4*>(M + r * d + k0 + (t & 1) * 4));
  return make_float4(0.f, 0.f, 0.f, 0.f);
}

__device__ __forceinline__ void store_slice(float (*S)[BM + PAD], float4 v) {
  const int t = threadIdx.x;
  const int r = t >> 1, kq = (t & 1) * 4;
  S[kq + 0][r] = v.x;
  S[kq + 1][r] = v.y;
  S[kq + 2][r] = v.z;
  S[kq + 3][r] = v.w;
}

// acc = X[row0 .. row0+127, :] . R[col0 .. col0+127, :]^T over K = d.
// Thread (tx = tid % 16, ty = tid / 16) owns rows ty*4 + {0..3} (+64) and
// columns tx*4 + {0..3} (+64): acc[i][j], i < 4 -> first row block.
__device__ __forceinline__ void gemm_tile(const float* __restrict__ X, int64_t row0, int64_t n_rows,
                                          const float* __restrict__ R, int col0, int d,
                                          GemmSmem& sm, float acc[8][8], int k0 = 0, int k1 = -1) {
  if (k1 < 0) k1 = d;  // the contraction covers coordinates [k0, k1)
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
  const int nk = (k1 - k0) / BK;
  float4 pa = load_slice(X, row0, n_rows, d, k0);
  float4 pb = load_slice(R, col0, d, d, k0);
  store_slice(sm.A[0], pa);
  store_slice(sm.B[0], pb);
  __syncthreads();
  for (int kt = 0; kt < nk; ++kt) {
    const int buf = kt & 1;
    if (kt + 1 < nk) {
      pa = load_slice(X, row0, n_rows, d, k0 + (kt + 1) * BK);
      pb = load_slice(R, col0, d, d, k0 + (kt + 1) * BK);
    }
#pragma unroll
    for (int k = 0; k < BK; ++k) {
      const float4 a0 = *reinterpret_cast<const float4*>(&sm.A[buf][k][ty * 4]);
      const float4 a1 = *reinterpret_cast<const float4*>(&sm.A[buf][k][64 + ty * 4]);
      const float4 b0 = *reinterpret_cast<const float4*>(&sm.B[buf][k][tx * 4]);
      const float4 b1 = *reinterpret_cast<const float4*>(&sm.B[buf][k][64 + tx * 4]);
      const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    if (kt + 1 < nk) {
      store_slice(sm.A[buf ^ 1], pa);
      store_slice(sm.B[buf ^ 1], pb);
    }
    __syncthreads();
  }
}

__device__ __forceinline__ int tile_row(int i) { return (i < 4 ? 0 : 64) + (threadIdx.x >> 4) * 4 + (i & 3); }
__device__ __forceinline__ int tile_col(int j) { return (j < 4 ? 0 : 64) + (threadIdx.x & 15) * 4 + (j & 3); }

struct EncodeSmem {
  GemmSmem g;
  uint8_t ctile[BM][BN + 8];  // row stride 136 B keeps 8-byte reads aligned
  float norm[BM], inv[BM], sum_c2[BM], sum_yc[BM];
  float bnd[255], cen[256];
  float cmu[BN], ca[BN], cinv[BN];  // TQ+ shift, scale and 1/scale of the tile's columns
};

// With CAL (a TQ+ calibration, Sec. II-B): the quantiser sees z = (y - mu) /
// a per coordinate, and the per-vector scalar is taken on the reconstruction
// a c + mu.
template <int BITS, bool CAL>
__global__ void __launch_bounds__(NT, 2)
k_encode(const float* __restrict__ X, int64_t n, int d, const float* __restrict__ R,
         const float* __restrict__ centroids, const float* __restrict__ boundaries, int scale_mode,
         const float* __restrict__ cal_mu, const float* __restrict__ cal_a,
         uint8_t* __restrict__ codes, float* __restrict__ scale) {
  constexpr int L = 1 << BITS;
  __shared__ EncodeSmem sm;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int i = tid; i < L; i += NT) sm.cen[i] = centroids[i];
  for (int i = tid; i < L - 1; i += NT) sm.bnd[i] = boundaries[i];
  const int64_t row_bytes = (int64_t)d * BITS / 8;
  const int64_t panels = (n + BM - 1) / BM;
  const int ntiles = (d + BN - 1) / BN;

  for (int64_t p = blockIdx.x; p < panels; p += gridDim.x) {
    const int64_t row0 = p * BM;
    // step 1: row norms (one warp per row, fixed summation order)
    for (int r = warp; r < BM; r += NT / 32) {
      float s = 0.f;
      if (row0 + r < n) {
        const float4* xr = reinterpret_cast<const float4*>(X + (row0 + r) * d);
        for (int j = lane; j < d / 4; j += 32) {
          const float4 v = __ldg(xr + j);
          s = fmaf(v.x, v.x, s);
          s = fmaf(v.y, v.y, s);
          s = fmaf(v.z, v.z, s);
          s = fmaf(v.w, v.w, s);
        }
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      if (lane == 0) {
        const float nr = sqrtf(s);
        sm.norm[r] = nr;
        sm.inv[r] = nr > 0.f ? 1.0f / nr : 0.f;
        sm.sum_c2[r] = 0.f;
        sm.sum_yc[r] = 0.f;
      }
    }
    __syncthreads();
    for (int nt = 0; nt < ntiles; ++nt) {
      const int col0 = nt * BN;
      if constexpr (CAL) {
        for (int c = tid; c < BN; c += NT) {
          const bool in = col0 + c < d;
          sm.cmu[c] = in ? cal_mu[col0 + c] : 0.f;
          sm.ca[c] = in ? cal_a[col0 + c] : 1.f;
          sm.cinv[c] = 1.0f / sm.ca[c];
        }  // read after gemm_tile's barriers
      }
      float acc[8][8];
      gemm_tile(X, row0, n, R, col0, d, sm.g, acc);
      // step 2-3: y = acc / ||x||, code = #{t < y} (of z = (y - mu) / a with TQ+)
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int r = tile_row(i);
        const float inv = sm.inv[r];
        float pc2 = 0.f, pyc = 0.f;
#pragma unroll
        for (int jh = 0; jh < 2; ++jh) {
          uint32_t packed4 = 0;
#pragma unroll
          for (int jj = 0; jj < 4; ++jj) {
            const int j = jh * 4 + jj;
            const float y = acc[i][j] * inv;
            const float zq = CAL ? (y - sm.cmu[tile_col(j)]) * sm.cinv[tile_col(j)] : y;
            int code = 0;
#pragma unroll
            for (int step = L / 2; step >= 1; step >>= 1)
              if (zq > sm.bnd[code + step - 1]) code += step;
            const float c = CAL ? fmaf(sm.ca[tile_col(j)], sm.cen[code], sm.cmu[tile_col(j)]) : sm.cen[code];
            if (col0 + tile_col(j) < d) {
              pc2 = fmaf(c, c, pc2);
              pyc = fmaf(y, c, pyc);
            }
            packed4 |= (uint32_t)code << (8 * jj);
          }
          *reinterpret_cast<uint32_t*>(&sm.ctile[r][tile_col(jh * 4)]) = packed4;
        }
#pragma unroll
        for (int o = 1; o < 16; o <<= 1) {
          pc2 += __shfl_xor_sync(0xffffffffu, pc2, o);
          pyc += __shfl_xor_sync(0xffffffffu, pyc, o);
        }
        if ((tid & 15) == 0) {
          sm.sum_c2[r] += pc2;
          sm.sum_yc[r] += pyc;
        }
      }
      __syncthreads();
      // step 4: pack 8 codes per item straight to HBM
      for (int item = tid; item < BM * (BN / 8); item += NT) {
        const int r = item / (BN / 8), g = item % (BN / 8);
        const int64_t row = row0 + r;
        const int dim0 = col0 + g * 8;
        if (row >= n || dim0 >= d) continue;
        const uint2 cc = *reinterpret_cast<const uint2*>(&sm.ctile[r][g * 8]);
        const uint64_t c8 = (uint64_t)cc.x | ((uint64_t)cc.y << 32);
        uint64_t bitsv = 0;
#pragma unroll
        for (int t = 0; t < 8; ++t) bitsv |= ((c8 >> (8 * t)) & (uint64_t)(L - 1)) << (BITS * t);
        uint8_t* dst = codes + row * row_bytes + (int64_t)dim0 * BITS / 8;
        if constexpr (BITS == 8) {
          *reinterpret_cast<uint64_t*>(dst) = bitsv;
        } else if constexpr (BITS == 4) {
          *reinterpret_cast<uint32_t*>(dst) = (uint32_t)bitsv;
        } else if constexpr (BITS == 2) {
          *reinterpret_cast<uint16_t*>(dst) = (uint16_t)bitsv;
        } else {
          dst[0] = (uint8_t)bitsv;
          dst[1] = (uint8_t)(bitsv >> 8);
          dst[2] = (uint8_t)(bitsv >> 16);
        }
      }
      __syncthreads();
    }
    // step 5: per-vector scalar
    for (int r = tid; r < BM; r += NT) {
      const int64_t row = row0 + r;
      if (row >= n) continue;
      const float nr = sm.norm[r];
      float s = 0.f;
      if (nr > 0.f) {
        if (scale_mode == TQ_SCALE_NONE) {
          s = nr;
        } else if (scale_mode == TQ_SCALE_NORM) {
          const float cn = sqrtf(sm.sum_c2[r]);
          s = cn > 0.f ? nr / cn : 0.f;
        } else {
          const float yc = sm.sum_yc[r];
          s = yc != 0.f ? nr / yc : 0.f;
        }
      }
      scale[row] = s;
    }
    __syncthreads();
  }
}

// Every search starts with the query rotation, which clears the search's
// status word and merge counters, and lets the kernel after it (launched as a
// programmatic dependent) start its prologue while the rotation runs.
__device__ __forceinline__ void search_start(int* status, int* counters, int64_t n_counters) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int64_t nb = (int64_t)gridDim.x * gridDim.y * gridDim.z;
  const int64_t b = blockIdx.x + (int64_t)gridDim.x * (blockIdx.y + (int64_t)gridDim.y * blockIdx.z);
  if (status && b == 0 && threadIdx.x == 0) *status = 0;
  if (counters)
    for (int64_t i = b * blockDim.x + threadIdx.x; i < n_counters; i += nb * blockDim.x) counters[i] = 0;
}

// Q' = Q R^T, plain store epilogue (nq > 256).
__global__ void __launch_bounds__(NT, 2)
k_rotate_gemm(const float* __restrict__ Q, int64_t nq, int d, const float* __restrict__ R,
              float* __restrict__ out, int* __restrict__ status, int* __restrict__ counters, int64_t n_counters) {
  __shared__ GemmSmem sm;
  search_start(status, counters, n_counters);
  const int64_t row0 = (int64_t)blockIdx.x * BM;
  const int col0 = blockIdx.y * BN;
  // gridDim.z = 2 splits the contraction in halves, each added onto the
  // zeroed output: two fp32 additions onto 0 give the same sum in either
  // order, so the result does not depend on which half lands first
  const int half = d / 2;
  float acc[8][8];
  if (gridDim.z == 2)
    gemm_tile(Q, row0, nq, R, col0, d, sm, acc, blockIdx.z * half, (blockIdx.z + 1) * half);
  else
    gemm_tile(Q, row0, nq, R, col0, d, sm, acc);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t r = row0 + tile_row(i);
    if (r >= nq) continue;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int c = col0 + tile_col(j);
      if (c >= d) continue;
      if (gridDim.z == 2) atomicAdd(out + r * d + c, acc[i][j]);
      else out[r * d + c] = acc[i][j];
    }
  }
}

// Q' = Q R^T for groups of NQ <= 8 queries: one warp per output coordinate,
// R read once per group.
template <int NQ>
__global__ void __launch_bounds__(256)
k_rotate_gemv(const float* __restrict__ Q, int64_t nq, int d, const float* __restrict__ R, float* __restrict__ out,
              int* __restrict__ status, int* __restrict__ counters, int64_t n_counters) {
  search_start(status, counters, n_counters);
  const int lane = threadIdx.x & 31;
  const int i = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (i >= d) return;
  // block row y handles queries NQ*y .. NQ*y + NQ - 1 (the last group may be short)
  const int64_t q0 = (int64_t)blockIdx.y * NQ;
  const int nqg = (int)min((int64_t)NQ, nq - q0);
  Q += q0 * d;
  out += q0 * d;
  float acc[NQ];
#pragma unroll
  for (int q = 0; q < NQ; ++q) acc[q] = 0.f;
  const float4* r4 = reinterpret_cast<const float4*>(R + (int64_t)i * d);
  const int d4 = d / 4;
  // R (d*d*4 bytes) is usually evicted from L2 by the corpus stream between
  // searches, so a lane issues all its row loads (16 for d = 2048) before
  // using any of them
  constexpr int RL = 16;
  for (int j0 = lane; j0 < d4; j0 += 32 * RL) {
    float4 rv[RL];
#pragma unroll
    for (int t = 0; t < RL; ++t) {
      const int j = j0 + 32 * t;
      rv[t] = j < d4 ? __ldg(r4 + j) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int t = 0; t < RL; ++t) {
      const int j = j0 + 32 * t;
      if (j >= d4) break;
#pragma unroll
      for (int q = 0; q < NQ; ++q) {
        if (q >= nqg) break;
        const float4 qv = __ldg(reinterpret_cast<const float4*>(Q + (int64_t)q * d) + j);
        acc[q] = fmaf(rv[t].x, qv.x, acc[q]);
        acc[q] = fmaf(rv[t].y, qv.y, acc[q]);
        acc[q] = fmaf(rv[t].z, qv.z, acc[q]);
        acc[q] = fmaf(rv[t].w, qv.w, acc[q]);
      }
    }
  }
#pragma unroll
  for (int q = 0; q < NQ; ++q) {
    float s = acc[q];
#pragma unroll
    for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0 && q < nqg) out[(int64_t)q * d + i] = s;
  }
}

// TQ+ calibration (Sec. II-B), pass 1: for each 128-row panel, the sums of y
// and y^2 (y = R x / ||x||) of every coordinate over the panel's non-zero
// rows, and their count.  Each CTA walks whole panels and sums in a fixed
// order, so the result does not depend on scheduling.  The sums are kept in
// double: y^2 of a float32 y is exact there, so a coordinate that takes one
// value over the batch comes out with a variance of exactly 0.
__global__ void __launch_bounds__(NT, 2)
k_calib_partial(const float* __restrict__ X, int64_t n, int d, const float* __restrict__ R,
                double* __restrict__ psum, double* __restrict__ psq, int* __restrict__ pcount) {
  __shared__ GemmSmem g;
  __shared__ float inv[BM];
  __shared__ int nz;
  __shared__ double red1[8][BN], red2[8][BN];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t panels = (n + BM - 1) / BM;
  const int ntiles = (d + BN - 1) / BN;
  for (int64_t p = blockIdx.x; p < panels; p += gridDim.x) {
    const int64_t row0 = p * BM;
    if (tid == 0) nz = 0;
    __syncthreads();
    for (int r = warp; r < BM; r += NT / 32) {
      float sq = 0.f;
      if (row0 + r < n) {
        const float4* xr = reinterpret_cast<const float4*>(X + (row0 + r) * d);
        for (int j = lane; j < d / 4; j += 32) {
          const float4 v = __ldg(xr + j);
          sq = fmaf(v.x, v.x, sq);
          sq = fmaf(v.y, v.y, sq);
          sq = fmaf(v.z, v.z, sq);
          sq = fmaf(v.w, v.w, sq);
        }
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
      if (lane == 0) {
        const float nr = sqrtf(sq);
        inv[r] = nr > 0.f ? 1.0f / nr : 0.f;
        if (nr > 0.f) atomicAdd(&nz, 1);
      }
    }
    __syncthreads();
    if (tid == 0) pcount[p] = nz;
    for (int nt = 0; nt < ntiles; ++nt) {
      const int col0 = nt * BN;
      float acc[8][8];
      gemm_tile(X, row0, n, R, col0, d, g, acc);
      double s1[8], s2[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        s1[j] = 0.0;
        s2[j] = 0.0;
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float iv = inv[tile_row(i)];  // 0 for a zero row or a row past n: adds nothing
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const double y = (double)(acc[i][j] * iv);
          s1[j] += y;
          s2[j] = fma(y, y, s2[j]);
        }
      }
      // rows ty (even) and ty + 1 (lanes 0-15 and 16-31 of one warp) first
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        s1[j] += __shfl_xor_sync(0xffffffffu, s1[j], 16);
        s2[j] += __shfl_xor_sync(0xffffffffu, s2[j], 16);
      }
      if ((lane & 16) == 0) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          red1[warp][tile_col(j)] = s1[j];
          red2[warp][tile_col(j)] = s2[j];
        }
      }
      __syncthreads();
      for (int c = tid; c < BN; c += NT) {
        if (col0 + c >= d) continue;
        double a = 0.0, b = 0.0;
        for (int t = 0; t < 8; ++t) {
          a += red1[t][c];
          b += red2[t][c];
        }
        psum[p * d + col0 + c] = a;
        psq[p * d + col0 + c] = b;
      }
      __syncthreads();
    }
  }
}

// Pass 2: per coordinate, the panels' sums added in panel order (in double):
// mu = mean, sigma = population standard deviation, a = sigma sqrt(d) (a = 1
// where sigma = 0; mu = 0, a = 1 without a non-zero row).
__global__ void k_calib_finish(const double* __restrict__ psum, const double* __restrict__ psq,
                               const int* __restrict__ pcount, int64_t panels, int d, float* __restrict__ mu,
                               float* __restrict__ a) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= d) return;
  double s1 = 0.0, s2 = 0.0;
  int64_t cnt = 0;
  for (int64_t p = 0; p < panels; ++p) {
    s1 += psum[p * d + j];
    s2 += psq[p * d + j];
    cnt += pcount[p];
  }
  if (cnt == 0) {
    mu[j] = 0.f;
    a[j] = 1.f;
    return;
  }
  const double m = s1 / (double)cnt;
  const double var = fmax(s2 / (double)cnt - m * m, 0.0);
  const double sg = sqrt(var);
  mu[j] = (float)m;
  a[j] = sg > 0.0 ? (float)(sg * sqrt((double)d)) : 1.f;
}

// A search over a TQ+ index: q''_j = a_j q'_j (in place) and the query's bias
// b = sum_j q'_j mu_j, so that scale * (q'' . c[code] + b) = scale * q' .
// (a c[code] + mu).  One block per query, fixed summation order.
__global__ void __launch_bounds__(256)
k_calib_query(float* __restrict__ qrot, int64_t nq, int d, const float* __restrict__ mu,
              const float* __restrict__ a, float* __restrict__ bias) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  __shared__ float red[8];
  const int64_t q = blockIdx.x;
  float* qq = qrot + q * d;
  float b = 0.f;
  for (int j = threadIdx.x; j < d; j += blockDim.x) {
    const float v = qq[j];
    b = fmaf(v, mu[j], b);
    qq[j] = v * a[j];
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) b += __shfl_xor_sync(0xffffffffu, b, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = b;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
    bias[q] = t;
  }
}

}  // namespace

// SM count of the current device, queried once per device.
int device_sm_count() {
  constexpr int kMaxDev = 64;
  static std::atomic<int> cache[kMaxDev];
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (dev >= 0 && dev < kMaxDev && (sms = cache[dev].load(std::memory_order_relaxed)) > 0) return sms;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1) return 1;
  if (dev >= 0 && dev < kMaxDev) cache[dev].store(sms, std::memory_order_relaxed);
  return sms;
}

// cudaFuncSetAttribute(MaxDynamicSharedMemorySize) once per kernel, device
// and size: the call is not free, and the searches launch on every request.
cudaError_t set_max_dynamic_smem(const void* func, int bytes) {
  struct Entry {
    const void* func;
    int dev, bytes;
  };
  static std::mutex mu;
  static Entry seen[256];
  static int nseen = 0;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  {
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < nseen; ++i)
      if (seen[i].func == func && seen[i].dev == dev && seen[i].bytes >= bytes) return cudaSuccess;
  }
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < nseen; ++i)
    if (seen[i].func == func && seen[i].dev == dev) {
      if (bytes > seen[i].bytes) seen[i].bytes = bytes;
      return cudaSuccess;
    }
  if (nseen < 256) seen[nseen++] = Entry{func, dev, bytes};
  return cudaSuccess;
}

cudaError_t launch_encode(const float* X, int64_t n, int d, const float* R, const float* centroids,
                          const float* boundaries, int bits, int scale_mode, const float* cal_mu,
                          const float* cal_a, uint8_t* codes, float* scale, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  const int64_t panels = (n + BM - 1) / BM;
  const int grid = (int)std::min<int64_t>(panels, (int64_t)device_sm_count() * 2);
  const bool cal = cal_mu != nullptr;
#define TQ_ENC_CASE(B)                                                                                       \
  case B:                                                                                                    \
    if (cal)                                                                                                 \
      k_encode<B, true><<<grid, NT, 0, s>>>(X, n, d, R, centroids, boundaries, scale_mode, cal_mu, cal_a,   \
                                            codes, scale);                                                   \
    else                                                                                                     \
      k_encode<B, false><<<grid, NT, 0, s>>>(X, n, d, R, centroids, boundaries, scale_mode, nullptr, nullptr, \
                                             codes, scale);                                                  \
    break;
  switch (bits) {
    TQ_ENC_CASE(2)
    TQ_ENC_CASE(3)
    TQ_ENC_CASE(4)
    TQ_ENC_CASE(8)
    default: return cudaErrorInvalidValue;
  }
#undef TQ_ENC_CASE
  return cudaGetLastError();
}

cudaError_t launch_rotate(const float* Q, int64_t nq, int d, const float* R, float* out, int* status,
                          int* counters, int64_t n_counters, cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  if (nq <= 8) {
    const dim3 grid((unsigned)((d + 7) / 8), 1);
    switch (nq) {
#define TQ_GEMV_CASE(N) \
  case N: k_rotate_gemv<N><<<grid, 256, 0, s>>>(Q, nq, d, R, out, status, counters, n_counters); break;
      TQ_GEMV_CASE(1) TQ_GEMV_CASE(2) TQ_GEMV_CASE(3) TQ_GEMV_CASE(4)
      TQ_GEMV_CASE(5) TQ_GEMV_CASE(6) TQ_GEMV_CASE(7) TQ_GEMV_CASE(8)
#undef TQ_GEMV_CASE
    }
    return cudaGetLastError();
  }
  if (nq <= 256) {  // groups of 8 queries: R stays in L2 across the groups; the GEMM would use few CTAs
    const dim3 grid((unsigned)((d + 7) / 8), (unsigned)((nq + 7) / 8));
    k_rotate_gemv<8><<<grid, 256, 0, s>>>(Q, nq, d, R, out, status, counters, n_counters);
    return cudaGetLastError();
  }
  // split the contraction in two when the tiles alone would leave SMs idle
  // (each half must be a whole number of BK slices)
  const int64_t tiles = ((nq + BM - 1) / BM) * ((d + BN - 1) / BN);
  const bool split = tiles < device_sm_count() && (d / 2) % BK == 0;
  if (split) {
    const cudaError_t e = cudaMemsetAsync(out, 0, (size_t)nq * d * sizeof(float), s);
    if (e != cudaSuccess) return e;
  }
  dim3 grid((unsigned)((nq + BM - 1) / BM), (unsigned)((d + BN - 1) / BN), split ? 2u : 1u);
  k_rotate_gemm<<<grid, NT, 0, s>>>(Q, nq, d, R, out, status, counters, n_counters);
  return cudaGetLastError();
}

}  // namespace tq

namespace tq {

size_t calibrate_workspace(int64_t n, int d) {
  const int64_t panels = (n + BM - 1) / BM;
  return (size_t)panels * d * 2 * sizeof(double) + (size_t)panels * sizeof(int);
}

cudaError_t launch_calibrate(const float* X, int64_t n, int d, const float* R, float* mu, float* a, void* ws,
                             cudaStream_t s) {
  const int64_t panels = (n + BM - 1) / BM;
  double* psum = static_cast<double*>(ws);
  double* psq = psum + (size_t)panels * d;
  int* pcount = reinterpret_cast<int*>(psq + (size_t)panels * d);
  const int grid = (int)std::min<int64_t>(panels, (int64_t)device_sm_count() * 2);
  k_calib_partial<<<grid, NT, 0, s>>>(X, n, d, R, psum, psq, pcount);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_calib_finish<<<(d + 255) / 256, 256, 0, s>>>(psum, psq, pcount, panels, d, mu, a);
  return cudaGetLastError();
}

cudaError_t launch_calib_query(float* qrot, int64_t nq, int d, const float* mu, const float* a, float* bias,
                               cudaStream_t s) {
  if (nq == 0) return cudaSuccess;
  k_calib_query<<<(unsigned)nq, 256, 0, s>>>(qrot, nq, d, mu, a, bias);
  return cudaGetLastError();
}

}  // namespace tq
