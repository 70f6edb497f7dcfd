// Internal declarations shared by the library's translation units.
#pragma once

#include <cstdarg>
#include <cstddef>
#include <cstdint>

#include "../../include/tq.h"

namespace tq {

// Records a thread-local error message and returns `st`.
tq_status fail(tq_status st, const char* fmt, ...);
// Clears the thread-local message and returns TQ_OK.
tq_status ok();

// Thread-local settings (tq_set_search_path / tq_profile_events).
int search_path();
void* profile_start();
void* profile_stop();

constexpr int kMaxK = 256;
constexpr int kMaxKMma = 64;     // per-thread top-k lists of the tensor-core scan
constexpr int kMmaMinBatch = 16; // AUTO uses the tensor-core scan from this batch size
constexpr int kMaxD = 8192;
constexpr int kRotTcMinBatch = 16;  // query batches rotated on the tensor cores from this size
// The fixed-point 4-bit centroid table (TQ_PATH_LUT_FIXED) applies from this
// d on: its rounding error is about 2^-16 of the largest centroid (~3.5 /
// sqrt(d)), so below it the exact fp32 table keeps unit-query scores within
// 1e-5.
constexpr int kFixMinD = 512;
// The query-folded 4-bit lookup scan (k_scan_fold, TQ_PATH_LUT_FOLD): largest k.
constexpr int kFoldMaxK = 32;
constexpr long long kWaitCyclesMax = 4000000000LL;  // the kernels' wait budget (~2 s at 2 GHz)

// Thread-local count of device allocations still to fail (tq_debug_fail_allocs).
int& fail_allocs();

inline bool valid_bits(int b) { return b == 2 || b == 3 || b == 4 || b == 8; }
inline int64_t row_bytes(int d, int bits) { return (int64_t)d * bits / 8; }
inline bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

}  // namespace tq
