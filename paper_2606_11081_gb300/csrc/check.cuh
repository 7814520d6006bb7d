// check.cuh -- index checks of the checked build.
//
// Compiled with -DGASLOC_CHECKED (build.build(checked=True) makes
// libgasloc_checked.so), the kernels test every global-memory row/column and
// every shared-memory slot they address against the extent of its buffer
// before the access.  A failed test records kDevBadIndex in the context's
// device error word -- the next synchronising call then returns
// GASLOC_EDEVICE -- and the access is skipped (a load yields zero).  Nothing
// traps and nothing waits.  In the normal build every test is the constant
// true and compiles to nothing.
#pragma once
#include <cstdint>

#include "internal.h"

namespace gasloc {

#ifdef GASLOC_CHECKED
constexpr bool kChecked = true;
#else
constexpr bool kChecked = false;
#endif

__device__ __forceinline__ bool report_bad(int32_t *err) {
    if (err) atomicCAS(err, static_cast<int32_t>(kDevOk), static_cast<int32_t>(kDevBadIndex));
    return false;
}

// [col, col + width) of row `row` inside `rows` rows of `stride` elements.
__device__ __forceinline__ bool row_ok(int64_t row, int64_t rows, int64_t col, int64_t width, int64_t stride,
                                       int32_t *err) {
    if (!kChecked) return true;
    const bool ok = row >= 0 && row < rows && col >= 0 && width >= 0 && col + width <= stride;
    return ok ? true : report_bad(err);
}

// [begin, end) inside [0, limit).
__device__ __forceinline__ bool span_ok(int64_t begin, int64_t end, int64_t limit, int32_t *err) {
    if (!kChecked) return true;
    const bool ok = begin >= 0 && begin <= end && end <= limit;
    return ok ? true : report_bad(err);
}

// A byte count or offset that is a multiple of 16 (TMA and bulk copies).
__device__ __forceinline__ bool aligned16_ok(int64_t bytes, int32_t *err) {
    if (!kChecked) return true;
    return bytes % 16 == 0 ? true : report_bad(err);
}

}  // namespace gasloc
