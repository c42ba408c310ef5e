// checked.cuh -- index checks of the checked build.
//
// compute-sanitizer is not available to this library's tests, so the
// hand-written kernels guard their shared-memory offsets, tensor-memory
// columns and global indices with SOMA_CHECK(cond, status).  In the default
// build the macro is the constant `true` (the condition is referenced, never
// evaluated) and costs nothing.  Built with
// -DSOMA_CHECKED (libsoma_checked.so), a failing check records
// SOMA_ERR_BOUNDS in the status word and the source line of the first
// failure in the word after it (the status pointer of every kernel points
// at a pair of words), and the guarded access is skipped: no trap, no
// fault, and the context stays usable.
#pragma once

#include "soma_device.cuh"

namespace soma {

constexpr int kStatusBounds = 7;  // mirrors SOMA_ERR_BOUNDS

}  // namespace soma

#ifdef SOMA_CHECKED
namespace soma {
__device__ __forceinline__ bool check_ok(bool ok, int* status, int line) {
  if (!ok) {
    atomicCAS(status, 0, kStatusBounds);
    atomicCAS(status + 1, 0, line);
  }
  return ok;
}
}  // namespace soma

#ifndef SOMA_CHECK_FILE
#define SOMA_CHECK_FILE 0
#endif
// the recorded position: 10000 * file id (SOMA_CHECK_FILE) + source line
#define SOMA_CHECK(cond, status) \
  (::soma::check_ok((cond), (status), 10000 * SOMA_CHECK_FILE + __LINE__))
#else
// the condition is not evaluated (sizeof), only referenced
#define SOMA_CHECK(cond, status) (static_cast<void>(sizeof(cond)), true)
#endif
