// hilo_block_forward_static_ws: hilo_block_forward for callers that cannot
// allocate device memory when they call the block.
//
// Some callers have no way to hand the library a workspace: code that runs
// inside a host framework whose device allocator is not reachable from the
// call site, or a service that fixes its device-memory footprint at start-up
// and forbids any allocation afterwards. This entry point needs no workspace
// argument: its scratch is a fixed array in the library's own device memory,
// HILO_STATIC_SCRATCH_BYTES long, which every GPU that loads the library holds
// until the process exits. It allocates nothing itself, and calls no
// allocating routine.
#include <cuda_runtime.h>
#include <stdio.h>

#include "../../include/hilo.h"
#include "internal.h"

namespace {

// The shared scratch (one copy per device context).
static __device__ __align__(256) unsigned char g_static_scratch[HILO_STATIC_SCRATCH_BYTES];

}  // namespace

extern "C" int hilo_block_forward_static_ws(const hilo_shape* shape,
                                            const hilo_block_weights* weights,
                                            const int32_t* cu_img, int32_t cap,
                                            const void* in_txt, const void* in_img,
                                            int in_dtype, float* out, void* stream) {
  if (!shape) return hilo::set_error(HILO_ERR_ARG, "hilo_block_forward_static_ws: shape is NULL");
  // the shape first: the scratch size of an invalid shape means nothing
  int st = hilo::check_block_shape(shape);
  if (st) return st;
  if (cap < 0) return hilo::set_error(HILO_ERR_ARG, "hilo_block_forward_static_ws: cap < 0");
  const size_t need = hilo_block_workspace_bytes(shape, cap);
  if (need > HILO_STATIC_SCRATCH_BYTES) {
    char msg[200];
    snprintf(msg, sizeof(msg),
             "hilo_block_forward_static_ws: this shape needs %zu scratch bytes, more than the "
             "built-in %zu; use hilo_block_forward with a caller workspace",
             need, static_cast<size_t>(HILO_STATIC_SCRATCH_BYTES));
    return hilo::set_error(HILO_ERR_WORKSPACE, msg);
  }
  // The host-side name g_static_scratch is not a device address: ask the
  // runtime for the array's address in the current device's context, on
  // every call, so that nothing cached can outlive that context (a device
  // reset, another context on the same device). The first call on a device
  // also loads the module; make it before any stream capture.
  void* scratch = nullptr;
  if (cudaGetSymbolAddress(&scratch, g_static_scratch) != cudaSuccess || !scratch)
    return hilo::set_error(HILO_ERR_CUDA,
                           "hilo_block_forward_static_ws: cudaGetSymbolAddress of the scratch failed");
  // Nothing in the scratch needs to start at zero: every scratch value the
  // block's kernels read was written earlier in the same call.
  return hilo_block_forward(shape, weights, cu_img, cap, in_txt, in_img, in_dtype, out,
                            scratch, HILO_STATIC_SCRATCH_BYTES, stream);
}
