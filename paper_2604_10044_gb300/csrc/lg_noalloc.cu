// lg_decode_attend_noalloc: lg_decode_attend without a caller-provided workspace.
//
// Some callers cannot allocate device memory at all: a plugin running inside a host framework
// that owns every device allocation, or a latency-critical serving loop where cudaMalloc's
// implicit synchronisation is not acceptable.  This entry point serves them: its scratch
// (the split-K partials, and the logits of the H2O accumulation) lives in one statically sized
// device array of this library, so the call itself allocates nothing.  The caller still
// passes every input and output.
#include <cuda_runtime.h>
#include <mutex>

#include "lg.h"

namespace {

// The scratch of every call on a device.  Every GPU that loads the library holds
// LG_NOALLOC_SCRATCH_BYTES of device memory for this array until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[LG_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
void *g_scratch_ptr[kMaxDevices] = {};

// Device address of the array for the current device, looked up once per device.  In host code
// the array's name is only a stand-in for the symbol, never a usable device address.
lg_status scratch_for_current_device(void **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return LG_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mutex);
  if (!g_scratch_ptr[dev]) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return LG_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return LG_OK;
}

}  // namespace

extern "C" lg_status lg_decode_attend_noalloc(const lg_cache *c, int layer0, int n_layers,
                                              const void *q, int H_q, float scale, void *out,
                                              float *stats, int suffix_w, int accumulate_h2o,
                                              int max_len, cudaStream_t s) {
  const size_t need = lg_workspace_size(c, H_q, n_layers, max_len, accumulate_h2o);
  if (need == 0) return LG_ERR_INVALID_ARG;
  if (need > (size_t)LG_NOALLOC_SCRATCH_BYTES) return LG_ERR_WORKSPACE;
  void *ws = nullptr;
  lg_status st = scratch_for_current_device(&ws);
  if (st != LG_OK) return st;
  // every byte of scratch the kernels read is written earlier in the same call (but the
  // pass-direction word, whose value never changes a result), so the contents left by a
  // previous call need no clearing
  return lg_decode_attend(c, layer0, n_layers, q, H_q, scale, out, stats, suffix_w,
                          accumulate_h2o, max_len, ws, (size_t)LG_NOALLOC_SCRATCH_BYTES, s);
}
