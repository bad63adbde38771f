// tadm_head_confidence_static: the fused output head + confidence for callers
// that cannot allocate device memory.  Such callers include code running
// inside a host framework that owns every device allocation and only hands
// out its input and output buffers, and latency-critical paths that forbid
// cudaMalloc because it can synchronise the whole device.  The per-row,
// per-column-tile partials that tadm_head_confidence keeps in caller scratch
// live here in a fixed array that is part of the library image.
#include <mutex>

#include "../../include/tadm.h"
#include "kernels.h"

namespace {

constexpr size_t kPartialBytes = TADM_HEAD_STATIC_SCRATCH_BYTES;

// The partials of one call.  Every GPU that loads the library holds this
// array (8 MiB) until the process exits.  In host code the name is only a
// host-side stand-in, never a device address: the device address comes from
// cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_head_partials[kPartialBytes];

constexpr int kMaxDevices = 256;
std::mutex g_mu;
void* g_addr[kMaxDevices] = {};

// Device address of g_head_partials on the current device, looked up once
// per device (with that device current) and remembered.  Like the rest of
// the library (whose GEMM launch attributes are also set once per process),
// this assumes one device per process and a context that lives as long as
// the process: after cudaDeviceReset the remembered address is stale, so the
// library must not be called again in that process.
tadm_status partials_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return TADM_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_head_partials) != cudaSuccess || !p) return TADM_ERR_CUDA;
    g_addr[dev] = p;
  }
  *out = g_addr[dev];
  return TADM_OK;
}

}  // namespace

extern "C" tadm_status tadm_head_confidence_static(const void* x, const void* w, int rows, int d, int vocab,
                                                   int mask_id, int dtype, float* conf, int32_t* tok,
                                                   tadm_stream stream) {
  size_t need = 0;
  if (tadm_head_scratch_size(rows, vocab, dtype, &need) != TADM_OK) return TADM_ERR_INVALID_ARG;
  // the argument checks of tadm_head_confidence, before the early return for rows == 0
  if (!x || !w || !conf || !tok || d <= 0 || mask_id < 0 || mask_id >= vocab) return TADM_ERR_INVALID_ARG;
  if (need > kPartialBytes) return TADM_ERR_INVALID_ARG;  // beyond the fixed array: use tadm_head_confidence
  if (rows == 0) return TADM_OK;
  void* scratch = nullptr;
  const tadm_status st = partials_address(&scratch);
  if (st != TADM_OK) return st;
  // Nothing in the array needs clearing: the GEMM epilogue writes every
  // partial that the merge kernel of the same call reads.
  return tadm_head_confidence(x, w, rows, d, vocab, mask_id, dtype, scratch, kPartialBytes, conf, tok, stream);
}
