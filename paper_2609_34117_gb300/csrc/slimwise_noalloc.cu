// slimwise_noalloc.cu -- decode MoE layer for callers that cannot allocate
// device memory.
//
// Some hosts of this library must not call cudaMalloc or any allocating
// routine during inference: a serving engine that sized and carved out all
// of its device memory up front, code that runs under a memory pool or
// allocator it does not control, or a plugin given only its inputs and
// outputs.  slimwise_moe_decode_noalloc serves them by running the same four
// kernels as slimwise_moe_decode with the scratch memory (routing state,
// grouped activations, expert outputs, counters) placed in a fixed device
// array that belongs to this library.
//
// The array is a file-scope __device__ variable of kNoAllocScratchBytes; every
// GPU that loads this library holds it until the process exits.  In host code
// its name is only a host-side stand-in, so its device address is looked up
// with cudaGetSymbolAddress, once per device, on the first call made with that
// device current.  That first call should therefore come before any stream
// capture.  All calls share the array, and it keeps what the last call left
// there: the kernels set every counter and flag they read at the start of
// each call, so nothing has to be cleared in between, but two calls whose
// kernels overlap on the GPU (different streams without ordering) race on it.
//
// The kernels record device-side errors (a repeated or out-of-range retained
// id, a bounded wait that gave up) in the error word at the head of the array;
// slimwise_moe_noalloc_device_status reads it, as slimwise_moe_device_status
// does for a caller's workspace.
//
// A launch that fails drops the cached address of the current device, so the
// next call looks it up again: after cudaDeviceReset, or once the primary
// context was destroyed and created anew, the array may sit at another
// device address.
#include <mutex>

#include "common.cuh"

namespace {

// Scratch limit: enough for the Qwen-class layer (H = 2048, E = 128,
// I = 768, top-8) at decode batches up to 151 tokens.
constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mu;
void *g_noalloc_ptr[64] = {};

}  // namespace

extern "C" int slimwise_moe_decode_noalloc(const void *hidden, const float *router_w,
                                           const int32_t *retained_idx, int32_t n_retained,
                                           const void *w_gate_up, const void *w_down,
                                           int32_t top_k, void *out, void *stream,
                                           const slimwise_moe_shape *shape) {
  if (!shape) return SLIMWISE_ERR_INVALID_ARG;
  size_t need = 0;
  int rc = slimwise_moe_workspace_size(shape, top_k, &need);
  if (rc != SLIMWISE_OK) return rc;
  // the problem's scratch must fit in the fixed array
  if (need > kNoAllocScratchBytes) return SLIMWISE_ERR_WORKSPACE;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return SLIMWISE_ERR_CUDA;
  void *scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
      void *p = nullptr;
      if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p)
        return SLIMWISE_ERR_CUDA;
      g_noalloc_ptr[dev] = p;
    }
    scratch = g_noalloc_ptr[dev];
  }
  rc = slimwise_moe_decode_ex(hidden, router_w, retained_idx, n_retained, w_gate_up, w_down,
                              top_k, out, stream, shape, scratch, kNoAllocScratchBytes, nullptr);
  if (rc == SLIMWISE_ERR_CUDA) {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    g_noalloc_ptr[dev] = nullptr;
  }
  return rc;
}

extern "C" int slimwise_moe_noalloc_device_status(void *stream, int32_t *flags) {
  if (!flags) return SLIMWISE_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int32_t v = 0;
  // the control words are the first region of the scratch layout
  if (cudaMemcpyFromSymbolAsync(&v, g_noalloc_scratch, sizeof(v),
                                slimwise::kCtrlErr * sizeof(int32_t), cudaMemcpyDeviceToHost,
                                st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return SLIMWISE_ERR_CUDA;
  *flags = v;
  return v ? SLIMWISE_ERR_DEVICE : SLIMWISE_OK;
}
