// dla_noalloc.cu -- dla_forward for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc at the point where they run the
// forward pass: a plugin inside an inference engine that owns every byte of
// device memory and hands out no workspace, or code that runs while another
// thread captures a CUDA graph in global mode, where an allocation is an
// error.  dla_forward_noalloc serves them with a fixed scratch region that is
// part of this library's device image: a file-scope static __device__ array of
// kScratchBytes (64 MiB).  Every GPU that loads the library holds that array
// until the process exits.
//
// Host code cannot use the array's name as a device address (in host code it
// names a host-side stand-in), so the first call on each device, with that
// device current, asks the runtime for the array's device address with
// cudaGetSymbolAddress and remembers it.  That first call should therefore come
// before any stream capture.  Nothing here calls cudaMalloc, cudaFree or any
// allocating routine; the work itself is the unchanged dla_forward, given the
// static array as its workspace.
#include <stdio.h>

#include <mutex>

#include "dla.h"
#include "dla_kernels.h"

namespace {

constexpr size_t kScratchBytes = (size_t)64 << 20;  // the stated maximum scratch
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

std::mutex g_mutex;
void* g_addr[kMaxDevices] = {};

}  // namespace

extern "C" dla_status dla_forward_noalloc(const dla_params* p, dla_dtype in_dtype, int B, int T, int H, int dk,
                                          int dv, const void* q, const void* k, const void* v, const float* lam,
                                          void* o, const dla_cache* cache, uint8_t* boundary, int32_t* merge_log,
                                          void* stream) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return dla::set_error(DLA_ERR_CUDA, "cudaGetDevice failed: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return dla::set_error(DLA_ERR_UNSUPPORTED, "device %d out of range", dev);
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_addr[dev]) {
      void* a = nullptr;
      e = cudaGetSymbolAddress(&a, g_noalloc_scratch);
      if (e != cudaSuccess || !a)
        return dla::set_error(DLA_ERR_CUDA, "cudaGetSymbolAddress of the static scratch failed: %s",
                              cudaGetErrorString(e));
      g_addr[dev] = a;
    }
    scratch = g_addr[dev];
  }
  dla_status s = dla_forward(p, in_dtype, B, T, H, dk, dv, q, k, v, lam, o, cache, boundary, merge_log, scratch,
                             kScratchBytes, stream);
  if (s == DLA_ERR_WORKSPACE) {
    char why[512];
    snprintf(why, sizeof(why), "%s", dla_last_error());
    return dla::set_error(DLA_ERR_WORKSPACE,
                          "this call needs more than the %zu bytes of static scratch of dla_forward_noalloc "
                          "(pass a cache and trace arrays, or use dla_forward with a larger workspace): %s",
                          kScratchBytes, why);
  }
  return s;
}
