// Top-k worker compression that allocates no device memory.
//
// Some callers cannot allocate device memory at all: code embedded in a host
// framework that owns every device allocation under a fixed memory plan, or
// a hot path that must never risk an allocation failure or an allocator
// synchronisation.  dqgan_create allocates (residuals, scratch), so such
// callers cannot use a handle.  This entry point runs the same top-k kernels
// as dqgan_worker_compress with DQGAN_TOPK, on a residual the caller owns,
// and takes its scratch from a fixed array in this library's device memory.
//
// The array below is reserved on every GPU that loads the library and stays
// reserved until the process exits.  In host code its name is only a
// host-side stand-in, not a device address: the device address is looked up
// with cudaGetSymbolAddress once per device, with that device current, and
// kept for the life of the process (so a device reset, which reloads the
// module, is not supported while this library is loaded).
#include <cmath>
#include <cstdio>
#include <mutex>

#include "internal.cuh"

namespace dq {
namespace {

// Largest d the fixed scratch supports, and the scratch itself (8.75 MiB;
// the one scratch row of a top-k worker at that d takes 8.01 MiB).  Both
// numbers are the ones dqgan.h states.
constexpr int64_t kNoAllocMaxD = DQGAN_NOALLOC_MAX_D;
constexpr size_t kNoAllocScratchBytes = (size_t)DQGAN_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char noalloc_scratch[kNoAllocScratchBytes];

std::mutex setup_mutex;
void* scratch_address[kMaxDevices] = {nullptr};

}  // namespace
}  // namespace dq

extern "C" int dqgan_topk_compress_noalloc(const float* g, float* e, void* out_msg, int64_t d, int64_t k,
                                           float lr, void* cuda_stream) {
  char why[256];
  if (d < 1 || d > dq::kNoAllocMaxD) {
    snprintf(why, sizeof why, "d = %lld outside [1, %lld] supported without allocation", (long long)d,
             (long long)dq::kNoAllocMaxD);
    return dq::set_thread_error(DQGAN_ERR_INVALID_ARG, why);
  }
  if (k < 1 || k > d) {
    snprintf(why, sizeof why, "k = %lld outside [1, d]", (long long)k);
    return dq::set_thread_error(DQGAN_ERR_INVALID_ARG, why);
  }
  if (!std::isfinite(lr)) return dq::set_thread_error(DQGAN_ERR_INVALID_ARG, "lr is not finite");
  if (!g || !e || !out_msg)
    return dq::set_thread_error(DQGAN_ERR_INVALID_ARG, "NULL gradient, residual or message pointer");
  if (((uintptr_t)g | (uintptr_t)e | (uintptr_t)out_msg) & 15u)
    return dq::set_thread_error(DQGAN_ERR_INVALID_ARG,
                                "gradient, residual and message must be 16-byte aligned");
  const size_t need = dq::topk_scratch_bytes(d, 1, 0);  // one row, no server tables
  if (need > dq::kNoAllocScratchBytes)
    return dq::set_thread_error(DQGAN_ERR_INVALID_ARG, "top-k scratch for this d exceeds the fixed array");

  int dev = 0;
  cudaError_t st = cudaGetDevice(&dev);
  if (st != cudaSuccess) {
    snprintf(why, sizeof why, "cudaGetDevice: %s", cudaGetErrorString(st));
    return dq::set_thread_error(DQGAN_ERR_CUDA, why);
  }
  if (dev < 0 || dev >= dq::kMaxDevices)
    return dq::set_thread_error(DQGAN_ERR_UNSUPPORTED, "device ordinal beyond the supported range");
  void* scratch = nullptr;
  {
    // first call on this device: look up the device address of the array
    std::lock_guard<std::mutex> lock(dq::setup_mutex);
    if (!dq::scratch_address[dev]) {
      void* ptr = nullptr;
      st = cudaGetSymbolAddress(&ptr, dq::noalloc_scratch);
      if (st != cudaSuccess || !ptr) {
        snprintf(why, sizeof why, "cudaGetSymbolAddress: %s", cudaGetErrorString(st));
        return dq::set_thread_error(DQGAN_ERR_CUDA, why);
      }
      dq::scratch_address[dev] = ptr;
    }
    scratch = dq::scratch_address[dev];
  }

  cudaStream_t stream = reinterpret_cast<cudaStream_t>(cuda_stream);
  // No clearing: the top-k kernels rewrite the tile counts, tile prefixes and
  // candidates of the row in full on every call.  The one word that carries
  // over is the candidate threshold of the previous call (zero in the array
  // as loaded, i.e. none); it decides how much work the first pass saves and
  // never changes a result, whatever d and k the previous call had.
  dq::CompressArgs a{};
  a.g = g;
  a.g_stride = 0;
  a.e = e;
  a.h = nullptr;
  a.ld = 0;
  a.msg = reinterpret_cast<uint8_t*>(out_msg);
  a.msg_stride = 0;
  a.d = d;
  a.lr = lr;
  a.worker0 = 0;
  a.nworkers = 1;
  a.row0 = 0;
  uint64_t launches = 0;
  st = dq::launch_topk_compress(a, k, false, scratch, stream, &launches);
  if (st != cudaSuccess) {
    snprintf(why, sizeof why, "top-k launch: %s", cudaGetErrorString(st));
    return dq::set_thread_error(DQGAN_ERR_CUDA, why);
  }
  return DQGAN_OK;
}
