// api.cu -- library-wide entry points of the MAPS C ABI: version, last CUDA
// error, and the sticky device status check.
#include "maps_internal.cuh"

namespace maps {

static thread_local int g_last_cuda_error = 0;

void set_last_cuda_error(cudaError_t e) { g_last_cuda_error = static_cast<int>(e); }

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 1;
  return n > 0 ? n : 1;
}

int max_smem_optin() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 48 * 1024;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
    return 48 * 1024;
  return n;
}

}  // namespace maps

extern "C" {

int maps_version(void) { return 100; }  // 0.1.0

int maps_last_cuda_error(void) { return maps::g_last_cuda_error; }

int maps_check(void *ws, void *stream) {
  if (ws == nullptr || !maps::aligned(ws, maps::kAlign)) return MAPS_E_INVALID;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  MAPS_TRY(maps::cuda_ok(cudaStreamSynchronize(s)));
  int32_t st = 0;
  MAPS_TRY(maps::cuda_ok(cudaMemcpy(&st, ws, sizeof(st), cudaMemcpyDeviceToHost)));
  if (st != MAPS_OK) {
    MAPS_TRY(maps::cuda_ok(cudaMemsetAsync(ws, 0, sizeof(int32_t), s)));
    MAPS_TRY(maps::cuda_ok(cudaStreamSynchronize(s)));
  }
  return st;
}

}  // extern "C"
