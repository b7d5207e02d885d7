// maps_internal.cuh -- helpers shared by the MAPS CUDA kernels (sm_103a).
//
// Nothing here is part of the public ABI (include/maps.h).
#pragma once

#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "maps.h"

namespace maps {

// ---------------------------------------------------------------------------
// Workspace: a 256-byte control block followed by per-call scratch carved in
// 256-byte aligned pieces.  The control block's first word is the sticky
// device status (MAPS_OK or the first error recorded by a kernel).
// ---------------------------------------------------------------------------
constexpr size_t kAlign = 256;
constexpr size_t kCtrlBytes = 256;

struct Carve {
  char *base;      // nullptr while only sizing
  size_t off = kCtrlBytes;
  explicit Carve(void *b) : base(static_cast<char *>(b)) {}
  template <class T>
  T *take(size_t count) {
    off = (off + kAlign - 1) / kAlign * kAlign;
    T *p = base ? reinterpret_cast<T *>(base + off) : nullptr;
    off += count * sizeof(T);
    return p;
  }
  size_t bytes() const { return (off + kAlign - 1) / kAlign * kAlign; }
};

inline int32_t *status_word(void *ws) { return static_cast<int32_t *>(ws); }

// First error wins; later errors do not overwrite it.
__device__ __forceinline__ void flag_error(int32_t *status, int code) {
  atomicCAS(status, 0, code);
}

// Bounded waits: a device-side wait gives up after this many polls (each poll
// sleeps briefly), records MAPS_E_TIMEOUT and lets the kernel finish.
constexpr uint32_t kSpinLimit = 1u << 22;

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long *p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_u64(unsigned long long *p, unsigned long long v) {
  asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t *p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_u32(uint32_t *p, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// A grid-wide barrier with a bounded wait, for kernels launched cooperatively
// (every block resident).  The words start at zero.  A block arrives with an
// acquire-release add (the block barrier before it orders every thread's
// writes before the release); the last to arrive resets the count and
// publishes the next generation with a release store; the others poll the
// generation with acquire loads.  After spin_limit polls a block records
// MAPS_E_TIMEOUT and the barrier returns false: the caller then returns at
// once, writing nothing more, so the kernel ends rather than hangs and no
// block works on data the barrier did not order.
struct GridBar {
  uint32_t arrived;
  uint32_t gen;
};
__device__ __forceinline__ uint32_t atom_add_acq_rel_u32(uint32_t *p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ bool grid_barrier(GridBar *b, int32_t *status, uint32_t spin_limit) {
  __shared__ int s_ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    const uint32_t g = ld_acquire_u32(&b->gen);
    if (atom_add_acq_rel_u32(&b->arrived, 1u) == gridDim.x - 1) {
      b->arrived = 0u;  // before the release below; nobody arrives until it
      st_release_u32(&b->gen, g + 1u);
    } else {
      uint32_t spins = 0;
      while (ld_acquire_u32(&b->gen) == g) {
        if (++spins > spin_limit) {
          atomicCAS(status, 0, MAPS_E_TIMEOUT);
          ok = 0;
          break;
        }
      }
    }
    s_ok = ok;
  }
  __syncthreads();
  return s_ok != 0;
}

// Programmatic dependent launch.  Every kernel of the library is launched
// with programmatic stream serialisation and starts with pdl_prologue():
// griddepcontrol.wait blocks until the previous grid on the stream has
// completed and its memory is visible (so nothing reads a predecessor's
// output early), and launch_dependents lets the next grid be scheduled once
// every CTA of this one has started, which hides the launch gap.
__device__ __forceinline__ void pdl_prologue() {
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
void set_last_cuda_error(cudaError_t e);

// Returns MAPS_OK or MAPS_E_CUDA (remembering the CUDA error).
inline int cuda_ok(cudaError_t e) {
  if (e == cudaSuccess) return MAPS_OK;
  set_last_cuda_error(e);
  return MAPS_E_CUDA;
}
inline int launch_ok() { return cuda_ok(cudaGetLastError()); }

// Launches `kernel` with programmatic stream serialisation (see pdl_prologue);
// errors surface through launch_ok().
template <typename... KArgs, typename... Args>
inline void launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  (void)cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

// A cooperative launch (every block resident at once, so the grid may wait at
// grid-wide barriers).  It is stream-ordered without programmatic overlap, so
// none of its blocks is placed while an earlier grid still holds resources.
// The caller sizes the grid within the occupancy limit; a launch the device
// refuses is reported.
template <typename... KArgs, typename... Args>
inline int launch_coop(void (*kernel)(KArgs...), int64_t grid, dim3 block, size_t smem,
                       cudaStream_t s, Args &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid < 1 ? 1 : grid));
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cuda_ok(cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...));
}

inline bool aligned(const void *p, size_t a) {
  return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

// Checks a caller workspace against a required size.
inline int check_ws(void *ws, size_t ws_bytes, size_t need) {
  if (ws == nullptr || !aligned(ws, kAlign)) return MAPS_E_INVALID;
  if (ws_bytes < need) return MAPS_E_WORKSPACE;
  return MAPS_OK;
}

// SEQUENTIAL horizon dispatch of J candidates on a dense K (the body of
// maps_dispatch's SEQUENTIAL mode, arguments already checked); mc ranks the
// decoders by headroom alone.  Uses the workspace past its control block.
int dispatch_sequential(int D, int H, int32_t *K, const int32_t *cap, int32_t *Q, int64_t J,
                        const int32_t *cp, const int32_t *cb, int32_t *choice, int64_t *headroom,
                        bool mc, void *ws, cudaStream_t s);

int sm_count();           // multiprocessors of the current device
int max_smem_optin();     // opt-in shared memory per block, bytes

#define MAPS_TRY(expr)            \
  do {                            \
    int maps_try_rc_ = (expr);    \
    if (maps_try_rc_ != MAPS_OK)  \
      return maps_try_rc_;        \
  } while (0)

}  // namespace maps
