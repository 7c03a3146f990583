// Shared helpers of the FL-GLM server library (sm_103a).
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/flglm.h"

#define FL_DEV __device__ __forceinline__

// Device status word codes (written by kernels, read by the host after a sync).
enum : int {
  FL_DEV_OK = 0,
  FL_DEV_TIMEOUT_FULL = 1,      // MMA waited too long for a TMA stage
  FL_DEV_TIMEOUT_EMPTY = 2,     // producer waited too long for a free stage
  FL_DEV_TIMEOUT_ACC_FULL = 3,  // epilogue waited too long for an accumulator
  FL_DEV_TIMEOUT_ACC_EMPTY = 4, // MMA waited too long for the epilogue
  FL_DEV_TIMEOUT_DRAIN = 5,     // teardown waited too long for in-flight work
  FL_DEV_BAD_ARG = 6,           // a kernel found an argument it cannot handle
};

// Bounded-wait budget: a wait gives up after this many nanoseconds of %globaltimer.
#ifndef FL_WAIT_NS
#define FL_WAIT_NS 2000000000ull
#endif

FL_DEV uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

// Programmatic dependent launch.  A kernel launched with fl_launch (programmatic stream
// serialization) may start while the previous kernel on the stream is still running; it
// calls pdl_wait() before its first access to global memory (which returns once that
// kernel has completed and its writes are visible) and then pdl_trigger(), which lets the
// next kernel's CTAs be scheduled as SMs free up.  Without the attribute both are no-ops.
FL_DEV void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
FL_DEV void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

FL_DEV void report_status(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

FL_DEV float bf2f(__nv_bfloat16 x) { return __bfloat162float(x); }
FL_DEV __nv_bfloat16 f2bf(float x) { return __float2bfloat16_rn(x); }

FL_DEV uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
FL_DEV float2 unpack_bf16x2(uint32_t u) {
  __nv_bfloat162 v = *reinterpret_cast<__nv_bfloat162*>(&u);
  return __bfloat1622float2(v);
}

// tanh-form GeLU and its derivative, with c = sqrt(2/pi), a = 0.044715.
// tanh by the hardware instruction (PTX tanh.approx.f32, relative error about 2^-11): the
// GeLU epilogues run on four warps per SM with nothing to hide an accurate tanhf's
// instruction latency behind, and their bf16 outputs cannot resolve the difference.
FL_DEV float tanh_hw(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
FL_DEV float gelu_tanh(float u) {
  const float c = 0.7978845608028654f, a = 0.044715f;
  float t = tanh_hw(c * (u + a * u * u * u));
  return 0.5f * u * (1.f + t);
}
FL_DEV float gelu_tanh_grad(float u) {
  const float c = 0.7978845608028654f, a = 0.044715f;
  float t = tanh_hw(c * (u + a * u * u * u));
  return 0.5f * (1.f + t) + 0.5f * u * (1.f - t * t) * c * (1.f + 3.f * a * u * u);
}

// Launches `kern` on `st` with programmatic stream serialization (see pdl_wait): the
// kernel must call pdl_wait() before touching global memory.
template <typename... KArgs, typename... Args>
cudaError_t fl_launch(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

#define FL_CUDA_TRY(expr)                                  \
  do {                                                     \
    cudaError_t _e = (expr);                               \
    if (_e != cudaSuccess) return fl_internal_cuda_error(_e, #expr, __FILE__, __LINE__); \
  } while (0)

// Records a CUDA error in the thread-local error string and returns FL_ERR_CUDA.
int fl_internal_cuda_error(cudaError_t e, const char* what, const char* file, int line);
int fl_internal_error(int code, const char* fmt, ...);

// Launch set-up shared by every launcher, kept per device and safe to call from several
// host threads (runtime.cu).  fl_sm_count: the current device's multiprocessor count.
// fl_func_smem: raises kernel `func`'s dynamic shared-memory limit to `bytes` on the
// current device (an attribute the driver keeps per device), once per (kernel, device,
// bytes); later calls return at once.
int fl_sm_count();
cudaError_t fl_func_smem(const void* func, int bytes);

// True when p is not a multiple of `bytes` (a power of two); a null p counts as aligned.
inline bool fl_misaligned(const void* p, uintptr_t bytes) { return (reinterpret_cast<uintptr_t>(p) & (bytes - 1)) != 0; }
