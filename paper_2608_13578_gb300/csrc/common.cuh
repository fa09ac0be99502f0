// Shared device helpers of the BCMT library: storage-type conversion, warp
// reductions, and the status bits a kernel sets when a bounded wait expires.
#pragma once

#include <atomic>

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

namespace bcmt {

typedef __nv_bfloat16 bf16;

// Bits OR-ed into the device status word.
enum : unsigned { kStatusTimeout = 1u, kStatusBadLaunch = 2u };

// Programmatic dependent launch.  Every kernel of the library is launched with
// programmatic stream serialisation (launch_k below) and starts with
// pdl_enter(): it lets the next kernel on the stream begin launching at once,
// then waits until the previous kernel has finished and its writes are
// visible.  Work placed before pdl_wait() (barrier init, TMEM allocation,
// tensor-map prefetch) overlaps the previous kernel; no global memory may be
// touched before it.  Both are no-ops for a launch without the attribute.
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_enter() {
  pdl_trigger();
  pdl_wait();
}

// Host: while `on`, this thread's launches on `stream` carry `priority`
// instead of the stream's own (the C-ABI calls raise their critical chain,
// which runs on the caller's stream, above the work they put beside it).
struct PriorityOverride {
  bool on = false;
  cudaStream_t stream = nullptr;
  int priority = 0;
};
inline PriorityOverride& priority_override() {
  static thread_local PriorityOverride p;
  return p;
}
inline int launch_priority(cudaStream_t stream) {
  const PriorityOverride& o = priority_override();
  if (o.on && o.stream == stream) return o.priority;
  int prio = 0;
  if (cudaStreamGetPriority(stream, &prio) != cudaSuccess) prio = 0;
  return prio;
}

// Host: launches `kernel` on `stream` with programmatic stream serialisation
// and launch_priority(stream) as the launch priority (so that the priority is
// kept when the launch is captured into a CUDA graph).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                            cudaStream_t stream, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  const int prio = launch_priority(stream);
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributePriority;
  attr[1].val.priority = prio;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Raises `kern`'s dynamic shared memory limit to `bytes` on the current device,
// once per device (function attributes belong to a device's context): `done`
// is the call site's bit set of devices already configured.
template <typename... KArgs>
inline cudaError_t smem_opt_in(void (*kern)(KArgs...), int bytes,
                               std::atomic<unsigned long long>* done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const unsigned long long bit = 1ull << (dev & 63);
  if (done->load() & bit) return cudaSuccess;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done->fetch_or(bit);
  return e;
}

// The same with thread-block clusters of `cluster_x` CTAs along x.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                    cudaStream_t stream, int cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  const int prio = launch_priority(stream);
  cudaLaunchAttribute attr[3];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = cluster_x;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  attr[2].id = cudaLaunchAttributePriority;
  attr[2].val.priority = prio;
  cfg.attrs = attr;
  cfg.numAttrs = 3;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

template <class T> __device__ __forceinline__ float to_f(T v);
template <> __device__ __forceinline__ float to_f<float>(float v) { return v; }
template <> __device__ __forceinline__ float to_f<bf16>(bf16 v) { return __bfloat162float(v); }

template <class T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float sigmoidf_(float u) { return 1.0f / (1.0f + expf(-u)); }
// Hardware-approximate sigmoid (ex2.approx and an approximate divide, a few
// ulp in fp32) for results stored in bf16, whose rounding is ~1000x coarser.
__device__ __forceinline__ float sigmoid_bf16out(float u) {
  return __fdividef(1.0f, 1.0f + __expf(-u));
}

// Loads that bypass L1 (ld.global.cg): for data written earlier in the same
// kernel by other CTAs (the phases of a cooperative kernel).
__device__ __forceinline__ void load8_cg(const float* p, float* v) {
  const float4 a = __ldcg(reinterpret_cast<const float4*>(p));
  const float4 b = __ldcg(reinterpret_cast<const float4*>(p) + 1);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

// Raw bf16 pairs, converted when used.
__device__ __forceinline__ void load8_raw(const bf16* p, uint4& raw) {
  raw = *reinterpret_cast<const uint4*>(p);
}
__device__ __forceinline__ void unpack8(const uint4& raw, float* v) {
  const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    __nv_bfloat162 h = *reinterpret_cast<const __nv_bfloat162*>(&w[i]);
    float2 f = __bfloat1622float2(h);
    v[2 * i] = f.x;
    v[2 * i + 1] = f.y;
  }
}

// Vector load/store of 4 consecutive elements (16 B for fp32, 8 B for bf16).
// The address must be aligned to the vector width.
__device__ __forceinline__ void load4(const float* p, float* v) {
  float4 t = *reinterpret_cast<const float4*>(p);
  v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
}
__device__ __forceinline__ void load4(const bf16* p, float* v) {
  uint2 t = *reinterpret_cast<const uint2*>(p);
  __nv_bfloat162 a = *reinterpret_cast<__nv_bfloat162*>(&t.x);
  __nv_bfloat162 b = *reinterpret_cast<__nv_bfloat162*>(&t.y);
  float2 fa = __bfloat1622float2(a), fb = __bfloat1622float2(b);
  v[0] = fa.x; v[1] = fa.y; v[2] = fb.x; v[3] = fb.y;
}
__device__ __forceinline__ void store4(float* p, const float* v) {
  *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
}
__device__ __forceinline__ void store4(bf16* p, const float* v) {
  __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]);
  __nv_bfloat162 b = __floats2bfloat162_rn(v[2], v[3]);
  uint2 t;
  t.x = *reinterpret_cast<uint32_t*>(&a);
  t.y = *reinterpret_cast<uint32_t*>(&b);
  *reinterpret_cast<uint2*>(p) = t;
}

// 8 consecutive elements (16 B for bf16, 32 B for fp32); 16-byte aligned.
__device__ __forceinline__ void load8(const float* p, float* v) {
  load4(p, v);
  load4(p + 4, v + 4);
}
__device__ __forceinline__ void load8(const bf16* p, float* v) {
  uint4 t = *reinterpret_cast<const uint4*>(p);
  const uint32_t w[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    __nv_bfloat162 h = *reinterpret_cast<const __nv_bfloat162*>(&w[i]);
    float2 f = __bfloat1622float2(h);
    v[2 * i] = f.x;
    v[2 * i + 1] = f.y;
  }
}
__device__ __forceinline__ void store8(float* p, const float* v) {
  store4(p, v);
  store4(p + 4, v + 4);
}
__device__ __forceinline__ void store8(bf16* p, const float* v) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
    w[i] = *reinterpret_cast<uint32_t*>(&h);
  }
  *reinterpret_cast<uint4*>(p) = make_uint4(w[0], w[1], w[2], w[3]);
}

}  // namespace bcmt
