// Shared device/host helpers of the JAGG library (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <stddef.h>

#include "../../include/jagg.h"

namespace jagg {

using bf16 = __nv_bfloat16;

// ------------------------------------------------------------------ status word
// Device-side status shared by every kernel of the library.  Bounded waits that give
// up set JAGG_DEV_TIMEOUT here instead of trapping; the host reads it through
// jagg_device_status().
// Each translation unit that sets it owns a copy (no relocatable device code is needed);
// jagg_device_status() combines them through the per-unit accessors declared below.
enum : unsigned { JAGG_DEV_OK = 0u, JAGG_DEV_TIMEOUT = 1u, JAGG_DEV_BADARG = 2u };
static __device__ unsigned g_device_status = 0;

// Reads (and optionally clears) this translation unit's status word.  Synchronous.
static inline int read_unit_status(unsigned* v, int clear) {
  if (cudaMemcpyFromSymbol(v, g_device_status, sizeof(unsigned)) != cudaSuccess) return -1;
  if (clear) {
    const unsigned zero = 0;
    if (cudaMemcpyToSymbol(g_device_status, &zero, sizeof(unsigned)) != cudaSuccess) return -1;
  }
  return 0;
}
int unit_status_gemm(unsigned* v, int clear);
int unit_status_signals(unsigned* v, int clear);
int unit_status_attention_tc(unsigned* v, int clear);
int unit_status_testing(unsigned* v, int clear);

__device__ __forceinline__ void set_device_status(unsigned bits) { atomicOr(&g_device_status, bits); }

// Wall-clock bound (ns) for every spin-wait in the library's kernels.
constexpr unsigned long long kWaitLimitNs = 2000000000ull;

__device__ __forceinline__ unsigned long long globaltimer_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ------------------------------------------------------------------ element access
template <typename T> struct Elem;
template <> struct Elem<float> {
  static __device__ __forceinline__ float load(const float* p) { return *p; }
  static __device__ __forceinline__ void store(float* p, float v) { *p = v; }
  static __device__ __forceinline__ float from(float v) { return v; }
};
template <> struct Elem<bf16> {
  static __device__ __forceinline__ float load(const bf16* p) { return __bfloat162float(*p); }
  static __device__ __forceinline__ void store(bf16* p, float v) { *p = __float2bfloat16_rn(v); }
  static __device__ __forceinline__ bf16 from(float v) { return __float2bfloat16_rn(v); }
};

template <typename T> __device__ __forceinline__ float ld(const T* p) { return Elem<T>::load(p); }
template <typename T> __device__ __forceinline__ void st(T* p, float v) { Elem<T>::store(p, v); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// tanh-approximated GELU and its derivative (the backbone's activation).
__device__ __forceinline__ float gelu_tanh(float u) {
  const float c = 0.7978845608028654f, a = 0.044715f;
  return 0.5f * u * (1.f + tanhf(c * (u + a * u * u * u)));
}
__device__ __forceinline__ float gelu_tanh_grad(float u) {
  const float c = 0.7978845608028654f, a = 0.044715f;
  float th = tanhf(c * (u + a * u * u * u));
  return 0.5f * (1.f + th) + 0.5f * u * (1.f - th * th) * c * (1.f + 3.f * a * u * u);
}
// gelu(u) and gelu'(u) sharing one tanh.
__device__ __forceinline__ void gelu_tanh_both(float u, float& g, float& dg) {
  const float c = 0.7978845608028654f, a = 0.044715f;
  const float th = tanhf(c * (u + a * u * u * u));
  g = 0.5f * u * (1.f + th);
  dg = 0.5f * (1.f + th) + 0.5f * u * (1.f - th * th) * c * (1.f + 3.f * a * u * u);
}
// The same pair with tanh from the hardware approximation (tanh.approx.f32, absolute
// error below 2^-10): for outputs rounded to bf16 (the tensor-core path).
__device__ __forceinline__ void gelu_tanh_both_approx(float u, float& g, float& dg) {
  const float c = 0.7978845608028654f, a = 0.044715f;
  float th;
  asm("tanh.approx.f32 %0, %1;" : "=f"(th) : "f"(c * (u + a * u * u * u)));
  g = 0.5f * u * (1.f + th);
  dg = 0.5f * (1.f + th) + 0.5f * u * (1.f - th * th) * c * (1.f + 3.f * a * u * u);
}
__device__ __forceinline__ float silu_f(float x) { return x / (1.f + expf(-x)); }
__device__ __forceinline__ float silu_grad_f(float x) {
  float s = 1.f / (1.f + expf(-x));
  return s * (1.f + x * (1.f - s));
}

inline int ceil_div(long long a, long long b) { return (int)((a + b - 1) / b); }

// ------------------------------------------------------------------ host errors
void set_last_error(const char* fmt, ...);
int cuda_status(cudaError_t e, const char* where);
int sm_count();

// ------------------------------------------------------------------ launch accounting
// Every kernel launch of the library is counted (jagg_launch_count).  While profiling is
// enabled (jagg_profile_enable), the launches of the path's kernels are also bracketed by
// CUDA events on their stream and attributed to a kernel family with their algorithmic
// FLOPs and bytes.
void count_launch();
enum ProfFamily : int {
  PROF_GEMM_TC = 0,
  PROF_GEMM_SIMT,
  PROF_ATTN_FWD,
  PROF_ATTN_BWD,
  PROF_LN_BWD,     // LayerNorm + gate backward
  PROF_ATTN_AUX,   // attention backward helpers (rowsum(dO O), dQ conversion)
  PROF_QKN_BWD,    // per-head RMSNorm + RoPE backward
  PROF_COLSUM,     // bias gradients (column sums)
  PROF_COPY,       // row copies between the stream and joint layouts
  PROF_SIGNALS,    // the step signals (with the aggregation when fused)
  PROF_GRAD_REDUCE,
  PROF_LN_FWD,     // LayerNorm + modulation forward
  PROF_QKN_FWD,    // per-head RMSNorm + RoPE forward
  PROF_FAMILIES
};
int prof_start(cudaStream_t s);  // returns a token, or -1 when profiling is off
void prof_stop(int token, cudaStream_t s, int family, double flops, double bytes, int m = 0, int n = 0, int k = 0);

}  // namespace jagg

#define JAGG_LAUNCHED()                                                         \
  do {                                                                          \
    JAGG_CUDA_TRY(cudaGetLastError());                                          \
    ::jagg::count_launch();                                                     \
  } while (0)

#define JAGG_CUDA_TRY(expr)                                                     \
  do {                                                                          \
    cudaError_t _e = (expr);                                                    \
    if (_e != cudaSuccess) return ::jagg::cuda_status(_e, #expr);               \
  } while (0)

#define JAGG_TRY(expr)                                                          \
  do {                                                                          \
    int _s = (expr);                                                            \
    if (_s != JAGG_OK) return _s;                                               \
  } while (0)

#define JAGG_CHECK_ARG(cond, ...)                                               \
  do {                                                                          \
    if (!(cond)) {                                                              \
      ::jagg::set_last_error(__VA_ARGS__);                                      \
      return JAGG_ERR_ARG;                                                      \
    }                                                                           \
  } while (0)
