// Joint softmax attention of the backbone: forward with saved log-sum-exp and the
// recomputing backward (the four N^2 d products of the appendix's Eqs. bwd_V .. bwd_QK).
#pragma once

#include "common.cuh"

namespace jagg {

// Row addressing of a [B, N, *] activation whose first n0 tokens of every sequence live in
// one buffer and the remaining N - n0 in another (the text and image streams of the
// MMDiT double blocks).  Single-stream layouts use n0 = N.
struct SegRows {
  void* p0;
  void* p1;
  int64_t ld0, ld1;
  int n0;
  __host__ __device__ __forceinline__ int64_t off(int b, int n, int N, int64_t elem_col) const {
    return n < n0 ? ((int64_t)b * n0 + n) * ld0 + elem_col : ((int64_t)b * (N - n0) + (n - n0)) * ld1 + elem_col;
  }
  __host__ __device__ __forceinline__ void* base(int n) const { return n < n0 ? p0 : p1; }
};

__host__ __device__ inline SegRows seg_single(void* p, int64_t ld, int N) { return SegRows{p, p, ld, ld, N}; }

struct AttnArgs {
  int B, N, heads, dh;
  float scale;  // 1/sqrt(dh)
  SegRows q, k, v;  // column offset of head h: col0 + h * dh
  int64_t q_col0, k_col0, v_col0;
  SegRows o;  // output, col h * dh
  float* lse;  // [B, heads, N] natural-log log-sum-exp of the scaled scores
  int dtype;
  int impl = 0;  // forward: 0 the library's choice; 1 warp-level MMA kernel; 2 tcgen05 kernel
};

struct AttnBwdArgs {
  AttnArgs f;  // forward inputs (q, k, v, o, lse)
  SegRows dO;  // upstream gradient of o, col h * dh
  float* Dv;   // [B, heads, N] rowsum(dO * O), filled by the launcher
  float* dq_acc;  // f32 [B*N, heads*dh] scratch, zeroed by the launcher
  SegRows dq, dk, dv;  // outputs (dtype), columns dq_col0 + h * dh etc.
  int64_t dq_col0, dk_col0, dv_col0;
  int impl = 0;  // 0: the library's choice; 1: warp-level MMA kernel; 2: tcgen05 kernel
};

int attention_fwd(const AttnArgs& a, cudaStream_t s);
// The tcgen05 forward (attention_tc.cu): bf16, head dim 64 / 128, stream boundary on a
// multiple of 128 tokens, 16-byte aligned views.
bool attention_fwd_tc_eligible(const AttnArgs& a);
int attention_fwd_tc(const AttnArgs& a, cudaStream_t s);
// The tcgen05 backward (attention_tc.cu): bf16, head dim 64 / 128, stream boundary on a
// multiple of 128 tokens, 16-byte aligned views.
bool attention_bwd_tc_eligible(const AttnBwdArgs& a);
int attention_bwd_tc(const AttnBwdArgs& a, cudaStream_t s);
// Scratch: Dv and dq_acc as described above.  dq_acc must be 16-byte aligned (it receives
// 16-byte vector reductions); attention_bwd_scratch places both in one buffer of
// attention_bwd_scratch_floats floats with dq_acc at a 256-byte boundary.
int attention_bwd(const AttnBwdArgs& a, cudaStream_t s);
int64_t attention_bwd_scratch_floats(int B, int N, int heads, int dh);
void attention_bwd_scratch(float* scratch, int B, int N, int heads, float** Dv, float** dq_acc);

}  // namespace jagg
