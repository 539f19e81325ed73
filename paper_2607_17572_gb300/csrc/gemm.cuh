// Dense products of the backbone: D[m, n] = sum_k A[m, k] B[n, k], f32 accumulate, with
// the fused epilogues the forward and backward passes need.
#pragma once

#include "common.cuh"

namespace jagg {

enum GemmEpi : int {
  EPI_STORE = 0,       // C = acc (+ bias[n])                     (C: dtype or f32)
  EPI_GELU = 1,        // u = acc + bias; C = gelu'(u) (C may be null); C2 = gelu(u)  (both dtype)
  EPI_GATE_RESID = 2,  // C = y = acc + bias; C2 = aux + gate[seq(m), n] * y  (C2, aux f32)
  EPI_MUL_AUX = 3,     // C = acc * aux                              (aux dtype)
  EPI_ACCUM = 4,       // C += acc (f32, atomic reduction; allows split-K)
};

struct GemmArgs {
  int M = 0, N = 0, K = 0;
  // Operand A: K-major A[m * lda + k], or MN-major A[k * lda + m].
  const void* A = nullptr;
  int64_t lda = 0;
  bool a_mn = false;
  int a_dtype = JAGG_DTYPE_BF16;
  // Operand B: K-major B[n * ldb + k], or MN-major B[k * ldb + n].
  const void* B = nullptr;
  int64_t ldb = 0;
  bool b_mn = false;
  int b_dtype = JAGG_DTYPE_BF16;

  int epi = EPI_STORE;
  const void* bias = nullptr;  // [N], in bias_dtype
  int bias_dtype = JAGG_DTYPE_BF16;
  void* C = nullptr;
  int64_t ldc = 0;
  int c_dtype = JAGG_DTYPE_BF16;  // EPI_ACCUM requires f32
  void* C2 = nullptr;
  int64_t ldc2 = 0;
  const void* aux = nullptr;
  int64_t ld_aux = 0;
  const float* gate = nullptr;  // gate[(m / rows_per_seq) * gate_stride + n]
  int64_t gate_stride = 0;
  int rows_per_seq = 1;
  // Optional row remap of C: row(m) = (m / remap_rows) * remap_stride + remap_offset + m % remap_rows
  int remap_rows = 0;
  int remap_offset = 0;
  int64_t remap_stride = 0;
  int split_k = 0;  // EPI_ACCUM only; 0 = choose
  // EPI_STORE / EPI_ACCUM only: element (m, n) goes to C[n * ldc + m] (a transposed output,
  // for products formulated as D^T so that the long dimension is M), and the bias is
  // indexed by m instead of n.
  bool c_trans = false;
  bool bias_m = false;
  int tile_n = 0;  // tensor-core tile width (64 / 128 / 256); 0 = chosen by the cost model
};

// Launches the product on `stream`.  bf16 x bf16 goes to the tcgen05 tensor-core kernel;
// anything involving f32 operands goes to the SIMT kernel.
int gemm(const GemmArgs& g, cudaStream_t stream);

// Forces the SIMT kernel (tests of the tensor-core path compare against it).
int gemm_simt(const GemmArgs& g, cudaStream_t stream);

}  // namespace jagg
