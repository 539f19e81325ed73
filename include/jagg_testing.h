/*
 * jagg_testing.h -- entry points that expose single kernels of the library to its tests.
 *
 * They are not part of the JAGG path; they let the tests check the dense-product and
 * attention kernels in isolation against a plain reference before the whole backbone is
 * compared with the oracle.  Same conventions as jagg.h (caller-owned device memory,
 * asynchronous on `stream`, status return).
 */
#ifndef JAGG_TESTING_H_
#define JAGG_TESTING_H_

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

/* D[m, n] = sum_k A[m, k] B[n, k] with the library's epilogues:
 *   epi 0 store:  C = D (+ bias[n])
 *   epi 1 gelu:   u = D + bias, C = gelu_tanh'(u), C2 = gelu_tanh(u)
 *   epi 2 gate:   C = y = D + bias, C2 = aux + gate[(m / rows_per_seq) * gate_stride + n] * y
 *   epi 3 mul:    C = D * aux
 *   epi 4 accum:  C += D (f32 C; split_k > 0 forces the number of K splits)
 * A is K-major (A[m*lda + k]) or MN-major (A[k*lda + m]); B is K-major (B[n*ldb + k]) or
 * MN-major (B[k*ldb + n]).  a_dtype/b_dtype/c_dtype/bias_dtype are JAGG_DTYPE_*; C2 and aux
 * follow c_dtype for gelu/dgelu and are f32 for gate.  force_simt selects the SIMT kernel
 * instead of the tcgen05 one (bf16 operands only take the tensor-core path).  For store and
 * accum, c_trans writes element (m, n) to C[n*ldc + m] and bias_m indexes the bias by m.
 * tile_n forces the tensor-core tile width (64, 128 or 256 columns; 0 = the library's
 * choice); a width the product cannot use returns JAGG_ERR_ARG. */
typedef struct jagg_gemm_desc {
  int32_t M, N, K;
  const void* A;
  int64_t lda;
  int32_t a_mn, a_dtype;
  const void* B;
  int64_t ldb;
  int32_t b_mn, b_dtype;
  int32_t epi;
  const void* bias;
  int32_t bias_dtype;
  void* C;
  int64_t ldc;
  int32_t c_dtype;
  void* C2;
  int64_t ldc2;
  const void* aux;
  int64_t ld_aux;
  const float* gate;
  int64_t gate_stride;
  int32_t rows_per_seq;
  int32_t split_k;
  int32_t force_simt;
  int32_t c_trans;
  int32_t bias_m;
  int32_t tile_n;
} jagg_gemm_desc;

int jagg_test_gemm(const jagg_gemm_desc* desc, cudaStream_t stream);

/* Joint softmax attention over qkv [B*N, 3*heads*dh] (q, k, v at column offsets 0, d, 2d;
 * dtype JAGG_DTYPE_*): o [B*N, d], lse [B, heads, N] f32.  The backward takes dO [B*N, d]
 * and writes dqkv [B*N, 3d] using scratch of jagg_test_attention_scratch_bytes bytes. */
int jagg_test_attention_fwd(const void* qkv, int B, int N, int heads, int dh, int dtype, void* o, float* lse,
                            cudaStream_t stream);
int64_t jagg_test_attention_scratch_bytes(int B, int N, int heads, int dh);
int jagg_test_attention_bwd(const void* qkv, const void* o, const float* lse, const void* dO, int B, int N,
                            int heads, int dh, int dtype, void* dqkv, void* scratch, cudaStream_t stream);
/* The backward over two-stream views, as the MMDiT double blocks use it: the first n0
 * tokens of every sequence live in qkv0 / o0 / dO0 / dqkv0 ([B*n0, 3d], [B*n0, d], ...),
 * the remaining N - n0 in qkv1 / o1 / dO1 / dqkv1 (n0 = N: one buffer, the *1 pointers
 * ignored).  impl: 0 the library's choice, 1 the warp-level MMA kernel, 2 the tcgen05
 * kernel (JAGG_ERR_ARG when it does not serve the call). */
/* The forward over two-stream views (same layout and impl codes as the backward below):
 * o0 / o1 receive the output rows of each stream, lse [B, heads, N]. */
int jagg_test_attention_fwd_streams(const void* qkv0, const void* qkv1, void* o0, void* o1, float* lse, int B,
                                    int N, int n0, int heads, int dh, int dtype, int impl, cudaStream_t stream);
int jagg_test_attention_bwd_streams(const void* qkv0, const void* qkv1, const void* o0, const void* o1,
                                    const float* lse, const void* dO0, const void* dO1, int B, int N, int n0,
                                    int heads, int dh, int dtype, void* dqkv0, void* dqkv1, void* scratch, int impl,
                                    cudaStream_t stream);

/* LayerNorm + modulation backward fused with the gate backward of the branch before it (the
 * per-row kernels of the joint VJP; the paper's Phase 4 reverse mode through adaLN), on M
 * rows of rows_per_seq rows per sequence, hidden size d (d % 4 == 0, d <= 3072).  Row m of
 * sequence b = m / rows_per_seq, all buffers row-major and contiguous (f32 unless noted):
 *   do_ln:   xh = (h - mean[m]) rstd[m]; e = dm (1 + scale[b]);
 *            dh_out = dh_in + rstd (e - mean_row(e) - xh mean_row(e xh));
 *            dshift[b] += sum_m dm, dscale[b] += sum_m dm xh   (dm [M, d] f32)
 *   do_gate: dy = gate[b] dh (dh = dh_out, or dh_in without do_ln); dgate[b] += sum_m dh y;
 *            dbias (nullable) += sum_b gate[b] sum_{m in b} dh   (y, dy [M, d] in `dtype`)
 * scale, gate: [M / rows_per_seq, d]; dshift, dscale, dgate: [M / rows_per_seq, d],
 * accumulated.  dh_out may alias dh_in.  JAGG_ERR_ARG for an unsupported d or rows that are
 * not whole sequences. */
int jagg_test_ln_gate_bwd(int M, int d, int rows_per_seq, int do_ln, int do_gate, const float* dm, const float* h,
                          const float* mean, const float* rstd, const float* scale, float* dshift, float* dscale,
                          const float* dh_in, float* dh_out, const void* y, const float* gate, float* dgate,
                          void* dy, float* dbias, int dtype, cudaStream_t stream);

/* Per-head RMSNorm of q and k (learned scale [dh], eps 1e-6) followed by 2D RoPE (the MMDiT
 * blocks' QK normalisation; the backbone reading of the paper's Flux / Qwen-Image models), on
 * M rows of N tokens per sequence whose first n_txt tokens are text (not rotated) and whose
 * image tokens lie on a grid gw wide.  qkv [M, ld_qkv] holds q at column 0 and k at column d
 * (d = heads * dh, dh <= 128 even), in `dtype`; qscale, kscale [dh] in `dtype`.
 * Forward: qk_out [M, 2d] = the normalised, rotated q then k; rq, rk [M, heads] f32 the
 * inverse RMS of each (row, head).  rope = 0 skips the rotation. */
int jagg_test_qk_norm_rope_fwd(const void* qkv, int64_t ld_qkv, int M, int N, int d, int heads, int n_txt, int gw,
                               const void* qscale, const void* kscale, int rope, void* qk_out, float* rq, float* rk,
                               int dtype, cudaStream_t stream);
/* Backward of the above: dqk [M, ld_dqk] (dtype) holds the gradient of the rotated q at column
 * 0 and of k at column d on entry and the gradient of the raw q, k on exit; dqscale,
 * dkscale [dh] f32 accumulate the scale gradients.  rq, rk from the forward. */
int jagg_test_qk_norm_rope_bwd(const void* qkv, int64_t ld_qkv, int M, int N, int d, int heads, int n_txt, int gw,
                               const void* qscale, const void* kscale, int rope, const float* rq, const float* rk,
                               void* dqk, int64_t ld_dqk, float* dqscale, float* dkscale, int dtype,
                               cudaStream_t stream);
/* Column sums db[c] += sum_r X[r * ld + c] (r < rows, c < cols; X f32 when x_f32 else bf16):
 * the bias gradients of the joint VJP. */
int jagg_test_colsum(const void* X, int x_f32, int rows, int cols, int64_t ld, float* db, cudaStream_t stream);

/* Failure detection of the bounded waits (every mbarrier wait of the library gives up after
 * a wall-clock limit instead of hanging): one CTA waits on an mbarrier that nothing arrives
 * at, with the limit limit_ns (0 < limit_ns <= 2 s, else JAGG_ERR_ARG) in place of the
 * library's 2 s.  The wait gives up, sets JAGG_DEV_STATUS_TIMEOUT in the device status word
 * (read and cleared by jagg_device_status) and the kernel returns; no copy or MMA is in
 * flight.  out device [2] u64: out[0] = 1 when the wait gave up, out[1] = the nanoseconds
 * it waited. */
int jagg_test_wait_timeout(unsigned long long limit_ns, unsigned long long* out, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* JAGG_TESTING_H_ */
