// Kernel-level entry points for the library's tests (include/jagg_testing.h).
#include "../../include/jagg_testing.h"
#include "attention.cuh"
#include "elementwise.cuh"
#include "gemm.cuh"
#include "ptx.cuh"

namespace jagg {
int unit_status_testing(unsigned* v, int clear) { return read_unit_status(v, clear); }
}  // namespace jagg

using namespace jagg;

namespace {
// One mbarrier that nothing ever arrives at: the library's bounded wait on it gives up after
// limit_ns, sets JAGG_DEV_TIMEOUT and returns.  No copy or MMA is in flight.
__global__ void wait_timeout_kernel(unsigned long long limit_ns, unsigned long long* out) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    ptx::mbar_init(&bar, 1);
    ptx::fence_mbar_init();
    const unsigned long long t0 = globaltimer_ns();
    const bool ok = ptx::mbar_wait_for(&bar, 0, limit_ns);
    out[0] = ok ? 0ull : 1ull;
    out[1] = globaltimer_ns() - t0;
  }
}
}  // namespace

extern "C" int jagg_test_wait_timeout(unsigned long long limit_ns, unsigned long long* out, cudaStream_t stream) {
  JAGG_CHECK_ARG(out, "jagg_test_wait_timeout: null output");
  JAGG_CHECK_ARG(limit_ns > 0 && limit_ns <= kWaitLimitNs, "jagg_test_wait_timeout: limit %llu ns outside (0, %llu]",
                 limit_ns, kWaitLimitNs);
  wait_timeout_kernel<<<1, 32, 0, stream>>>(limit_ns, out);
  JAGG_LAUNCHED();
  return JAGG_OK;
}

extern "C" int jagg_test_gemm(const jagg_gemm_desc* d, cudaStream_t stream) {
  JAGG_CHECK_ARG(d, "jagg_test_gemm: null descriptor");
  GemmArgs g;
  g.M = d->M; g.N = d->N; g.K = d->K;
  g.A = d->A; g.lda = d->lda; g.a_mn = d->a_mn != 0; g.a_dtype = d->a_dtype;
  g.B = d->B; g.ldb = d->ldb; g.b_mn = d->b_mn != 0; g.b_dtype = d->b_dtype;
  g.epi = d->epi;
  g.bias = d->bias; g.bias_dtype = d->bias_dtype;
  g.C = d->C; g.ldc = d->ldc; g.c_dtype = d->c_dtype;
  g.C2 = d->C2; g.ldc2 = d->ldc2;
  g.aux = d->aux; g.ld_aux = d->ld_aux;
  g.gate = d->gate; g.gate_stride = d->gate_stride; g.rows_per_seq = d->rows_per_seq;
  g.split_k = d->split_k;
  g.c_trans = d->c_trans != 0;
  g.bias_m = d->bias_m != 0;
  g.tile_n = d->tile_n;
  return d->force_simt ? gemm_simt(g, stream) : gemm(g, stream);
}

static AttnArgs make_args(const void* qkv, int B, int N, int heads, int dh, int dtype, void* o, float* lse) {
  AttnArgs a;
  const int d = heads * dh;
  a.B = B; a.N = N; a.heads = heads; a.dh = dh; a.scale = 1.f / sqrtf((float)dh);
  a.q = a.k = a.v = seg_single(const_cast<void*>(qkv), 3 * d, N);
  a.q_col0 = 0; a.k_col0 = d; a.v_col0 = 2 * d;
  a.o = seg_single(o, d, N);
  a.lse = lse;
  a.dtype = dtype;
  return a;
}

extern "C" int jagg_test_attention_fwd(const void* qkv, int B, int N, int heads, int dh, int dtype, void* o,
                                       float* lse, cudaStream_t stream) {
  JAGG_CHECK_ARG(qkv && o && lse, "jagg_test_attention_fwd: null pointer");
  return attention_fwd(make_args(qkv, B, N, heads, dh, dtype, o, lse), stream);
}

extern "C" int64_t jagg_test_attention_scratch_bytes(int B, int N, int heads, int dh) {
  return attention_bwd_scratch_floats(B, N, heads, dh) * 4;
}

extern "C" int jagg_test_attention_bwd(const void* qkv, const void* o, const float* lse, const void* dO, int B, int N,
                                       int heads, int dh, int dtype, void* dqkv, void* scratch,
                                       cudaStream_t stream) {
  JAGG_CHECK_ARG(qkv && o && lse && dO && dqkv && scratch, "jagg_test_attention_bwd: null pointer");
  AttnBwdArgs ab;
  ab.f = make_args(qkv, B, N, heads, dh, dtype, const_cast<void*>(o), const_cast<float*>(lse));
  const int d = heads * dh;
  ab.dO = seg_single(const_cast<void*>(dO), d, N);
  attention_bwd_scratch(static_cast<float*>(scratch), B, N, heads, &ab.Dv, &ab.dq_acc);
  ab.dq = ab.dk = ab.dv = seg_single(dqkv, 3 * d, N);
  ab.dq_col0 = 0; ab.dk_col0 = d; ab.dv_col0 = 2 * d;
  return attention_bwd(ab, stream);
}

extern "C" int jagg_test_attention_fwd_streams(const void* qkv0, const void* qkv1, void* o0, void* o1, float* lse,
                                               int B, int N, int n0, int heads, int dh, int dtype, int impl,
                                               cudaStream_t stream) {
  JAGG_CHECK_ARG(qkv0 && o0 && lse, "jagg_test_attention_fwd_streams: null pointer");
  JAGG_CHECK_ARG(n0 > 0 && n0 <= N, "jagg_test_attention_fwd_streams: n0 = %d", n0);
  const bool two = n0 < N;
  JAGG_CHECK_ARG(!two || (qkv1 && o1), "jagg_test_attention_fwd_streams: null second stream");
  const int d = heads * dh;
  auto view = [&](const void* p0, const void* p1, int64_t ld) {
    return SegRows{const_cast<void*>(p0), const_cast<void*>(two ? p1 : p0), ld, ld, two ? n0 : N};
  };
  AttnArgs f;
  f.B = B; f.N = N; f.heads = heads; f.dh = dh; f.scale = 1.f / sqrtf((float)dh);
  f.q = f.k = f.v = view(qkv0, qkv1, 3 * d);
  f.q_col0 = 0; f.k_col0 = d; f.v_col0 = 2 * d;
  f.o = view(o0, o1, d);
  f.lse = lse;
  f.dtype = dtype;
  f.impl = impl;
  return attention_fwd(f, stream);
}

extern "C" int jagg_test_attention_bwd_streams(const void* qkv0, const void* qkv1, const void* o0, const void* o1,
                                               const float* lse, const void* dO0, const void* dO1, int B, int N,
                                               int n0, int heads, int dh, int dtype, void* dqkv0, void* dqkv1,
                                               void* scratch, int impl, cudaStream_t stream) {
  JAGG_CHECK_ARG(qkv0 && o0 && lse && dO0 && dqkv0 && scratch, "jagg_test_attention_bwd_streams: null pointer");
  JAGG_CHECK_ARG(n0 > 0 && n0 <= N, "jagg_test_attention_bwd_streams: n0 = %d", n0);
  const bool two = n0 < N;
  JAGG_CHECK_ARG(!two || (qkv1 && o1 && dO1 && dqkv1), "jagg_test_attention_bwd_streams: null second stream");
  const int d = heads * dh;
  auto view = [&](const void* p0, const void* p1, int64_t ld) {
    return SegRows{const_cast<void*>(p0), const_cast<void*>(two ? p1 : p0), ld, ld, two ? n0 : N};
  };
  AttnBwdArgs ab;
  AttnArgs& f = ab.f;
  f.B = B; f.N = N; f.heads = heads; f.dh = dh; f.scale = 1.f / sqrtf((float)dh);
  f.q = f.k = f.v = view(qkv0, qkv1, 3 * d);
  f.q_col0 = 0; f.k_col0 = d; f.v_col0 = 2 * d;
  f.o = view(o0, o1, d);
  f.lse = const_cast<float*>(lse);
  f.dtype = dtype;
  ab.dO = view(dO0, dO1, d);
  attention_bwd_scratch(static_cast<float*>(scratch), B, N, heads, &ab.Dv, &ab.dq_acc);
  ab.dq = ab.dk = ab.dv = view(dqkv0, dqkv1, 3 * d);
  ab.dq_col0 = 0; ab.dk_col0 = d; ab.dv_col0 = 2 * d;
  ab.impl = impl;
  return attention_bwd(ab, stream);
}

extern "C" int jagg_test_ln_gate_bwd(int M, int d, int rows_per_seq, int do_ln, int do_gate, const float* dm,
                                     const float* h, const float* mean, const float* rstd, const float* scale,
                                     float* dshift, float* dscale, const float* dh_in, float* dh_out, const void* y,
                                     const float* gate, float* dgate, void* dy, float* dbias, int dtype,
                                     cudaStream_t stream) {
  JAGG_CHECK_ARG(M > 0 && rows_per_seq > 0, "jagg_test_ln_gate_bwd: M=%d rows_per_seq=%d", M, rows_per_seq);
  JAGG_CHECK_ARG(dtype == JAGG_DTYPE_F32 || dtype == JAGG_DTYPE_BF16, "jagg_test_ln_gate_bwd: bad dtype");
  JAGG_CHECK_ARG(!do_ln || (dm && h && mean && rstd && scale && dshift && dscale && dh_out),
                 "jagg_test_ln_gate_bwd: null LayerNorm operand");
  JAGG_CHECK_ARG(!do_gate || (y && gate && dgate && dy), "jagg_test_ln_gate_bwd: null gate operand");
  JAGG_CHECK_ARG(dh_in, "jagg_test_ln_gate_bwd: null dh_in");
  LnGateBwd a{};
  a.M = M; a.d = d; a.rows_per_seq = rows_per_seq;
  a.do_ln = do_ln; a.dm = dm; a.dm_f32 = 1; a.h = h; a.mean = mean; a.rstd = rstd;
  a.scale = scale; a.mod_stride = d; a.dshift = dshift; a.dscale = dscale; a.dmod_stride = d;
  a.dh_in = dh_in; a.dh_out = dh_out;
  a.do_gate = do_gate; a.y = y; a.gate = gate; a.dgate = dgate; a.dy = dy; a.dbias = dbias;
  a.dtype = dtype;
  return launch_ln_gate_bwd(a, stream);
}

static QkNormRope qkn_args(const void* qkv, int64_t ld_qkv, int M, int N, int d, int heads, int n_txt, int gw,
                           const void* qscale, const void* kscale, int rope, int dtype) {
  QkNormRope q{};
  q.qkv = qkv; q.ld_qkv = ld_qkv;
  q.M = M; q.N = N; q.d = d; q.heads = heads; q.n_txt = n_txt; q.gw = gw;
  q.qscale_txt = q.qscale_img = qscale;
  q.kscale_txt = q.kscale_img = kscale;
  q.rope = rope;
  q.dtype = dtype;
  return q;
}

static int qkn_check(const char* name, int M, int N, int d, int heads, int n_txt, int gw, int rope, int dtype) {
  JAGG_CHECK_ARG(M > 0 && N > 0 && M % N == 0, "%s: M=%d not a whole number of %d-token sequences", name, M, N);
  JAGG_CHECK_ARG(dtype == JAGG_DTYPE_F32 || dtype == JAGG_DTYPE_BF16, "%s: bad dtype", name);
  JAGG_CHECK_ARG(n_txt >= 0 && n_txt <= N, "%s: n_txt=%d outside [0, %d]", name, n_txt, N);
  JAGG_CHECK_ARG(!rope || (gw > 0 && (N - n_txt) % gw == 0), "%s: %d image tokens not a grid %d wide", name,
                 N - n_txt, gw);
  (void)d; (void)heads;
  return JAGG_OK;
}

extern "C" int jagg_test_qk_norm_rope_fwd(const void* qkv, int64_t ld_qkv, int M, int N, int d, int heads, int n_txt,
                                          int gw, const void* qscale, const void* kscale, int rope, void* qk_out,
                                          float* rq, float* rk, int dtype, cudaStream_t stream) {
  JAGG_TRY(qkn_check("jagg_test_qk_norm_rope_fwd", M, N, d, heads, n_txt, gw, rope, dtype));
  JAGG_CHECK_ARG(qkv && qscale && kscale && qk_out && rq && rk, "jagg_test_qk_norm_rope_fwd: null pointer");
  QkNormRope q = qkn_args(qkv, ld_qkv, M, N, d, heads, n_txt, gw, qscale, kscale, rope, dtype);
  q.qk_out = qk_out; q.rq = rq; q.rk = rk;
  return launch_qk_norm_rope_fwd(q, stream);
}

extern "C" int jagg_test_qk_norm_rope_bwd(const void* qkv, int64_t ld_qkv, int M, int N, int d, int heads, int n_txt,
                                          int gw, const void* qscale, const void* kscale, int rope, const float* rq,
                                          const float* rk, void* dqk, int64_t ld_dqk, float* dqscale, float* dkscale,
                                          int dtype, cudaStream_t stream) {
  JAGG_TRY(qkn_check("jagg_test_qk_norm_rope_bwd", M, N, d, heads, n_txt, gw, rope, dtype));
  JAGG_CHECK_ARG(qkv && qscale && kscale && rq && rk && dqk && dqscale && dkscale,
                 "jagg_test_qk_norm_rope_bwd: null pointer");
  QkNormRopeBwd b{};
  b.f = qkn_args(qkv, ld_qkv, M, N, d, heads, n_txt, gw, qscale, kscale, rope, dtype);
  b.f.rq = const_cast<float*>(rq); b.f.rk = const_cast<float*>(rk);
  b.dqk = dqk; b.ld_dqk = ld_dqk;
  b.dqs_txt = b.dqs_img = dqscale;
  b.dks_txt = b.dks_img = dkscale;
  return launch_qk_norm_rope_bwd(b, stream);
}

extern "C" int jagg_test_colsum(const void* X, int x_f32, int rows, int cols, int64_t ld, float* db,
                                cudaStream_t stream) {
  JAGG_CHECK_ARG(X && db && rows > 0 && cols > 0 && ld >= cols, "jagg_test_colsum: bad arguments");
  return launch_colsum(X, x_f32, x_f32 ? JAGG_DTYPE_F32 : JAGG_DTYPE_BF16, rows, cols, ld, db, stream);
}
