// GRPO step signals (Phase 2), JAGG aggregation (Phase 3) and gradient reductions.
//
// Both backbone families of Eq. logprob have a transition mean that is affine in the model
// output y_j (the velocity v_j or the noise prediction eps_j): mu_j = a_j z_j + c_j y_j, with
//   rectified flow       a_j = 1,                        c_j = t_{j+1} - t_j;
//   epsilon prediction   a_j = alpha_{j+1} / alpha_j,    c_j = -alpha_{j+1} (sigma_j / alpha_j
//                                                               - sigma_{j+1} / alpha_{j+1})
// ((alpha, sigma) the diffusion schedule at the window's times).  So r_ij = z_{j+1} - mu_j and
// d logp / d y_ij = r_ij c_j / sigma_j^2 for both, and one set of kernels serves both.
//
// grpo_step_signals runs in three launches:
//   1. advantages A_i (Eq. advantage) from the group's rewards, and the W pairs (a_j, c_j);
//   2. ||r_ij||^2, one CTA per (i, j, chunk of D), partial sums in f64 written to the
//      workspace (fixed order: deterministic);
//   3. per (i, j): log-prob (Eq. logprob), ratio, clip decision (Eq. grpo_loss), the
//      coefficient k_ij = scale (-A_i) rho_ij c_j / sigma_j^2 (0 when clipped); then one
//      elementwise pass writes s_ij = k_ij r_ij and/or the aggregated cotangents
//      sum_j (1 - alpha_j) s_ij and sum_j alpha_j s_ij (Eq. alpha, Eq. s_base_corr).
// The v-hat / z tiles of a window are read twice; at the paper's shapes they fit in L2.
#include <mutex>

#include "common.cuh"

namespace jagg {

int unit_status_signals(unsigned* v, int clear) { return read_unit_status(v, clear); }

namespace {

constexpr int SIG_THREADS = 256;
constexpr int SIG_PER_THREAD = 32;
constexpr int SIG_CHUNK = SIG_THREADS * SIG_PER_THREAD;  // elements of D per CTA in pass 2

__device__ __forceinline__ float ldv_any(const void* p, int64_t i, int is_f32) {
  return is_f32 ? static_cast<const float*>(p)[i] : __bfloat162float(static_cast<const bf16*>(p)[i]);
}

// An f64 mean coefficient as an unevaluated sum of two floats (hi + lo).  Rounding a_j or c_j
// to one float shifts r_ij by the same relative amount at every element, an error that does
// not average out over D and reaches the log-prob as ~1e-7 * sqrt(D) |z| |r| / sigma^2.
struct Coef2 {
  float hi, lo;
};
__device__ __forceinline__ Coef2 split_coef(double x) {
  const float hi = (float)x;
  return Coef2{hi, (float)(x - (double)hi)};
}
// r = z1 - a z0 - c y: the hi products cancel most of z1 exactly inside the first two fmas; the
// lo terms are small corrections.
__device__ __forceinline__ float resid(float z1, float z0, float y, Coef2 a, Coef2 c) {
  float r = fmaf(-a.hi, z0, z1);
  r = fmaf(-c.hi, y, r);
  r = fmaf(-a.lo, z0, r);
  return fmaf(-c.lo, y, r);
}

// The mean coefficients (a_j, c_j) of one step: the flow Euler step, or (eps) the DDIM step
// of the schedule values a0 = alpha_j, a1 = alpha_{j+1}, s0 = sigma_j, s1 = sigma_{j+1}.
// False (and a = c = 0) when an alpha is not positive.  The step signals and the rollout
// sampler both take their coefficients from here, so both see the same f64 values.
__device__ __forceinline__ bool mean_coef(double t0, double t1, bool eps, double a0, double a1, double s0, double s1,
                                          double* a, double* c) {
  if (!eps) {
    *a = 1.0;
    *c = t1 - t0;
    return true;
  }
  if (a0 > 0.0 && a1 > 0.0) {
    *a = a1 / a0;
    *c = -a1 * (s0 / a0 - s1 / a1);
    return true;
  }
  *a = 0.0;
  *c = 0.0;
  return false;
}

// One warp.  Lane 0: the advantages.  All lanes: the mean coefficients mc[j] = a_j,
// mc[W + j] = c_j; sched_alpha == nullptr selects the rectified-flow step.
__global__ void prep_kernel(const float* rewards, int G, double adv_eps, double adv_clip, double* adv, const double* t,
                            const double* sched_alpha, const double* sched_sigma, int W, double* mc) {
  if (blockIdx.x != 0) return;
  for (int j = threadIdx.x; j < W; j += 32) {
    const bool eps = sched_alpha != nullptr;
    double a, c;
    if (!mean_coef(t[j], t[j + 1], eps, eps ? sched_alpha[j] : 0.0, eps ? sched_alpha[j + 1] : 0.0,
                   eps ? sched_sigma[j] : 0.0, eps ? sched_sigma[j + 1] : 0.0, &a, &c))
      set_device_status(JAGG_DEV_BADARG);
    mc[j] = a;
    mc[W + j] = c;
  }
  if (threadIdx.x != 0) return;
  double mu = 0.0;
  for (int i = 0; i < G; ++i) mu += (double)rewards[i];
  mu /= G;
  double ss = 0.0;
  for (int i = 0; i < G; ++i) {
    const double d = (double)rewards[i] - mu;
    ss += d * d;
  }
  const double sd = G > 1 ? sqrt(ss / (G - 1)) : 0.0;
  for (int i = 0; i < G; ++i) {
    double a = ((double)rewards[i] - mu) / (sd + adv_eps);
    a = a > adv_clip ? adv_clip : (a < -adv_clip ? -adv_clip : a);
    adv[i] = a;
  }
}

// sum of r(k)^2 over the CTA's chunk of D (k = blockIdx.x * SIG_CHUNK + ...), valid in thread
// 0: f32 partial sums folded into f64 every 8 terms, then a fixed-order block reduction.  The
// rollout sampler and the step signals share it, so equal residuals give equal log-probs.
template <class R>
__device__ __forceinline__ double chunk_sq_sum(int64_t D, R r_at) {
  const int64_t k0 = (int64_t)blockIdx.x * SIG_CHUNK;
  double acc = 0.0;
  float part = 0.f;
#pragma unroll 4
  for (int u = 0; u < SIG_PER_THREAD; ++u) {
    const int64_t k = k0 + threadIdx.x + (int64_t)u * SIG_THREADS;
    if (k < D) {
      const float r = r_at(k);
      part = fmaf(r, r, part);
    }
    if ((u & 7) == 7) {  // fold every 8 terms into the f64 accumulator
      acc += (double)part;
      part = 0.f;
    }
  }
  acc += (double)part;
  acc = warp_sum(acc);
  __shared__ double red[SIG_THREADS / 32];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x / 32] = acc;
  __syncthreads();
  double s = 0.0;
  if (threadIdx.x == 0)
    for (int w = 0; w < SIG_THREADS / 32; ++w) s += red[w];
  return s;
}

// Eq. logprob from the squared residual norm.  Written with explicitly rounded operations so
// that no call site contracts it into a different fused multiply-add: the rollout sampler
// and the step signals must agree to the last bit.
__device__ __forceinline__ double gauss_logp(double rr, double sg, int64_t D) {
  const double quad = __ddiv_rn(rr, __dmul_rn(2.0, __dmul_rn(sg, sg)));
  const double norm = __dmul_rn((double)D, log(__dmul_rn(sqrt(2.0 * 3.14159265358979323846), sg)));
  return __dsub_rn(-quad, norm);
}

// grid: (chunks, G*W)
__global__ void __launch_bounds__(SIG_THREADS) resid_norm_kernel(const void* v, int v_f32, const float* z,
                                                                 const double* mc, int W, int64_t D, double* partial) {
  const int ij = blockIdx.y;
  const int i = ij / W, j = ij % W;
  const Coef2 a = split_coef(mc[j]), c = split_coef(mc[W + j]);
  const float* z0 = z + ((int64_t)i * (W + 1) + j) * D;
  const float* z1 = z0 + D;
  const int64_t vb = ((int64_t)i * W + j) * D;
  const double s =
      chunk_sq_sum(D, [&](int64_t k) { return resid(z1[k], z0[k], ldv_any(v, vb + k, v_f32), a, c); });
  if (threadIdx.x == 0) partial[(int64_t)ij * gridDim.x + blockIdx.x] = s;
}

// One thread per (i, j).
__global__ void logprob_kernel(const double* partial, int chunks, const double* mc, const double* sigma,
                               const double* logp_old, const double* adv, int G, int W, int64_t D, double clip_eps,
                               double scale, double* logp_new, double* ratio, uint8_t* clipped, float* coef) {
  const int ij = blockIdx.x * blockDim.x + threadIdx.x;
  if (ij >= G * W) return;
  const int i = ij / W, j = ij % W;
  double rr = 0.0;
  for (int c = 0; c < chunks; ++c) rr += partial[(int64_t)ij * chunks + c];
  const double sg = sigma[j];
  const double c = mc[W + j];
  const double lp = gauss_logp(rr, sg, D);
  const double rho = exp(lp - logp_old[ij]);
  const double a = adv[i];
  const bool clip = (a > 0.0 && rho > 1.0 + clip_eps) || (a < 0.0 && rho < 1.0 - clip_eps);
  logp_new[ij] = lp;
  ratio[ij] = rho;
  clipped[ij] = clip ? 1 : 0;
  coef[ij] = clip ? 0.f : (float)(scale * (-a) * rho * c / (sg * sg));
}

// grid: (ceil(D / SIG_THREADS / 4), G).  Each thread: 4 consecutive elements of D.
__global__ void __launch_bounds__(SIG_THREADS) apply_kernel(const void* v, int v_f32, const float* z, const double* t,
                                                            const double* mc, const float* coef, int G, int W,
                                                            int64_t D, float* s_out, float* cot_out) {
  const int i = blockIdx.y;
  const int64_t kbase = ((int64_t)blockIdx.x * SIG_THREADS + threadIdx.x) * 4;
  if (kbase >= D) return;
  const double den = t[0] - t[W - 1];
  float base[4] = {0.f, 0.f, 0.f, 0.f}, corr[4] = {0.f, 0.f, 0.f, 0.f};
  for (int j = 0; j < W; ++j) {
    const Coef2 ma = split_coef(mc[j]), mcj = split_coef(mc[W + j]);
    const float c = coef[i * W + j];
    const float al = cot_out ? (den != 0.0 ? (float)((t[0] - t[j]) / den) : 0.f) : 0.f;
    const float* z0 = z + ((int64_t)i * (W + 1) + j) * D;
    const float* z1 = z0 + D;
    const int64_t vb = ((int64_t)i * W + j) * D;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int64_t k = kbase + e;
      if (k < D) {
        const float r = resid(z1[k], z0[k], ldv_any(v, vb + k, v_f32), ma, mcj);
        const float s = c * r;
        if (s_out) s_out[vb + k] = s;
        base[e] += (1.f - al) * s;
        corr[e] += al * s;
      }
    }
  }
  if (cot_out) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int64_t k = kbase + e;
      if (k < D) {
        cot_out[(int64_t)i * D + k] = base[e];
        cot_out[((int64_t)G + i) * D + k] = corr[e];
      }
    }
  }
}

// Rollout sampler step.  grid: (chunks, G).  z_{j+1} = a z_j + c y + sigma xi, rounded to f32
// and stored, then its residual against the mean enters the same chunk sums as the signals.
struct RolloutStep {
  const void* y;
  int y_f32;
  const float* z_cur;
  const float* xi;
  float* z_next;
  void* z_model;  // optional dense [G, D] copy of z_next in the model's dtype (next forward's input)
  int zm_f32;
  int64_t D, z_ld, y_ld, xi_ld;
  double t0, t1, sigma, a0, a1, s0, s1;
  int eps;
  double* partial;
};

__global__ void __launch_bounds__(SIG_THREADS) rollout_step_kernel(RolloutStep p) {
  const int i = blockIdx.y;
  double ad, cd;
  if (!mean_coef(p.t0, p.t1, p.eps != 0, p.a0, p.a1, p.s0, p.s1, &ad, &cd) && blockIdx.x == 0 && i == 0 &&
      threadIdx.x == 0)
    set_device_status(JAGG_DEV_BADARG);
  const Coef2 a = split_coef(ad), c = split_coef(cd);
  const float sg = (float)p.sigma;
  const float* z0 = p.z_cur + (int64_t)i * p.z_ld;
  float* z1 = p.z_next + (int64_t)i * p.z_ld;
  const float* xi = p.xi + (int64_t)i * p.xi_ld;
  const int64_t yb = (int64_t)i * p.y_ld;
  const double s = chunk_sq_sum(p.D, [&](int64_t k) {
    const float zk = z0[k], yk = ldv_any(p.y, yb + k, p.y_f32);
    float m = fmaf(a.lo, zk, c.lo * yk);
    m = fmaf(c.hi, yk, m);
    m = fmaf(a.hi, zk, m);
    const float zn = fmaf(sg, xi[k], m);
    z1[k] = zn;
    if (p.z_model) {
      if (p.zm_f32)
        static_cast<float*>(p.z_model)[(int64_t)i * p.D + k] = zn;
      else
        static_cast<bf16*>(p.z_model)[(int64_t)i * p.D + k] = __float2bfloat16_rn(zn);
    }
    return resid(zn, zk, yk, a, c);
  });
  if (threadIdx.x == 0) p.partial[(int64_t)i * gridDim.x + blockIdx.x] = s;
}

__global__ void rollout_logp_kernel(const double* partial, int chunks, double sigma, int G, int64_t D,
                                    double* logp, int64_t logp_ld) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= G) return;
  double rr = 0.0;
  for (int c = 0; c < chunks; ++c) rr += partial[(int64_t)i * chunks + c];
  logp[(int64_t)i * logp_ld] = gauss_logp(rr, sigma, D);
}

__global__ void check_alpha_kernel(const double* t, int W) {
  if (threadIdx.x == 0 && blockIdx.x == 0 && !(t[0] - t[W - 1] != 0.0)) set_device_status(JAGG_DEV_BADARG);
}

__global__ void aggregate_kernel(const float* s, const double* t, int G, int W, int64_t D, float* cot) {
  const int i = blockIdx.y;
  const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= D) return;
  const double den = t[0] - t[W - 1];
  float base = 0.f, corr = 0.f;
  if (den != 0.0) {
    for (int j = 0; j < W; ++j) {
      const float al = (float)((t[0] - t[j]) / den);
      const float v = s[((int64_t)i * W + j) * D + k];
      base += (1.f - al) * v;
      corr += al * v;
    }
  }
  cot[(int64_t)i * D + k] = base;
  cot[((int64_t)G + i) * D + k] = corr;
}

__global__ void aggregate_span_kernel(const float* s, int64_t ld, const double* t, double t_first, double t_last, int G,
                                      int n, int64_t D, float* cot, int accumulate) {
  const int i = blockIdx.y;
  const int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= D) return;
  const double den = t_first - t_last;
  float base = 0.f, corr = 0.f;
  for (int j = 0; j < n; ++j) {
    const float al = (float)((t_first - t[j]) / den);
    const float v = s[(int64_t)i * ld + (int64_t)j * D + k];
    base += (1.f - al) * v;
    corr += al * v;
  }
  float* b = cot + (int64_t)i * D + k;
  float* c = cot + ((int64_t)G + i) * D + k;
  if (accumulate) {
    *b += base;
    *c += corr;
  } else {
    *b = base;
    *c = corr;
  }
}

// ------------------------------------------------------------------ grad_reduce
constexpr int GR_BLOCKS = 1024;
constexpr int GR_THREADS = 256;

// HAS_B: a second vector b (else <a, b> = |b|^2 = |a|^2 and b is not read); HAS_ACC: the
// update acc += alpha a.  Each thread loads a run of 8 float4 of each input before using any
// of them, so 8 (16) loads per thread are in flight; f32 sums over a run fold into f64.
template <bool HAS_B, bool HAS_ACC>
__global__ void __launch_bounds__(GR_THREADS) grad_reduce_kernel(const float* a, const float* b, int64_t P,
                                                                 float alpha, float* acc, double* partial) {
  double sab = 0.0, saa = 0.0, sbb = 0.0;
  const int64_t nvec = P / 4;
  const float4* a4 = reinterpret_cast<const float4*>(a);
  const float4* b4 = reinterpret_cast<const float4*>(b);
  float4* c4 = reinterpret_cast<float4*>(acc);
  const int64_t stride = (int64_t)GR_BLOCKS * GR_THREADS;
  const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int64_t idx = (int64_t)blockIdx.x * GR_THREADS + threadIdx.x; idx < nvec; idx += 8 * stride) {
    float4 x[8], y[8];
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      const int64_t q = idx + (int64_t)r * stride;
      x[r] = q < nvec ? a4[q] : zero;
      if constexpr (HAS_B) y[r] = q < nvec ? b4[q] : zero;
    }
    float fab = 0.f, faa = 0.f, fbb = 0.f;
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      faa += x[r].x * x[r].x + x[r].y * x[r].y + x[r].z * x[r].z + x[r].w * x[r].w;
      if constexpr (HAS_B) {
        fab += x[r].x * y[r].x + x[r].y * y[r].y + x[r].z * y[r].z + x[r].w * y[r].w;
        fbb += y[r].x * y[r].x + y[r].y * y[r].y + y[r].z * y[r].z + y[r].w * y[r].w;
      }
    }
    if constexpr (HAS_ACC) {
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        const int64_t q = idx + (int64_t)r * stride;
        if (q < nvec) {
          float4 c = c4[q];
          c.x += alpha * x[r].x; c.y += alpha * x[r].y; c.z += alpha * x[r].z; c.w += alpha * x[r].w;
          c4[q] = c;
        }
      }
    }
    if constexpr (!HAS_B) fab = fbb = faa;
    sab += fab;
    saa += faa;
    sbb += fbb;
  }
  // scalar tail (P % 4), handled by block 0
  if (blockIdx.x == 0) {
    for (int64_t k = nvec * 4 + threadIdx.x; k < P; k += GR_THREADS) {
      const float x = a[k], y = b ? b[k] : a[k];
      sab += (double)x * y;
      saa += (double)x * x;
      sbb += (double)y * y;
      if (acc) acc[k] += alpha * x;
    }
  }
  if (!partial) return;
  sab = warp_sum(sab);
  saa = warp_sum(saa);
  sbb = warp_sum(sbb);
  __shared__ double red[3][GR_THREADS / 32];
  const int w = threadIdx.x / 32;
  if ((threadIdx.x & 31) == 0) {
    red[0][w] = sab;
    red[1][w] = saa;
    red[2][w] = sbb;
  }
  __syncthreads();
  if (threadIdx.x < 3) {
    double s = 0.0;
    for (int i = 0; i < GR_THREADS / 32; ++i) s += red[threadIdx.x][i];
    partial[(int64_t)blockIdx.x * 3 + threadIdx.x] = s;
  }
}

__global__ void grad_reduce_final(const double* partial, double* out3) {
  if (threadIdx.x < 3) {
    double s = 0.0;
    for (int i = 0; i < GR_BLOCKS; ++i) s += partial[(int64_t)i * 3 + threadIdx.x];
    out3[threadIdx.x] = s;
  }
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// The (a_j, c_j) pairs at the head of the signals workspace, padded to 16 bytes.
int64_t mean_coef_bytes(int W) { return ((int64_t)2 * W * 8 + 15) / 16 * 16; }

}  // namespace

}  // namespace jagg

using namespace jagg;

// ------------------------------------------------------------------ C ABI
extern "C" int64_t jagg_signals_workspace_bytes(int G, int W, int64_t D) {
  if (G <= 0 || W <= 0 || D <= 0) return 0;
  const int64_t chunks = (D + SIG_CHUNK - 1) / SIG_CHUNK;
  return mean_coef_bytes(W) + (int64_t)G * W * chunks * 8 + (int64_t)G * W * 4 + 64;
}

namespace jagg {
namespace {
int step_signals(const char* name, const void* v_hat, int v_dtype, const float* z, const double* t,
                 const double* sched_alpha, const double* sched_sigma, const double* sigma, const double* logp_old,
                 const float* rewards, int G, int W, int64_t D, double clip_eps, double adv_clip, double adv_eps,
                 double scale, float* s_out, float* cot_out, double* logp_new, double* ratio, uint8_t* clipped,
                 double* adv_out, void* ws, size_t ws_bytes, cudaStream_t stream) {
  JAGG_CHECK_ARG(G > 0 && W > 0 && D > 0, "%s: G=%d W=%d D=%lld must be positive", name, G, W, (long long)D);
  JAGG_CHECK_ARG(G <= 65535 && (int64_t)G * W <= 65535, "%s: G*W too large", name);
  JAGG_CHECK_ARG(v_dtype == JAGG_DTYPE_F32 || v_dtype == JAGG_DTYPE_BF16, "%s: bad v_dtype", name);
  JAGG_CHECK_ARG(v_hat && z && t && sigma && logp_old && rewards && logp_new && ratio && clipped && adv_out && ws,
                 "%s: null pointer", name);
  JAGG_CHECK_ARG(!cot_out || W >= 2, "%s: aggregation needs W >= 2", name);
  JAGG_CHECK_ARG(clip_eps >= 0.0 && adv_clip >= 0.0 && adv_eps >= 0.0, "%s: negative constant", name);
  const int64_t need = jagg_signals_workspace_bytes(G, W, D);
  if ((int64_t)ws_bytes < need) {
    set_last_error("%s: workspace %zu < %lld bytes", name, ws_bytes, (long long)need);
    return JAGG_ERR_WORKSPACE;
  }
  JAGG_CHECK_ARG(aligned16(ws), "%s: workspace not 16-byte aligned", name);
  const int chunks = (int)((D + SIG_CHUNK - 1) / SIG_CHUNK);
  double* mc = static_cast<double*>(ws);
  double* partial = reinterpret_cast<double*>(static_cast<char*>(ws) + mean_coef_bytes(W));
  float* coef = reinterpret_cast<float*>(partial + (int64_t)G * W * chunks);
  const int vf32 = v_dtype == JAGG_DTYPE_F32;
  const int tok = prof_start(stream);
  prep_kernel<<<1, 32, 0, stream>>>(rewards, G, adv_eps, adv_clip, adv_out, t, sched_alpha, sched_sigma, W, mc);
  JAGG_LAUNCHED();
  resid_norm_kernel<<<dim3(chunks, G * W), SIG_THREADS, 0, stream>>>(v_hat, vf32, z, mc, W, D, partial);
  JAGG_LAUNCHED();
  logprob_kernel<<<ceil_div((int64_t)G * W, 128), 128, 0, stream>>>(partial, chunks, mc, sigma, logp_old, adv_out, G,
                                                                     W, D, clip_eps, scale, logp_new, ratio, clipped,
                                                                     coef);
  JAGG_LAUNCHED();
  if (s_out || cot_out) {
    if (cot_out) {
      check_alpha_kernel<<<1, 32, 0, stream>>>(t, W);
      JAGG_LAUNCHED();
    }
    const int gx = ceil_div(D, (int64_t)SIG_THREADS * 4);
    apply_kernel<<<dim3(gx, G), SIG_THREADS, 0, stream>>>(v_hat, vf32, z, t, mc, coef, G, W, D, s_out,
                                                          cot_out);
    JAGG_LAUNCHED();
  }
  // algorithmic bytes: v-hat and the W + 1 latents of every sample read once, the signals
  // (G W rows) or the cotangents (2G rows) written in f32
  const double out_rows = s_out ? (double)G * W : (cot_out ? 2.0 * G : 0.0);
  prof_stop(tok, stream, PROF_SIGNALS, 0.0,
            (double)D * ((double)G * W * (vf32 ? 4.0 : 2.0) + (double)G * (W + 1) * 4.0 + out_rows * 4.0));
  return JAGG_OK;
}
}  // namespace
}  // namespace jagg

extern "C" int grpo_step_signals(const void* v_hat, int v_dtype, const float* z, const double* t, const double* sigma,
                                 const double* logp_old, const float* rewards, int G, int W, int64_t D,
                                 double clip_eps, double adv_clip, double adv_eps, double scale, float* s_out,
                                 float* cot_out, double* logp_new, double* ratio, uint8_t* clipped, double* adv_out,
                                 void* ws, size_t ws_bytes, cudaStream_t stream) {
  return step_signals("grpo_step_signals", v_hat, v_dtype, z, t, nullptr, nullptr, sigma, logp_old, rewards, G, W, D,
                      clip_eps, adv_clip, adv_eps, scale, s_out, cot_out, logp_new, ratio, clipped, adv_out, ws,
                      ws_bytes, stream);
}

extern "C" int grpo_step_signals_eps(const void* eps_hat, int eps_dtype, const float* z, const double* t,
                                     const double* sched_alpha, const double* sched_sigma, const double* sigma,
                                     const double* logp_old, const float* rewards, int G, int W, int64_t D,
                                     double clip_eps, double adv_clip, double adv_eps, double scale, float* s_out,
                                     float* cot_out, double* logp_new, double* ratio, uint8_t* clipped,
                                     double* adv_out, void* ws, size_t ws_bytes, cudaStream_t stream) {
  JAGG_CHECK_ARG(sched_alpha && sched_sigma, "grpo_step_signals_eps: null schedule");
  return step_signals("grpo_step_signals_eps", eps_hat, eps_dtype, z, t, sched_alpha, sched_sigma, sigma, logp_old,
                      rewards, G, W, D, clip_eps, adv_clip, adv_eps, scale, s_out, cot_out, logp_new, ratio, clipped,
                      adv_out, ws, ws_bytes, stream);
}

extern "C" int64_t jagg_rollout_workspace_bytes(int G, int64_t D) {
  if (G <= 0 || D <= 0) return 0;
  return (int64_t)G * ((D + SIG_CHUNK - 1) / SIG_CHUNK) * 8 + 64;
}

extern "C" int jagg_rollout_step(const void* y_hat, int y_dtype, int64_t y_sample_stride, const float* z_cur,
                                 float* z_next, int64_t z_sample_stride, const float* xi, int64_t xi_sample_stride,
                                 int G, int64_t D, double t_cur, double t_next, double sigma, const double* sched,
                                 double* logp, int64_t logp_stride, void* z_model, int z_model_dtype, void* ws,
                                 size_t ws_bytes, cudaStream_t stream) {
  JAGG_CHECK_ARG(y_hat && z_cur && z_next && xi && logp && ws, "jagg_rollout_step: null pointer");
  JAGG_CHECK_ARG(G > 0 && G <= 65535 && D > 0, "jagg_rollout_step: bad G=%d or D=%lld", G, (long long)D);
  JAGG_CHECK_ARG(y_dtype == JAGG_DTYPE_F32 || y_dtype == JAGG_DTYPE_BF16, "jagg_rollout_step: bad y_dtype");
  JAGG_CHECK_ARG(sigma > 0.0, "jagg_rollout_step: sigma %g must be positive", sigma);
  const int64_t zl = z_sample_stride ? z_sample_stride : D, yl = y_sample_stride ? y_sample_stride : D,
                xl = xi_sample_stride ? xi_sample_stride : D;
  JAGG_CHECK_ARG(zl >= D && yl >= D && xl >= D, "jagg_rollout_step: a sample stride is below D");
  JAGG_CHECK_ARG(logp_stride >= 1, "jagg_rollout_step: logp_stride must be >= 1");
  JAGG_CHECK_ARG(!z_model || z_model_dtype == JAGG_DTYPE_F32 || z_model_dtype == JAGG_DTYPE_BF16,
                 "jagg_rollout_step: bad z_model_dtype");
  const int64_t need = jagg_rollout_workspace_bytes(G, D);
  if ((int64_t)ws_bytes < need) {
    set_last_error("jagg_rollout_step: workspace %zu < %lld bytes", ws_bytes, (long long)need);
    return JAGG_ERR_WORKSPACE;
  }
  JAGG_CHECK_ARG(aligned16(ws), "jagg_rollout_step: workspace not 16-byte aligned");
  const int chunks = (int)((D + SIG_CHUNK - 1) / SIG_CHUNK);
  RolloutStep p{y_hat, y_dtype == JAGG_DTYPE_F32, z_cur, xi, z_next, z_model, z_model_dtype == JAGG_DTYPE_F32,
                D, zl, yl, xl, t_cur, t_next, sigma,
                sched ? sched[0] : 0.0, sched ? sched[1] : 0.0, sched ? sched[2] : 0.0, sched ? sched[3] : 0.0,
                sched ? 1 : 0, static_cast<double*>(ws)};
  rollout_step_kernel<<<dim3(chunks, G), SIG_THREADS, 0, stream>>>(p);
  JAGG_LAUNCHED();
  rollout_logp_kernel<<<ceil_div((int64_t)G, 128), 128, 0, stream>>>(static_cast<double*>(ws), chunks, sigma, G, D,
                                                                      logp, logp_stride);
  JAGG_LAUNCHED();
  return JAGG_OK;
}

extern "C" int jagg_aggregate(const float* s, const double* t_window, int G, int W, int64_t D, float* cot,
                              cudaStream_t stream) {
  JAGG_CHECK_ARG(s && t_window && cot, "jagg_aggregate: null pointer");
  JAGG_CHECK_ARG(G > 0 && G <= 65535 && D > 0, "jagg_aggregate: bad G=%d or D=%lld", G, (long long)D);
  JAGG_CHECK_ARG(W >= 2, "jagg_aggregate: W=%d, the endpoints must differ (W >= 2)", W);
  check_alpha_kernel<<<1, 32, 0, stream>>>(t_window, W);
  JAGG_LAUNCHED();
  aggregate_kernel<<<dim3(ceil_div(D, 256), G), 256, 0, stream>>>(s, t_window, G, W, D, cot);
  JAGG_LAUNCHED();
  return JAGG_OK;
}

extern "C" int jagg_aggregate_span(const float* s, int64_t s_sample_stride, const double* t_steps, double t_first,
                                   double t_last, int G, int n, int64_t D, float* cot, int accumulate,
                                   cudaStream_t stream) {
  JAGG_CHECK_ARG(s && t_steps && cot, "jagg_aggregate_span: null pointer");
  JAGG_CHECK_ARG(G > 0 && G <= 65535 && n > 0 && D > 0, "jagg_aggregate_span: bad G=%d, n=%d or D=%lld", G, n,
                 (long long)D);
  JAGG_CHECK_ARG(t_first != t_last, "jagg_aggregate_span: the window endpoints must differ");
  const int64_t ld = s_sample_stride ? s_sample_stride : (int64_t)n * D;
  JAGG_CHECK_ARG(ld >= (int64_t)n * D, "jagg_aggregate_span: sample stride %lld below n * D", (long long)ld);
  aggregate_span_kernel<<<dim3(ceil_div(D, 256), G), 256, 0, stream>>>(s, ld, t_steps, t_first, t_last, G, n, D, cot,
                                                                       accumulate);
  JAGG_LAUNCHED();
  return JAGG_OK;
}

extern "C" int jagg_route(int n_windows, double jagg_frac, const double* cos, double tau, uint8_t* route,
                          double* derived_frac) {
  JAGG_CHECK_ARG(n_windows > 0 && route, "jagg_route: n_windows=%d / null route", n_windows);
  if (!cos) {
    JAGG_CHECK_ARG(jagg_frac >= 0.0 && jagg_frac <= 1.0, "jagg_route: jagg_frac %g outside [0, 1]", jagg_frac);
    int n_jagg = (int)floor(jagg_frac * n_windows + 1e-9);
    if (n_jagg > n_windows) n_jagg = n_windows;
    for (int w = 0; w < n_windows; ++w) route[w] = w < n_jagg ? 1 : 0;
    if (derived_frac) *derived_frac = (double)n_jagg / n_windows;
    return JAGG_OK;
  }
  int prefix = 0;
  bool in_prefix = true;
  for (int w = 0; w < n_windows; ++w) {
    route[w] = cos[w] >= tau ? 1 : 0;
    if (in_prefix && route[w])
      ++prefix;
    else
      in_prefix = false;
  }
  if (derived_frac) *derived_frac = (double)prefix / n_windows;
  return JAGG_OK;
}

extern "C" int64_t jagg_grad_reduce_workspace_bytes(int64_t P) {
  (void)P;
  return (int64_t)GR_BLOCKS * 3 * 8;
}

extern "C" int grad_reduce(const float* a, const float* b, int64_t P, float alpha, float* acc, double* out3, void* ws,
                           size_t ws_bytes, cudaStream_t stream) {
  JAGG_CHECK_ARG(a && P > 0, "grad_reduce: null input or P=%lld", (long long)P);
  JAGG_CHECK_ARG(aligned16(a) && (!b || aligned16(b)) && (!acc || aligned16(acc)),
                 "grad_reduce: buffers must be 16-byte aligned");
  if (!acc && !out3) return JAGG_OK;
  if (out3) {
    if (!ws || (int64_t)ws_bytes < jagg_grad_reduce_workspace_bytes(P)) {
      set_last_error("grad_reduce: workspace too small");
      return JAGG_ERR_WORKSPACE;
    }
  }
  const int tok = prof_start(stream);
  double* part = out3 ? static_cast<double*>(ws) : nullptr;
  if (b && acc)
    grad_reduce_kernel<true, true><<<GR_BLOCKS, GR_THREADS, 0, stream>>>(a, b, P, alpha, acc, part);
  else if (b)
    grad_reduce_kernel<true, false><<<GR_BLOCKS, GR_THREADS, 0, stream>>>(a, b, P, alpha, acc, part);
  else if (acc)
    grad_reduce_kernel<false, true><<<GR_BLOCKS, GR_THREADS, 0, stream>>>(a, b, P, alpha, acc, part);
  else
    grad_reduce_kernel<false, false><<<GR_BLOCKS, GR_THREADS, 0, stream>>>(a, b, P, alpha, acc, part);
  JAGG_LAUNCHED();
  if (out3) {
    grad_reduce_final<<<1, 32, 0, stream>>>(static_cast<const double*>(ws), out3);
    JAGG_LAUNCHED();
  }
  // algorithmic bytes: a (and b) read, acc read and written
  prof_stop(tok, stream, PROF_GRAD_REDUCE, 0.0, 4.0 * P * (1.0 + (b ? 1.0 : 0.0) + (acc ? 2.0 : 0.0)));
  return JAGG_OK;
}

// ------------------------------------------------------------------ allocation-free variant
// Scratch for grpo_step_signals_static: compiled into the library, one copy per device.
static __device__ __align__(256) unsigned char g_signals_scratch[JAGG_SIGNALS_STATIC_SCRATCH_BYTES];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// The array's device address for the device of `stream`, which must be the current device
// (the address comes from a runtime query on the current device), looked up once per device.
// In host code `g_signals_scratch` names a host-side stand-in, never the device memory itself.
int scratch_for_stream(cudaStream_t stream, void** out) {
  int dev = 0, sdev = 0;
  JAGG_CUDA_TRY(cudaGetDevice(&dev));
  JAGG_CUDA_TRY(cudaStreamGetDevice(stream, &sdev));
  JAGG_CHECK_ARG(sdev == dev, "grpo_step_signals_static: the stream belongs to device %d, the current device is %d",
                 sdev, dev);
  JAGG_CHECK_ARG(dev >= 0 && dev < kMaxDevices, "grpo_step_signals_static: device %d out of range", dev);
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    JAGG_CUDA_TRY(cudaGetSymbolAddress(&p, g_signals_scratch));
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return JAGG_OK;
}
}  // namespace

extern "C" int grpo_step_signals_static(const void* v_hat, int v_dtype, const float* z, const double* t,
                                        const double* sigma, const double* logp_old, const float* rewards, int G,
                                        int W, int64_t D, double clip_eps, double adv_clip, double adv_eps,
                                        double scale, float* s_out, float* cot_out, double* logp_new,
                                        double* ratio, uint8_t* clipped, double* adv_out, cudaStream_t stream) {
  JAGG_CHECK_ARG(G > 0 && W > 0 && D > 0, "grpo_step_signals_static: G=%d W=%d D=%lld must be positive", G, W,
                 (long long)D);
  const int64_t need = jagg_signals_workspace_bytes(G, W, D);
  if (need > (int64_t)JAGG_SIGNALS_STATIC_SCRATCH_BYTES) {
    set_last_error("grpo_step_signals_static: needs %lld scratch bytes, more than the %d compiled in",
                   (long long)need, (int)JAGG_SIGNALS_STATIC_SCRATCH_BYTES);
    return JAGG_ERR_WORKSPACE;
  }
  void* scratch = nullptr;
  JAGG_TRY(scratch_for_stream(stream, &scratch));
  return jagg::step_signals("grpo_step_signals_static", v_hat, v_dtype, z, t, nullptr, nullptr, sigma, logp_old,
                            rewards, G, W, D, clip_eps, adv_clip, adv_eps, scale, s_out, cot_out, logp_new, ratio,
                            clipped, adv_out, scratch, (size_t)JAGG_SIGNALS_STATIC_SCRATCH_BYTES, stream);
}
