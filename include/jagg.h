/*
 * jagg.h -- C ABI of the JAGG backward library for GB300 (sm_103a).
 *
 * JAGG (Jacobian-Aggregated Group Gradient, arxiv 2607.17572) replaces the W per-step
 * DiT backward passes of one window of W sampling steps of diffusion GRPO with one
 * joint vector-Jacobian product at the two window endpoints (Sec. 3.3, Algorithm 1).
 * This library is that update-stage hot path on one GPU:
 *
 *   dit_forward_save   Phase 1: v = DiT(z, t, txt), keeping what Phase 4 needs
 *   grpo_step_signals  Phase 2: s_j = dL_j/dv_j through Eq. logprob and Eq. grpo_loss
 *                      (grpo_step_signals_eps: the same for an epsilon-prediction model)
 *   jagg_aggregate     Phase 3: Eq. alpha and Eq. s_base_corr
 *                      (jagg_aggregate_span: over a span of a window's steps)
 *   jagg_route         jagg_frac routing (Sec. 3.3 and the gradient-quality appendix)
 *   jagg_rollout_step  one rollout sampler step with the log-prob of its sample
 *   dit_joint_vjp      Phase 4: grad += sum_rows J(z_row, t_row)^T cot_row
 *   grad_reduce        gradient accumulation and the cosine / norm-ratio reductions
 *
 * Conventions shared by every entry point:
 *   - Memory is owned by the caller.  Pointers documented "device" must be device
 *     memory of the current CUDA device; "host" pointers are ordinary host memory.
 *     Device buffers must be 16-byte aligned and contiguous, row-major.
 *   - Calls are asynchronous on `stream` unless stated otherwise; results are valid
 *     once the stream has reached them.
 *   - The return value is a status: JAGG_OK (0) or a negative JAGG_ERR_* code.  Argument
 *     errors are detected on the host before anything is launched; jagg_last_error()
 *     returns a description of the most recent error of the calling thread.
 *   - No entry point allocates device memory except jagg_model_create (a small table).
 *     Scratch space is a caller-provided workspace sized by the *_workspace_bytes calls.
 *   - Waits inside kernels are bounded; a wait that gives up sets a device status bit
 *     (read with jagg_device_status) instead of hanging or trapping.
 *
 * bf16 is IEEE bfloat16 stored as uint16; f32/f64 are IEEE float/double.
 */
#ifndef JAGG_H_
#define JAGG_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ----------------------------------------------------------------- status codes */
#define JAGG_OK 0
#define JAGG_ERR_ARG (-1)          /* invalid pointer, size, alignment or config     */
#define JAGG_ERR_UNSUPPORTED (-2)  /* valid request the library does not implement   */
#define JAGG_ERR_CUDA (-3)         /* a CUDA runtime/driver call failed               */
#define JAGG_ERR_TIMEOUT (-4)      /* a bounded device wait gave up                   */
#define JAGG_ERR_WORKSPACE (-5)    /* workspace or saved arena smaller than required  */

#define JAGG_DTYPE_F32 0
#define JAGG_DTYPE_BF16 1

#define JAGG_ARCH_DIT 0    /* single-stream adaLN DiT blocks                           */
#define JAGG_ARCH_MMDIT 1  /* double-stream MMDiT blocks followed by Flux-style single  */

/* Device status bits (jagg_device_status). */
#define JAGG_DEV_STATUS_TIMEOUT 1u
#define JAGG_DEV_STATUS_BADARG 2u

/* Text of the most recent error of the calling thread ("" if none). */
const char* jagg_last_error(void);

/* Reads the device status word (synchronises the device); clears it when `clear` != 0. */
int jagg_device_status(unsigned* status_out, int clear);

/* Number of kernels the library has launched in this process (host-side counter). */
int64_t jagg_launch_count(void);

/* Kernel timing by family.  jagg_profile_enable(1) clears earlier records and starts
 * bracketing the launches of the path's kernels with CUDA events on their stream (this
 * adds two event records per launch); jagg_profile_enable(0) stops.  Families, in this
 * order: gemm_tcgen05, gemm_simt, attention_fwd, attention_bwd, ln_gate_bwd,
 * attention_bwd_aux, qk_norm_rope_bwd, colsum, copy_rows, step_signals, grad_reduce,
 * ln_mod_fwd, qk_norm_rope_fwd (step_signals and grad_reduce cover a whole call of the
 * entry point).  jagg_profile_read synchronises the device and fills up to `cap` entries,
 * one per family: launches, summed device milliseconds, summed algorithmic FLOPs (2 per
 * multiply-add of the products the operation defines) and algorithmic bytes (each input
 * read once, each output written once). */
typedef struct jagg_profile_stat {
  char family[32];
  int64_t launches;
  double ms;
  double flops;
  double bytes;
} jagg_profile_stat;
int jagg_profile_enable(int on);
int jagg_profile_read(jagg_profile_stat* out, int cap, int* n_out);
/* The recorded launches one by one, in launch order (up to `cap`): family, the product's
 * M, N, K (0 for other families), device milliseconds, algorithmic FLOPs and bytes.
 * Synchronises. */
typedef struct jagg_profile_launch {
  char family[32];
  int32_t m, n, k;
  double ms;
  double flops;
  double bytes;
} jagg_profile_launch;
int jagg_profile_launches(jagg_profile_launch* out, int cap, int* n_out);

/* ------------------------------------------------------------------ backbone
 * The velocity network v_theta(z, t, txt).  The paper trains Flux and Qwen-Image
 * (Sec. 4) without describing them; the library implements the pinned DiT / MMDiT of
 * the project's design notes: patch embedding, text projection, sinusoidal t-embedding
 * MLP, adaLN-modulated blocks with tanh-GELU MLPs and joint [txt; img] softmax
 * attention (per-head RMSNorm and 2D RoPE in the MMDiT), and a modulated final layer.
 */
typedef struct jagg_config {
  int32_t arch;          /* JAGG_ARCH_DIT or JAGG_ARCH_MMDIT                          */
  int32_t dtype;         /* storage/compute type of weights and activations           */
  int32_t hidden;        /* d (multiple of 64)                                        */
  int32_t heads;         /* d / heads = head dim: 16 (f32 only), 64 or 128             */
  int32_t mlp;           /* MLP width (multiple of 64)                                */
  int32_t depth;         /* DiT blocks (DIT) or Flux-style single blocks (MMDIT)      */
  int32_t depth_double;  /* double-stream blocks (MMDIT), 0 for DIT                   */
  int32_t in_channels;   /* latent channels C                                         */
  int32_t latent_h;      /* latent height H (multiple of patch)                       */
  int32_t latent_w;      /* latent width W (multiple of patch)                        */
  int32_t patch;         /* patch size p                                              */
  int32_t txt_len;       /* text tokens per sequence                                  */
  int32_t txt_dim;       /* text embedding width (multiple of 8)                      */
  int32_t freq_dim;      /* sinusoidal t-embedding width (256)                        */
} jagg_config;

typedef struct jagg_model* jagg_model_t;

/* Number of scalar parameters, and of parameter tensors, of a configuration. */
int64_t jagg_param_count(const jagg_config* cfg);
int jagg_param_tensor_count(const jagg_config* cfg);

/* Describes parameter tensor `index` (0 <= index < jagg_param_tensor_count): its name
 * (e.g. "blocks.3.qkv.w", NUL-terminated into name[name_cap]), its element offset in
 * the flat parameter buffer and its shape (rows x cols; cols = 1 for vectors).  Matrices
 * are stored [out, in] row-major.  The same offsets index the fp32 gradient buffer. */
int jagg_param_info(const jagg_config* cfg, int index, char* name, size_t name_cap,
                    int64_t* offset, int64_t* rows, int64_t* cols);

/* Creates a model over caller-owned device weights (jagg_param_count elements of
 * cfg->dtype laid out as jagg_param_info describes).  The weights must stay valid and
 * unchanged while the model is used.  Synchronous; allocates a small host table. */
int jagg_model_create(const jagg_config* cfg, const void* weights, jagg_model_t* model_out);
int jagg_model_destroy(jagg_model_t model);

/* Bytes of the saved-activation arena for a forward over B sequences, and of the
 * workspace that dit_forward_save / dit_joint_vjp need for B sequences. */
int64_t jagg_saved_bytes(jagg_model_t model, int B);
int64_t jagg_workspace_bytes(jagg_model_t model, int B);

/* Phase 1 (Sec. 3.3, Algorithm 1): v_out = DiT(z, t, txt) for B sequences.
 *   z      device [B, C, H, W] cfg dtype       network input latents
 *   t      device [B] f32                      network-input times
 *   txt    device [B, txt_len, txt_dim] dtype  text embeddings
 *   v_out  device [B, C, H, W] cfg dtype       predicted velocities
 *   saved  device arena of >= jagg_saved_bytes(B) bytes, or NULL for a forward that
 *          keeps nothing (the middle steps of a window run this way)
 *   ws     device workspace of >= jagg_workspace_bytes(B) bytes                        */
int dit_forward_save(jagg_model_t model, const void* z, const float* t, const void* txt,
                     int B, void* v_out, void* saved, size_t saved_bytes, void* ws,
                     size_t ws_bytes, cudaStream_t stream);

/* Phase 4 (Sec. 3.3 "Joint backward", Algorithm 1): grad += sum_b J(z_b, t_b)^T cot_b,
 * the parameter VJP of every row of a saved forward, in one pass.  For a JAGG window the
 * rows are [z_0 of each sample; z_{W-1} of each sample] and cot = [s_base; s_corr]
 * (Eq. s_base_corr); for the exact per-step path they are the W*G step inputs and cot
 * holds each s_j.  No gradient flows to z or txt (they are fixed samples, Phase 2).
 *   saved  the arena of a dit_forward_save over the same B rows
 *   cot    device [B, C, H, W] f32 cotangents (rounded to cfg dtype inside)
 *   grad   device f32 [jagg_param_count], accumulated (+=), same layout as the weights */
int dit_joint_vjp(jagg_model_t model, const void* saved, size_t saved_bytes, int B,
                  const float* cot, float* grad, void* ws, size_t ws_bytes,
                  cudaStream_t stream);

/* ------------------------------------------------------------------ GRPO signals
 * Phase 2 (Sec. 3.3): for sample i and step j of a window,
 *   r_ij   = z_{i,j+1} - z_{i,j} - v_ij (t_{j+1} - t_j)
 *   logp   = -||r_ij||^2 / (2 sigma_j^2) - D log(sqrt(2 pi) sigma_j)        (Eq. logprob)
 *   rho    = exp(logp - logp_old_ij)
 *   A_i    = clamp((r_i - mean) / (std + adv_eps), +-adv_clip), unbiased std (Eq. advantage)
 *   s_ij   = scale * d max(-A rho, -A clip(rho, 1-eps, 1+eps)) / d v_ij          (Eq. grpo_loss)
 *          = scale * (-A_i) rho r_ij (t_{j+1}-t_j) / sigma_j^2, or 0 when the clipped branch
 *            is strictly larger (A>0 and rho>1+eps, or A<0 and rho<1-eps).
 * The squared norms are accumulated in f64 and logp / rho are f64.
 *   v_hat     device [G, W, D] (v_dtype)   model outputs of the window's steps
 *   z         device [G, W+1, D] f32       trajectory states z_0 .. z_W of the window
 *   t         device [W+1] f64             network-input times t_0 .. t_W
 *   sigma     device [W] f64               per-step noise scale
 *   logp_old  device [G, W] f64            rollout log-probs
 *   rewards   device [G] f32
 *   s_out     device [G, W, D] f32 or NULL
 *   cot_out   device [2G, D] f32 or NULL: if given, the aggregated JAGG cotangents
 *             (jagg_aggregate over t_0..t_{W-1}) are written in the same pass; needs W >= 2
 *   logp_new, ratio device [G, W] f64; clipped device [G, W] u8; adv_out device [G] f64
 *   ws        device workspace of >= jagg_signals_workspace_bytes(G, W, D) bytes       */
int64_t jagg_signals_workspace_bytes(int G, int W, int64_t D);
int grpo_step_signals(const void* v_hat, int v_dtype, const float* z, const double* t,
                      const double* sigma, const double* logp_old, const float* rewards,
                      int G, int W, int64_t D, double clip_eps, double adv_clip,
                      double adv_eps, double scale, float* s_out, float* cot_out,
                      double* logp_new, double* ratio, uint8_t* clipped, double* adv_out,
                      void* ws, size_t ws_bytes, cudaStream_t stream);

/* Phase 2 for an epsilon-prediction backbone (Eq. logprob, epsilon case): the transition
 * mean is the deterministic DDIM step of the diffusion schedule (alpha_t, sigma_t),
 *   mu_ij = alpha_{j+1} (z_{i,j} / alpha_j - (sigma_j / alpha_j - sigma_{j+1} / alpha_{j+1}) eps_ij)
 *         = a_j z_{i,j} + c_j eps_ij,
 * and every other quantity is as in grpo_step_signals with r_ij = z_{i,j+1} - mu_ij and
 *   s_ij = scale * (-A_i) rho r_ij c_j / sigma_j^2 (0 when clipped),
 * the derivative with respect to the model output eps_ij.  The schedule's sigma_t is the noise
 * level of z_t = alpha_t x + sigma_t eps; sigma (the step's noise scale) enters the density
 * only.  t is used for the aggregation weights alone (cot_out).
 *   eps_hat      device [G, W, D] (eps_dtype)   noise predictions of the window's steps
 *   sched_alpha  device [W+1] f64 alpha_t at t_0 .. t_W, all > 0 (checked on device: otherwise
 *                JAGG_DEV_STATUS_BADARG is set and the outputs are meaningless)
 *   sched_sigma  device [W+1] f64 sigma_t at t_0 .. t_W
 * Workspace: jagg_signals_workspace_bytes(G, W, D), as for grpo_step_signals.           */
int grpo_step_signals_eps(const void* eps_hat, int eps_dtype, const float* z, const double* t,
                          const double* sched_alpha, const double* sched_sigma, const double* sigma,
                          const double* logp_old, const float* rewards, int G, int W, int64_t D,
                          double clip_eps, double adv_clip, double adv_eps, double scale, float* s_out,
                          float* cot_out, double* logp_new, double* ratio, uint8_t* clipped,
                          double* adv_out, void* ws, size_t ws_bytes, cudaStream_t stream);

/* grpo_step_signals for callers that cannot allocate device memory (no counterpart in the
 * paper: an interface convenience of this library).  Some callers have no way to obtain a
 * workspace: code that runs where cudaMalloc is not allowed or not wanted, such as an
 * embedding runtime with a fixed, pre-planned memory budget or a host that owns no
 * device allocator.  This entry point takes the same arguments as grpo_step_signals
 * except the workspace, and uses instead a scratch array compiled into the library
 * (JAGG_SIGNALS_STATIC_SCRATCH_BYTES bytes of device memory, held by every GPU that loads
 * the library until the process exits).  It allocates nothing.
 *   - Requests whose scratch need (jagg_signals_workspace_bytes(G, W, D)) exceeds
 *     JAGG_SIGNALS_STATIC_SCRATCH_BYTES fail with JAGG_ERR_WORKSPACE before any launch.
 *   - The stream must belong to the current device (JAGG_ERR_ARG otherwise).
 *   - The first call on a device looks up the array's device address (a synchronous
 *     runtime query) and keeps it for the life of the process; make that first call before
 *     any stream capture on that device.  A device reset (cudaDeviceReset) after it is not
 *     supported: the kept address would be stale.
 *   - Every call shares the one array: calls whose kernels may overlap on the GPU (on
 *     different streams without ordering between them) race and give wrong results.
 *     Nothing in the array needs to start at zero; each call overwrites what it reads. */
#define JAGG_SIGNALS_STATIC_SCRATCH_BYTES (1 << 20)
int grpo_step_signals_static(const void* v_hat, int v_dtype, const float* z, const double* t,
                             const double* sigma, const double* logp_old, const float* rewards,
                             int G, int W, int64_t D, double clip_eps, double adv_clip,
                             double adv_eps, double scale, float* s_out, float* cot_out,
                             double* logp_new, double* ratio, uint8_t* clipped, double* adv_out,
                             cudaStream_t stream);

/* Phase 3 (Eq. alpha, Eq. s_base_corr): alpha_j = (t_0 - t_j) / (t_0 - t_{W-1}),
 *   cot[i]     = sum_j (1 - alpha_j) s[i, j]   (s_base, endpoint j = 0)
 *   cot[G + i] = sum_j alpha_j s[i, j]         (s_corr, endpoint j = W-1)
 *   s      device [G, W, D] f32;  t_window device [W] f64 network-input times
 *   cot    device [2G, D] f32.  Requires W >= 2 and t_0 != t_{W-1} (checked on device:
 *   a zero denominator sets JAGG_DEV_STATUS_BADARG and writes zeros).                */
int jagg_aggregate(const float* s, const double* t_window, int G, int W, int64_t D,
                   float* cot, cudaStream_t stream);

/* Phase 3 over a span of a window's steps, alpha taken against the window's endpoint times
 * (Eq. alpha, Eq. s_base_corr): alpha_j = (t_first - t_j) / (t_first - t_last),
 *   cot[i]     (+)= sum_j (1 - alpha_j) s[i, j]
 *   cot[G + i] (+)= sum_j alpha_j s[i, j]          over the n steps given.
 * Serves the sequential-graph variant (Sec. 3.4, Algorithm 2: s_base from steps 0..W-2 is
 * complete before the last step's forward, whose s_{W-1} then adds to s_corr alone) and the
 * endpoint-only ablation of Sec. 4 (the span {0, W-1} with t_first = t_0, t_last = t_{W-1}
 * maps s_0 and s_{W-1} to the two rows unweighted).  jagg_aggregate is the span of all W
 * steps with accumulate = 0.
 *   s        device f32, step j of sample i at s[i * s_sample_stride + j * D] (s_sample_stride =
 *            0: n * D, a [G, n, D] array; W * D addresses n steps inside a [G, W, D] window)
 *   t_steps  device [n] f64 network-input times of the steps
 *   t_first, t_last  host f64 window endpoint times (must differ: JAGG_ERR_ARG otherwise)
 *   cot      device [2G, D] f32, overwritten (accumulate = 0) or added to (accumulate != 0) */
int jagg_aggregate_span(const float* s, int64_t s_sample_stride, const double* t_steps, double t_first,
                        double t_last, int G, int n, int64_t D, float* cot, int accumulate, cudaStream_t stream);

/* One step of the rollout sampler (the stochastic transition that Eq. logprob scores, Sec. 3.1
 * and Sec. 3.2), fused with the log-probability of the sample it draws (the rollout's old
 * log-prob that Eq. grpo_loss divides by):
 *   z_next_i = mu_i + sigma xi_i,  mu_i = a z_cur_i + c y_i,  stored in f32;
 *   logp_i   = -||z_next_i - mu_i||^2 / (2 sigma^2) - D log(sqrt(2 pi) sigma)
 * with (a, c) = (1, t_next - t_cur) for a rectified-flow velocity y (Euler-Maruyama step),
 * or the DDIM step of grpo_step_signals_eps for a noise prediction y when sched is given.
 * The residual and its sum are evaluated by the same device code as grpo_step_signals, so
 * scoring the stored step there with the same y gives exactly this logp (ratio exactly 1).
 *   y_hat    device [G, D] (y_dtype) model outputs at z_cur, row i at y_hat + i * y_sample_stride
 *   z_cur    device f32, row i at z_cur + i * z_sample_stride; z_next likewise (may be the next
 *            step of the same [G, T+1, D] trajectory buffer: z_sample_stride = (T+1) D)
 *   xi       device f32 standard-normal draws, row i at xi + i * xi_sample_stride
 *            (a stride of 0 means D for y_hat, z and xi)
 *   t_cur, t_next, sigma  host f64 (sigma > 0)
 *   sched    host [4] f64 = {alpha_cur, alpha_next, sigma_cur, sigma_next} or NULL (flow);
 *            an alpha <= 0 sets JAGG_DEV_STATUS_BADARG (outputs then meaningless)
 *   logp     device f64, sample i at logp[i * logp_stride]
 *   z_model  device [G, D] (z_model_dtype) or NULL: z_next rounded to the model's storage type,
 *            the input of the next step's forward
 *   ws       device workspace of >= jagg_rollout_workspace_bytes(G, D) bytes            */
int64_t jagg_rollout_workspace_bytes(int G, int64_t D);
int jagg_rollout_step(const void* y_hat, int y_dtype, int64_t y_sample_stride, const float* z_cur,
                      float* z_next, int64_t z_sample_stride, const float* xi, int64_t xi_sample_stride,
                      int G, int64_t D, double t_cur, double t_next, double sigma, const double* sched,
                      double* logp, int64_t logp_stride, void* z_model, int z_model_dtype, void* ws,
                      size_t ws_bytes, cudaStream_t stream);

/* jagg_frac routing (Sec. 3.3 "High-noise vs. low-noise scheduling"; rule of the
 * gradient-quality appendix).  Host-only, synchronous.
 *   cos == NULL: schedule mode, route[w] = (w < floor(jagg_frac * n_windows + 1e-9)).
 *   cos != NULL: calibration mode, route[w] = (cos[w] >= tau) and *derived_frac (if not
 *   NULL) = longest qualifying prefix / n_windows.  jagg_frac is ignored.
 *   route  host [n_windows] u8: 1 = JAGG window, 0 = exact per-step window.           */
int jagg_route(int n_windows, double jagg_frac, const double* cos, double tau,
               uint8_t* route, double* derived_frac);

/* Gradient reductions (gradient-quality appendix: cos(g_JAGG, g_exact) and
 * rho = ||g_JAGG|| / ||g_exact||; accumulation of window gradients).
 *   acc != NULL: acc[k] += alpha * a[k]
 *   out3 != NULL: out3 = { <a,b>, <a,a>, <b,b> } in f64 (b may be NULL: then <a,a> thrice)
 *   a, b, acc device f32 [P]; out3 device f64 [3]
 *   ws device workspace of >= jagg_grad_reduce_workspace_bytes(P) bytes (when out3)   */
int64_t jagg_grad_reduce_workspace_bytes(int64_t P);
int grad_reduce(const float* a, const float* b, int64_t P, float alpha, float* acc,
                double* out3, void* ws, size_t ws_bytes, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* JAGG_H_ */
