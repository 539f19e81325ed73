// Bandwidth-bound kernels of the backbone's forward and backward passes.
#pragma once

#include "common.cuh"

namespace jagg {

// Latent <-> token layout (token n = r*(W/p) + c; feature f = ch*p*p + py*p + px).
// in_f32 / out_f32 select f32, otherwise the storage type `dtype`.
int launch_patchify(const void* z, int in_f32, void* xp, int out_f32, int dtype, int B, int C, int H, int W, int p,
                    cudaStream_t s);
int launch_unpatchify(const void* xp, void* z, int dtype, int B, int C, int H, int W, int p, cudaStream_t s);

// phi[b] = [cos(1000 t_b w_k), sin(1000 t_b w_k)], w_k = 10000^(-k/half); f32 [B, dim].
int launch_timestep_embedding(const float* t, float* phi, int B, int dim, cudaStream_t s);

// out = silu(in) (f32 -> f32), n elements.
int launch_silu(const float* in, float* out, int64_t n, cudaStream_t s);
// g[i] *= silu'(x[i]) (f32).
int launch_mul_silu_grad(float* g, const float* x, int64_t n, cudaStream_t s);

// h[b, row0 + n, :] += 2D sin-cos position table of patch n (gh x gw grid), f32.
int launch_add_pos_embed(float* h, int B, int rows_per_seq, int row0, int gh, int gw, int d, cudaStream_t s);

// LayerNorm (no affine, eps 1e-6) + adaLN modulation:
//   out[m] = (x - mean) rstd (1 + scale[b]) + shift[b],   x = h[in_row(m)] (f32)
// in_row(m) = (m / seg) * seg_stride + seg_off + m % seg (seg = 0: in_row = m);
// b = m / rows_per_seq; shift/scale f32 rows of length >= d with stride mod_stride.
// Saves mean and rstd per output row (f32).
struct LnModFwd {
  const float* h;
  int seg, seg_off;
  int64_t seg_stride;
  int M, d, rows_per_seq;
  const float* shift;
  const float* scale;
  int64_t mod_stride;
  void* out;
  int dtype;
  float* mean;
  float* rstd;
};
int launch_ln_mod_fwd(const LnModFwd& a, cudaStream_t s);

// Backward of LayerNorm + modulation, optionally followed by the backward of the gated
// residual branch that produced the normalised input (all per row m of one sequence b):
//   ln:   dxh = dm (1 + scale[b]);  dh[out_row] = dh_in[out_row] + rstd (dxh - mean(dxh)
//         - xh mean(dxh xh));  dshift[b] += sum_m dm;  dscale[b] += sum_m dm xh
//   gate: with dh the resulting residual gradient: dgate[b] += sum_m dh y;
//         dy = gate[b] dh (dtype);  dbias += sum_m dy
// h/mean/rstd are the forward's LN input and statistics; in_row() remaps as in LnModFwd
// and also addresses dh_in / dh_out.
struct LnGateBwd {
  int M, d, rows_per_seq;
  int seg, seg_off;
  int64_t seg_stride;
  // LayerNorm part (do_ln)
  int do_ln;
  const void* dm;
  int dm_f32;
  const float* h;
  const float* mean;
  const float* rstd;
  const float* scale;
  int64_t mod_stride;
  float* dshift;  // f32 rows, stride dmod_stride
  float* dscale;
  int64_t dmod_stride;
  const float* dh_in;  // may alias dh_out
  float* dh_out;
  // gate part (do_gate)
  int do_gate;
  const void* y;  // dtype [M, d] (rows m, not remapped)
  const float* gate;
  float* dgate;
  void* dy;  // dtype [M, d]
  float* dbias;  // f32 [d] or nullptr
  int dtype;
};
int launch_ln_gate_bwd(const LnGateBwd& a, cudaStream_t s);

// db[n] += sum_r X[r * ld + n], r < rows, n < cols (X f32 or dtype).
int launch_colsum(const void* X, int x_f32, int dtype, int rows, int cols, int64_t ld, float* db, cudaStream_t s);

// out[r', :] = in[in_row(r'), :] converted f32 -> dtype, r' < rows; in_row as LnModFwd.
int launch_gather_rows(const float* in, int64_t ld_in, int seg, int seg_off, int64_t seg_stride, void* out,
                       int dtype, int rows, int cols, cudaStream_t s);

// Copies rows between two buffers of the same element type with independent segment maps
// (used to interleave the text and image streams).  elem_bytes 2 or 4.
int launch_copy_rows(const void* in, int64_t ld_in, int in_seg, int in_seg_off, int64_t in_seg_stride, void* out,
                     int64_t ld_out, int out_seg, int out_seg_off, int64_t out_seg_stride, int rows, int cols,
                     int elem_bytes, cudaStream_t s);

// Attention helper: Dv[b, head, n] = sum_c dO[row, head*dh + c] * O[row, head*dh + c].
int launch_attn_rowdot(const void* dO, const void* O, int64_t ld, float* Dv, int B, int N, int heads, int dh,
                       int dtype, cudaStream_t s);

// Per-head RMSNorm (learned scale, eps 1e-6) followed by 2D RoPE on q and k of a qkv buffer,
// writing the transformed q/k into qk_out [M, 2d] (dtype); saves 1/rms for q and k.
struct QkNormRope {
  const void* qkv;  // [M, ld_qkv] dtype: q at col 0, k at col d
  int64_t ld_qkv;
  int M, N, d, heads, n_txt, gw;
  const void* qscale_txt;  // [dh] weights dtype
  const void* kscale_txt;
  const void* qscale_img;
  const void* kscale_img;
  int rope;
  void* qk_out;  // [M, 2d]
  float* rq;     // [M, heads]
  float* rk;
  int dtype;
};
int launch_qk_norm_rope_fwd(const QkNormRope& a, cudaStream_t s);
// Backward: given dq, dk of the transformed q/k (inside dqkv [M, ld] at cols 0 and d, f32 or
// dtype), writes d(raw q), d(raw k) into the same place (dtype) and accumulates the scale
// gradients (f32 [dh] each) into dqs_txt/dks_txt/dqs_img/dks_img.
struct QkNormRopeBwd {
  QkNormRope f;
  void* dqk;  // [M, ld_dqk] dtype, in place
  int64_t ld_dqk;
  float* dqs_txt;
  float* dks_txt;
  float* dqs_img;
  float* dks_img;
};
int launch_qk_norm_rope_bwd(const QkNormRopeBwd& a, cudaStream_t s);

}  // namespace jagg
