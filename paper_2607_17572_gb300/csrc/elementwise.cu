// Bandwidth-bound kernels: layout transforms, embeddings, LayerNorm + adaLN modulation
// (forward and backward fused with the gated-residual backward), bias reductions,
// QK RMSNorm + 2D RoPE.
#include "elementwise.cuh"

namespace jagg {

namespace {

__device__ __forceinline__ float ldx(const void* p, int64_t i, int is_f32) {
  return is_f32 ? static_cast<const float*>(p)[i] : __bfloat162float(static_cast<const bf16*>(p)[i]);
}
__device__ __forceinline__ void stx(void* p, int64_t i, int is_f32, float v) {
  if (is_f32)
    static_cast<float*>(p)[i] = v;
  else
    static_cast<bf16*>(p)[i] = __float2bfloat16_rn(v);
}
__device__ __forceinline__ int64_t seg_row(int m, int seg, int seg_off, int64_t seg_stride) {
  return seg ? (int64_t)(m / seg) * seg_stride + seg_off + m % seg : (int64_t)m;
}

int grid_for(int64_t n, int threads) {
  int64_t b = (n + threads - 1) / threads;
  return (int)(b < 1 ? 1 : (b > 1048576 ? 1048576 : b));
}

// ------------------------------------------------------------------ layouts
__global__ void patchify_kernel(const void* z, int in_f32, void* xp, int out_f32, int B, int C, int H, int W, int p) {
  const int gw = W / p, gh = H / p;
  const int pd = C * p * p;
  const int64_t total = (int64_t)B * gh * gw * pd;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int f = (int)(i % pd);
    const int64_t tok = i / pd;
    const int n = (int)(tok % (gh * gw));
    const int b = (int)(tok / (gh * gw));
    const int r = n / gw, c = n % gw;
    const int ch = f / (p * p), py = (f / p) % p, px = f % p;
    const int64_t zi = (((int64_t)b * C + ch) * H + (r * p + py)) * W + (c * p + px);
    stx(xp, i, out_f32, ldx(z, zi, in_f32));
  }
}

__global__ void unpatchify_kernel(const void* xp, void* z, int is_f32, int B, int C, int H, int W, int p) {
  const int gw = W / p, gh = H / p;
  const int pd = C * p * p;
  const int64_t total = (int64_t)B * C * H * W;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int x = (int)(i % W);
    const int y = (int)((i / W) % H);
    const int ch = (int)((i / ((int64_t)W * H)) % C);
    const int b = (int)(i / ((int64_t)W * H * C));
    const int r = y / p, py = y % p, c = x / p, px = x % p;
    const int64_t xi = ((int64_t)b * gh * gw + r * gw + c) * pd + ch * p * p + py * p + px;
    stx(z, i, is_f32, ldx(xp, xi, is_f32));
  }
}

__global__ void temb_kernel(const float* t, float* phi, int B, int dim) {
  const int half = dim / 2;
  const int total = B * half;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
    const int b = i / half, k = i % half;
    // w_k = 10000^(-k/half) evaluated in double so the argument 1000 t w_k is accurate
    const double w = exp(-log(10000.0) * (double)k / (double)half);
    const double a = 1000.0 * (double)t[b] * w;
    phi[(int64_t)b * dim + k] = (float)cos(a);
    phi[(int64_t)b * dim + half + k] = (float)sin(a);
  }
}

__global__ void silu_kernel(const float* in, float* out, int64_t n) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    out[i] = silu_f(in[i]);
}
__global__ void mul_silu_grad_kernel(float* g, const float* x, int64_t n) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    g[i] *= silu_grad_f(x[i]);
}

__global__ void pos_embed_kernel(float* h, int B, int rows_per_seq, int row0, int gh, int gw, int d) {
  const int q = d / 4;
  const int64_t total = (int64_t)B * gh * gw * d;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int c = (int)(i % d);
    const int64_t tok = i / d;
    const int n = (int)(tok % (gh * gw));
    const int b = (int)(tok / (gh * gw));
    const int half = c / (d / 2);         // 0: row, 1: column
    const int cc = c % (d / 2);
    const int k = cc % q;
    const double pos = half == 0 ? (double)(n / gw) : (double)(n % gw);
    const double a = pos * exp(-log(10000.0) * (double)k / (double)q);
    const float v = (float)(cc < q ? sin(a) : cos(a));
    h[((int64_t)b * rows_per_seq + row0 + n) * d + c] += v;
  }
}

// ------------------------------------------------------------------ LayerNorm + modulation
// One warp per row; the row stays in registers (d <= 32 * 4 * LN_MAXV).
constexpr int LN_MAXV = 24;  // d <= 3072

__global__ void ln_mod_fwd_kernel(LnModFwd a) {
  const int warps = blockDim.x / 32;
  const int m = blockIdx.x * warps + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (m >= a.M) return;
  const int nv = (a.d + 127) / 128;  // float4 slots per lane; slot (i*32 + lane) covers 4 columns
  const float* x = a.h + seg_row(m, a.seg, a.seg_off, a.seg_stride) * a.d;
  float4 v[LN_MAXV];
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < LN_MAXV; ++i) {
    v[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i < nv && (i * 32 + lane) * 4 < a.d) {
      v[i] = reinterpret_cast<const float4*>(x)[i * 32 + lane];
      s += v[i].x + v[i].y + v[i].z + v[i].w;
    }
  }
  const float mean = warp_sum(s) / a.d;
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < LN_MAXV; ++i)
    if (i < nv && (i * 32 + lane) * 4 < a.d) {
      float dx = v[i].x - mean, dy = v[i].y - mean, dz = v[i].z - mean, dw = v[i].w - mean;
      ss += dx * dx + dy * dy + dz * dz + dw * dw;
    }
  const float rstd = rsqrtf(warp_sum(ss) / a.d + 1e-6f);
  const int b = m / a.rows_per_seq;
  const float* sh = a.shift + (int64_t)b * a.mod_stride;
  const float* sc = a.scale + (int64_t)b * a.mod_stride;
  const int is_f32 = a.dtype == JAGG_DTYPE_F32;
#pragma unroll
  for (int i = 0; i < LN_MAXV; ++i)
    if (i < nv && (i * 32 + lane) * 4 < a.d) {
      const int c = (i * 32 + lane) * 4;
      float4 s4 = *reinterpret_cast<const float4*>(sc + c);
      float4 h4 = *reinterpret_cast<const float4*>(sh + c);
      float o0 = (v[i].x - mean) * rstd * (1.f + s4.x) + h4.x;
      float o1 = (v[i].y - mean) * rstd * (1.f + s4.y) + h4.y;
      float o2 = (v[i].z - mean) * rstd * (1.f + s4.z) + h4.z;
      float o3 = (v[i].w - mean) * rstd * (1.f + s4.w) + h4.w;
      if (is_f32) {
        *reinterpret_cast<float4*>(static_cast<float*>(a.out) + (int64_t)m * a.d + c) = make_float4(o0, o1, o2, o3);
      } else {
        __nv_bfloat162 p0 = __floats2bfloat162_rn(o0, o1), p1 = __floats2bfloat162_rn(o2, o3);
        uint2 raw;
        raw.x = *reinterpret_cast<uint32_t*>(&p0);
        raw.y = *reinterpret_cast<uint32_t*>(&p1);
        *reinterpret_cast<uint2*>(static_cast<bf16*>(a.out) + (int64_t)m * a.d + c) = raw;
      }
    }
  if (lane == 0) {
    a.mean[m] = mean;
    a.rstd[m] = rstd;
  }
}

// Backward: a block of LNB_THREADS threads walks LNB_ROWS consecutive rows of one sequence;
// thread t owns columns t, t + LNB_THREADS, ...; per-row statistics via block reductions;
// per-column partial sums stay in registers and are flushed with atomics at the end.
constexpr int LNB_THREADS = 256;
constexpr int LNB_ROWS = 32;
constexpr int LNB_MAXC = 12;  // d <= 3072

__device__ __forceinline__ float2 block_sum2(float2 v, float2* red) {
  v.x = warp_sum(v.x);
  v.y = warp_sum(v.y);
  const int w = threadIdx.x / 32, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float2 r = make_float2(0.f, 0.f);
  for (int i = 0; i < LNB_THREADS / 32; ++i) {
    r.x += red[i].x;
    r.y += red[i].y;
  }
  return r;
}

__global__ void __launch_bounds__(LNB_THREADS) ln_gate_bwd_kernel(LnGateBwd a) {
  __shared__ float2 red[LNB_THREADS / 32];
  const int chunks_per_seq = (a.rows_per_seq + LNB_ROWS - 1) / LNB_ROWS;
  const int b = blockIdx.x / chunks_per_seq;
  const int r0 = b * a.rows_per_seq + (blockIdx.x % chunks_per_seq) * LNB_ROWS;
  const int r1 = min(r0 + LNB_ROWS, (b + 1) * a.rows_per_seq);
  const int nc = (a.d + LNB_THREADS - 1) / LNB_THREADS;
  const int is_f32 = a.dtype == JAGG_DTYPE_F32;
  float psh[LNB_MAXC], psc[LNB_MAXC], pg[LNB_MAXC], pb[LNB_MAXC];
  float scl[LNB_MAXC], gt[LNB_MAXC];
#pragma unroll
  for (int i = 0; i < LNB_MAXC; ++i) {
    psh[i] = psc[i] = pg[i] = pb[i] = 0.f;
    const int c = threadIdx.x + i * LNB_THREADS;
    scl[i] = (a.do_ln && i < nc && c < a.d) ? a.scale[(int64_t)b * a.mod_stride + c] : 0.f;
    gt[i] = (a.do_gate && i < nc && c < a.d) ? a.gate[(int64_t)b * a.mod_stride + c] : 0.f;
  }
  for (int m = r0; m < r1; ++m) {
    const int64_t hr = seg_row(m, a.seg, a.seg_off, a.seg_stride);
    float dhv[LNB_MAXC];
    if (a.do_ln) {
      const float mu = a.mean[m], rs = a.rstd[m];
      float dm[LNB_MAXC], xh[LNB_MAXC];
      float2 acc = make_float2(0.f, 0.f);
#pragma unroll
      for (int i = 0; i < LNB_MAXC; ++i) {
        const int c = threadIdx.x + i * LNB_THREADS;
        dm[i] = xh[i] = 0.f;
        if (i < nc && c < a.d) {
          dm[i] = ldx(a.dm, (int64_t)m * a.d + c, a.dm_f32);
          xh[i] = (a.h[hr * a.d + c] - mu) * rs;
          const float dxh = dm[i] * (1.f + scl[i]);
          acc.x += dxh;
          acc.y += dxh * xh[i];
          psh[i] += dm[i];
          psc[i] += dm[i] * xh[i];
        }
      }
      const float2 tot = block_sum2(acc, red);
      const float m1 = tot.x / a.d, m2 = tot.y / a.d;
#pragma unroll
      for (int i = 0; i < LNB_MAXC; ++i) {
        const int c = threadIdx.x + i * LNB_THREADS;
        dhv[i] = 0.f;
        if (i < nc && c < a.d) {
          const float dxh = dm[i] * (1.f + scl[i]);
          const float v = a.dh_in[hr * a.d + c] + rs * (dxh - m1 - xh[i] * m2);
          a.dh_out[hr * a.d + c] = v;
          dhv[i] = v;
        }
      }
    } else {
#pragma unroll
      for (int i = 0; i < LNB_MAXC; ++i) {
        const int c = threadIdx.x + i * LNB_THREADS;
        dhv[i] = (i < nc && c < a.d) ? a.dh_in[hr * a.d + c] : 0.f;
      }
    }
    if (a.do_gate) {
#pragma unroll
      for (int i = 0; i < LNB_MAXC; ++i) {
        const int c = threadIdx.x + i * LNB_THREADS;
        if (i < nc && c < a.d) {
          const float yv = ldx(a.y, (int64_t)m * a.d + c, is_f32);
          pg[i] += dhv[i] * yv;
          const float dy = gt[i] * dhv[i];
          stx(a.dy, (int64_t)m * a.d + c, is_f32, dy);
          pb[i] += is_f32 ? dy : __bfloat162float(__float2bfloat16_rn(dy));
        }
      }
    }
  }
#pragma unroll
  for (int i = 0; i < LNB_MAXC; ++i) {
    const int c = threadIdx.x + i * LNB_THREADS;
    if (i < nc && c < a.d) {
      if (a.do_ln) {
        atomicAdd(a.dshift + (int64_t)b * a.dmod_stride + c, psh[i]);
        atomicAdd(a.dscale + (int64_t)b * a.dmod_stride + c, psc[i]);
      }
      if (a.do_gate) {
        atomicAdd(a.dgate + (int64_t)b * a.dmod_stride + c, pg[i]);
        if (a.dbias) atomicAdd(a.dbias + c, pb[i]);
      }
    }
  }
}

// ------------------------------------------------------------------ reductions / copies
constexpr int CS_ROWS = 64;
__global__ void colsum_kernel(const void* X, int x_f32, int rows, int cols, int64_t ld, float* db) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  const int r0 = blockIdx.y * CS_ROWS;
  if (c >= cols) return;
  const int r1 = min(r0 + CS_ROWS, rows);
  float s = 0.f;
  for (int r = r0; r < r1; ++r) s += ldx(X, (int64_t)r * ld + c, x_f32);
  atomicAdd(db + c, s);
}

__global__ void gather_rows_kernel(const float* in, int64_t ld_in, int seg, int seg_off, int64_t seg_stride, void* out,
                                   int out_f32, int rows, int cols) {
  const int64_t total = (int64_t)rows * cols;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int r = (int)(i / cols), c = (int)(i % cols);
    stx(out, i, out_f32, in[seg_row(r, seg, seg_off, seg_stride) * ld_in + c]);
  }
}

template <typename E>
__global__ void copy_rows_kernel(const E* in, int64_t ld_in, int is, int io, int64_t iss, E* out, int64_t ld_out,
                                 int os, int oo, int64_t oss, int rows, int cols) {
  const int64_t total = (int64_t)rows * cols;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int r = (int)(i / cols), c = (int)(i % cols);
    out[seg_row(r, os, oo, oss) * ld_out + c] = in[seg_row(r, is, io, iss) * ld_in + c];
  }
}

__global__ void attn_rowdot_kernel(const void* dO, const void* O, int64_t ld, float* Dv, int B, int N, int heads,
                                   int dh, int is_f32) {
  // one warp per (row, head)
  const int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) / 32;
  const int lane = threadIdx.x & 31;
  const int64_t total = (int64_t)B * N * heads;
  if (w >= total) return;
  const int hd = (int)(w % heads);
  const int64_t row = w / heads;  // b * N + n
  float s = 0.f;
  for (int c = lane; c < dh; c += 32) {
    const int64_t i = row * ld + (int64_t)hd * dh + c;
    s += ldx(dO, i, is_f32) * ldx(O, i, is_f32);
  }
  s = warp_sum(s);
  if (lane == 0) {
    const int64_t b = row / N, n = row % N;
    Dv[(b * heads + hd) * N + n] = s;
  }
}

// ------------------------------------------------------------------ QK RMSNorm + RoPE
// One warp per (row, head) handles q and k; dh <= 128 -> up to 4 elements per lane as
// two rotated pairs.
__device__ __forceinline__ void rope_angle(int n, int n_txt, int gw, int dh, int pair, float& cs, float& sn) {
  // pair index within the head: first dh/4 pairs rotate by the patch row, the rest by the column
  const int hd = dh / 2, npair = hd / 2;
  if (n < n_txt) {
    cs = 1.f;
    sn = 0.f;
    return;
  }
  const int tok = n - n_txt;
  const int axis = pair / npair, i = pair % npair;
  const double pos = axis == 0 ? (double)(tok / gw) : (double)(tok % gw);
  const double th = exp(-log(10000.0) * 2.0 * (double)i / (double)hd);
  double s, c;
  sincos(pos * th, &s, &c);
  cs = (float)c;
  sn = (float)s;
}

__global__ void qk_norm_rope_fwd_kernel(QkNormRope a) {
  const int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) / 32;
  const int lane = threadIdx.x & 31;
  if (w >= (int64_t)a.M * a.heads) return;
  const int hd = (int)(w % a.heads);
  const int m = (int)(w / a.heads);
  const int n = m % a.N;
  const int dh = a.d / a.heads;
  const int is_f32 = a.dtype == JAGG_DTYPE_F32;
  const bool txt = n < a.n_txt;
  for (int which = 0; which < 2; ++which) {
    const void* scl = which == 0 ? (txt ? a.qscale_txt : a.qscale_img) : (txt ? a.kscale_txt : a.kscale_img);
    const int64_t base = (int64_t)m * a.ld_qkv + which * a.d + hd * dh;
    float x[4] = {0.f, 0.f, 0.f, 0.f};
    float ss = 0.f;
    for (int j = 0; j < 2; ++j) {
      const int pair = lane + 32 * j;
      if (2 * pair < dh) {
        x[2 * j] = ldx(a.qkv, base + 2 * pair, is_f32);
        x[2 * j + 1] = ldx(a.qkv, base + 2 * pair + 1, is_f32);
        ss += x[2 * j] * x[2 * j] + x[2 * j + 1] * x[2 * j + 1];
      }
    }
    const float r = rsqrtf(warp_sum(ss) / dh + 1e-6f);
    for (int j = 0; j < 2; ++j) {
      const int pair = lane + 32 * j;
      if (2 * pair < dh) {
        const float y0 = x[2 * j] * r * ldx(scl, 2 * pair, is_f32);
        const float y1 = x[2 * j + 1] * r * ldx(scl, 2 * pair + 1, is_f32);
        float cs = 1.f, sn = 0.f;
        if (a.rope) rope_angle(n, a.n_txt, a.gw, dh, pair, cs, sn);
        const int64_t o = (int64_t)m * 2 * a.d + which * a.d + hd * dh + 2 * pair;
        stx(a.qk_out, o, is_f32, y0 * cs - y1 * sn);
        stx(a.qk_out, o + 1, is_f32, y0 * sn + y1 * cs);
      }
    }
    if (lane == 0) (which == 0 ? a.rq : a.rk)[(int64_t)m * a.heads + hd] = r;
  }
}

__global__ void qk_norm_rope_bwd_kernel(QkNormRopeBwd b) {
  const QkNormRope& a = b.f;
  const int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) / 32;
  const int lane = threadIdx.x & 31;
  if (w >= (int64_t)a.M * a.heads) return;
  const int hd = (int)(w % a.heads);
  const int m = (int)(w / a.heads);
  const int n = m % a.N;
  const int dh = a.d / a.heads;
  const int is_f32 = a.dtype == JAGG_DTYPE_F32;
  const bool txt = n < a.n_txt;
  for (int which = 0; which < 2; ++which) {
    const void* scl = which == 0 ? (txt ? a.qscale_txt : a.qscale_img) : (txt ? a.kscale_txt : a.kscale_img);
    float* dscl = which == 0 ? (txt ? b.dqs_txt : b.dqs_img) : (txt ? b.dks_txt : b.dks_img);
    const float r = (which == 0 ? a.rq : a.rk)[(int64_t)m * a.heads + hd];
    const int64_t xb = (int64_t)m * a.ld_qkv + which * a.d + hd * dh;
    const int64_t gb = (int64_t)m * b.ld_dqk + which * a.d + hd * dh;
    float x[4] = {0.f, 0.f, 0.f, 0.f}, u[4] = {0.f, 0.f, 0.f, 0.f}, gsc[4] = {0.f, 0.f, 0.f, 0.f};
    float xu = 0.f;
    for (int j = 0; j < 2; ++j) {
      const int pair = lane + 32 * j;
      if (2 * pair < dh) {
        // undo the rotation of the incoming gradient (rotate by -angle)
        const float g0 = ldx(b.dqk, gb + 2 * pair, is_f32), g1 = ldx(b.dqk, gb + 2 * pair + 1, is_f32);
        float cs = 1.f, sn = 0.f;
        if (a.rope) rope_angle(n, a.n_txt, a.gw, dh, pair, cs, sn);
        const float dy0 = g0 * cs + g1 * sn;
        const float dy1 = -g0 * sn + g1 * cs;
        x[2 * j] = ldx(a.qkv, xb + 2 * pair, is_f32);
        x[2 * j + 1] = ldx(a.qkv, xb + 2 * pair + 1, is_f32);
        gsc[2 * j] = ldx(scl, 2 * pair, is_f32);
        gsc[2 * j + 1] = ldx(scl, 2 * pair + 1, is_f32);
        atomicAdd(dscl + 2 * pair, dy0 * x[2 * j] * r);
        atomicAdd(dscl + 2 * pair + 1, dy1 * x[2 * j + 1] * r);
        u[2 * j] = dy0 * gsc[2 * j];
        u[2 * j + 1] = dy1 * gsc[2 * j + 1];
        xu += x[2 * j] * u[2 * j] + x[2 * j + 1] * u[2 * j + 1];
      }
    }
    xu = warp_sum(xu);
    for (int j = 0; j < 2; ++j) {
      const int pair = lane + 32 * j;
      if (2 * pair < dh) {
        for (int e = 0; e < 2; ++e) {
          const float dx = r * u[2 * j + e] - x[2 * j + e] * r * r * r * xu / dh;
          stx(b.dqk, gb + 2 * pair + e, is_f32, dx);
        }
      }
    }
  }
}

}  // namespace

// ------------------------------------------------------------------ launchers
int launch_patchify(const void* z, int in_f32, void* xp, int out_f32, int dtype, int B, int C, int H, int W, int p,
                    cudaStream_t s) {
  (void)dtype;
  const int64_t n = (int64_t)B * C * H * W;
  patchify_kernel<<<grid_for(n, 256), 256, 0, s>>>(z, in_f32, xp, out_f32, B, C, H, W, p);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_unpatchify(const void* xp, void* z, int dtype, int B, int C, int H, int W, int p, cudaStream_t s) {
  const int64_t n = (int64_t)B * C * H * W;
  unpatchify_kernel<<<grid_for(n, 256), 256, 0, s>>>(xp, z, dtype == JAGG_DTYPE_F32, B, C, H, W, p);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_timestep_embedding(const float* t, float* phi, int B, int dim, cudaStream_t s) {
  temb_kernel<<<grid_for((int64_t)B * dim / 2, 256), 256, 0, s>>>(t, phi, B, dim);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_silu(const float* in, float* out, int64_t n, cudaStream_t s) {
  silu_kernel<<<grid_for(n, 256), 256, 0, s>>>(in, out, n);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_mul_silu_grad(float* g, const float* x, int64_t n, cudaStream_t s) {
  mul_silu_grad_kernel<<<grid_for(n, 256), 256, 0, s>>>(g, x, n);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_add_pos_embed(float* h, int B, int rows_per_seq, int row0, int gh, int gw, int d, cudaStream_t s) {
  pos_embed_kernel<<<grid_for((int64_t)B * gh * gw * d, 256), 256, 0, s>>>(h, B, rows_per_seq, row0, gh, gw, d);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_ln_mod_fwd(const LnModFwd& a, cudaStream_t s) {
  JAGG_CHECK_ARG(a.d % 4 == 0 && a.d <= 128 * LN_MAXV, "ln_mod: hidden %d unsupported", a.d);
  const int warps = 8;
  ln_mod_fwd_kernel<<<ceil_div(a.M, warps), warps * 32, 0, s>>>(a);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_ln_gate_bwd(const LnGateBwd& a, cudaStream_t s) {
  JAGG_CHECK_ARG(a.d <= LNB_THREADS * LNB_MAXC, "ln_gate_bwd: hidden %d unsupported", a.d);
  JAGG_CHECK_ARG(a.M % a.rows_per_seq == 0, "ln_gate_bwd: rows not a whole number of sequences");
  const int seqs = a.M / a.rows_per_seq;
  const int chunks = ceil_div(a.rows_per_seq, LNB_ROWS);
  ln_gate_bwd_kernel<<<seqs * chunks, LNB_THREADS, 0, s>>>(a);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_colsum(const void* X, int x_f32, int dtype, int rows, int cols, int64_t ld, float* db, cudaStream_t s) {
  (void)dtype;
  dim3 grid(ceil_div(cols, 256), ceil_div(rows, CS_ROWS));
  colsum_kernel<<<grid, 256, 0, s>>>(X, x_f32, rows, cols, ld, db);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_gather_rows(const float* in, int64_t ld_in, int seg, int seg_off, int64_t seg_stride, void* out,
                       int dtype, int rows, int cols, cudaStream_t s) {
  gather_rows_kernel<<<grid_for((int64_t)rows * cols, 256), 256, 0, s>>>(in, ld_in, seg, seg_off, seg_stride, out,
                                                                         dtype == JAGG_DTYPE_F32, rows, cols);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_copy_rows(const void* in, int64_t ld_in, int in_seg, int in_seg_off, int64_t in_seg_stride, void* out,
                     int64_t ld_out, int out_seg, int out_seg_off, int64_t out_seg_stride, int rows, int cols,
                     int elem_bytes, cudaStream_t s) {
  const int g = grid_for((int64_t)rows * cols, 256);
  if (elem_bytes == 4)
    copy_rows_kernel<float><<<g, 256, 0, s>>>(static_cast<const float*>(in), ld_in, in_seg, in_seg_off, in_seg_stride,
                                             static_cast<float*>(out), ld_out, out_seg, out_seg_off, out_seg_stride,
                                             rows, cols);
  else
    copy_rows_kernel<uint16_t><<<g, 256, 0, s>>>(static_cast<const uint16_t*>(in), ld_in, in_seg, in_seg_off,
                                                in_seg_stride, static_cast<uint16_t*>(out), ld_out, out_seg,
                                                out_seg_off, out_seg_stride, rows, cols);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_attn_rowdot(const void* dO, const void* O, int64_t ld, float* Dv, int B, int N, int heads, int dh,
                       int dtype, cudaStream_t s) {
  const int64_t warps = (int64_t)B * N * heads;
  attn_rowdot_kernel<<<grid_for(warps * 32, 256), 256, 0, s>>>(dO, O, ld, Dv, B, N, heads, dh,
                                                              dtype == JAGG_DTYPE_F32);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_qk_norm_rope_fwd(const QkNormRope& a, cudaStream_t s) {
  JAGG_CHECK_ARG(a.d / a.heads <= 128, "qk_norm: head dim too large");
  const int64_t warps = (int64_t)a.M * a.heads;
  qk_norm_rope_fwd_kernel<<<grid_for(warps * 32, 256), 256, 0, s>>>(a);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
int launch_qk_norm_rope_bwd(const QkNormRopeBwd& a, cudaStream_t s) {
  const int64_t warps = (int64_t)a.f.M * a.f.heads;
  qk_norm_rope_bwd_kernel<<<grid_for(warps * 32, 256), 256, 0, s>>>(a);
  JAGG_LAUNCHED();
  return JAGG_OK;
}

}  // namespace jagg
