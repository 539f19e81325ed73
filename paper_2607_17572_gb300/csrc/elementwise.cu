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
    // f32 is enough here (|argument| < grid size, error ~1e-6); f64 is slow on this part
    const float pos = half == 0 ? (float)(n / gw) : (float)(n % gw);
    const float a = pos * expf(-9.210340371976184f * (float)k / (float)q);  // ln(10000)
    const float v = cc < q ? sinf(a) : cosf(a);
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

// Backward of LayerNorm + modulation and of a gated residual branch.
__device__ __forceinline__ void load4(const void* p, int64_t i, int is_f32, float (&v)[4]) {
  if (is_f32) {
    const float4 f = *reinterpret_cast<const float4*>(static_cast<const float*>(p) + i);
    v[0] = f.x; v[1] = f.y; v[2] = f.z; v[3] = f.w;
  } else {
    const uint2 raw = *reinterpret_cast<const uint2*>(static_cast<const bf16*>(p) + i);
    const bf16* h = reinterpret_cast<const bf16*>(&raw);
    v[0] = __bfloat162float(h[0]); v[1] = __bfloat162float(h[1]);
    v[2] = __bfloat162float(h[2]); v[3] = __bfloat162float(h[3]);
  }
}
__device__ __forceinline__ void store4(void* p, int64_t i, int is_f32, const float (&v)[4]) {
  if (is_f32) {
    *reinterpret_cast<float4*>(static_cast<float*>(p) + i) = make_float4(v[0], v[1], v[2], v[3]);
  } else {
    __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]), b = __floats2bfloat162_rn(v[2], v[3]);
    uint2 raw;
    raw.x = *reinterpret_cast<uint32_t*>(&a);
    raw.y = *reinterpret_cast<uint32_t*>(&b);
    *reinterpret_cast<uint2*>(static_cast<bf16*>(p) + i) = raw;
  }
}

// One pass per row tile: a block of 8 warps takes LNF_ROWS rows of one sequence, each warp
// LNF_R of them.  Per row: the LayerNorm input-gradient (added to the residual gradient
// dh) and dy = gate * dh.  The per-sequence column sums (dshift, dscale, dgate, and sum dh
// for the bias gradient: sum_m dy = gate * sum_m dh) are summed over a warp's rows in
// registers, then over the block in shared memory (laid out [quantity][element][d/4] so a
// warp's atomics hit consecutive words), then flushed with one global atomic per column.
constexpr int LNF_R = 4;
constexpr int LNF_ROWS = 8 * LNF_R;

// Persistent: the grid walks the (sequence, row-chunk) units, so no wave tail.  NVT > 0
// fixes the number of float4 column groups per lane (d = 128 NVT) at compile time, so the
// column loops unroll and a warp's loads for its rows are issued together.
#ifndef LNF_MIN_BLOCKS
#define LNF_MIN_BLOCKS 3
#endif
template <int NVT>
__global__ void __launch_bounds__(256, LNF_MIN_BLOCKS) ln_gate_fused_kernel(LnGateBwd a) {
  extern __shared__ float part[];  // [4 quantities][4][d/4]
  const int d = a.d, d4 = a.d / 4;
  const int chunks = (a.rows_per_seq + LNF_ROWS - 1) / LNF_ROWS;
  const int units = (a.M / a.rows_per_seq) * chunks;
  const int warp = threadIdx.x / 32, lane = threadIdx.x & 31;
  const int is_f32 = a.dtype == JAGG_DTYPE_F32;
  const int nv = NVT > 0 ? NVT : (d + 127) / 128;
  for (int unit = blockIdx.x; unit < units; unit += gridDim.x) {
    const int b = unit / chunks;
    const int r0 = (unit % chunks) * LNF_ROWS;
    for (int i = threadIdx.x; i < 4 * d; i += blockDim.x) part[i] = 0.f;
    __syncthreads();
    const float* gate = a.do_gate ? a.gate + (int64_t)b * a.mod_stride : nullptr;
    const float* sc = a.do_ln ? a.scale + (int64_t)b * a.mod_stride : nullptr;
    int mrow[LNF_R];
    int64_t hrow[LNF_R];
    bool live[LNF_R];
    float mu[LNF_R], rs[LNF_R], s1[LNF_R], s2[LNF_R];
#pragma unroll
    for (int k = 0; k < LNF_R; ++k) {
      const int r = r0 + warp * LNF_R + k;
      live[k] = r < a.rows_per_seq;
      mrow[k] = b * a.rows_per_seq + (live[k] ? r : 0);
      hrow[k] = seg_row(mrow[k], a.seg, a.seg_off, a.seg_stride);
      mu[k] = rs[k] = s1[k] = s2[k] = 0.f;
    }
    if (a.do_ln) {
#pragma unroll
      for (int k = 0; k < LNF_R; ++k) {
        if (live[k]) {
          mu[k] = a.mean[mrow[k]];
          rs[k] = a.rstd[mrow[k]];
        }
      }
#pragma unroll
      for (int i = 0; i < (NVT > 0 ? NVT : 1); ++i) {
        for (int ii = i; ii < (NVT > 0 ? i + 1 : nv); ++ii) {
          const int c = (ii * 32 + lane) * 4;
          if (c >= d) continue;
          const float4 s4 = *reinterpret_cast<const float4*>(sc + c);
          const float sv[4] = {s4.x, s4.y, s4.z, s4.w};
#pragma unroll
          for (int k = 0; k < LNF_R; ++k) {
            if (!live[k]) continue;
            float dm[4];
            load4(a.dm, (int64_t)mrow[k] * d + c, a.dm_f32, dm);
            const float4 h4 = *reinterpret_cast<const float4*>(a.h + hrow[k] * d + c);
            const float hv[4] = {h4.x, h4.y, h4.z, h4.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float dxh = dm[e] * (1.f + sv[e]);
              s1[k] += dxh;
              s2[k] += dxh * (hv[e] - mu[k]) * rs[k];
            }
          }
        }
      }
#pragma unroll
      for (int k = 0; k < LNF_R; ++k) {
        s1[k] = warp_sum(s1[k]) / d;
        s2[k] = warp_sum(s2[k]) / d;
      }
    }
#pragma unroll
    for (int i = 0; i < (NVT > 0 ? NVT : 1); ++i) {
      for (int ii = i; ii < (NVT > 0 ? i + 1 : nv); ++ii) {
        const int c = (ii * 32 + lane) * 4;
        if (c >= d) continue;
        float acc[4][4];  // [quantity][element]
#pragma unroll
        for (int q = 0; q < 4; ++q)
#pragma unroll
          for (int e = 0; e < 4; ++e) acc[q][e] = 0.f;
        float sv[4] = {0.f, 0.f, 0.f, 0.f}, gv[4] = {0.f, 0.f, 0.f, 0.f};
        if (a.do_ln) {
          const float4 s4 = *reinterpret_cast<const float4*>(sc + c);
          sv[0] = s4.x; sv[1] = s4.y; sv[2] = s4.z; sv[3] = s4.w;
        }
        if (gate) {
          const float4 g4 = *reinterpret_cast<const float4*>(gate + c);
          gv[0] = g4.x; gv[1] = g4.y; gv[2] = g4.z; gv[3] = g4.w;
        }
#pragma unroll
        for (int k = 0; k < LNF_R; ++k) {
          if (!live[k]) continue;
          const float4 d4v = *reinterpret_cast<const float4*>(a.dh_in + hrow[k] * d + c);
          float dh[4] = {d4v.x, d4v.y, d4v.z, d4v.w};
          if (a.do_ln) {
            float dm[4];
            load4(a.dm, (int64_t)mrow[k] * d + c, a.dm_f32, dm);
            const float4 h4 = *reinterpret_cast<const float4*>(a.h + hrow[k] * d + c);
            const float hv[4] = {h4.x, h4.y, h4.z, h4.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float xh = (hv[e] - mu[k]) * rs[k];
              dh[e] += rs[k] * (dm[e] * (1.f + sv[e]) - s1[k] - xh * s2[k]);
              acc[0][e] += dm[e];
              acc[1][e] += dm[e] * xh;
            }
            *reinterpret_cast<float4*>(a.dh_out + hrow[k] * d + c) = make_float4(dh[0], dh[1], dh[2], dh[3]);
          }
          if (gate) {
            const float dy[4] = {gv[0] * dh[0], gv[1] * dh[1], gv[2] * dh[2], gv[3] * dh[3]};
            store4(a.dy, (int64_t)mrow[k] * d + c, is_f32, dy);
            float yv[4];
            load4(a.y, (int64_t)mrow[k] * d + c, is_f32, yv);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              acc[2][e] += dh[e] * yv[e];
              acc[3][e] += dh[e];
            }
          }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          if (q < 2 ? !a.do_ln : !gate) continue;
#pragma unroll
          for (int e = 0; e < 4; ++e) atomicAdd(&part[(q * 4 + e) * d4 + c / 4], acc[q][e]);
        }
      }
    }
    __syncthreads();
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
      auto P = [&](int q) { return part[(q * 4 + c % 4) * d4 + c / 4]; };
      if (a.do_ln) {
        atomicAdd(a.dshift + (int64_t)b * a.dmod_stride + c, P(0));
        atomicAdd(a.dscale + (int64_t)b * a.dmod_stride + c, P(1));
      }
      if (a.do_gate) {
        atomicAdd(a.dgate + (int64_t)b * a.dmod_stride + c, P(2));
        if (a.dbias) atomicAdd(a.dbias + c, gate[c] * P(3));
      }
    }
    __syncthreads();  // the partials are re-zeroed by the next unit
  }
}

// Row-in-registers variant for d = 128 NV <= 768, with the LayerNorm part always present and
// dm in f32 (GATE: the gate part too; YBF: y and dy in bf16).  A warp issues every load of
// one row at once (dh, dm, h, y: float4-wide groups per 128 columns), forms the row
// statistics with two warp reductions and updates the row without a second pass.  The
// sequence's scale and gate vectors sit in shared memory for the whole segment.  The
// per-sequence column sums go to a warp-private shared-memory slab ([4 quantities][d],
// plain read-modify-write, no atomics), summed over the block's 8 warps and flushed with
// atomics once per sequence segment.  Each CTA owns a contiguous, equal share of the rows
// (at most a few sequence segments), so every CTA finishes at the same time.
template <int NV, bool GATE, bool YBF>
__global__ void __launch_bounds__(256, 2) ln_gate_rowreg_kernel(LnGateBwd a) {
  extern __shared__ float part[];  // [8 warps][4 quantities][d], then scale[d], gate[d]
  constexpr int d = 128 * NV;
  const int warp = threadIdx.x / 32, lane = threadIdx.x & 31;
  float* mine = part + warp * 4 * d;
  float* sc_s = part + 8 * 4 * d;
  float* gt_s = sc_s + d;
  const int row_begin = (int)((int64_t)a.M * blockIdx.x / gridDim.x);
  const int row_end = (int)((int64_t)a.M * (blockIdx.x + 1) / gridDim.x);
  for (int seg0 = row_begin; seg0 < row_end;) {
    const int b = seg0 / a.rows_per_seq;
    const int seg1 = min(row_end, (b + 1) * a.rows_per_seq);
    for (int i = lane; i < 4 * d; i += 32) mine[i] = 0.f;
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
      sc_s[c] = 1.f + a.scale[(int64_t)b * a.mod_stride + c];
      if (GATE) gt_s[c] = a.gate[(int64_t)b * a.mod_stride + c];
    }
    __syncthreads();
#pragma unroll 1
    for (int m = seg0 + warp; m < seg1; m += 8) {
      const int64_t hr = seg_row(m, a.seg, a.seg_off, a.seg_stride);
      const float mu = a.mean[m], rs = a.rstd[m];
      float4 dh[NV], dm[NV], hv[NV];
      uint2 yb[NV];
      float4 yf[NV];
#pragma unroll
      for (int i = 0; i < NV; ++i) {
        const int c = (i * 32 + lane) * 4;
        dh[i] = *reinterpret_cast<const float4*>(a.dh_in + hr * d + c);
        dm[i] = *reinterpret_cast<const float4*>(static_cast<const float*>(a.dm) + (int64_t)m * d + c);
        hv[i] = *reinterpret_cast<const float4*>(a.h + hr * d + c);
        if (GATE) {
          if (YBF)
            yb[i] = *reinterpret_cast<const uint2*>(static_cast<const bf16*>(a.y) + (int64_t)m * d + c);
          else
            yf[i] = *reinterpret_cast<const float4*>(static_cast<const float*>(a.y) + (int64_t)m * d + c);
        }
      }
      float s1 = 0.f, s2 = 0.f;
#pragma unroll
      for (int i = 0; i < NV; ++i) {
        const float4 sv = *reinterpret_cast<const float4*>(sc_s + (i * 32 + lane) * 4);
        hv[i].x = (hv[i].x - mu) * rs; hv[i].y = (hv[i].y - mu) * rs;  // now x-hat
        hv[i].z = (hv[i].z - mu) * rs; hv[i].w = (hv[i].w - mu) * rs;
        const float e0 = dm[i].x * sv.x, e1 = dm[i].y * sv.y, e2 = dm[i].z * sv.z, e3 = dm[i].w * sv.w;
        s1 += (e0 + e1) + (e2 + e3);
        s2 += (e0 * hv[i].x + e1 * hv[i].y) + (e2 * hv[i].z + e3 * hv[i].w);
      }
      s1 = warp_sum(s1) / d;
      s2 = warp_sum(s2) / d;
#pragma unroll
      for (int i = 0; i < NV; ++i) {
        const int c = (i * 32 + lane) * 4;
        const float4 sv = *reinterpret_cast<const float4*>(sc_s + c);
        dh[i].x += rs * (dm[i].x * sv.x - s1 - hv[i].x * s2);
        dh[i].y += rs * (dm[i].y * sv.y - s1 - hv[i].y * s2);
        dh[i].z += rs * (dm[i].z * sv.z - s1 - hv[i].z * s2);
        dh[i].w += rs * (dm[i].w * sv.w - s1 - hv[i].w * s2);
        *reinterpret_cast<float4*>(a.dh_out + hr * d + c) = dh[i];
        float4* q0 = reinterpret_cast<float4*>(mine + c);
        float4* q1 = reinterpret_cast<float4*>(mine + d + c);
        float4 u = *q0, w = *q1;
        u.x += dm[i].x; u.y += dm[i].y; u.z += dm[i].z; u.w += dm[i].w;
        w.x += dm[i].x * hv[i].x; w.y += dm[i].y * hv[i].y; w.z += dm[i].z * hv[i].z; w.w += dm[i].w * hv[i].w;
        *q0 = u;
        *q1 = w;
        if (GATE) {
          float y0, y1, y2, y3;
          if (YBF) {
            const bf16* h = reinterpret_cast<const bf16*>(&yb[i]);
            y0 = __bfloat162float(h[0]); y1 = __bfloat162float(h[1]);
            y2 = __bfloat162float(h[2]); y3 = __bfloat162float(h[3]);
          } else {
            y0 = yf[i].x; y1 = yf[i].y; y2 = yf[i].z; y3 = yf[i].w;
          }
          const float4 g4 = *reinterpret_cast<const float4*>(gt_s + c);
          const float dy[4] = {g4.x * dh[i].x, g4.y * dh[i].y, g4.z * dh[i].z, g4.w * dh[i].w};
          store4(a.dy, (int64_t)m * d + c, !YBF, dy);
          float4* q2 = reinterpret_cast<float4*>(mine + 2 * d + c);
          float4* q3 = reinterpret_cast<float4*>(mine + 3 * d + c);
          float4 u2 = *q2, w2 = *q3;
          u2.x += dh[i].x * y0; u2.y += dh[i].y * y1; u2.z += dh[i].z * y2; u2.w += dh[i].w * y3;
          w2.x += dh[i].x; w2.y += dh[i].y; w2.z += dh[i].z; w2.w += dh[i].w;
          *q2 = u2;
          *q3 = w2;
        }
      }
    }
    __syncthreads();
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
      float P[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int w = 0; w < 8; ++w)
#pragma unroll
        for (int q = 0; q < (GATE ? 4 : 2); ++q) P[q] += part[(w * 4 + q) * d + c];
      atomicAdd(a.dshift + (int64_t)b * a.dmod_stride + c, P[0]);
      atomicAdd(a.dscale + (int64_t)b * a.dmod_stride + c, P[1]);
      if (GATE) {
        atomicAdd(a.dgate + (int64_t)b * a.dmod_stride + c, P[2]);
        if (a.dbias) atomicAdd(a.dbias + c, gt_s[c] * P[3]);
      }
    }
    __syncthreads();  // the slabs and vectors are rewritten for the next segment
    seg0 = seg1;
  }
}

// Row-per-CTA variant for d = 1024 NV4 (d = 3072 at the Flux and Qwen widths; bf16 y and
// dy, dm in f32 when the LayerNorm part is present).  The 256 threads of a block take one row at a time,
// each holding NV4 float4 column groups of every operand in registers, so every row is read
// once and written once.  The row statistics are two block reductions: warp shuffles, then
// the 8 warp partials through a shared slot double-buffered by row parity (one barrier per
// row).  Each CTA owns a contiguous, equal share of the rows and each thread the same columns
// for all of them, so the per-sequence column sums (dshift, dscale, dgate, sum dh for the
// bias gradient) stay in registers and leave by one global atomic per column and quantity
// at each sequence boundary.
template <int NV4, bool LN, bool GATE>
__global__ void __launch_bounds__(256, 2) ln_gate_rowcta_kernel(LnGateBwd a) {
  constexpr int d = 1024 * NV4;
  __shared__ float red[2][2][8];  // [row parity][s1, s2][warp]
  __shared__ __align__(16) float sc_s[LN ? d : 4], gt_s[GATE ? d : 4];  // 1 + scale, gate of the sequence
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int row_begin = (int)((int64_t)a.M * blockIdx.x / gridDim.x);
  const int row_end = (int)((int64_t)a.M * (blockIdx.x + 1) / gridDim.x);
  int parity = 0;
  for (int seg0 = row_begin; seg0 < row_end;) {
    const int b = seg0 / a.rows_per_seq;
    const int seg1 = min(row_end, (b + 1) * a.rows_per_seq);
    float4 acc[4][NV4];
    __syncthreads();  // the previous segment's readers of the vectors are done
#pragma unroll
    for (int i = 0; i < NV4; ++i) {
      const int c = (i * 256 + tid) * 4;
      if (LN) {
        float4 v = *reinterpret_cast<const float4*>(a.scale + (int64_t)b * a.mod_stride + c);
        v.x += 1.f; v.y += 1.f; v.z += 1.f; v.w += 1.f;
        *reinterpret_cast<float4*>(sc_s + c) = v;
      }
      if (GATE) *reinterpret_cast<float4*>(gt_s + c) = *reinterpret_cast<const float4*>(a.gate + (int64_t)b * a.mod_stride + c);
#pragma unroll
      for (int q = 0; q < 4; ++q) acc[q][i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    __syncthreads();
#pragma unroll 1
    for (int m = seg0; m < seg1; ++m) {
      const int64_t hr = seg_row(m, a.seg, a.seg_off, a.seg_stride);
      float4 dh[NV4], dm[NV4], hv[NV4];
      uint2 yb[NV4];  // y in bf16
#pragma unroll
      for (int i = 0; i < NV4; ++i) {
        const int c = (i * 256 + tid) * 4;
        dh[i] = *reinterpret_cast<const float4*>(a.dh_in + hr * d + c);
        if (LN) {
          dm[i] = *reinterpret_cast<const float4*>(static_cast<const float*>(a.dm) + (int64_t)m * d + c);
          hv[i] = *reinterpret_cast<const float4*>(a.h + hr * d + c);
        }
        if (GATE) yb[i] = *reinterpret_cast<const uint2*>(static_cast<const bf16*>(a.y) + (int64_t)m * d + c);
      }
      if (LN) {
        const float mu = a.mean[m], rs = a.rstd[m];
        float s1 = 0.f, s2 = 0.f;
#pragma unroll
        for (int i = 0; i < NV4; ++i) {
          hv[i].x = (hv[i].x - mu) * rs; hv[i].y = (hv[i].y - mu) * rs;  // now x-hat
          hv[i].z = (hv[i].z - mu) * rs; hv[i].w = (hv[i].w - mu) * rs;
          const float4 sv = *reinterpret_cast<const float4*>(sc_s + (i * 256 + tid) * 4);
          const float e0 = dm[i].x * sv.x, e1 = dm[i].y * sv.y, e2 = dm[i].z * sv.z, e3 = dm[i].w * sv.w;
          s1 += (e0 + e1) + (e2 + e3);
          s2 += (e0 * hv[i].x + e1 * hv[i].y) + (e2 * hv[i].z + e3 * hv[i].w);
        }
        s1 = warp_sum(s1);
        s2 = warp_sum(s2);
        if (lane == 0) {
          red[parity][0][warp] = s1;
          red[parity][1][warp] = s2;
        }
        __syncthreads();
        s1 = 0.f;
        s2 = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) {
          s1 += red[parity][0][w];
          s2 += red[parity][1][w];
        }
        s1 /= d;
        s2 /= d;
        parity ^= 1;
#pragma unroll
        for (int i = 0; i < NV4; ++i) {
          const int c = (i * 256 + tid) * 4;
          const float4 sv = *reinterpret_cast<const float4*>(sc_s + c);
          dh[i].x += rs * (dm[i].x * sv.x - s1 - hv[i].x * s2);
          dh[i].y += rs * (dm[i].y * sv.y - s1 - hv[i].y * s2);
          dh[i].z += rs * (dm[i].z * sv.z - s1 - hv[i].z * s2);
          dh[i].w += rs * (dm[i].w * sv.w - s1 - hv[i].w * s2);
          *reinterpret_cast<float4*>(a.dh_out + hr * d + c) = dh[i];
          acc[0][i].x += dm[i].x; acc[0][i].y += dm[i].y; acc[0][i].z += dm[i].z; acc[0][i].w += dm[i].w;
          acc[1][i].x += dm[i].x * hv[i].x; acc[1][i].y += dm[i].y * hv[i].y;
          acc[1][i].z += dm[i].z * hv[i].z; acc[1][i].w += dm[i].w * hv[i].w;
        }
      }
      if (GATE) {
#pragma unroll
        for (int i = 0; i < NV4; ++i) {
          const int c = (i * 256 + tid) * 4;
          const float4 g4 = *reinterpret_cast<const float4*>(gt_s + c);
          const float dy[4] = {g4.x * dh[i].x, g4.y * dh[i].y, g4.z * dh[i].z, g4.w * dh[i].w};
          store4(a.dy, (int64_t)m * d + c, 0, dy);
          const bf16* yh = reinterpret_cast<const bf16*>(&yb[i]);
          acc[2][i].x += dh[i].x * __bfloat162float(yh[0]); acc[2][i].y += dh[i].y * __bfloat162float(yh[1]);
          acc[2][i].z += dh[i].z * __bfloat162float(yh[2]); acc[2][i].w += dh[i].w * __bfloat162float(yh[3]);
          acc[3][i].x += dh[i].x; acc[3][i].y += dh[i].y; acc[3][i].z += dh[i].z; acc[3][i].w += dh[i].w;
        }
      }
    }
#pragma unroll
    for (int i = 0; i < NV4; ++i) {
      const int c = (i * 256 + tid) * 4;
      const float* q0 = &acc[0][i].x;
      const float* q1 = &acc[1][i].x;
      const float* q2 = &acc[2][i].x;
      const float* q3 = &acc[3][i].x;
      const float* g4 = gt_s + c;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if (LN) {
          atomicAdd(a.dshift + (int64_t)b * a.dmod_stride + c + e, q0[e]);
          atomicAdd(a.dscale + (int64_t)b * a.dmod_stride + c + e, q1[e]);
        }
        if (GATE) {
          atomicAdd(a.dgate + (int64_t)b * a.dmod_stride + c + e, q2[e]);
          if (a.dbias) atomicAdd(a.dbias + c + e, g4[e] * q3[e]);
        }
      }
    }
    seg0 = seg1;
  }
}

template <int NV4, bool LN, bool GATE>
int launch_ln_gate_rowcta_t(const LnGateBwd& a, cudaStream_t s) {
  static int per_sm = 0;
  if (!per_sm) {
    JAGG_CUDA_TRY(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ln_gate_rowcta_kernel<NV4, LN, GATE>, 256, 0));
    if (per_sm < 1) per_sm = 1;
  }
  // equal row shares of at least 8 rows per CTA, at most one wave of resident CTAs
  const int cap = per_sm * sm_count();
  const int want = ceil_div(a.M, 8);
  ln_gate_rowcta_kernel<NV4, LN, GATE><<<want < cap ? want : cap, 256, 0, s>>>(a);
  JAGG_LAUNCHED();
  return JAGG_OK;
}

template <int NV4>
int launch_ln_gate_rowcta(const LnGateBwd& a, cudaStream_t s) {
  if (a.do_ln) return a.do_gate ? launch_ln_gate_rowcta_t<NV4, true, true>(a, s)
                                : launch_ln_gate_rowcta_t<NV4, true, false>(a, s);
  return launch_ln_gate_rowcta_t<NV4, false, true>(a, s);
}

template <int NV, bool GATE, bool YBF>
int launch_ln_gate_rowreg_t(const LnGateBwd& a, cudaStream_t s) {
  const int smem = (8 * 4 + 2) * 128 * NV * (int)sizeof(float);
  static bool attr = false;
  if (!attr) {
    JAGG_CUDA_TRY(cudaFuncSetAttribute(ln_gate_rowreg_kernel<NV, GATE, YBF>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    attr = true;
  }
  static int per_sm = 0;
  if (!per_sm) {
    JAGG_CUDA_TRY(
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ln_gate_rowreg_kernel<NV, GATE, YBF>, 256, smem));
    if (per_sm < 1) per_sm = 1;
  }
  // equal row shares of at least 16 rows per CTA, at most one wave of resident CTAs
  const int cap = per_sm * sm_count();
  const int want = ceil_div(a.M, 16);
  ln_gate_rowreg_kernel<NV, GATE, YBF><<<want < cap ? want : cap, 256, smem, s>>>(a);
  JAGG_LAUNCHED();
  return JAGG_OK;
}

template <int NVT>
int launch_ln_gate_nv(const LnGateBwd& a, int smem, cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    JAGG_CUDA_TRY(cudaFuncSetAttribute(ln_gate_fused_kernel<NVT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       4 * 3072 * (int)sizeof(float)));
    attr = true;
  }
  static int per_sm = 0;
  if (!per_sm) {
    JAGG_CUDA_TRY(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ln_gate_fused_kernel<NVT>, 256,
                                                                4 * 3072 * (int)sizeof(float)));
    if (per_sm < 1) per_sm = 1;
  }
  const int units = (a.M / a.rows_per_seq) * ceil_div(a.rows_per_seq, LNF_ROWS);
  const int cap = per_sm * sm_count();
  ln_gate_fused_kernel<NVT><<<units < cap ? units : cap, 256, smem, s>>>(a);
  JAGG_LAUNCHED();
  return JAGG_OK;
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

// Column sums of a bf16 matrix, 8 columns (one 16-byte load) per thread: block = 32 column
// groups (256 columns) x 8 row slices over CSV_ROWS rows; the 8 slices meet in shared memory
// and each column gets one atomic add per block.
constexpr int CSV_ROWS = 256;
__global__ void __launch_bounds__(256) colsum_bf16x8_kernel(const bf16* X, int rows, int cols, int64_t ld, float* db) {
  __shared__ float part[8][257];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const int c0 = (blockIdx.x * 32 + tx) * 8;
  const int r0 = blockIdx.y * CSV_ROWS;
  const int r1 = min(r0 + CSV_ROWS, rows);
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (c0 < cols) {
#pragma unroll 4
    for (int r = r0 + ty; r < r1; r += 8) {
      const uint4 raw = *reinterpret_cast<const uint4*>(X + (int64_t)r * ld + c0);
      const bf16* h = reinterpret_cast<const bf16*>(&raw);
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] += __bfloat162float(h[i]);
    }
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) part[ty][tx * 8 + i] = acc[i];
  __syncthreads();
  const int c = blockIdx.x * 256 + threadIdx.x;
  if (c < cols) {
    float t = 0.f;
#pragma unroll
    for (int y = 0; y < 8; ++y) t += part[y][threadIdx.x];
    atomicAdd(db + c, t);
  }
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

// Whole rows in 16-byte vectors, a row per block iteration (row pitches, row bytes and both
// bases 16-byte aligned).
__global__ void copy_rows_v16_kernel(const uint8_t* in, int64_t ld_in_b, int is, int io, int64_t iss, uint8_t* out,
                                     int64_t ld_out_b, int os, int oo, int64_t oss, int rows, int nvec) {
  for (int r = blockIdx.x; r < rows; r += gridDim.x) {
    const uint4* src = reinterpret_cast<const uint4*>(in + seg_row(r, is, io, iss) * ld_in_b);
    uint4* dst = reinterpret_cast<uint4*>(out + seg_row(r, os, oo, oss) * ld_out_b);
    for (int c = threadIdx.x; c < nvec; c += blockDim.x) dst[c] = __ldg(src + c);
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
  // f32: the angle pos * theta (pos < grid size) is off by a few 1e-6 rad at most
  const float pos = axis == 0 ? (float)(tok / gw) : (float)(tok % gw);
  const float th = exp2f(-13.287712379549449f * 2.f * (float)i / (float)hd);  // 10000^(-2i/hd)
  sincosf(pos * th, &sn, &cs);
}

// Grid-stride over (row, head) items, one warp per item; lane j owns the rotated pairs j
// and j + 32 of the head.
constexpr int QKN_THREADS = 256, QKN_WARPS = QKN_THREADS / 32;

__global__ void __launch_bounds__(QKN_THREADS) qk_norm_rope_fwd_kernel(QkNormRope a) {
  const int lane = threadIdx.x & 31;
  const int dh = a.d / a.heads;
  const int is_f32 = a.dtype == JAGG_DTYPE_F32;
  const int64_t items = (int64_t)a.M * a.heads;
  for (int64_t w = (int64_t)blockIdx.x * QKN_WARPS + threadIdx.x / 32; w < items;
       w += (int64_t)gridDim.x * QKN_WARPS) {
    const int hd = (int)(w % a.heads);
    const int m = (int)(w / a.heads);
    const int n = m % a.N;
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
}

// The scale gradients sum over every (row, head): each lane keeps its elements' partial
// sums in registers (q / k x text / image), the block adds its warps' partials in shared
// memory and issues one atomic per element.
__global__ void __launch_bounds__(QKN_THREADS) qk_norm_rope_bwd_kernel(QkNormRopeBwd b) {
  const QkNormRope& a = b.f;
  __shared__ float part[QKN_WARPS][4][128];
  const int lane = threadIdx.x & 31, warp = threadIdx.x / 32;
  const int dh = a.d / a.heads;
  const int is_f32 = a.dtype == JAGG_DTYPE_F32;
  float acc[4][4];  // [which * 2 + stream][element]
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[i][e] = 0.f;
  const int64_t items = (int64_t)a.M * a.heads;
  for (int64_t w = (int64_t)blockIdx.x * QKN_WARPS + warp; w < items; w += (int64_t)gridDim.x * QKN_WARPS) {
    const int hd = (int)(w % a.heads);
    const int m = (int)(w / a.heads);
    const int n = m % a.N;
    const bool txt = n < a.n_txt;
#pragma unroll
    for (int which = 0; which < 2; ++which) {
      const void* scl = which == 0 ? (txt ? a.qscale_txt : a.qscale_img) : (txt ? a.kscale_txt : a.kscale_img);
      const float r = (which == 0 ? a.rq : a.rk)[(int64_t)m * a.heads + hd];
      const int64_t xb = (int64_t)m * a.ld_qkv + which * a.d + hd * dh;
      const int64_t gb = (int64_t)m * b.ld_dqk + which * a.d + hd * dh;
      float x[4] = {0.f, 0.f, 0.f, 0.f}, u[4] = {0.f, 0.f, 0.f, 0.f}, dsc[4] = {0.f, 0.f, 0.f, 0.f};
      float xu = 0.f;
#pragma unroll
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
          dsc[2 * j] = dy0 * x[2 * j] * r;
          dsc[2 * j + 1] = dy1 * x[2 * j + 1] * r;
          u[2 * j] = dy0 * ldx(scl, 2 * pair, is_f32);
          u[2 * j + 1] = dy1 * ldx(scl, 2 * pair + 1, is_f32);
          xu += x[2 * j] * u[2 * j] + x[2 * j + 1] * u[2 * j + 1];
        }
      }
      const int slot = which * 2 + (txt ? 0 : 1);
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[slot][e] += dsc[e];
      xu = warp_sum(xu);
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int pair = lane + 32 * j;
        if (2 * pair < dh) {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const float dx = r * u[2 * j + e] - x[2 * j + e] * r * r * r * xu / dh;
            stx(b.dqk, gb + 2 * pair + e, is_f32, dx);
          }
        }
      }
    }
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int pair = lane + 32 * j;
      if (2 * pair < dh) {
        part[warp][i][2 * pair] = acc[i][2 * j];
        part[warp][i][2 * pair + 1] = acc[i][2 * j + 1];
      }
    }
  __syncthreads();
  float* dst[4] = {b.dqs_txt, b.dqs_img, b.dks_txt, b.dks_img};
  for (int t = threadIdx.x; t < 4 * dh; t += QKN_THREADS) {
    const int i = t / dh, c = t % dh;
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < QKN_WARPS; ++w) s += part[w][i][c];
    if (s != 0.f) atomicAdd(dst[i] + c, s);
  }
}

// Head dim 128 in bf16 (the Flux and Qwen widths): lane l owns the 4 consecutive elements
// [4l, 4l + 4) of q and of k, i.e. the rotated pairs 2l and 2l + 1, so every operand moves
// in 8-byte vectors and each lane's RMSNorm scales and RoPE frequencies are fixed for the
// whole kernel.  The angles are the ones rope_angle forms (same expressions), so the forward
// rotation and its inverse in the backward agree bit for bit.  A warp walks rows, each row's
// heads two (backward) or four (forward) at a time: 2 KB of loads in flight per warp.
constexpr int QKV_ITEMS = 2;      // heads per warp iteration of the backward
constexpr int QKV_ITEMS_FWD = 4;  // and of the forward (fewer live registers)

__device__ __forceinline__ void bf16x4_load(const bf16* p, float (&v)[4]) {
  const uint2 raw = *reinterpret_cast<const uint2*>(p);
  const bf16* h = reinterpret_cast<const bf16*>(&raw);
  v[0] = __bfloat162float(h[0]); v[1] = __bfloat162float(h[1]);
  v[2] = __bfloat162float(h[2]); v[3] = __bfloat162float(h[3]);
}
__device__ __forceinline__ void bf16x4_store(bf16* p, const float (&v)[4]) {
  __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]), b = __floats2bfloat162_rn(v[2], v[3]);
  uint2 raw;
  raw.x = *reinterpret_cast<uint32_t*>(&a);
  raw.y = *reinterpret_cast<uint32_t*>(&b);
  *reinterpret_cast<uint2*>(p) = raw;
}
// RoPE angles of head dim 128 as a table in shared memory, filled by each block: entry
// [pos][i] = (cos, sin) of pos * theta_i for the 32 frequencies of one axis, pos below the
// larger grid side; the values are rope_angle's (same expressions), so the forward rotation
// and its inverse agree bit for bit.  QKN_TABLE_MAX bounds the grid side the table serves.
constexpr int QKN_TABLE_MAX = 128;
__device__ __forceinline__ int rope_table_side(const QkNormRope& a) {
  const int gh = (a.N - a.n_txt) / a.gw;
  return gh > a.gw ? gh : a.gw;
}
__device__ __forceinline__ void rope_table_fill(const QkNormRope& a, float2* tab) {
  const int side = rope_table_side(a);
  for (int t = threadIdx.x; t < side * 32; t += blockDim.x) {
    const int pos = t / 32, i = t % 32;
    const float th = exp2f(-13.287712379549449f * 2.f * (float)i / 64.f);  // 10000^(-2i/64)
    float sn, cs;
    sincosf((float)pos * th, &sn, &cs);
    tab[t] = make_float2(cs, sn);
  }
}
// cos / sin of the lane's two pairs (2 lane, 2 lane + 1: axis lane / 16, frequencies
// 2 lane % 32 and + 1) for token n; identity for text tokens
__device__ __forceinline__ void rope_lane(const QkNormRope& a, const float2* tab, int n, int lane, float (&cs)[2],
                                          float (&sn)[2]) {
  cs[0] = cs[1] = 1.f;
  sn[0] = sn[1] = 0.f;
  if (!a.rope || n < a.n_txt) return;
  const int tok = n - a.n_txt;
  const int pos = lane < 16 ? tok / a.gw : tok % a.gw;
  const float4 v = *reinterpret_cast<const float4*>(tab + pos * 32 + ((2 * lane) & 31));
  cs[0] = v.x; sn[0] = v.y; cs[1] = v.z; sn[1] = v.w;
}

__global__ void __launch_bounds__(QKN_THREADS) qk_norm_rope_fwd_v_kernel(QkNormRope a) {
  extern __shared__ __align__(16) float2 rope_tab[];  // [side][32] when a.rope
  if (a.rope) rope_table_fill(a, rope_tab);
  __syncthreads();
  const int lane = threadIdx.x & 31;
  float scl[4][4];  // q txt, q img, k txt, k img: this lane's 4 elements
  bf16x4_load(static_cast<const bf16*>(a.qscale_txt) + 4 * lane, scl[0]);
  bf16x4_load(static_cast<const bf16*>(a.qscale_img) + 4 * lane, scl[1]);
  bf16x4_load(static_cast<const bf16*>(a.kscale_txt) + 4 * lane, scl[2]);
  bf16x4_load(static_cast<const bf16*>(a.kscale_img) + 4 * lane, scl[3]);
  // one row per warp, its heads two at a time: the token's stream and angles once per row
  for (int m = blockIdx.x * QKN_WARPS + threadIdx.x / 32; m < a.M; m += gridDim.x * QKN_WARPS) {
    const int n = m % a.N;
    const bool txt = n < a.n_txt;
    float cs[2], sn[2];
    rope_lane(a, rope_tab, n, lane, cs, sn);
    const bf16* row = static_cast<const bf16*>(a.qkv) + (int64_t)m * a.ld_qkv + 4 * lane;
    bf16* out = static_cast<bf16*>(a.qk_out) + (int64_t)m * 2 * a.d + 4 * lane;
    for (int h0 = 0; h0 < a.heads; h0 += QKV_ITEMS_FWD) {
      float x[QKV_ITEMS_FWD][2][4];
#pragma unroll
      for (int it = 0; it < QKV_ITEMS_FWD; ++it) {
        const int hd = h0 + it < a.heads ? h0 + it : h0;
#pragma unroll
        for (int which = 0; which < 2; ++which) bf16x4_load(row + which * a.d + hd * 128, x[it][which]);
      }
#pragma unroll
      for (int it = 0; it < QKV_ITEMS_FWD; ++it) {
        const int hd = h0 + it;
        if (hd >= a.heads) break;
#pragma unroll
        for (int which = 0; which < 2; ++which) {
          float sc[4];  // selected per element: the array index stays a compile-time constant
#pragma unroll
          for (int e = 0; e < 4; ++e) sc[e] = txt ? scl[which * 2][e] : scl[which * 2 + 1][e];
          const float* xv = x[it][which];
          const float r =
              rsqrtf(warp_sum(xv[0] * xv[0] + xv[1] * xv[1] + xv[2] * xv[2] + xv[3] * xv[3]) / 128.f + 1e-6f);
          float o[4];
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const float y0 = xv[2 * e] * r * sc[2 * e], y1 = xv[2 * e + 1] * r * sc[2 * e + 1];
            o[2 * e] = y0 * cs[e] - y1 * sn[e];
            o[2 * e + 1] = y0 * sn[e] + y1 * cs[e];
          }
          bf16x4_store(out + which * a.d + hd * 128, o);
          if (lane == 0) (which == 0 ? a.rq : a.rk)[(int64_t)m * a.heads + hd] = r;
        }
      }
    }
  }
}

__global__ void __launch_bounds__(QKN_THREADS, 3) qk_norm_rope_bwd_v_kernel(QkNormRopeBwd b) {
  const QkNormRope& a = b.f;
  __shared__ float part[QKN_WARPS][4][128];
  extern __shared__ __align__(16) float2 rope_tab[];  // [side][32] when a.rope
  if (a.rope) rope_table_fill(a, rope_tab);
  const int lane = threadIdx.x & 31, warp = threadIdx.x / 32;
  __shared__ __align__(16) float scl[4][128];  // q txt, q img, k txt, k img
  for (int t = threadIdx.x; t < 4 * 128; t += QKN_THREADS) {
    const void* p = t < 128 ? a.qscale_txt : t < 256 ? a.qscale_img : t < 384 ? a.kscale_txt : a.kscale_img;
    scl[t / 128][t % 128] = __bfloat162float(static_cast<const bf16*>(p)[t % 128]);
  }
  // scale gradients of the warp's rows, [which * 2 + stream][element]: one read-modify-write
  // of the lane's 4 elements per row
  float4* wpart = reinterpret_cast<float4*>(&part[warp][0][0]);
#pragma unroll
  for (int i = 0; i < 4; ++i) wpart[i * 32 + lane] = make_float4(0.f, 0.f, 0.f, 0.f);
  __syncthreads();
  // one row per warp, its heads two at a time: the token's stream and angles once per row
  for (int m = blockIdx.x * QKN_WARPS + warp; m < a.M; m += gridDim.x * QKN_WARPS) {
    const int n = m % a.N;
    const bool txt = n < a.n_txt;
    float cs[2], sn[2];
    rope_lane(a, rope_tab, n, lane, cs, sn);
    const bf16* xrow = static_cast<const bf16*>(a.qkv) + (int64_t)m * a.ld_qkv + 4 * lane;
    bf16* grow = static_cast<bf16*>(b.dqk) + (int64_t)m * b.ld_dqk + 4 * lane;
    float rowacc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};  // q, k scale gradients of the row
    for (int h0 = 0; h0 < a.heads; h0 += QKV_ITEMS) {
      float x[QKV_ITEMS][2][4], g[QKV_ITEMS][2][4];
#pragma unroll
      for (int it = 0; it < QKV_ITEMS; ++it) {
        const int hd = h0 + it < a.heads ? h0 + it : h0;
#pragma unroll
        for (int which = 0; which < 2; ++which) {
          bf16x4_load(xrow + which * a.d + hd * 128, x[it][which]);
          bf16x4_load(grow + which * a.d + hd * 128, g[it][which]);
        }
      }
#pragma unroll
      for (int it = 0; it < QKV_ITEMS; ++it) {
        const int hd = h0 + it;
        if (hd >= a.heads) break;
#pragma unroll
        for (int which = 0; which < 2; ++which) {
          const float4 sc4 = *reinterpret_cast<const float4*>(&scl[which * 2 + (txt ? 0 : 1)][4 * lane]);
          const float sc[4] = {sc4.x, sc4.y, sc4.z, sc4.w};
          const float* xv = x[it][which];
          const float r = (which == 0 ? a.rq : a.rk)[(int64_t)m * a.heads + hd];
          float u[4], dy[4];
#pragma unroll
          for (int e = 0; e < 2; ++e) {  // undo the rotation of the incoming gradient
            const float g0 = g[it][which][2 * e], g1 = g[it][which][2 * e + 1];
            dy[2 * e] = g0 * cs[e] + g1 * sn[e];
            dy[2 * e + 1] = -g0 * sn[e] + g1 * cs[e];
          }
          float xu = 0.f;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            rowacc[which][e] += dy[e] * xv[e] * r;
            u[e] = dy[e] * sc[e];
            xu += xv[e] * u[e];
          }
          xu = warp_sum(xu);
          float dx[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) dx[e] = r * u[e] - xv[e] * r * r * r * xu / 128.f;
          bf16x4_store(grow + which * a.d + hd * 128, dx);
        }
      }
    }
#pragma unroll
    for (int which = 0; which < 2; ++which) {
      float4& q = wpart[(which * 2 + (txt ? 0 : 1)) * 32 + lane];
      q.x += rowacc[which][0]; q.y += rowacc[which][1]; q.z += rowacc[which][2]; q.w += rowacc[which][3];
    }
  }
  __syncthreads();
  for (int t = threadIdx.x; t < 4 * 128; t += QKN_THREADS) {
    const int i = t / 128, c = t % 128;
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < QKN_WARPS; ++w) s += part[w][i][c];
    float* dst = i == 0 ? b.dqs_txt : i == 1 ? b.dqs_img : i == 2 ? b.dks_txt : b.dks_img;
    if (s != 0.f) atomicAdd(dst + c, s);
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
  const int tok = prof_start(s);
  ln_mod_fwd_kernel<<<ceil_div(a.M, warps), warps * 32, 0, s>>>(a);
  JAGG_LAUNCHED();
  // algorithmic bytes: h read (f32), the modulated output written (storage type), statistics
  prof_stop(tok, s, PROF_LN_FWD, 0.0,
            (double)a.M * (a.d * (4.0 + (a.dtype == JAGG_DTYPE_F32 ? 4.0 : 2.0)) + 8.0));
  return JAGG_OK;
}
// The row-in-registers kernel serves LayerNorm backwards with an f32 dm (with or without the
// gate); the rest go to the persistent kernel.
template <int NV>
int launch_ln_gate_rowreg(const LnGateBwd& a, int smem_fused, cudaStream_t s) {
  if (!a.do_ln || !a.dm_f32) return launch_ln_gate_nv<0>(a, smem_fused, s);
  if (!a.do_gate) return launch_ln_gate_rowreg_t<NV, false, false>(a, s);
  return a.dtype == JAGG_DTYPE_F32 ? launch_ln_gate_rowreg_t<NV, true, false>(a, s)
                                   : launch_ln_gate_rowreg_t<NV, true, true>(a, s);
}

int launch_ln_gate_bwd(const LnGateBwd& a, cudaStream_t s) {
  JAGG_CHECK_ARG(a.d % 4 == 0 && a.d <= 3072, "ln_gate_bwd: hidden %d unsupported", a.d);
  JAGG_CHECK_ARG(a.M % a.rows_per_seq == 0, "ln_gate_bwd: rows not a whole number of sequences");
  if (!a.do_ln && !a.do_gate) return JAGG_OK;
  const int smem = 4 * a.d * (int)sizeof(float);
  const int tok = prof_start(s);
  int st;
  switch (a.d % 128 == 0 ? a.d / 128 : 0) {
    case 3: st = launch_ln_gate_rowreg<3>(a, smem, s); break;
    case 4: st = launch_ln_gate_rowreg<4>(a, smem, s); break;
    case 6: st = launch_ln_gate_rowreg<6>(a, smem, s); break;
    case 8: st = launch_ln_gate_nv<8>(a, smem, s); break;
    case 12: st = launch_ln_gate_nv<12>(a, smem, s); break;
    case 24:
      st = (!a.do_ln || a.dm_f32) && a.dtype == JAGG_DTYPE_BF16 ? launch_ln_gate_rowcta<3>(a, s)
                                                                  : launch_ln_gate_nv<24>(a, smem, s);
      break;
    default: st = launch_ln_gate_nv<0>(a, smem, s); break;
  }
  JAGG_TRY(st);
  // algorithmic bytes: dh read + write (f32), dm (f32), h (f32), y and dy (storage type)
  const double elem = (double)a.M * a.d;
  prof_stop(tok, s, PROF_LN_BWD, 0.0,
            elem * ((a.do_ln ? 16.0 : 4.0) + (a.do_gate ? 2.0 * (a.dtype == JAGG_DTYPE_F32 ? 4 : 2) : 0.0)));
  return JAGG_OK;
}
int launch_colsum(const void* X, int x_f32, int dtype, int rows, int cols, int64_t ld, float* db, cudaStream_t s) {
  (void)dtype;
  const int tok = prof_start(s);
  // algorithmic bytes: X read once, db read and written
  const double bytes = (double)rows * cols * (x_f32 ? 4 : 2) + 8.0 * cols;
  if (!x_f32 && cols % 8 == 0 && ld % 8 == 0 && (reinterpret_cast<uintptr_t>(X) & 15) == 0) {
    dim3 grid(ceil_div(cols, 256), ceil_div(rows, CSV_ROWS));
    colsum_bf16x8_kernel<<<grid, 256, 0, s>>>(static_cast<const bf16*>(X), rows, cols, ld, db);
    JAGG_LAUNCHED();
    prof_stop(tok, s, PROF_COLSUM, 0.0, bytes);
    return JAGG_OK;
  }
  dim3 grid(ceil_div(cols, 256), ceil_div(rows, CS_ROWS));
  colsum_kernel<<<grid, 256, 0, s>>>(X, x_f32, rows, cols, ld, db);
  JAGG_LAUNCHED();
  prof_stop(tok, s, PROF_COLSUM, 0.0, bytes);
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
  const int tok = prof_start(s);
  const int64_t row_b = (int64_t)cols * elem_bytes;
  const bool v16 = row_b % 16 == 0 && (ld_in * elem_bytes) % 16 == 0 && (ld_out * elem_bytes) % 16 == 0 &&
                   (reinterpret_cast<uintptr_t>(in) & 15) == 0 && (reinterpret_cast<uintptr_t>(out) & 15) == 0;
  const int g = grid_for((int64_t)rows * cols, 256);
  if (v16 && rows > 0) {
    const int nb = rows < 8 * sm_count() ? rows : 8 * sm_count();
    copy_rows_v16_kernel<<<nb, 256, 0, s>>>(static_cast<const uint8_t*>(in), ld_in * elem_bytes, in_seg, in_seg_off,
                                            in_seg_stride, static_cast<uint8_t*>(out), ld_out * elem_bytes, out_seg,
                                            out_seg_off, out_seg_stride, rows, (int)(row_b / 16));
  } else if (elem_bytes == 4)
    copy_rows_kernel<float><<<g, 256, 0, s>>>(static_cast<const float*>(in), ld_in, in_seg, in_seg_off, in_seg_stride,
                                             static_cast<float*>(out), ld_out, out_seg, out_seg_off, out_seg_stride,
                                             rows, cols);
  else
    copy_rows_kernel<uint16_t><<<g, 256, 0, s>>>(static_cast<const uint16_t*>(in), ld_in, in_seg, in_seg_off,
                                                in_seg_stride, static_cast<uint16_t*>(out), ld_out, out_seg,
                                                out_seg_off, out_seg_stride, rows, cols);
  JAGG_LAUNCHED();
  prof_stop(tok, s, PROF_COPY, 0.0, 2.0 * rows * cols * elem_bytes);
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
// The vectorised kernels serve head dim 128 in bf16 with 8-byte aligned rows and scales.
static bool aligned8(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 7) == 0; }
static int qkn_table_bytes(const QkNormRope& a) {
  if (!a.rope) return 0;
  const int gh = (a.N - a.n_txt) / a.gw;
  return (gh > a.gw ? gh : a.gw) * 32 * (int)sizeof(float2);
}
static bool qkn_vector(const QkNormRope& a) {
  if (a.rope && (a.gw <= 0 || (a.N - a.n_txt) % a.gw || (a.N - a.n_txt) / a.gw > QKN_TABLE_MAX ||
                 a.gw > QKN_TABLE_MAX))
    return false;
  return a.dtype == JAGG_DTYPE_BF16 && a.heads > 0 && a.d == 128 * a.heads && a.ld_qkv % 4 == 0 &&
         aligned8(a.qkv) && aligned8(a.qk_out) && aligned8(a.qscale_txt) && aligned8(a.qscale_img) &&
         aligned8(a.kscale_txt) && aligned8(a.kscale_img);
}
int launch_qk_norm_rope_fwd(const QkNormRope& a, cudaStream_t s) {
  JAGG_CHECK_ARG(a.heads > 0 && a.d % a.heads == 0 && a.d / a.heads <= 128 && (a.d / a.heads) % 2 == 0,
                 "qk_norm: head dim unsupported");
  if (a.M <= 0) return JAGG_OK;
  const int64_t blocks = ((int64_t)a.M * a.heads + QKN_WARPS - 1) / QKN_WARPS;
  const int tok = prof_start(s);
  if (qkn_vector(a)) {
    const int64_t vb = ceil_div((int64_t)a.M, (int64_t)QKN_WARPS);
    const int cap = 3 * sm_count();  // the resident blocks (77 registers, 3 per SM)
    qk_norm_rope_fwd_v_kernel<<<(int)(vb < cap ? vb : cap), QKN_THREADS, qkn_table_bytes(a), s>>>(a);
  } else {
    qk_norm_rope_fwd_kernel<<<(int)(blocks < 65536 ? blocks : 65536), QKN_THREADS, 0, s>>>(a);
  }
  JAGG_LAUNCHED();
  // algorithmic bytes: raw q, k read, transformed q, k written (storage type), 1/rms of both
  const double esz = a.dtype == JAGG_DTYPE_F32 ? 4.0 : 2.0;
  prof_stop(tok, s, PROF_QKN_FWD, 0.0, (double)a.M * (4.0 * a.d * esz + 8.0 * a.heads));
  return JAGG_OK;
}
int launch_qk_norm_rope_bwd(const QkNormRopeBwd& a, cudaStream_t s) {
  const QkNormRope& f = a.f;
  JAGG_CHECK_ARG(f.heads > 0 && f.d % f.heads == 0 && f.d / f.heads <= 128 && (f.d / f.heads) % 2 == 0,
                 "qk_norm: head dim unsupported");
  JAGG_CHECK_ARG(a.dqs_txt && a.dks_txt && a.dqs_img && a.dks_img, "qk_norm: null scale gradient");
  if (f.M <= 0) return JAGG_OK;
  // a few blocks per SM: each block ends in 4 dh atomics
  const int64_t blocks = ((int64_t)f.M * f.heads + QKN_WARPS - 1) / QKN_WARPS;
  const int cap = 4 * sm_count();
  const int tok = prof_start(s);
  if (qkn_vector(f) && a.ld_dqk % 4 == 0 && aligned8(a.dqk)) {
    // a few blocks per SM: each block ends in 4 x 128 scale-gradient atomics
    const int64_t vb = ceil_div((int64_t)f.M, (int64_t)QKN_WARPS);
    const int vcap = 3 * sm_count();  // the resident blocks (80 registers, 3 per SM)
    qk_norm_rope_bwd_v_kernel<<<(int)(vb < vcap ? vb : vcap), QKN_THREADS, qkn_table_bytes(f), s>>>(a);
  } else {
    qk_norm_rope_bwd_kernel<<<(int)(blocks < cap ? blocks : cap), QKN_THREADS, 0, s>>>(a);
  }
  JAGG_LAUNCHED();
  // algorithmic bytes: dq, dk read and rewritten in place, raw q, k read (storage type), 1/rms
  const double esz = f.dtype == JAGG_DTYPE_F32 ? 4.0 : 2.0;
  prof_stop(tok, s, PROF_QKN_BWD, 0.0, (double)f.M * (6.0 * f.d * esz + 8.0 * f.heads));
  return JAGG_OK;
}

}  // namespace jagg
