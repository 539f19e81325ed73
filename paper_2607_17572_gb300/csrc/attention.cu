// Joint softmax attention, forward (saving the log-sum-exp) and backward (recomputing the
// probabilities from it).
//
// bf16, head dim 64 / 128: flash-style kernels on the warp-level tensor-core MMA
// (m16n8k16, f32 accumulate).  Forward: a CTA owns 64 queries (16 per warp) and streams
// 64-key tiles with an online softmax.  Backward: a CTA owns 64 keys (16 per warp) and
// streams 64-query tiles: S^T = K Q^T, P^T = exp(S^T - lse), dP^T = V dO^T,
// dS^T = P^T (dP^T - rowsum(dO O)), dV += P^T dO, dK += dS^T Q, and dQ += dS K through
// shared memory and f32 atomics (appendix, Eqs. bwd_V .. bwd_QK).
//
// f32 (and any head dim): straightforward SIMT kernels, one thread per query (forward)
// or per key (backward).
#include <algorithm>

#include "attention.cuh"
#include "ptx.cuh"

namespace jagg {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ float ldx(const void* p, int64_t i, int is_f32) {
  return is_f32 ? static_cast<const float*>(p)[i] : __bfloat162float(static_cast<const bf16*>(p)[i]);
}
__device__ __forceinline__ void stx(void* p, int64_t i, int is_f32, float v) {
  if (is_f32)
    static_cast<float*>(p)[i] = v;
  else
    static_cast<bf16*>(p)[i] = __float2bfloat16_rn(v);
}

// ------------------------------------------------------------------ warp MMA helpers
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(ptx::smem_u32(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(ptx::smem_u32(p)));
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(ptx::smem_u32(dst)), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

constexpr int TILE = 64;

// Shared memory of the backward kernel: K, V, NBUF x (Q, dO), dS^T, NBUF x (lse, rowsum).
template <int D>
struct BwdCfg {
  static constexpr int NBUF = D <= 64 ? 2 : 1;
  static constexpr int SMEM = (2 + 2 * NBUF) * TILE * (D + 8) * 2 + TILE * (TILE + 8) * 2 + 2 * NBUF * TILE * 4;
};

// Copies rows n0 .. n0+63 (zero beyond N) of one head's D columns into smem with pitch D+8.
template <int D>
__device__ __forceinline__ void load_tile(bf16* sm, const SegRows& sr, int b, int n0, int N, int64_t col) {
  constexpr int CH = D / 8;
  for (int idx = threadIdx.x; idx < TILE * CH; idx += blockDim.x) {
    const int r = idx / CH, c = idx % CH;
    const int n = n0 + r;
    const bool valid = n < N;
    const bf16* src = valid ? static_cast<const bf16*>(sr.base(n)) + sr.off(b, n, N, col + c * 8)
                            : static_cast<const bf16*>(sr.p0);
    cp_async16(sm + r * (D + 8) + c * 8, src, valid);
  }
}

// ------------------------------------------------------------------ bf16 forward
template <int D>
__global__ void __launch_bounds__(128) fa_fwd_kernel(AttnArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  constexpr int P = D + 8;
  bf16* sQ = reinterpret_cast<bf16*>(smem);
  bf16* sK = sQ + TILE * P;
  bf16* sV = sK + TILE * P;
  const int N = a.N;
  const int qt = blockIdx.x, bh = blockIdx.y;
  const int b = bh / a.heads, h = bh % a.heads;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, tig = lane & 3;
  const float sl2 = a.scale * kLog2e;

  load_tile<D>(sQ, a.q, b, qt * TILE, N, a.q_col0 + (int64_t)h * D);
  cp_async_wait_all();
  __syncthreads();
  uint32_t qf[D / 16][4];
#pragma unroll
  for (int kc = 0; kc < D / 16; ++kc)
    ldsm_x4(qf[kc], sQ + (warp * 16 + (lane & 7) + 8 * ((lane >> 3) & 1)) * P + kc * 16 + 8 * (lane >> 4));

  float o[D / 8][4];
#pragma unroll
  for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};

  const int nkt = (N + TILE - 1) / TILE;
  for (int kt = 0; kt < nkt; ++kt) {
    __syncthreads();
    load_tile<D>(sK, a.k, b, kt * TILE, N, a.k_col0 + (int64_t)h * D);
    load_tile<D>(sV, a.v, b, kt * TILE, N, a.v_col0 + (int64_t)h * D);
    cp_async_wait_all();
    __syncthreads();
    float s[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int kc = 0; kc < D / 16; ++kc) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t kb[4];
        ldsm_x4(kb, sK + (np * 16 + (lane & 7) + 8 * (lane >> 4)) * P + kc * 16 + 8 * ((lane >> 3) & 1));
        mma16816(s[2 * np], qf[kc], kb[0], kb[1]);
        mma16816(s[2 * np + 1], qf[kc], kb[2], kb[3]);
      }
    }
    float mx[2] = {mrow[0], mrow[1]};
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kt * TILE + nt * 8 + 2 * tig + (e & 1);
        s[nt][e] = key < N ? s[nt][e] * sl2 : -INFINITY;
      }
      mx[0] = fmaxf(mx[0], fmaxf(s[nt][0], s[nt][1]));
      mx[1] = fmaxf(mx[1], fmaxf(s[nt][2], s[nt][3]));
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
    }
    const float corr0 = exp2f(mrow[0] - mx[0]), corr1 = exp2f(mrow[1] - mx[1]);
    mrow[0] = mx[0];
    mrow[1] = mx[1];
    float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      s[nt][0] = exp2f(s[nt][0] - mx[0]);
      s[nt][1] = exp2f(s[nt][1] - mx[0]);
      s[nt][2] = exp2f(s[nt][2] - mx[1]);
      s[nt][3] = exp2f(s[nt][3] - mx[1]);
      rs0 += s[nt][0] + s[nt][1];
      rs1 += s[nt][2] + s[nt][3];
    }
    lrow[0] = lrow[0] * corr0 + rs0;
    lrow[1] = lrow[1] * corr1 + rs1;
#pragma unroll
    for (int dt = 0; dt < D / 8; ++dt) {
      o[dt][0] *= corr0;
      o[dt][1] *= corr0;
      o[dt][2] *= corr1;
      o[dt][3] *= corr1;
    }
#pragma unroll
    for (int kc = 0; kc < 4; ++kc) {
      uint32_t pa[4] = {pack_bf16(s[2 * kc][0], s[2 * kc][1]), pack_bf16(s[2 * kc][2], s[2 * kc][3]),
                        pack_bf16(s[2 * kc + 1][0], s[2 * kc + 1][1]), pack_bf16(s[2 * kc + 1][2], s[2 * kc + 1][3])};
#pragma unroll
      for (int dp = 0; dp < D / 16; ++dp) {
        uint32_t vb[4];
        ldsm_x4_t(vb, sV + (kc * 16 + (lane & 7) + 8 * ((lane >> 3) & 1)) * P + dp * 16 + 8 * (lane >> 4));
        mma16816(o[2 * dp], pa, vb[0], vb[1]);
        mma16816(o[2 * dp + 1], pa, vb[2], vb[3]);
      }
    }
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
  }
  const float inv0 = 1.f / lrow[0], inv1 = 1.f / lrow[1];
  const int q0 = qt * TILE + warp * 16 + g, q1 = q0 + 8;
#pragma unroll
  for (int dt = 0; dt < D / 8; ++dt) {
    const int64_t col = (int64_t)h * D + dt * 8 + 2 * tig;
    if (q0 < N)
      *reinterpret_cast<uint32_t*>(static_cast<bf16*>(a.o.base(q0)) + a.o.off(b, q0, N, col)) =
          pack_bf16(o[dt][0] * inv0, o[dt][1] * inv0);
    if (q1 < N)
      *reinterpret_cast<uint32_t*>(static_cast<bf16*>(a.o.base(q1)) + a.o.off(b, q1, N, col)) =
          pack_bf16(o[dt][2] * inv1, o[dt][3] * inv1);
  }
  if (tig == 0) {
    if (q0 < N) a.lse[(int64_t)bh * N + q0] = (mrow[0] + log2f(lrow[0])) * kLn2;
    if (q1 < N) a.lse[(int64_t)bh * N + q1] = (mrow[1] + log2f(lrow[1])) * kLn2;
  }
}

// ------------------------------------------------------------------ bf16 backward
template <int D>
__global__ void __launch_bounds__(128) fa_bwd_kernel(AttnBwdArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  constexpr int P = D + 8;
  constexpr int PS = TILE + 8;
  // Query-side tiles (Q, dO, lse, rowsum) are double-buffered for head dim 64: the next
  // tile's cp.async copies overlap the current tile's products.  (At 128 the second buffer
  // would halve the CTAs per SM.)
  constexpr int NBUF = BwdCfg<D>::NBUF;
  bf16* sK = reinterpret_cast<bf16*>(smem);
  bf16* sV = sK + TILE * P;
  bf16* sQ0 = sV + TILE * P;            // NBUF tiles of Q
  bf16* sdO0 = sQ0 + NBUF * TILE * P;   // NBUF tiles of dO
  bf16* sdS = sdO0 + NBUF * TILE * P;   // [key][query], pitch PS
  float* sL0 = reinterpret_cast<float*>(sdS + TILE * PS);  // NBUF x (lse * log2e, +inf beyond N)
  float* sDv0 = sL0 + NBUF * TILE;
  const AttnArgs& f = a.f;
  const int N = f.N;
  const int kt = blockIdx.x, bh = blockIdx.y;
  const int b = bh / f.heads, h = bh % f.heads;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, tig = lane & 3;
  const float sl2 = f.scale * kLog2e;

  auto fetch_queries = [&](int qt) {
    const int buf = qt % NBUF;
    load_tile<D>(sQ0 + buf * TILE * P, f.q, b, qt * TILE, N, f.q_col0 + (int64_t)h * D);
    load_tile<D>(sdO0 + buf * TILE * P, a.dO, b, qt * TILE, N, (int64_t)h * D);
    cp_async_commit();
    for (int i = threadIdx.x; i < TILE; i += blockDim.x) {
      const int q = qt * TILE + i;
      sL0[buf * TILE + i] = q < N ? f.lse[(int64_t)bh * N + q] * kLog2e : INFINITY;
      sDv0[buf * TILE + i] = q < N ? a.Dv[(int64_t)bh * N + q] : 0.f;
    }
  };

  load_tile<D>(sK, f.k, b, kt * TILE, N, f.k_col0 + (int64_t)h * D);
  load_tile<D>(sV, f.v, b, kt * TILE, N, f.v_col0 + (int64_t)h * D);
  cp_async_commit();

  float dk[D / 8][4], dv[D / 8][4];
#pragma unroll
  for (int i = 0; i < D / 8; ++i) {
    dk[i][0] = dk[i][1] = dk[i][2] = dk[i][3] = 0.f;
    dv[i][0] = dv[i][1] = dv[i][2] = dv[i][3] = 0.f;
  }
  const int nqt = (N + TILE - 1) / TILE;
  if (NBUF == 2) fetch_queries(0);
  for (int qt = 0; qt < nqt; ++qt) {
    __syncthreads();  // every warp is done with the buffer about to be refilled
    if (NBUF == 1) {
      fetch_queries(qt);
      cp_async_wait<0>();
    } else if (qt + 1 < nqt) {
      fetch_queries(qt + 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const bf16* sQ = sQ0 + (qt % NBUF) * TILE * P;
    const bf16* sdO = sdO0 + (qt % NBUF) * TILE * P;
    const float* sL = sL0 + (qt % NBUF) * TILE;
    const float* sDv = sDv0 + (qt % NBUF) * TILE;

    // S^T = K_w Q^T and dP^T = V_w dO^T: 16 keys x 64 queries per warp
    float st[8][4], dpt[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      st[i][0] = st[i][1] = st[i][2] = st[i][3] = 0.f;
      dpt[i][0] = dpt[i][1] = dpt[i][2] = dpt[i][3] = 0.f;
    }
#pragma unroll
    for (int kc = 0; kc < D / 16; ++kc) {
      uint32_t ka[4], va[4];
      const int arow = (warp * 16 + (lane & 7) + 8 * ((lane >> 3) & 1)) * P + kc * 16 + 8 * (lane >> 4);
      ldsm_x4(ka, sK + arow);
      ldsm_x4(va, sV + arow);
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        const int brow = (np * 16 + (lane & 7) + 8 * (lane >> 4)) * P + kc * 16 + 8 * ((lane >> 3) & 1);
        uint32_t qb[4], ob[4];
        ldsm_x4(qb, sQ + brow);
        ldsm_x4(ob, sdO + brow);
        mma16816(st[2 * np], ka, qb[0], qb[1]);
        mma16816(st[2 * np + 1], ka, qb[2], qb[3]);
        mma16816(dpt[2 * np], va, ob[0], ob[1]);
        mma16816(dpt[2 * np + 1], va, ob[2], ob[3]);
      }
    }
    // P^T and dS^T
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int q = nt * 8 + 2 * tig + (e & 1);
        const float p = exp2f(st[nt][e] * sl2 - sL[q]);
        st[nt][e] = p;
        dpt[nt][e] = p * (dpt[nt][e] - sDv[q]);
      }
    // dV += P^T dO, dK += dS^T Q
#pragma unroll
    for (int kc = 0; kc < 4; ++kc) {
      uint32_t pa[4] = {pack_bf16(st[2 * kc][0], st[2 * kc][1]), pack_bf16(st[2 * kc][2], st[2 * kc][3]),
                        pack_bf16(st[2 * kc + 1][0], st[2 * kc + 1][1]),
                        pack_bf16(st[2 * kc + 1][2], st[2 * kc + 1][3])};
      uint32_t da[4] = {pack_bf16(dpt[2 * kc][0], dpt[2 * kc][1]), pack_bf16(dpt[2 * kc][2], dpt[2 * kc][3]),
                        pack_bf16(dpt[2 * kc + 1][0], dpt[2 * kc + 1][1]),
                        pack_bf16(dpt[2 * kc + 1][2], dpt[2 * kc + 1][3])};
#pragma unroll
      for (int dp = 0; dp < D / 16; ++dp) {
        const int trow = (kc * 16 + (lane & 7) + 8 * ((lane >> 3) & 1)) * P + dp * 16 + 8 * (lane >> 4);
        uint32_t ob[4], qb[4];
        ldsm_x4_t(ob, sdO + trow);
        ldsm_x4_t(qb, sQ + trow);
        mma16816(dv[2 * dp], pa, ob[0], ob[1]);
        mma16816(dv[2 * dp + 1], pa, ob[2], ob[3]);
        mma16816(dk[2 * dp], da, qb[0], qb[1]);
        mma16816(dk[2 * dp + 1], da, qb[2], qb[3]);
      }
    }
    // dS^T -> shared memory for the dQ product
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      *reinterpret_cast<uint32_t*>(sdS + (warp * 16 + g) * PS + nt * 8 + 2 * tig) = pack_bf16(dpt[nt][0], dpt[nt][1]);
      *reinterpret_cast<uint32_t*>(sdS + (warp * 16 + g + 8) * PS + nt * 8 + 2 * tig) =
          pack_bf16(dpt[nt][2], dpt[nt][3]);
    }
    __syncthreads();
    // dQ rows warp*16 .. +15 of this query tile = dS K over the 64 keys, 64 columns at a time
    const int q0 = qt * TILE + warp * 16 + g, q1 = q0 + 8;
#pragma unroll
    for (int dc = 0; dc < D / 64; ++dc) {
      float dq[8][4];
#pragma unroll
      for (int i = 0; i < 8; ++i) dq[i][0] = dq[i][1] = dq[i][2] = dq[i][3] = 0.f;
#pragma unroll
      for (int kc = 0; kc < 4; ++kc) {
        uint32_t sa[4];
        ldsm_x4_t(sa, sdS + (kc * 16 + (lane & 7) + 8 * (lane >> 4)) * PS + warp * 16 + 8 * ((lane >> 3) & 1));
#pragma unroll
        for (int dp = 0; dp < 4; ++dp) {
          uint32_t kb[4];
          ldsm_x4_t(kb, sK + (kc * 16 + (lane & 7) + 8 * ((lane >> 3) & 1)) * P + dc * 64 + dp * 16 + 8 * (lane >> 4));
          mma16816(dq[2 * dp], sa, kb[0], kb[1]);
          mma16816(dq[2 * dp + 1], sa, kb[2], kb[3]);
        }
      }
      // Lanes tig and tig^1 swap halves so that each issues one 16-byte reduction: even
      // lanes add row q0, columns 2tig..2tig+3; odd lanes add row q1, columns 2tig-2..2tig+1.
      // (dq_acc is 16-byte aligned and its row pitch a multiple of 4 floats: checked on launch.)
      const bool even = (tig & 1) == 0;
      const int64_t ld = (int64_t)f.heads * D;
#pragma unroll
      for (int dt = 0; dt < 8; ++dt) {
        const float s0 = even ? dq[dt][2] : dq[dt][0];
        const float s1 = even ? dq[dt][3] : dq[dt][1];
        const float r0 = __shfl_xor_sync(0xffffffffu, s0, 1);
        const float r1 = __shfl_xor_sync(0xffffffffu, s1, 1);
        const int qrow = even ? q0 : q1;
        const int col = h * D + dc * 64 + dt * 8 + 2 * (even ? tig : tig - 1);
        if (qrow < N) {
          float* p = a.dq_acc + ((int64_t)b * N + qrow) * ld + col;
          if (even)
            ptx::red_add_v4(p, dq[dt][0] * f.scale, dq[dt][1] * f.scale, r0 * f.scale, r1 * f.scale);
          else
            ptx::red_add_v4(p, r0 * f.scale, r1 * f.scale, dq[dt][2] * f.scale, dq[dt][3] * f.scale);
        }
      }
    }
  }
  // dK (times the softmax scale) and dV for this CTA's keys
  const int k0 = kt * TILE + warp * 16 + g, k1 = k0 + 8;
#pragma unroll
  for (int dt = 0; dt < D / 8; ++dt) {
    const int64_t c = (int64_t)h * D + dt * 8 + 2 * tig;
    if (k0 < N) {
      *reinterpret_cast<uint32_t*>(static_cast<bf16*>(a.dk.base(k0)) + a.dk.off(b, k0, N, a.dk_col0 + c)) =
          pack_bf16(dk[dt][0] * f.scale, dk[dt][1] * f.scale);
      *reinterpret_cast<uint32_t*>(static_cast<bf16*>(a.dv.base(k0)) + a.dv.off(b, k0, N, a.dv_col0 + c)) =
          pack_bf16(dv[dt][0], dv[dt][1]);
    }
    if (k1 < N) {
      *reinterpret_cast<uint32_t*>(static_cast<bf16*>(a.dk.base(k1)) + a.dk.off(b, k1, N, a.dk_col0 + c)) =
          pack_bf16(dk[dt][2] * f.scale, dk[dt][3] * f.scale);
      *reinterpret_cast<uint32_t*>(static_cast<bf16*>(a.dv.base(k1)) + a.dv.off(b, k1, N, a.dv_col0 + c)) =
          pack_bf16(dv[dt][2], dv[dt][3]);
    }
  }
}

// ------------------------------------------------------------------ SIMT (any dtype)
template <int D>
__global__ void attn_fwd_simt(AttnArgs a) {
  const int bh = blockIdx.y, b = bh / a.heads, h = bh % a.heads;
  const int q = blockIdx.x * blockDim.x + threadIdx.x;
  const int N = a.N;
  const int f32 = a.dtype == JAGG_DTYPE_F32;
  if (q >= N) return;
  float qv[D], o[D];
  const int64_t qo = a.q.off(b, q, N, a.q_col0 + (int64_t)h * D);
  for (int c = 0; c < D; ++c) {
    qv[c] = ldx(a.q.base(q), qo + c, f32) * a.scale;
    o[c] = 0.f;
  }
  float m = -INFINITY, l = 0.f;
  for (int j = 0; j < N; ++j) {
    const int64_t ko = a.k.off(b, j, N, a.k_col0 + (int64_t)h * D);
    float s = 0.f;
    for (int c = 0; c < D; ++c) s += qv[c] * ldx(a.k.base(j), ko + c, f32);
    const float mn = fmaxf(m, s);
    const float corr = expf(m - mn), p = expf(s - mn);
    l = l * corr + p;
    const int64_t vo = a.v.off(b, j, N, a.v_col0 + (int64_t)h * D);
    for (int c = 0; c < D; ++c) o[c] = o[c] * corr + p * ldx(a.v.base(j), vo + c, f32);
    m = mn;
  }
  const int64_t oo = a.o.off(b, q, N, (int64_t)h * D);
  for (int c = 0; c < D; ++c) stx(a.o.base(q), oo + c, f32, o[c] / l);
  a.lse[(int64_t)bh * N + q] = m + logf(l);
}

template <int D>
__global__ void attn_bwd_simt(AttnBwdArgs a) {
  const AttnArgs& f = a.f;
  const int bh = blockIdx.y, b = bh / f.heads, h = bh % f.heads;
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  const int N = f.N;
  const int f32 = f.dtype == JAGG_DTYPE_F32;
  if (j >= N) return;
  float kv[D], vv[D], dk[D], dv[D];
  const int64_t ko = f.k.off(b, j, N, f.k_col0 + (int64_t)h * D);
  const int64_t vo = f.v.off(b, j, N, f.v_col0 + (int64_t)h * D);
  for (int c = 0; c < D; ++c) {
    kv[c] = ldx(f.k.base(j), ko + c, f32);
    vv[c] = ldx(f.v.base(j), vo + c, f32);
    dk[c] = dv[c] = 0.f;
  }
  const int64_t ld = (int64_t)f.heads * D;
  for (int i = 0; i < N; ++i) {
    const int64_t qo = f.q.off(b, i, N, f.q_col0 + (int64_t)h * D);
    const int64_t go = a.dO.off(b, i, N, (int64_t)h * D);
    float s = 0.f, dp = 0.f;
    for (int c = 0; c < D; ++c) {
      s += ldx(f.q.base(i), qo + c, f32) * kv[c];
      dp += ldx(a.dO.base(i), go + c, f32) * vv[c];
    }
    const float p = expf(s * f.scale - f.lse[(int64_t)bh * N + i]);
    const float ds = p * (dp - a.Dv[(int64_t)bh * N + i]);
    float* dq = a.dq_acc + ((int64_t)b * N + i) * ld + (int64_t)h * D;
    for (int c = 0; c < D; ++c) {
      dv[c] += p * ldx(a.dO.base(i), go + c, f32);
      dk[c] += ds * ldx(f.q.base(i), qo + c, f32);
      atomicAdd(dq + c, ds * kv[c] * f.scale);
    }
  }
  const int64_t dko = a.dk.off(b, j, N, a.dk_col0 + (int64_t)h * D);
  const int64_t dvo = a.dv.off(b, j, N, a.dv_col0 + (int64_t)h * D);
  for (int c = 0; c < D; ++c) {
    stx(a.dk.base(j), dko + c, f32, dk[c] * f.scale);
    stx(a.dv.base(j), dvo + c, f32, dv[c]);
  }
}

// Before the backward: Dv[b, h, n] = sum_c dO[n, h*D + c] O[n, h*D + c] and dq_acc = 0.
// One thread per (row, 8 columns); the D/8 threads of a head are adjacent lanes and
// combine their partial dots with shuffles.
__global__ void rowdot_zero_kernel(AttnBwdArgs a) {
  const AttnArgs& f = a.f;
  const int d = f.heads * f.dh;
  const int cpr = d / 8;  // 8-column chunks per row
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  const int row = idx / cpr, ch = idx % cpr;
  const bool live = row < f.B * f.N;
  const int b = live ? row / f.N : 0, n = live ? row % f.N : 0;
  const int col = ch * 8;
  float s = 0.f;
  if (live) {
    const int64_t go = a.dO.off(b, n, f.N, col), oo = f.o.off(b, n, f.N, col);
    if (f.dtype == JAGG_DTYPE_F32) {
      const float4* g4 = reinterpret_cast<const float4*>(static_cast<const float*>(a.dO.base(n)) + go);
      const float4* o4 = reinterpret_cast<const float4*>(static_cast<const float*>(f.o.base(n)) + oo);
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const float4 x = g4[k], y = o4[k];
        s += x.x * y.x + x.y * y.y + x.z * y.z + x.w * y.w;
      }
    } else {
      const uint4 gr = *reinterpret_cast<const uint4*>(static_cast<const bf16*>(a.dO.base(n)) + go);
      const uint4 orr = *reinterpret_cast<const uint4*>(static_cast<const bf16*>(f.o.base(n)) + oo);
      const bf16* gh = reinterpret_cast<const bf16*>(&gr);
      const bf16* oh = reinterpret_cast<const bf16*>(&orr);
#pragma unroll
      for (int k = 0; k < 8; ++k) s += __bfloat162float(gh[k]) * __bfloat162float(oh[k]);
    }
    float4* z = reinterpret_cast<float4*>(a.dq_acc + (int64_t)row * d + col);
    z[0] = make_float4(0.f, 0.f, 0.f, 0.f);
    z[1] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  const int per_head = f.dh / 8;  // a power of two <= 32
  for (int o = per_head / 2; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (live && ch % per_head == 0) a.Dv[((int64_t)b * f.heads + ch / per_head) * f.N + n] = s;
}

// dq (storage type, segment rows) <- dq_acc (f32); one thread per (row, 8 columns).
__global__ void dq_store_kernel(AttnBwdArgs a) {
  const AttnArgs& f = a.f;
  const int d = f.heads * f.dh;
  const int cpr = d / 8;
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  const int row = idx / cpr, col = (idx % cpr) * 8;
  if (row >= f.B * f.N) return;
  const int b = row / f.N, n = row % f.N;
  const float4* src = reinterpret_cast<const float4*>(a.dq_acc + (int64_t)row * d + col);
  const float4 x = src[0], y = src[1];
  const int64_t o = a.dq.off(b, n, f.N, a.dq_col0 + col);
  if (f.dtype == JAGG_DTYPE_F32) {
    float4* dst = reinterpret_cast<float4*>(static_cast<float*>(a.dq.base(n)) + o);
    dst[0] = x;
    dst[1] = y;
  } else {
    uint4 raw;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&raw);
    h[0] = __floats2bfloat162_rn(x.x, x.y);
    h[1] = __floats2bfloat162_rn(x.z, x.w);
    h[2] = __floats2bfloat162_rn(y.x, y.y);
    h[3] = __floats2bfloat162_rn(y.z, y.w);
    *reinterpret_cast<uint4*>(static_cast<bf16*>(a.dq.base(n)) + o) = raw;
  }
}

template <int D>
int fwd_tc(const AttnArgs& a, cudaStream_t s) {
  const int smem = 3 * TILE * (D + 8) * 2;
  static bool set = false;
  if (!set) {
    JAGG_CUDA_TRY(cudaFuncSetAttribute(fa_fwd_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    set = true;
  }
  dim3 grid(ceil_div(a.N, TILE), a.B * a.heads);
  const int tok = prof_start(s);
  fa_fwd_kernel<D><<<grid, 128, smem, s>>>(a);
  JAGG_LAUNCHED();
  // QK^T and PV: 2 N^2 d multiply-adds per (sequence, head)
  prof_stop(tok, s, PROF_ATTN_FWD, 4.0 * a.B * a.heads * (double)a.N * a.N * D,
            2.0 * a.B * (double)a.N * a.heads * D * 4);
  return JAGG_OK;
}
template <int D>
int bwd_tc(const AttnBwdArgs& a, cudaStream_t s) {
  const int smem = BwdCfg<D>::SMEM;
  static bool set = false;
  if (!set) {
    JAGG_CUDA_TRY(cudaFuncSetAttribute(fa_bwd_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    set = true;
  }
  dim3 grid(ceil_div(a.f.N, TILE), a.f.B * a.f.heads);
  const int tok = prof_start(s);
  fa_bwd_kernel<D><<<grid, 128, smem, s>>>(a);
  JAGG_LAUNCHED();
  // dV = P^T dO, dP = dO V^T, dQ = dS K, dK = dS^T Q: 4 N^2 d multiply-adds per (sequence,
  // head); the recomputation of S is not counted
  prof_stop(tok, s, PROF_ATTN_BWD, 8.0 * a.f.B * a.f.heads * (double)a.f.N * a.f.N * D,
            2.0 * a.f.B * (double)a.f.N * a.f.heads * D * 7);
  return JAGG_OK;
}

template <int D>
int fwd_simt(const AttnArgs& a, cudaStream_t s) {
  dim3 grid(ceil_div(a.N, 64), a.B * a.heads);
  attn_fwd_simt<D><<<grid, 64, 0, s>>>(a);
  JAGG_LAUNCHED();
  return JAGG_OK;
}
template <int D>
int bwd_simt(const AttnBwdArgs& a, cudaStream_t s) {
  dim3 grid(ceil_div(a.f.N, 64), a.f.B * a.f.heads);
  attn_bwd_simt<D><<<grid, 64, 0, s>>>(a);
  JAGG_LAUNCHED();
  return JAGG_OK;
}

}  // namespace

static int64_t dv_floats_padded(int B, int N, int heads) { return ((int64_t)B * heads * N + 63) / 64 * 64; }

int64_t attention_bwd_scratch_floats(int B, int N, int heads, int dh) {
  return dv_floats_padded(B, N, heads) + (int64_t)B * N * heads * dh;
}

void attention_bwd_scratch(float* scratch, int B, int N, int heads, float** Dv, float** dq_acc) {
  *Dv = scratch;
  *dq_acc = scratch + dv_floats_padded(B, N, heads);
}

int attention_fwd(const AttnArgs& a, cudaStream_t s) {
  JAGG_CHECK_ARG(a.B > 0 && a.N > 0 && a.heads > 0, "attention: empty shape");
  JAGG_CHECK_ARG(a.impl >= 0 && a.impl <= 2, "attention: bad implementation %d", a.impl);
  const bool tc = attention_fwd_tc_eligible(a);
  JAGG_CHECK_ARG(a.impl != 2 || tc, "attention: the tcgen05 forward does not serve this call");
  if (tc && a.impl != 1) {
    const int tok = prof_start(s);
    JAGG_TRY(attention_fwd_tc(a, s));
    // QK^T and PV: 2 N^2 d multiply-adds per (sequence, head); the second S pass is not counted
    prof_stop(tok, s, PROF_ATTN_FWD, 4.0 * a.B * a.heads * (double)a.N * a.N * a.dh,
              2.0 * a.B * (double)a.N * a.heads * a.dh * 4);
    return JAGG_OK;
  }
  if (a.dtype == JAGG_DTYPE_BF16) {
    if (a.dh == 64) return fwd_tc<64>(a, s);
    if (a.dh == 128) return fwd_tc<128>(a, s);
  }
  switch (a.dh) {
    case 16: return fwd_simt<16>(a, s);
    case 32: return fwd_simt<32>(a, s);
    case 64: return fwd_simt<64>(a, s);
    case 128: return fwd_simt<128>(a, s);
  }
  set_last_error("attention: head dim %d unsupported", a.dh);
  return JAGG_ERR_UNSUPPORTED;
}

int attention_bwd(const AttnBwdArgs& a, cudaStream_t s) {
  const AttnArgs& f = a.f;
  JAGG_CHECK_ARG(f.B > 0 && f.N > 0 && f.heads > 0, "attention: empty shape");
  JAGG_CHECK_ARG((reinterpret_cast<uintptr_t>(a.dq_acc) & 15) == 0 && (f.heads * f.dh) % 4 == 0,
                 "attention: dq accumulator must be 16-byte aligned with a row pitch of 4k floats");
  JAGG_CHECK_ARG(f.dh % 8 == 0 && f.dh <= 256, "attention: head dim %d unsupported", f.dh);
  const int64_t chunks = (int64_t)f.B * f.N * f.heads * f.dh / 8;
  JAGG_CHECK_ARG(chunks < (1ll << 31), "attention: too many rows");
  int tok = prof_start(s);
  rowdot_zero_kernel<<<(int)((chunks + 255) / 256), 256, 0, s>>>(a);
  JAGG_LAUNCHED();
  prof_stop(tok, s, PROF_ATTN_AUX, 0.0, 4.0 * f.B * f.N * f.heads * f.dh * 1.5);
  int st = JAGG_ERR_UNSUPPORTED;
  JAGG_CHECK_ARG(a.impl >= 0 && a.impl <= 2, "attention: bad implementation %d", a.impl);
  const bool tc = attention_bwd_tc_eligible(a);
  JAGG_CHECK_ARG(a.impl != 2 || tc, "attention: the tcgen05 backward does not serve this call");
  if (tc && a.impl != 1) {
    tok = prof_start(s);
    st = attention_bwd_tc(a, s);
    prof_stop(tok, s, PROF_ATTN_BWD, 8.0 * f.B * f.heads * (double)f.N * f.N * f.dh,
              2.0 * f.B * (double)f.N * f.heads * f.dh * 7);
  } else if (f.dtype == JAGG_DTYPE_BF16 && f.dh == 64)
    st = bwd_tc<64>(a, s);
  else if (f.dtype == JAGG_DTYPE_BF16 && f.dh == 128)
    st = bwd_tc<128>(a, s);
  else if (f.dh == 16)
    st = bwd_simt<16>(a, s);
  else if (f.dh == 32)
    st = bwd_simt<32>(a, s);
  else if (f.dh == 64)
    st = bwd_simt<64>(a, s);
  else if (f.dh == 128)
    st = bwd_simt<128>(a, s);
  if (st != JAGG_OK) {
    if (st == JAGG_ERR_UNSUPPORTED) set_last_error("attention: head dim %d unsupported", f.dh);
    return st;
  }
  const int64_t total = (int64_t)f.B * f.N * f.heads * f.dh;
  tok = prof_start(s);
  dq_store_kernel<<<(int)((chunks + 255) / 256), 256, 0, s>>>(a);
  JAGG_LAUNCHED();
  prof_stop(tok, s, PROF_ATTN_AUX, 0.0, 6.0 * total);
  return JAGG_OK;
}

}  // namespace jagg
