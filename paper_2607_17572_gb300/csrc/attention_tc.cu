// Attention on the fifth-generation tensor cores (tcgen05, TMEM accumulators, TMA-fed
// shared-memory operands), bf16: the backward (appendix, Eqs. bwd_V .. bwd_QK, with the
// softmax recomputed from the saved log-sum-exp) for head dims 128 and 64
// (fa_bwd_tc128_kernel, fa_bwd_tc64_kernel), and the forward, one pass with an online
// softmax at head dim 128 (fa_fwd_tc128_kernel), two passes at 64 (fa_fwd_tc_kernel<64>).
// Ragged ends and the MMDiT text / image split: 3D tensor maps [sequence][token][column]
// per stream buffer make TMA read zeros past the last token and drop dQ rows past it.
#include <cuda.h>

#include "attention.cuh"
#include "ptx.cuh"
#include "tmap.cuh"

namespace jagg {

int unit_status_attention_tc(unsigned* v, int clear) { return read_unit_status(v, clear); }
namespace {

constexpr float kLog2eTc = 1.4426950408889634f;
// Tensor maps of one backward call: per stream buffer (0: the first n0 tokens of every
// sequence, 1: the rest) the query, key, value and output-gradient views, and the dQ
// accumulator.
struct FbMaps {
  CUtensorMap q[2], k[2], v[2], dO[2], dq;
};

struct FbParams {
  int B, N, heads, n0;
  float scale;
  int64_t q_col0, k_col0, v_col0, dk_col0, dv_col0;
  const float* lse;
  const float* Dv;
  SegRows dk, dv;
};

// Shared-memory descriptor of a 128-byte-swizzled operand; k-step `k` (16 elements of K).
// K-major: `rows` rows of 128 B per 64-element K chunk, chunks rows * 128 B apart.
// MN-major: the K dimension runs down the rows (8-row atoms 1024 B apart), 64-element MN
// chunks `chunk_bytes` apart.
// The descriptor of step k is that of the operand's base plus the step's byte offset / 16:
// the start-address field holds address / 16 in its low 14 bits and every operand lies below
// 2^18 bytes of shared memory, so the addition never carries out of the field.  With the
// k-loops unrolled, the base descriptor is formed once per operand and each step costs one
// add in the single issuing thread.
__device__ __forceinline__ uint64_t kmajor_desc(uint32_t base, int rows, int k) {
  return ptx::sdesc_sw128(base, 16, 1024) + (uint64_t)(((k >> 2) * (rows * 128) + (k & 3) * 32) >> 4);
}
__device__ __forceinline__ uint64_t mnmajor_desc(uint32_t base, int chunk_bytes, int k) {
  return ptx::sdesc_sw128(base, chunk_bytes, 1024) + (uint64_t)(k * 128);
}

__device__ __forceinline__ uint32_t pack2_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Writes columns c0 .. c0 + 31 of row r (16 packed bf16 pairs) into a K-major
// 128-byte-swizzled tile of 64-column chunks, `rows` rows per chunk.
__device__ __forceinline__ void st_row32_packed(uint8_t* tile, int rows, int r, int c0, const uint32_t* h) {
  uint8_t* row = tile + (c0 >> 6) * (rows * 128) + r * 128;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int j16 = ((c0 & 63) >> 3) + u;
    *reinterpret_cast<uint4*>(row + ((j16 ^ (r & 7)) << 4)) =
        make_uint4(h[4 * u], h[4 * u + 1], h[4 * u + 2], h[4 * u + 3]);
  }
}

// ================================================================== backward, head dims 128 and 64
// 128-key x 64-query tiles with S^T and dP^T double-buffered in tensor memory.  One CTA per
// SM, persistent over (128-key tile, sequence, head) units; per unit the sequence's query
// tiles stream through three Q / dO stages.  Tensor memory (512 columns), buffer b = tile % 2:
//   S_b   [128 b, 128 b + 64)        S^T (f32); P^T written over it (bf16, two per column)
//   dP_b  [128 b + 64, 128 b + 128)  dP^T (f32); dS^T written over it; then dQ^T (f32)
//   [256, 384) dV, [384, 512) dK     accumulated over the whole sequence
// Products of tile g (buffer b), in issue order (one thread; the tensor pipe runs them in
// order):
//   dV += P^T dO, dK += dS^T Q        A from tensor memory, B (dO, Q) from shared memory
//   dQ^T = K^T dS^T                   both from shared memory (dS^T in a double-buffered
//                                     shared tile); over dS^T in dP_b
//   S^T(g+2) = K Q^T                  over P^T(g) in S_b
//   dP^T(g+2) = V dO^T                once the dQ warps have read dQ^T(g) out of dP_b
// The 8 P / dS warps form P^T of tile g+1 as soon as its S^T lands and dS^T once its dP^T
// lands, while the products of tile g run; each writes only over the f32 columns it has read
// (32 keys x 32 queries per warp), so no warp waits for another and nothing waits for a
// product to release a shared P / dS tile.  The 4 dQ warps move dQ^T through shared memory
// into TMA f32 reduce-adds and store each unit's dK, dV at its end.
// Head dim 64 (fa_bwd_tc64_kernel): the same schedule with dV in [256, 320), dK in [320, 384);
// dQ^T has 64 rows, so its product takes M = 128 over the stacked A operand [K^T; V^T] (the V
// tile follows the K tile in shared memory: the second 64-row chunk of A) and lanes 64-127 of
// the result, V^T dS^T, are not read.  A 64-column product takes as long as a 128-row one on
// this tensor pipe, so the stacking costs nothing.
constexpr int FB2_THREADS = 448;  // 14 warps

template <int D_>
struct Fb2 {
  static constexpr int D = D_, BK = 128, BQ = 64, NS = 3;
  static constexpr int KV_BYTES = BK * D * 2;  // 32 KB at D = 128 (two 64-column chunks), 16 KB at 64
  static constexpr int QT_BYTES = BQ * D * 2;  // 16 KB, 8 KB
  static constexpr int DS_BYTES = BK * BQ * 2; // 16 KB
  static constexpr int DQ_WARP_BYTES = 32 * 32 * 4;
  static constexpr int OFF_K = 0;
  static constexpr int OFF_V = OFF_K + KV_BYTES;
  static constexpr int OFF_Q = OFF_V + KV_BYTES;         // NS stages
  static constexpr int OFF_DO = OFF_Q + NS * QT_BYTES;   // NS stages
  static constexpr int OFF_DS = OFF_DO + NS * QT_BYTES;  // 2 buffers
  static constexpr int OFF_DQ = OFF_DS + 2 * DS_BYTES;
  static constexpr int OFF_LSE = OFF_DQ + 4 * DQ_WARP_BYTES;
  static constexpr int OFF_RD = OFF_LSE + NS * BQ * 4;
  static constexpr int OFF_BAR = OFF_RD + NS * BQ * 4;
  static constexpr int NBAR = 24;
  static constexpr int SMEM = OFF_BAR + NBAR * 8 + 16 + 1024;  // + alignment of the base to 1024 bytes
  static_assert(SMEM <= 232448, "shared memory budget");
  __host__ __device__ static constexpr uint32_t t_s(int b) { return 128u * b; }
  __host__ __device__ static constexpr uint32_t t_dp(int b) { return 128u * b + 64u; }
  static constexpr uint32_t T_DV = 256, T_DK = 256 + D;
  static_assert(OFF_V == OFF_K + BK * 128 * (D / 64), "the dQ^T A operand's second chunk");
};

template <int D_>
__device__ __forceinline__ void fa_bwd_v3(const FbMaps& maps, const FbParams& p, uint8_t* smem_fb2) {
  using C = Fb2<D_>;
  constexpr int BK = C::BK, BQ = C::BQ, D = C::D, NS = C::NS;
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_fb2) + 1023) & ~uintptr_t(1023));
  uint8_t* sK = sm + C::OFF_K;
  uint8_t* sV = sm + C::OFF_V;
  uint8_t* sQ = sm + C::OFF_Q;
  uint8_t* sdO = sm + C::OFF_DO;
  uint8_t* sdS = sm + C::OFF_DS;
  uint8_t* sDQ = sm + C::OFF_DQ;
  float* sLse = reinterpret_cast<float*>(sm + C::OFF_LSE);
  float* sRd = reinterpret_cast<float*>(sm + C::OFF_RD);
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + C::OFF_BAR);
  uint64_t* full = bar;              // [NS] Q, dO, lse, rowsum(dO O) of a stage landed
  uint64_t* empty = bar + NS;        // [NS] the stage's products are done
  uint64_t* bar_s = bar + 2 * NS;    // [2] S^T of a tile in S_b
  uint64_t* bar_dp = bar_s + 2;      // [2] dP^T of a tile in dP_b
  uint64_t* bar_p = bar_s + 4;       // [2] P^T written (8 warps)
  uint64_t* bar_ds = bar_s + 6;      // [2] dS^T written to TMEM and shared memory (8 warps)
  uint64_t* bar_dq = bar_s + 8;      // [2] dQ^T of a tile in dP_b
  uint64_t* dqfree = bar_s + 10;     // [2] the dQ warps have read it (4 warps)
  uint64_t* bar_kv = bar_s + 12;     // a unit's K, V landed
  uint64_t* kv_free = bar_s + 13;    // a unit's products are done (K, V reusable)
  uint64_t* bar_fin = bar_s + 14;    // a unit's dK, dV are final
  uint64_t* kvout = bar_s + 15;      // the dQ warps have read them (4 warps)
  uint64_t* bar_drain = bar_s + 16;  // the MMA thread's drain after a give-up
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar + C::NBAR);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int N = p.N;
  const int nkt = (N + BK - 1) / BK;
  const int units = nkt * p.B * p.heads;
  const int nq = (N + BQ - 1) / BQ;
  // unit u: key tile u % nkt of sequence-head u / nkt
  auto unit_of = [&](int u, int& k0, int& b, int& h) {
    const int bh = u / nkt;
    k0 = (u % nkt) * BK;
    b = bh / p.heads;
    h = bh % p.heads;
  };
  auto seg_of = [&](int r) { return r < p.n0 ? 0 : 1; };
  auto row_in = [&](int r) { return r < p.n0 ? r : r - p.n0; };

  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < NS; ++i) {
      ptx::mbar_init(&full[i], 1 + 32);  // the TMA's expect-tx arrival + one per producer lane's copies
      ptx::mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      ptx::mbar_init(&bar_s[i], 1);
      ptx::mbar_init(&bar_dp[i], 1);
      ptx::mbar_init(&bar_p[i], 8);
      ptx::mbar_init(&bar_ds[i], 8);
      ptx::mbar_init(&bar_dq[i], 1);
      ptx::mbar_init(&dqfree[i], 4);
    }
    ptx::mbar_init(bar_kv, 1);
    ptx::mbar_init(kv_free, 1);
    ptx::mbar_init(bar_fin, 1);
    ptx::mbar_init(kvout, 4);
    ptx::mbar_init(bar_drain, 1);
    ptx::fence_mbar_init();
    for (int sg = 0; sg < 2; ++sg) {
      ptx::prefetch_tmap(&maps.q[sg]);
      ptx::prefetch_tmap(&maps.k[sg]);
      ptx::prefetch_tmap(&maps.v[sg]);
      ptx::prefetch_tmap(&maps.dO[sg]);
    }
    ptx::prefetch_tmap(&maps.dq);
  }
  if (warp == 1) {
    ptx::tmem_alloc(tmem_slot, 512);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    int i = 0;
    int i_last = -1, g_last = -1;  // the last unit whose K, V and the last tile whose Q, dO were issued
    for (int u = blockIdx.x; u < units && !*abort_flag; u += gridDim.x, ++i) {
      int k0, b, h;
      unit_of(u, k0, b, h);
      const int bh = b * p.heads + h;
      bool ok = true;
      if (lane == 0) {
        ok = ptx::mbar_wait(kv_free, (i & 1) ^ 1);
        if (ok) {
          const int sg = seg_of(k0), r = row_in(k0);
          ptx::mbar_arrive_expect_tx(bar_kv, 2 * C::KV_BYTES);
#pragma unroll
          for (int c = 0; c < D / 64; ++c) {
            ptx::tma_load_3d(sK + c * BK * 128, &maps.k[sg], bar_kv, (int)(p.k_col0 + h * D + c * 64), r, b);
            ptx::tma_load_3d(sV + c * BK * 128, &maps.v[sg], bar_kv, (int)(p.v_col0 + h * D + c * 64), r, b);
          }
          i_last = i;
        }
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      if (!ok) { *abort_flag = 1; break; }
      for (int j = 0; j < nq; ++j) {
        const int g = i * nq + j;
        const int st = g % NS;
        if (lane == 0) ok = ptx::mbar_wait(&empty[st], ((g / NS) & 1) ^ 1);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        if (!ok || *abort_flag) { *abort_flag = 1; break; }
        const int q0 = j * BQ;
        // lse and rowsum(dO O) of the tile's queries by 4-byte copies the stage barrier tracks
        // (their rows need not be 16-byte aligned); +inf / 0 past the last query
        for (int t = lane; t < BQ; t += 32) {
          const int q = q0 + t;
          if (q < N) {
            ptx::cp_async4(sLse + st * BQ + t, p.lse + (int64_t)bh * N + q);
            ptx::cp_async4(sRd + st * BQ + t, p.Dv + (int64_t)bh * N + q);
          } else {
            sLse[st * BQ + t] = INFINITY;
            sRd[st * BQ + t] = 0.f;
          }
        }
        ptx::cp_async_arrive_noinc(&full[st]);
        __syncwarp();
        if (lane == 0) {
          const int sg = seg_of(q0), r = row_in(q0);
          ptx::mbar_arrive_expect_tx(&full[st], 2 * C::QT_BYTES);
#pragma unroll
          for (int c = 0; c < D / 64; ++c) {
            ptx::tma_load_3d(sQ + st * C::QT_BYTES + c * BQ * 128, &maps.q[sg], &full[st],
                             (int)(p.q_col0 + h * D + c * 64), r, b);
            ptx::tma_load_3d(sdO + st * C::QT_BYTES + c * BQ * 128, &maps.dO[sg], &full[st], h * D + c * 64, r,
                             b);
          }
        }
        g_last = g;
      }
      if (*abort_flag) break;
    }
    // After a give-up anywhere in the CTA, copies already issued may still be landing in
    // shared memory: wait (bounded) for the last phase of every buffer before exiting.
    if (*abort_flag && lane == 0) {
      if (i_last >= 0) ptx::mbar_wait(bar_kv, i_last & 1);
      for (int k = 0; k < NS && g_last - k >= 0; ++k)
        ptx::mbar_wait(&full[(g_last - k) % NS], ((g_last - k) / NS) & 1);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (ptx::elect_one()) {
      constexpr uint32_t id_s = ptx::idesc_bf16(128, BQ, false, false);  // S^T, dP^T
      constexpr uint32_t id_acc = ptx::idesc_bf16(128, D, false, true);  // dV, dK (A from TMEM)
      constexpr uint32_t id_dq = ptx::idesc_bf16(128, BQ, true, true);   // dQ^T
      const uint32_t aK = ptx::smem_u32(sK), aV = ptx::smem_u32(sV);
      auto issue_s = [&](int g) {  // S^T = K Q^T into S_b
        const uint32_t aQ = ptx::smem_u32(sQ + (g % NS) * C::QT_BYTES);
#pragma unroll
        for (int k = 0; k < D / 16; ++k)
          ptx::umma_bf16(tmem + C::t_s(g & 1), kmajor_desc(aK, BK, k), kmajor_desc(aQ, BQ, k), id_s, k > 0);
        ptx::umma_commit(&bar_s[g & 1]);
      };
      auto issue_dp = [&](int g) {  // dP^T = V dO^T into dP_b
        const uint32_t adO = ptx::smem_u32(sdO + (g % NS) * C::QT_BYTES);
#pragma unroll
        for (int k = 0; k < D / 16; ++k)
          ptx::umma_bf16(tmem + C::t_dp(g & 1), kmajor_desc(aV, BK, k), kmajor_desc(adO, BQ, k), id_s, k > 0);
        ptx::umma_commit(&bar_dp[g & 1]);
      };
      bool ok = true;
      int i = 0;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++i) {
        if (!ptx::mbar_wait(bar_kv, i & 1)) { ok = false; break; }
        // the unit's first two tiles
        for (int j = 0; j < 2 && j < nq && ok; ++j) {
          const int g = i * nq + j;
          if (!ptx::mbar_wait(&full[g % NS], (g / NS) & 1)) { ok = false; break; }
          ptx::tc_fence_after();
          issue_s(g);
          // dP_b held dQ^T of the buffer's previous tile (an earlier unit's): drained
          if (g >= 2 && !ptx::mbar_wait(&dqfree[g & 1], ((g - 2) >> 1) & 1)) { ok = false; break; }
          ptx::tc_fence_after();
          issue_dp(g);
        }
        for (int j = 0; j < nq && ok; ++j) {
          const int g = i * nq + j;
          const int st = g % NS, bb = g & 1;
          const uint32_t aQ = ptx::smem_u32(sQ + st * C::QT_BYTES), adO = ptx::smem_u32(sdO + st * C::QT_BYTES);
          const uint32_t adS = ptx::smem_u32(sdS + bb * C::DS_BYTES);
          if (!ptx::mbar_wait(&bar_p[bb], (g >> 1) & 1)) { ok = false; break; }
          ptx::tc_fence_after();
          // the first dV, dK products of a unit overwrite the accumulators: the dQ warps have
          // read the previous unit's
          if (j == 0 && i > 0) {
            if (!ptx::mbar_wait(kvout, (i - 1) & 1)) { ok = false; break; }
            ptx::tc_fence_after();
          }
          // P^T of queries [32 hf, 32 hf + 32) sits in columns S_b + 32 hf + [0, 16)
#pragma unroll
          for (int k = 0; k < BQ / 16; ++k)
            ptx::umma_bf16_ts(tmem + C::T_DV, tmem + C::t_s(bb) + (k >> 1) * 32 + (k & 1) * 8,
                              mnmajor_desc(adO, BQ * 128, k), id_acc, (j > 0 || k > 0) ? 1u : 0u);
          if (!ptx::mbar_wait(&bar_ds[bb], (g >> 1) & 1)) { ok = false; break; }
          ptx::tc_fence_after();
#pragma unroll
          for (int k = 0; k < BQ / 16; ++k)
            ptx::umma_bf16_ts(tmem + C::T_DK, tmem + C::t_dp(bb) + (k >> 1) * 32 + (k & 1) * 8,
                              mnmajor_desc(aQ, BQ * 128, k), id_acc, (j > 0 || k > 0) ? 1u : 0u);
          ptx::umma_commit(&empty[st]);
          // dQ^T[d][q] = sum_key K[key][d] dS^T[key][q], over dS^T in dP_b
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            ptx::umma_bf16(tmem + C::t_dp(bb), mnmajor_desc(aK, BK * 128, k), mnmajor_desc(adS, BK * 128, k),
                           id_dq, k > 0);
          ptx::umma_commit(&bar_dq[bb]);
          if (j + 2 < nq) {
            const int g2 = g + 2;
            if (!ptx::mbar_wait(&full[g2 % NS], (g2 / NS) & 1)) { ok = false; break; }
            ptx::tc_fence_after();
            issue_s(g2);
            if (!ptx::mbar_wait(&dqfree[bb], (g >> 1) & 1)) { ok = false; break; }
            ptx::tc_fence_after();
            issue_dp(g2);
          }
        }
        ptx::umma_commit(kv_free);
        ptx::umma_commit(bar_fin);
      }
      if (!ok) *abort_flag = 1;
      if (*abort_flag) {  // MMAs of this thread may still run: drain them before TMEM is freed
        ptx::umma_commit(bar_drain);
        ptx::mbar_wait(bar_drain, 0);
      }
    }
  } else if (warp < 10) {
    // ---------------------------------------------------------------- P / dS
    const int quarter = warp & 3, hf = (warp - 2) >> 2;
    const int r = quarter * 32 + lane;  // key row of the tile = TMEM lane
    const int c0 = hf * 32;             // this warp's query columns
    const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
    const float c1 = p.scale * kLog2eTc;
    bool ok = true;
    int i = 0;
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++i) {
      for (int j = 0; j < nq; ++j) {
        const int g = i * nq + j;
        const int st = g % NS, bb = g & 1;
        ok = ptx::mbar_wait(&bar_s[bb], (g >> 1) & 1) && ptx::mbar_wait(&full[st], (g / NS) & 1);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok || *abort_flag) { ok = false; *abort_flag = 1; break; }
        ptx::tc_fence_after();
        const float* lse = sLse + st * BQ + c0;
        const float* rd = sRd + st * BQ + c0;
        uint32_t hp[16];  // P^T of this thread's 32 queries, bf16 pairs
        {
          uint32_t rs[32];
          ptx::tmem_ld_32x32b_x32(trow + C::t_s(bb) + c0, rs);
          ptx::tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; e += 4) {
            const float4 l4 = *reinterpret_cast<const float4*>(lse + e);
            const float p0 = ptx::ex2_approx(fmaf(__uint_as_float(rs[e]), c1, -l4.x * kLog2eTc));
            const float p1 = ptx::ex2_approx(fmaf(__uint_as_float(rs[e + 1]), c1, -l4.y * kLog2eTc));
            const float p2 = ptx::ex2_approx(fmaf(__uint_as_float(rs[e + 2]), c1, -l4.z * kLog2eTc));
            const float p3 = ptx::ex2_approx(fmaf(__uint_as_float(rs[e + 3]), c1, -l4.w * kLog2eTc));
            hp[e / 2] = pack2_bf16(p0, p1);
            hp[e / 2 + 1] = pack2_bf16(p2, p3);
          }
        }
        // over this warp's own S^T columns, read already
        ptx::tmem_st_32x32b_x16(trow + C::t_s(bb) + c0, hp);
        ptx::tmem_st_wait();
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&bar_p[bb]);
        ok = __all_sync(0xffffffffu, ptx::mbar_wait(&bar_dp[bb], (g >> 1) & 1));
        if (!ok || *abort_flag) { ok = false; *abort_flag = 1; break; }
        ptx::tc_fence_after();
        uint32_t hd[16];
        {
          uint32_t rp[32];
          ptx::tmem_ld_32x32b_x32(trow + C::t_dp(bb) + c0, rp);
          ptx::tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; e += 4) {
            const float4 r4 = *reinterpret_cast<const float4*>(rd + e);
            const uint32_t a = hp[e / 2], a2 = hp[e / 2 + 1];
            hd[e / 2] = pack2_bf16(__uint_as_float(a << 16) * (__uint_as_float(rp[e]) - r4.x),
                                   __uint_as_float(a & 0xffff0000u) * (__uint_as_float(rp[e + 1]) - r4.y));
            hd[e / 2 + 1] = pack2_bf16(__uint_as_float(a2 << 16) * (__uint_as_float(rp[e + 2]) - r4.z),
                                       __uint_as_float(a2 & 0xffff0000u) * (__uint_as_float(rp[e + 3]) - r4.w));
          }
        }
        ptx::tmem_st_32x32b_x16(trow + C::t_dp(bb) + c0, hd);
        // the B operand of dQ^T: row = key, columns = queries (the product that read this
        // buffer two tiles ago finished before this tile's dP^T)
        st_row32_packed(sdS + bb * C::DS_BYTES, BK, r, c0, hd);
        ptx::tmem_st_wait();
        ptx::fence_proxy_async_smem();
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&bar_ds[bb]);
      }
      if (!ok) break;
    }
  } else {
    // ---------------------------------------------------------------- dQ -> f32 reduce-add; dK, dV
    const int quarter = warp & 3;
    const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
    uint8_t* stg = sDQ + quarter * C::DQ_WARP_BYTES;
    bool ok = true;
    int i = 0;
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++i) {
      int k0, b, h;
      unit_of(u, k0, b, h);
      for (int j = 0; j < nq; ++j) {
        const int g = i * nq + j;
        const int bb = g & 1;
        ok = __all_sync(0xffffffffu, ptx::mbar_wait(&bar_dq[bb], (g >> 1) & 1));
        if (!ok || *abort_flag) { ok = false; *abort_flag = 1; break; }
        ptx::tc_fence_after();
        uint32_t rq[64];
        ptx::tmem_ld_32x32b_x32(trow + C::t_dp(bb), *reinterpret_cast<uint32_t(*)[32]>(rq));
        ptx::tmem_ld_32x32b_x32(trow + C::t_dp(bb) + 32, *reinterpret_cast<uint32_t(*)[32]>(rq + 32));
        ptx::tmem_ld_wait();
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&dqfree[bb]);
        const int q0 = j * BQ;
        // dQ^T: lane = head-dim index, columns = the tile's 64 queries; two 32 x 32 boxes
        // (box rows = queries) through one staging box (head dim 64: lane quarters 0, 1 only)
        if (quarter * 32 >= D) continue;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          if (lane == 0) ptx::bulk_wait_read<0>();
          __syncwarp();
#pragma unroll
          for (int q = 0; q < 32; ++q)
            *reinterpret_cast<float*>(stg + q * 128 + (((lane >> 2) ^ (q & 7)) << 4) + (lane & 3) * 4) =
                __uint_as_float(rq[hh * 32 + q]) * p.scale;
          ptx::fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            const int row = q0 + hh * 32;
            if (row < N) {
              ptx::tma_reduce_add_3d(&maps.dq, stg, h * D + quarter * 32, row, b);
              ptx::bulk_commit();
            }
          }
        }
      }
      if (!ok) break;
      // the unit's dK, dV (key rows of this warp's lane quarter)
      ok = __all_sync(0xffffffffu, ptx::mbar_wait(bar_fin, i & 1));
      if (!ok || *abort_flag) { ok = false; *abort_flag = 1; break; }
      ptx::tc_fence_after();
      const int key = k0 + quarter * 32 + lane;
#pragma unroll 1
      for (int c = 0; c < D / 32; ++c) {
        uint32_t rv[32], rk[32];
        ptx::tmem_ld_32x32b_x32(trow + C::T_DV + c * 32, rv);
        ptx::tmem_ld_32x32b_x32(trow + C::T_DK + c * 32, rk);
        ptx::tmem_ld_wait();
        if (key < N) {
          bf16* dv = static_cast<bf16*>(p.dv.base(key)) + p.dv.off(b, key, N, p.dv_col0 + h * D + c * 32);
          bf16* dk = static_cast<bf16*>(p.dk.base(key)) + p.dk.off(b, key, N, p.dk_col0 + h * D + c * 32);
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            uint4 a, bb;
            a.x = pack2_bf16(__uint_as_float(rv[8 * t]), __uint_as_float(rv[8 * t + 1]));
            a.y = pack2_bf16(__uint_as_float(rv[8 * t + 2]), __uint_as_float(rv[8 * t + 3]));
            a.z = pack2_bf16(__uint_as_float(rv[8 * t + 4]), __uint_as_float(rv[8 * t + 5]));
            a.w = pack2_bf16(__uint_as_float(rv[8 * t + 6]), __uint_as_float(rv[8 * t + 7]));
            bb.x = pack2_bf16(__uint_as_float(rk[8 * t]) * p.scale, __uint_as_float(rk[8 * t + 1]) * p.scale);
            bb.y = pack2_bf16(__uint_as_float(rk[8 * t + 2]) * p.scale, __uint_as_float(rk[8 * t + 3]) * p.scale);
            bb.z = pack2_bf16(__uint_as_float(rk[8 * t + 4]) * p.scale, __uint_as_float(rk[8 * t + 5]) * p.scale);
            bb.w = pack2_bf16(__uint_as_float(rk[8 * t + 6]) * p.scale, __uint_as_float(rk[8 * t + 7]) * p.scale);
            *reinterpret_cast<uint4*>(dv + 8 * t) = a;
            *reinterpret_cast<uint4*>(dk + 8 * t) = bb;
          }
        }
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(kvout);
    }
    if (lane == 0) ptx::bulk_wait<0>();
    __syncwarp();
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 512);
  }
}

__global__ void __launch_bounds__(FB2_THREADS, 1) fa_bwd_tc128_kernel(const __grid_constant__ FbMaps maps,
                                                                      FbParams p) {
  extern __shared__ uint8_t smem_fb2[];
  fa_bwd_v3<128>(maps, p, smem_fb2);
}
__global__ void __launch_bounds__(FB2_THREADS, 1) fa_bwd_tc64_kernel(const __grid_constant__ FbMaps maps,
                                                                     FbParams p) {
  extern __shared__ uint8_t smem_fb2[];
  fa_bwd_v3<64>(maps, p, smem_fb2);
}

// ================================================================== forward, head dim 64
// Persistent over (128-query tile, sequence, head) units, two passes over the sequence's
// 128-key tiles per unit:
//   pass 1   S = Q K^T (TMEM), the exact row maximum m of the scaled scores;
//   pass 2   S again, P = exp(scale (S - m)) (f32 row sums l; bf16 P to shared memory),
//            O += P V (TMEM, never rescaled);
//   then     O / l -> bf16 output, lse = scale m + ln l.
// The extra S product (half the forward's tensor work again) buys a softmax with no running
// rescale of O.  Warp roles: 0 TMA producer (Q once per unit, K in pass 1, K and V in pass 2),
// 1 MMA issuer, 2-9 softmax and output (two warps per TMEM lane quarter = 32 query rows,
// 64 key columns each; they exchange row maxima and sums through shared memory).
constexpr int FF_THREADS = 320;  // 10 warps

template <int D>
struct FfCfg {
  static_assert(D == 64, "head dim 128 has fa_fwd_tc128_kernel");
  static constexpr int BQ = 128, BK = 128;
  static constexpr int NS = 3;  // K (pass 1) / K, V (pass 2) stages
  static constexpr int NP = 2;  // P buffers
  static constexpr int Q_BYTES = BQ * D * 2;
  static constexpr int KV_BYTES = BK * D * 2;
  static constexpr int P_BYTES = BQ * BK * 2;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + Q_BYTES;
  static constexpr int OFF_V = OFF_K + NS * KV_BYTES;
  static constexpr int OFF_P = OFF_V + NS * KV_BYTES;
  static constexpr int OFF_RED = OFF_P + NP * P_BYTES;  // [2: max, sum][2 halves][128 rows] f32
  static constexpr int OFF_BAR = OFF_RED + 2 * 2 * 128 * 4;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  static constexpr int T_O = 256;  // TMEM: S buffers at columns 0 and 128, O at 256
  static_assert(SMEM <= 232448, "shared memory budget");
};

struct FfMaps {
  CUtensorMap q[2], k[2], v[2];
};

struct FfParams {
  int B, N, heads, n0;
  float scale;
  int64_t q_col0, k_col0, v_col0;
  SegRows o;
  float* lse;
};

__device__ __forceinline__ void named_bar(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

template <int D>
__global__ void __launch_bounds__(FF_THREADS, 1) fa_fwd_tc_kernel(const __grid_constant__ FfMaps maps, FfParams p) {
  using C = FfCfg<D>;
  constexpr int BQ = C::BQ, BK = C::BK, NS = C::NS, NP = C::NP;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = sm + C::OFF_Q;
  uint8_t* sK = sm + C::OFF_K;
  uint8_t* sV = sm + C::OFF_V;
  uint8_t* sP = sm + C::OFF_P;
  float* red = reinterpret_cast<float*>(sm + C::OFF_RED);
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + C::OFF_BAR);
  uint64_t* full = bar;              // [NS] a K (and V) stage landed
  uint64_t* empty = full + NS;       // [NS] its products are done
  uint64_t* qfull = empty + NS;      // the unit's Q landed
  uint64_t* qfree = qfull + 1;       // the unit's last S product is done
  uint64_t* bar_s = qfree + 1;       // [2] S in TMEM buffer b
  uint64_t* sfree = bar_s + 2;       // [2] the 8 warps have read it
  uint64_t* pready = sfree + 2;      // [NP] P written by the 8 warps
  uint64_t* pfree = pready + NP;     // [NP] the product reading P is done
  uint64_t* bar_o = pfree + NP;      // the unit's O is complete
  uint64_t* ofree = bar_o + 1;       // the 8 warps have read O
  uint64_t* bar_drain = ofree + 1;   // the MMA thread's drain after a give-up
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar_drain + 1);
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int N = p.N;
  const int nk = (N + BK - 1) / BK;
  const int nq = (N + BQ - 1) / BQ;
  const int units = nq * p.B * p.heads;
  // unit u: query tile u % nq of sequence-head u / nq
  auto unit_of = [&](int u, int& q0, int& b, int& h) {
    const int bh = u / nq;
    q0 = (u % nq) * BQ;
    b = bh / p.heads;
    h = bh % p.heads;
  };
  auto seg_of = [&](int r) { return r < p.n0 ? 0 : 1; };
  auto row_in = [&](int r) { return r < p.n0 ? r : r - p.n0; };

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int i = 0; i < NS; ++i) {
      ptx::mbar_init(&full[i], 1);
      ptx::mbar_init(&empty[i], 1);
    }
    ptx::mbar_init(qfull, 1);
    ptx::mbar_init(qfree, 1);
    for (int i = 0; i < 2; ++i) {
      ptx::mbar_init(&bar_s[i], 1);
      ptx::mbar_init(&sfree[i], 8);
    }
    for (int i = 0; i < NP; ++i) {
      ptx::mbar_init(&pready[i], 8);
      ptx::mbar_init(&pfree[i], 1);
    }
    ptx::mbar_init(bar_o, 1);
    ptx::mbar_init(ofree, 8);
    ptx::mbar_init(bar_drain, 1);
    ptx::fence_mbar_init();
    for (int sg = 0; sg < 2; ++sg) {
      ptx::prefetch_tmap(&maps.q[sg]);
      ptx::prefetch_tmap(&maps.k[sg]);
      ptx::prefetch_tmap(&maps.v[sg]);
    }
  }
  if (warp == 1) {
    ptx::tmem_alloc(tmem_slot, 512);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      int g = 0, i = 0, iq_last = -1;  // g: K / V tiles issued; iq_last: the last unit whose Q was issued
      bool ok = true;
      for (int u = blockIdx.x; u < units && ok && !abort_flag; u += gridDim.x, ++i) {
        int q0, b, h;
        unit_of(u, q0, b, h);
        if (i > 0 && !ptx::mbar_wait(qfree, (i - 1) & 1)) { ok = false; break; }
        iq_last = i;
        ptx::mbar_arrive_expect_tx(qfull, C::Q_BYTES);
#pragma unroll
        for (int c = 0; c < D / 64; ++c)
          ptx::tma_load_3d(sQ + c * BQ * 128, &maps.q[seg_of(q0)], qfull, (int)(p.q_col0 + h * D + c * 64),
                           row_in(q0), b);
        for (int pass = 0; pass < 2 && ok; ++pass) {
          for (int j = 0; j < nk; ++j, ++g) {
            const int st = g % NS;
            if (g >= NS && !ptx::mbar_wait(&empty[st], ((g / NS) & 1) ^ 1)) { ok = false; break; }
            const int k0 = j * BK, sg = seg_of(k0), r = row_in(k0);
            ptx::mbar_arrive_expect_tx(&full[st], (pass + 1) * C::KV_BYTES);
#pragma unroll
            for (int c = 0; c < D / 64; ++c) {
              ptx::tma_load_3d(sK + st * C::KV_BYTES + c * BK * 128, &maps.k[sg], &full[st],
                               (int)(p.k_col0 + h * D + c * 64), r, b);
              if (pass == 1)
                ptx::tma_load_3d(sV + st * C::KV_BYTES + c * BK * 128, &maps.v[sg], &full[st],
                                 (int)(p.v_col0 + h * D + c * 64), r, b);
            }
          }
        }
      }
      if (!ok) abort_flag = 1;
      // after a give-up: wait (bounded) for the copies still landing before exiting
      if (abort_flag) {
        if (iq_last >= 0) ptx::mbar_wait(qfull, iq_last & 1);
        for (int k = 0; k < NS && g - 1 - k >= 0; ++k) ptx::mbar_wait(&full[(g - 1 - k) % NS], ((g - 1 - k) / NS) & 1);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (ptx::elect_one()) {
      constexpr uint32_t id_s = ptx::idesc_bf16(128, BK, false, false);
      constexpr uint32_t id_o = ptx::idesc_bf16(128, D, false, true);
      const uint32_t aQ = ptx::smem_u32(sQ);
      bool ok = true;
      int g = 0, sc = 0, pc = 0, i = 0;
      auto issue_s = [&](int st) {  // S of the stage's key tile into TMEM buffer sc % 2
        const int sb = sc & 1;
        if (sc >= 2 && !ptx::mbar_wait(&sfree[sb], ((sc >> 1) & 1) ^ 1)) return false;
        ptx::tc_fence_after();
        const uint32_t aK = ptx::smem_u32(sK + st * C::KV_BYTES);
#pragma unroll
        for (int k = 0; k < D / 16; ++k)
          ptx::umma_bf16(tmem + sb * 128, kmajor_desc(aQ, BQ, k), kmajor_desc(aK, BK, k), id_s, k > 0);
        ptx::umma_commit(&bar_s[sb]);
        ++sc;
        return true;
      };
      auto issue_pv = [&](int st, bool first) {  // O += P V of the stage's value tile
        const int pb = pc % NP;
        if (!ptx::mbar_wait(&pready[pb], (pc / NP) & 1)) return false;
        ptx::tc_fence_after();
        const uint32_t aP = ptx::smem_u32(sP + pb * C::P_BYTES);
        const uint32_t aV = ptx::smem_u32(sV + st * C::KV_BYTES);
#pragma unroll
        for (int k = 0; k < BK / 16; ++k)
          ptx::umma_bf16(tmem + C::T_O, kmajor_desc(aP, BQ, k), mnmajor_desc(aV, BK * 128, k), id_o,
                         (!first || k > 0) ? 1u : 0u);
        ptx::umma_commit(&pfree[pb]);
        ptx::umma_commit(&empty[st]);
        ++pc;
        return true;
      };
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++i) {
        if (!ptx::mbar_wait(qfull, i & 1)) { ok = false; break; }
        // pass 1
        for (int j = 0; j < nk && ok; ++j, ++g) {
          const int st = g % NS;
          if (!ptx::mbar_wait(&full[st], (g / NS) & 1)) { ok = false; break; }
          ok = issue_s(st);
          ptx::umma_commit(&empty[st]);
        }
        // pass 2: S of tile j, then P V of tile j - 1
        int prev_st = -1;
        for (int j = 0; j < nk && ok; ++j, ++g) {
          const int st = g % NS;
          if (!ptx::mbar_wait(&full[st], (g / NS) & 1)) { ok = false; break; }
          if (!issue_s(st)) { ok = false; break; }
          if (j == nk - 1) ptx::umma_commit(qfree);
          if (j > 0) {
            if (j == 1 && i > 0 && !ptx::mbar_wait(ofree, (i - 1) & 1)) { ok = false; break; }
            if (!issue_pv(prev_st, j == 1)) { ok = false; break; }
          }
          prev_st = st;
        }
        if (!ok) break;
        if (nk == 1 && i > 0 && !ptx::mbar_wait(ofree, (i - 1) & 1)) { ok = false; break; }
        if (!issue_pv(prev_st, nk == 1)) { ok = false; break; }
        ptx::umma_commit(bar_o);
      }
      if (!ok) abort_flag = 1;
      if (abort_flag) {  // MMAs of this thread may still run: drain them before TMEM is freed
        ptx::umma_commit(bar_drain);
        ptx::mbar_wait(bar_drain, 0);
      }
    }
  } else {
    // ---------------------------------------------------------------- softmax, output
    // The two warps of a lane quarter meet at named barriers, so neither leaves the unit
    // loop early: after a failed (timed-out) wait a warp runs on without waiting.
    const int quarter = warp & 3, half = (warp - 2) >> 2;
    const int r = quarter * 32 + lane;  // query row of the tile = TMEM lane
    const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
    const float c2 = p.scale * kLog2eTc;
    float* red_m = red;
    float* red_l = red + 2 * 128;
    bool ok = true;
    auto wait = [&](uint64_t* b, uint32_t phase) {
      if (ok) ok = __all_sync(0xffffffffu, ptx::mbar_wait(b, phase));
      if (!ok) abort_flag = 1;
    };
    int sc = 0, pc = 0, i = 0;
    for (int u = blockIdx.x; u < units; u += gridDim.x, ++i) {
      int q0, b, h;
      unit_of(u, q0, b, h);
      // pass 1: the row maximum over the valid keys
      float m = -INFINITY;
      for (int j = 0; j < nk; ++j, ++sc) {
        const int sb = sc & 1;
        wait(&bar_s[sb], (sc >> 1) & 1);
        ptx::tc_fence_after();
        uint32_t rs[64];
        ptx::tmem_ld_32x32b_x32(trow + sb * 128 + half * 64, *reinterpret_cast<uint32_t(*)[32]>(rs));
        ptx::tmem_ld_32x32b_x32(trow + sb * 128 + half * 64 + 32, *reinterpret_cast<uint32_t(*)[32]>(rs + 32));
        ptx::tmem_ld_wait();
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0 && ok) ptx::mbar_arrive(&sfree[sb]);
        const int kv = N - (j * BK + half * 64);  // valid keys among this warp's 64
#pragma unroll
        for (int c = 0; c < 64; ++c)
          if (c < kv) m = fmaxf(m, __uint_as_float(rs[c]));
      }
      red_m[half * 128 + r] = m;
      named_bar(1 + quarter, 64);
      m = fmaxf(m, red_m[(1 - half) * 128 + r]);
      // pass 2: P, its row sums, O += P V
      float l = 0.f;
      for (int j = 0; j < nk; ++j, ++sc, ++pc) {
        const int sb = sc & 1, pb = pc % NP;
        wait(&bar_s[sb], (sc >> 1) & 1);
        ptx::tc_fence_after();
        uint32_t hp[32];
        const int kv = N - (j * BK + half * 64);
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
          uint32_t rs[32];
          ptx::tmem_ld_32x32b_x32(trow + sb * 128 + half * 64 + cc * 32, rs);
          ptx::tmem_ld_wait();
#pragma unroll
          for (int c = 0; c < 32; c += 2) {
            const float p0 = cc * 32 + c < kv ? ptx::ex2_approx((__uint_as_float(rs[c]) - m) * c2) : 0.f;
            const float p1 = cc * 32 + c + 1 < kv ? ptx::ex2_approx((__uint_as_float(rs[c + 1]) - m) * c2) : 0.f;
            l += p0 + p1;
            hp[cc * 16 + c / 2] = pack2_bf16(p0, p1);
          }
        }
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0 && ok) ptx::mbar_arrive(&sfree[sb]);
        if (pc >= NP) wait(&pfree[pb], ((pc - NP) / NP) & 1);
        uint8_t* tile = sP + pb * C::P_BYTES;
        st_row32_packed(tile, BQ, r, half * 64, hp);
        st_row32_packed(tile, BQ, r, half * 64 + 32, hp + 16);
        ptx::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0 && ok) ptx::mbar_arrive(&pready[pb]);
      }
      red_l[half * 128 + r] = l;
      named_bar(1 + quarter, 64);
      l += red_l[(1 - half) * 128 + r];
      // the unit's output: O / l, and the log-sum-exp
      wait(bar_o, i & 1);
      ptx::tc_fence_after();
      const int q = q0 + r;
      const float inv = 1.f / l;
#pragma unroll
      for (int cc = 0; cc < D / 64; ++cc) {
        uint32_t ro[32];
        ptx::tmem_ld_32x32b_x32(trow + C::T_O + half * (D / 2) + cc * 32, ro);
        ptx::tmem_ld_wait();
        if (q < N && ok) {
          bf16* o = static_cast<bf16*>(p.o.base(q)) + p.o.off(b, q, N, (int64_t)h * D + half * (D / 2) + cc * 32);
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            uint4 w;
            w.x = pack2_bf16(__uint_as_float(ro[8 * v]) * inv, __uint_as_float(ro[8 * v + 1]) * inv);
            w.y = pack2_bf16(__uint_as_float(ro[8 * v + 2]) * inv, __uint_as_float(ro[8 * v + 3]) * inv);
            w.z = pack2_bf16(__uint_as_float(ro[8 * v + 4]) * inv, __uint_as_float(ro[8 * v + 5]) * inv);
            w.w = pack2_bf16(__uint_as_float(ro[8 * v + 6]) * inv, __uint_as_float(ro[8 * v + 7]) * inv);
            *reinterpret_cast<uint4*>(o + 8 * v) = w;
          }
        }
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0 && ok) ptx::mbar_arrive(ofree);
      if (half == 0 && q < N && ok) p.lse[((int64_t)b * p.heads + h) * N + q] = p.scale * m + logf(l);
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 512);
  }
}

// ================================================================== forward, head dim 128
// One pass over the keys with an online softmax.  Persistent over (pair of 128-query tiles A
// and B, sequence, head) units; per unit the sequence's 128-key tiles stream through a K ring
// and a V ring, each K and V tile serving both query tiles.  Tensor memory (512 columns):
//   S_A [0, 128), S_B [128, 256)   S = Q K^T (f32); P written over it (bf16, two per column)
//   O_A [256, 384), O_B [384, 512) O += P V (f32), accumulated over the keys
// Issue order per key tile j: PV_A(j-1), S_A(j), PV_B(j-1), S_B(j), so the softmax of one
// query tile runs while the products of the other do.  Softmax warps 2-5 own tile A, 6-9 tile
// B, a thread per query row (no exchange between warps).  Each row keeps a reference maximum m: P = exp(scale (S - m)); when a tile's maximum
// exceeds m by more than 8 / (scale log2 e) (P would pass 2^8), m moves up and the row's O (once
// the previous P V product has finished) and running sum l are rescaled, so O is rescaled only
// while the maximum is still climbing.  P goes to tensor memory over S columns 64-127 (read
// into registers first) and is the A operand of P V, whose key blocks follow that placement.
// Row maxima take the three-input max, the scale-shift and the row sums the paired f32 forms.
// At the end O / l leaves in bf16 and lse = scale m + ln l.
constexpr int FF2_THREADS = 320;  // 10 warps

struct Ff2 {
  static constexpr int D = 128, BQ = 128, BK = 128, NKS = 2, NVS = 3;
  static constexpr int TILE = 128 * 128 * 2;  // 32 KB: 128 rows x 128 bf16, two 64-column chunks
  static constexpr int OFF_Q = 0;             // Q_A, Q_B
  static constexpr int OFF_K = OFF_Q + 2 * TILE;
  static constexpr int OFF_V = OFF_K + NKS * TILE;
  static constexpr int OFF_BAR = OFF_V + NVS * TILE;
  static constexpr int NBAR = 24;
  static constexpr int SMEM = OFF_BAR + NBAR * 8 + 16 + 1024;  // + alignment of the base to 1024 bytes
  static_assert(SMEM <= 232448, "shared memory budget");
  static constexpr uint32_t T_S = 0, T_O = 256;  // S_X at 128 X, O_X at 256 + 128 X
  // Column (within S_X) of P of keys 16 kb .. 16 kb + 15, two bf16 per column: key blocks 4-7
  // at 64-95, 0-3 at 96-127.
  static __host__ __device__ constexpr uint32_t p_col(int kb) { return 64 + 8 * ((kb + 4) & 7); }
};

// Keys at or past `kv` (columns col0 + c of the tile) -> -inf.
template <int n>
__device__ __forceinline__ void mask_keys(uint32_t (&r)[n], int col0, int kv) {
#pragma unroll
  for (int c = 0; c < n; ++c)
    if (col0 + c >= kv) r[c] = 0xff800000u;
}
// Running maxima of n f32 values in four independent chains.
template <int n>
__device__ __forceinline__ void row_max4(const uint32_t (&r)[n], float (&mx)[4]) {
#pragma unroll
  for (int c = 0; c < n; c += 8) {
    mx[0] = ptx::max3(mx[0], __uint_as_float(r[c]), __uint_as_float(r[c + 1]));
    mx[1] = ptx::max3(mx[1], __uint_as_float(r[c + 2]), __uint_as_float(r[c + 3]));
    mx[2] = ptx::max3(mx[2], __uint_as_float(r[c + 4]), __uint_as_float(r[c + 5]));
    mx[3] = ptx::max3(mx[3], __uint_as_float(r[c + 6]), __uint_as_float(r[c + 7]));
  }
}
// p = 2^(s c2 - m c2) of n f32 values, packed in place two per word (bf16) into r[0, n/2);
// the f32 values are added into acc0, acc1.
template <int n>
__device__ __forceinline__ void exp_pack(uint32_t (&r)[n], float2 vc2, float2 vmc, float2& acc0, float2& acc1) {
#pragma unroll
  for (int c = 0; c < n; c += 4) {
    const float2 t0 = ptx::fma2(make_float2(__uint_as_float(r[c]), __uint_as_float(r[c + 1])), vc2, vmc);
    const float2 t1 = ptx::fma2(make_float2(__uint_as_float(r[c + 2]), __uint_as_float(r[c + 3])), vc2, vmc);
    const float2 p0 = make_float2(ptx::ex2_approx(t0.x), ptx::ex2_approx(t0.y));
    const float2 p1 = make_float2(ptx::ex2_approx(t1.x), ptx::ex2_approx(t1.y));
    acc0 = ptx::add2(acc0, p0);
    acc1 = ptx::add2(acc1, p1);
    r[c / 2] = pack2_bf16(p0.x, p0.y);
    r[c / 2 + 1] = pack2_bf16(p1.x, p1.y);
  }
}

__global__ void __launch_bounds__(FF2_THREADS, 1) fa_fwd_tc128_kernel(const __grid_constant__ FfMaps maps,
                                                                      FfParams p) {
  using C = Ff2;
  constexpr int BQ = C::BQ, BK = C::BK, D = C::D, NKS = C::NKS, NVS = C::NVS;
  extern __shared__ uint8_t smem_ff2[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_ff2) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = sm + C::OFF_Q;
  uint8_t* sK = sm + C::OFF_K;
  uint8_t* sV = sm + C::OFF_V;
  uint64_t* bar = reinterpret_cast<uint64_t*>(sm + C::OFF_BAR);
  uint64_t* kfull = bar;                // [NKS] a K tile landed
  uint64_t* kempty = kfull + NKS;       // [NKS] both S products reading it are done
  uint64_t* vfull = kempty + NKS;       // [NVS] a V tile landed
  uint64_t* vempty = vfull + NVS;       // [NVS] both P V products reading it are done
  uint64_t* qfull = vempty + NVS;       // the unit's Q_A, Q_B landed
  uint64_t* qfree = qfull + 1;          // the unit's last S products are done
  uint64_t* bar_s = qfree + 1;          // [2] S_X of a key tile in TMEM
  uint64_t* pready = bar_s + 2;         // [2] P_X written (and O_X rescaled) by tile X's 4 warps
  uint64_t* bar_pv = pready + 2;        // [2] the P_X V product of a key tile is done
  uint64_t* ofree = bar_pv + 2;         // [2] tile X's 4 warps have read O_X
  uint64_t* bar_drain = ofree + 2;      // the MMA thread's drain after a give-up
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar + C::NBAR);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int N = p.N;
  const int nk = (N + BK - 1) / BK;
  const int nq = (N + BQ - 1) / BQ;
  const int npair = (nq + 1) / 2;
  const int units = npair * p.B * p.heads;
  // unit u: query tiles 2 (u % npair) and + 1 of sequence-head u / npair
  auto unit_of = [&](int u, int& q0, int& b, int& h) {
    const int bh = u / npair;
    q0 = (u % npair) * 2 * BQ;
    b = bh / p.heads;
    h = bh % p.heads;
  };
  auto seg_of = [&](int r) { return r < p.n0 ? 0 : 1; };
  auto row_in = [&](int r) { return r < p.n0 ? r : r - p.n0; };

  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < NKS; ++i) {
      ptx::mbar_init(&kfull[i], 1);
      ptx::mbar_init(&kempty[i], 1);
    }
    for (int i = 0; i < NVS; ++i) {
      ptx::mbar_init(&vfull[i], 1);
      ptx::mbar_init(&vempty[i], 1);
    }
    ptx::mbar_init(qfull, 1);
    ptx::mbar_init(qfree, 1);
    for (int x = 0; x < 2; ++x) {
      ptx::mbar_init(&bar_s[x], 1);
      ptx::mbar_init(&pready[x], 4);
      ptx::mbar_init(&bar_pv[x], 1);
      ptx::mbar_init(&ofree[x], 4);
    }
    ptx::mbar_init(bar_drain, 1);
    ptx::fence_mbar_init();
    for (int sg = 0; sg < 2; ++sg) {
      ptx::prefetch_tmap(&maps.q[sg]);
      ptx::prefetch_tmap(&maps.k[sg]);
      ptx::prefetch_tmap(&maps.v[sg]);
    }
  }
  if (warp == 1) {
    ptx::tmem_alloc(tmem_slot, 512);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      int gk = 0, gv = 0, i = 0, iq_last = -1;  // K / V tiles issued; the last unit whose Q was issued
      bool ok = true;
      for (int u = blockIdx.x; u < units && ok && !*abort_flag; u += gridDim.x, ++i) {
        int q0, b, h;
        unit_of(u, q0, b, h);
        if (!ptx::mbar_wait(qfree, (i & 1) ^ 1)) { ok = false; break; }
        iq_last = i;
        ptx::mbar_arrive_expect_tx(qfull, 2 * C::TILE);
        for (int x = 0; x < 2; ++x) {
          // query tile B past the last query (odd tile count): a tile of zeros
          const int qx = q0 + x * BQ < N ? q0 + x * BQ : q0;
#pragma unroll
          for (int c = 0; c < D / 64; ++c)
            ptx::tma_load_3d(sQ + x * C::TILE + c * BQ * 128, &maps.q[seg_of(qx)], qfull,
                             (int)(p.q_col0 + h * D + c * 64), row_in(qx), b);
        }
        for (int j = 0; j < nk && ok; ++j, ++gk, ++gv) {
          const int k0 = j * BK, sg = seg_of(k0), r = row_in(k0);
          const int ks = gk % NKS, vs = gv % NVS;
          if (!ptx::mbar_wait(&kempty[ks], ((gk / NKS) & 1) ^ 1)) { ok = false; break; }
          ptx::mbar_arrive_expect_tx(&kfull[ks], C::TILE);
#pragma unroll
          for (int c = 0; c < D / 64; ++c)
            ptx::tma_load_3d(sK + ks * C::TILE + c * BK * 128, &maps.k[sg], &kfull[ks],
                             (int)(p.k_col0 + h * D + c * 64), r, b);
          if (!ptx::mbar_wait(&vempty[vs], ((gv / NVS) & 1) ^ 1)) { ok = false; ++gk; break; }
          ptx::mbar_arrive_expect_tx(&vfull[vs], C::TILE);
#pragma unroll
          for (int c = 0; c < D / 64; ++c)
            ptx::tma_load_3d(sV + vs * C::TILE + c * BK * 128, &maps.v[sg], &vfull[vs],
                             (int)(p.v_col0 + h * D + c * 64), r, b);
        }
      }
      if (!ok) *abort_flag = 1;
      // after a give-up: wait (bounded) for the copies still landing before exiting
      if (*abort_flag) {
        if (iq_last >= 0) ptx::mbar_wait(qfull, iq_last & 1);
        for (int k = 0; k < NKS && gk - 1 - k >= 0; ++k)
          ptx::mbar_wait(&kfull[(gk - 1 - k) % NKS], ((gk - 1 - k) / NKS) & 1);
        for (int k = 0; k < NVS && gv - 1 - k >= 0; ++k)
          ptx::mbar_wait(&vfull[(gv - 1 - k) % NVS], ((gv - 1 - k) / NVS) & 1);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (ptx::elect_one()) {
      constexpr uint32_t id_s = ptx::idesc_bf16(128, BK, false, false);  // S = Q K^T
      constexpr uint32_t id_o = ptx::idesc_bf16(128, D, false, true);    // O += P V (A from TMEM)
      bool ok = true;
      int gk = 0, gv = 0, i = 0;
      uint32_t pr_phase[2] = {0u, 0u};  // pready[X] phases consumed
      auto issue_s = [&](int x, int ks) {  // S_X = Q_X K^T of K stage ks
        const uint32_t aQ = ptx::smem_u32(sQ + x * C::TILE), aK = ptx::smem_u32(sK + ks * C::TILE);
#pragma unroll
        for (int k = 0; k < D / 16; ++k)
          ptx::umma_bf16(tmem + C::T_S + x * 128, kmajor_desc(aQ, BQ, k), kmajor_desc(aK, BK, k), id_s, k > 0);
        ptx::umma_commit(&bar_s[x]);
      };
      auto issue_pv = [&](int x, int vs, bool first) {  // O_X += P_X V of V stage vs
        const uint32_t aV = ptx::smem_u32(sV + vs * C::TILE);
#pragma unroll
        for (int k = 0; k < BK / 16; ++k)
          ptx::umma_bf16_ts(tmem + C::T_O + x * 128, tmem + C::T_S + x * 128 + C::p_col(k),
                            mnmajor_desc(aV, BK * 128, k), id_o, (!first || k > 0) ? 1u : 0u);
        ptx::umma_commit(&bar_pv[x]);
      };
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++i) {
        if (!ptx::mbar_wait(qfull, i & 1)) { ok = false; break; }
        // key tile 0: S_A, S_B
        if (!ptx::mbar_wait(&kfull[gk % NKS], (gk / NKS) & 1)) { ok = false; break; }
        ptx::tc_fence_after();
        issue_s(0, gk % NKS);
        issue_s(1, gk % NKS);
        ptx::umma_commit(&kempty[gk % NKS]);
        if (nk == 1) ptx::umma_commit(qfree);
        ++gk;
        for (int j = 1; j <= nk && ok; ++j) {
          const int vs = gv % NVS;
          for (int x = 0; x < 2 && ok; ++x) {
            // P_X of key tile j - 1, then (j < nk) S_X of key tile j over it
            if (!ptx::mbar_wait(&pready[x], pr_phase[x])) { ok = false; break; }
            pr_phase[x] ^= 1u;
            ptx::tc_fence_after();
            if (j == 1 && i > 0) {  // O_X of the previous unit has been read
              if (!ptx::mbar_wait(&ofree[x], (i - 1) & 1)) { ok = false; break; }
              ptx::tc_fence_after();
            }
            if (x == 0 && !ptx::mbar_wait(&vfull[vs], (gv / NVS) & 1)) { ok = false; break; }
            ptx::tc_fence_after();
            issue_pv(x, vs, j == 1);
            if (j < nk) {
              if (x == 0 && !ptx::mbar_wait(&kfull[gk % NKS], (gk / NKS) & 1)) { ok = false; break; }
              ptx::tc_fence_after();
              issue_s(x, gk % NKS);
            }
          }
          if (!ok) break;
          ptx::umma_commit(&vempty[vs]);
          ++gv;
          if (j < nk) {
            ptx::umma_commit(&kempty[gk % NKS]);
            if (j == nk - 1) ptx::umma_commit(qfree);
            ++gk;
          }
        }
      }
      if (!ok) *abort_flag = 1;
      if (*abort_flag) {  // MMAs of this thread may still run: drain them before TMEM is freed
        ptx::umma_commit(bar_drain);
        ptx::mbar_wait(bar_drain, 0);
      }
    }
  } else {
    // ---------------------------------------------------------------- softmax, output
    const int x = (warp - 2) >> 2;       // query tile A (warps 2-5) or B (6-9)
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;   // query row of the tile = TMEM lane
    const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
    const uint32_t tS = trow + C::T_S + x * 128, tO = trow + C::T_O + x * 128;
    const float c2 = p.scale * kLog2eTc;
    const float kRescale = 8.f / c2;      // P stays below 2^8 between rescales
    bool ok = true;
    int i = 0;
    uint32_t s_phase = 0, pv_phase = 0;  // bar_s[x] / bar_pv[x] phases consumed
    for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++i) {
      int q0, b, h;
      unit_of(u, q0, b, h);
      float m = -INFINITY, l = 0.f;
      for (int j = 0; j < nk; ++j) {
        ok = __all_sync(0xffffffffu, ptx::mbar_wait(&bar_s[x], s_phase));
        s_phase ^= 1u;
        if (!ok || *abort_flag) { ok = false; *abort_flag = 1; break; }
        ptx::tc_fence_after();
        // The row maximum: keys 0-63 (read again below), then 64-127 (kept in registers).
        const int kv = N - j * BK;  // valid keys of the tile (at least one)
        const bool ragged = kv < BK;
        uint32_t rh[64];
        float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
        ptx::tmem_ld_32x32b_x32(tS, *reinterpret_cast<uint32_t(*)[32]>(rh));
        ptx::tmem_ld_32x32b_x32(tS + 32, *reinterpret_cast<uint32_t(*)[32]>(rh + 32));
        ptx::tmem_ld_wait();
        if (ragged) mask_keys(rh, 0, kv);
        row_max4(rh, mx);
        ptx::tmem_ld_32x32b_x32(tS + 64, *reinterpret_cast<uint32_t(*)[32]>(rh));
        ptx::tmem_ld_32x32b_x32(tS + 96, *reinterpret_cast<uint32_t(*)[32]>(rh + 32));
        ptx::tmem_ld_wait();
        if (ragged) mask_keys(rh, 64, kv);
        row_max4(rh, mx);
        const float tmax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
        if (j == 0) {
          m = tmax;
        } else if (__any_sync(0xffffffffu, tmax > m + kRescale)) {
          // the maximum of some row of the warp moved up: the whole warp (the tensor-memory
          // accesses are warp-wide) rescales O and l to the new references once the previous
          // P V product has finished; rows whose maximum stayed take the factor 1
          const float mn = fmaxf(m, tmax);
          const float f = ptx::ex2_approx((m - mn) * c2);
          ok = __all_sync(0xffffffffu, ptx::mbar_wait(&bar_pv[x], pv_phase));
          if (!ok) { *abort_flag = 1; break; }
          ptx::tc_fence_after();
#pragma unroll 1
          for (int c = 0; c < D / 16; ++c) {  // 16 columns at a time: the S row stays in registers
            uint32_t ro[16];
            ptx::tmem_ld_32x32b_x16(tO + c * 16, ro);
            ptx::tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 16; ++e) ro[e] = __float_as_uint(__uint_as_float(ro[e]) * f);
            ptx::tmem_st_32x32b_x16(tO + c * 16, ro);
          }
          l *= f;
          m = mn;
        }
        // P = exp(scale (S - m)) (at most 2^8) in bf16 at the columns Ff2::p_col gives: keys 64-127 over the
        // S columns 64-95 (already in registers), keys 0-63 over 96-127, so keys 0-63 can be
        // read again while keys 64-127 are exponentiated
        const float mc = m * c2;
        const float2 vc2 = make_float2(c2, c2), vmc = make_float2(-mc, -mc);
        float2 l0 = make_float2(0.f, 0.f), l1 = make_float2(0.f, 0.f);
        uint32_t ra[32];
        ptx::tmem_ld_32x32b_x32(tS, ra);
        exp_pack(rh, vc2, vmc, l0, l1);
        ptx::tmem_st_32x32b_x16(tS + C::p_col(4), *reinterpret_cast<const uint32_t(*)[16]>(rh));
        ptx::tmem_st_32x32b_x16(tS + C::p_col(6), *reinterpret_cast<const uint32_t(*)[16]>(rh + 16));
        uint32_t(&rb)[32] = *reinterpret_cast<uint32_t(*)[32]>(rh + 32);
        ptx::tmem_ld_32x32b_x32(tS + 32, rb);
        ptx::tmem_ld_wait();
        if (ragged) {
          mask_keys(ra, 0, kv);
          mask_keys(rb, 32, kv);
        }
        exp_pack(ra, vc2, vmc, l0, l1);
        ptx::tmem_st_32x32b_x16(tS + C::p_col(0), *reinterpret_cast<const uint32_t(*)[16]>(ra));
        exp_pack(rb, vc2, vmc, l0, l1);
        ptx::tmem_st_32x32b_x16(tS + C::p_col(2), *reinterpret_cast<const uint32_t(*)[16]>(rb));
        l += (l0.x + l0.y) + (l1.x + l1.y);
        ptx::tmem_st_wait();
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&pready[x]);
        // the P V product of this tile completes phase pv_phase of bar_pv[x] (the rescale
        // above waits on the previous tile's)
        if (j > 0) pv_phase ^= 1u;
      }
      if (!ok) break;
      // the unit's output: O / l once the last P V product is done, and the log-sum-exp
      ok = __all_sync(0xffffffffu, ptx::mbar_wait(&bar_pv[x], pv_phase));
      pv_phase ^= 1u;
      if (!ok || *abort_flag) { ok = false; *abort_flag = 1; break; }
      ptx::tc_fence_after();
      const int q = q0 + x * BQ + r;
      const float inv = 1.f / l;
#pragma unroll 1
      for (int c = 0; c < D / 32; ++c) {
        uint32_t ro[32];
        ptx::tmem_ld_32x32b_x32(tO + c * 32, ro);
        ptx::tmem_ld_wait();
        if (q < N) {
          bf16* o = static_cast<bf16*>(p.o.base(q)) + p.o.off(b, q, N, (int64_t)h * D + c * 32);
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            uint4 w;
            w.x = pack2_bf16(__uint_as_float(ro[8 * v]) * inv, __uint_as_float(ro[8 * v + 1]) * inv);
            w.y = pack2_bf16(__uint_as_float(ro[8 * v + 2]) * inv, __uint_as_float(ro[8 * v + 3]) * inv);
            w.z = pack2_bf16(__uint_as_float(ro[8 * v + 4]) * inv, __uint_as_float(ro[8 * v + 5]) * inv);
            w.w = pack2_bf16(__uint_as_float(ro[8 * v + 6]) * inv, __uint_as_float(ro[8 * v + 7]) * inv);
            *reinterpret_cast<uint4*>(o + 8 * v) = w;
          }
        }
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(&ofree[x]);
      if (q < N) p.lse[((int64_t)b * p.heads + h) * N + q] = p.scale * m + logf(l);
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, 512);
  }
}

// 3D view [sequence][token][column] of a stream buffer (bf16), boxes of 64 columns x `rows`.
int seg_map(CUtensorMap* m, const void* base, int64_t ld, int ntok, int B, int rows) {
  const uint64_t dims[3] = {(uint64_t)ld, (uint64_t)ntok, (uint64_t)B};
  const uint64_t strides[2] = {(uint64_t)ld * 2, (uint64_t)ld * 2 * ntok};
  const uint32_t box[3] = {64, (uint32_t)rows, 1};
  return encode_tmap(m, false, 3, base, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// The pipelined backward (fa_bwd_tc128_kernel, fa_bwd_tc64_kernel).
template <int D>
int launch_v3(const AttnBwdArgs& a, cudaStream_t s) {
  using C = Fb2<D>;
  auto kernel = D == 128 ? fa_bwd_tc128_kernel : fa_bwd_tc64_kernel;
  const AttnArgs& f = a.f;
  const int n0 = f.q.n0, N = f.N;
  const int n1 = N - n0;
  FbMaps maps;
  for (int sg = 0; sg < 2; ++sg) {
    const int nt = sg == 0 ? n0 : n1;
    if (nt <= 0) {  // single stream: the second views are unused copies
      maps.q[1] = maps.q[0];
      maps.k[1] = maps.k[0];
      maps.v[1] = maps.v[0];
      maps.dO[1] = maps.dO[0];
      break;
    }
    JAGG_TRY(seg_map(&maps.q[sg], sg ? f.q.p1 : f.q.p0, sg ? f.q.ld1 : f.q.ld0, nt, f.B, C::BQ));
    JAGG_TRY(seg_map(&maps.k[sg], sg ? f.k.p1 : f.k.p0, sg ? f.k.ld1 : f.k.ld0, nt, f.B, C::BK));
    JAGG_TRY(seg_map(&maps.v[sg], sg ? f.v.p1 : f.v.p0, sg ? f.v.ld1 : f.v.ld0, nt, f.B, C::BK));
    JAGG_TRY(seg_map(&maps.dO[sg], sg ? a.dO.p1 : a.dO.p0, sg ? a.dO.ld1 : a.dO.ld0, nt, f.B, C::BQ));
  }
  {
    const int64_t cols = (int64_t)f.heads * C::D;
    const uint64_t dims[3] = {(uint64_t)cols, (uint64_t)N, (uint64_t)f.B};
    const uint64_t strides[2] = {(uint64_t)cols * 4, (uint64_t)cols * 4 * N};
    const uint32_t box[3] = {32, 32, 1};
    JAGG_TRY(encode_tmap(&maps.dq, true, 3, a.dq_acc, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B));
  }
  FbParams p;
  p.B = f.B; p.N = N; p.heads = f.heads; p.n0 = n0 > 0 && n0 < N ? n0 : N;
  p.scale = f.scale;
  p.q_col0 = f.q_col0; p.k_col0 = f.k_col0; p.v_col0 = f.v_col0;
  p.dk_col0 = a.dk_col0; p.dv_col0 = a.dv_col0;
  p.lse = f.lse; p.Dv = a.Dv;
  p.dk = a.dk; p.dv = a.dv;
  static bool attr = false;
  if (!attr) {
    JAGG_CUDA_TRY(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM));
    attr = true;
  }
  const int units = ceil_div(N, C::BK) * f.B * f.heads;
  const int nsm = sm_count();
  kernel<<<units < nsm ? units : nsm, FB2_THREADS, C::SMEM, s>>>(maps, p);
  JAGG_LAUNCHED();
  return JAGG_OK;
}

template <int D>
int launch_fwd(const AttnArgs& f, cudaStream_t s) {
  using C = FfCfg<D>;
  const int n0 = f.q.n0, N = f.N;
  const int n1 = N - n0;
  FfMaps maps;
  for (int sg = 0; sg < 2; ++sg) {
    const int nt = sg == 0 ? n0 : n1;
    if (nt <= 0) {  // single stream: the second views are unused copies
      maps.q[1] = maps.q[0];
      maps.k[1] = maps.k[0];
      maps.v[1] = maps.v[0];
      break;
    }
    JAGG_TRY(seg_map(&maps.q[sg], sg ? f.q.p1 : f.q.p0, sg ? f.q.ld1 : f.q.ld0, nt, f.B, C::BQ));
    JAGG_TRY(seg_map(&maps.k[sg], sg ? f.k.p1 : f.k.p0, sg ? f.k.ld1 : f.k.ld0, nt, f.B, C::BK));
    JAGG_TRY(seg_map(&maps.v[sg], sg ? f.v.p1 : f.v.p0, sg ? f.v.ld1 : f.v.ld0, nt, f.B, C::BK));
  }
  FfParams p;
  p.B = f.B; p.N = N; p.heads = f.heads; p.n0 = n0 > 0 && n0 < N ? n0 : N;
  p.scale = f.scale;
  p.q_col0 = f.q_col0; p.k_col0 = f.k_col0; p.v_col0 = f.v_col0;
  p.o = f.o;
  p.lse = f.lse;
  static bool attr = false;
  if (!attr) {
    JAGG_CUDA_TRY(cudaFuncSetAttribute(fa_fwd_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM));
    attr = true;
  }
  const int units = ceil_div(N, C::BQ) * f.B * f.heads;
  const int nsm = sm_count();
  fa_fwd_tc_kernel<D><<<units < nsm ? units : nsm, FF_THREADS, C::SMEM, s>>>(maps, p);
  JAGG_LAUNCHED();
  return JAGG_OK;
}

}  // namespace

// Whether the tensor-core forward serves the call: bf16, head dim 64 / 128, the stream
// boundary on a 128-token multiple, 16-byte aligned operands and output rows.
bool attention_fwd_tc_eligible(const AttnArgs& f) {
  if (f.dtype != JAGG_DTYPE_BF16 || (f.dh != 64 && f.dh != 128) || !f.lse) return false;
  const int n0 = f.q.n0;
  const bool single = n0 >= f.N;
  if (!single && (n0 <= 0 || n0 % 128)) return false;
  const SegRows* views[4] = {&f.q, &f.k, &f.v, &f.o};
  for (const SegRows* v : views) {
    if (v->n0 != n0) return false;
    if (!aligned16(v->p0) || v->ld0 % 8) return false;
    if (!single && (!aligned16(v->p1) || v->ld1 % 8)) return false;
  }
  return f.q_col0 % 8 == 0 && f.k_col0 % 8 == 0 && f.v_col0 % 8 == 0;
}

// The head-dim-128 forward (fa_fwd_tc128_kernel).
int launch_fwd128(const AttnArgs& f, cudaStream_t s) {
  using C = Ff2;
  const int n0 = f.q.n0, N = f.N;
  const int n1 = N - n0;
  FfMaps maps;
  for (int sg = 0; sg < 2; ++sg) {
    const int nt = sg == 0 ? n0 : n1;
    if (nt <= 0) {  // single stream: the second views are unused copies
      maps.q[1] = maps.q[0];
      maps.k[1] = maps.k[0];
      maps.v[1] = maps.v[0];
      break;
    }
    JAGG_TRY(seg_map(&maps.q[sg], sg ? f.q.p1 : f.q.p0, sg ? f.q.ld1 : f.q.ld0, nt, f.B, C::BQ));
    JAGG_TRY(seg_map(&maps.k[sg], sg ? f.k.p1 : f.k.p0, sg ? f.k.ld1 : f.k.ld0, nt, f.B, C::BK));
    JAGG_TRY(seg_map(&maps.v[sg], sg ? f.v.p1 : f.v.p0, sg ? f.v.ld1 : f.v.ld0, nt, f.B, C::BK));
  }
  FfParams p;
  p.B = f.B; p.N = N; p.heads = f.heads; p.n0 = n0 > 0 && n0 < N ? n0 : N;
  p.scale = f.scale;
  p.q_col0 = f.q_col0; p.k_col0 = f.k_col0; p.v_col0 = f.v_col0;
  p.o = f.o;
  p.lse = f.lse;
  static bool attr = false;
  if (!attr) {
    JAGG_CUDA_TRY(cudaFuncSetAttribute(fa_fwd_tc128_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM));
    attr = true;
  }
  const int units = ceil_div(ceil_div(N, C::BQ), 2) * f.B * f.heads;
  const int nsm = sm_count();
  fa_fwd_tc128_kernel<<<units < nsm ? units : nsm, FF2_THREADS, C::SMEM, s>>>(maps, p);
  JAGG_LAUNCHED();
  return JAGG_OK;
}

int attention_fwd_tc(const AttnArgs& f, cudaStream_t s) {
  return f.dh == 64 ? launch_fwd<64>(f, s) : launch_fwd128(f, s);
}

// Whether the tensor-core backward serves the call: bf16, head dim 64 / 128, the stream
// boundary on a 128-token multiple, 16-byte aligned buffers with 16-byte row pitches.
bool attention_bwd_tc_eligible(const AttnBwdArgs& a) {
  const AttnArgs& f = a.f;
  if (f.dtype != JAGG_DTYPE_BF16 || (f.dh != 64 && f.dh != 128)) return false;
  const int n0 = f.q.n0;
  const bool single = n0 >= f.N;
  if (!single && (n0 <= 0 || n0 % 128)) return false;
  const SegRows* views[4] = {&f.q, &f.k, &f.v, &a.dO};
  for (const SegRows* v : views) {
    if (v->n0 != n0) return false;
    if (!aligned16(v->p0) || v->ld0 % 8) return false;
    if (!single && (!aligned16(v->p1) || v->ld1 % 8)) return false;
  }
  if (f.q_col0 % 8 || f.k_col0 % 8 || f.v_col0 % 8) return false;
  return aligned16(a.dq_acc) && (a.dk_col0 % 8 == 0) && (a.dv_col0 % 8 == 0) && a.dk.ld0 % 8 == 0 &&
         a.dv.ld0 % 8 == 0 && (single || (a.dk.ld1 % 8 == 0 && a.dv.ld1 % 8 == 0));
}

int attention_bwd_tc(const AttnBwdArgs& a, cudaStream_t s) {
  return a.f.dh == 64 ? launch_v3<64>(a, s) : launch_v3<128>(a, s);
}

}  // namespace jagg
