// Dense products of the backbone on sm_103a.
//
// bf16 x bf16 -> f32: a persistent, warp-specialised tcgen05 kernel.  One CTA per SM;
// warp 0 issues TMA loads of 128-byte-swizzled tiles into a multi-stage shared-memory
// ring, warp 1 (one elected thread) issues tcgen05.mma into a double-buffered TMEM
// accumulator, warps 2-9 (two per TMEM lane quarter) drain TMEM with tcgen05.ld and run the fused epilogue while
// the next tile's MMAs proceed.  Both operands may be K-major or MN-major, so the
// forward (X W^T), input-gradient (dY W) and weight-gradient (dY^T X) products all read
// their operands in place, without transposes.
//
// f32 operands (the fp32 configuration and the per-sequence modulation / t-embedding
// products with B rows): a tiled SIMT kernel with the same epilogue.
#include <cuda.h>
#include <mutex>

#include "gemm.cuh"
#include "ptx.cuh"
#include "tmap.cuh"

namespace jagg {

int unit_status_gemm(unsigned* v, int clear) { return read_unit_status(v, clear); }

// ------------------------------------------------------------------ epilogue
struct EpiParams {
  int M, N, epi;
  const void* bias;
  int bias_bf16;
  void* C;
  int64_t ldc;
  int c_bf16;
  void* C2;
  int64_t ldc2;
  const void* aux;
  int64_t ld_aux;
  const float* gate;
  int64_t gate_stride;
  int rows_per_seq;
  int remap_rows, remap_offset;
  int64_t remap_stride;
  int vec_ok;  // 8-wide vector accesses are aligned
  int c_trans, bias_m;
};

__device__ __forceinline__ float ldv(const void* p, int64_t i, int is_bf16) {
  return is_bf16 ? __bfloat162float(static_cast<const bf16*>(p)[i]) : static_cast<const float*>(p)[i];
}
__device__ __forceinline__ void stv(void* p, int64_t i, int is_bf16, float v) {
  if (is_bf16)
    static_cast<bf16*>(p)[i] = __float2bfloat16_rn(v);
  else
    static_cast<float*>(p)[i] = v;
}

__device__ __forceinline__ int64_t epi_crow(const EpiParams& e, int m) {
  return e.remap_rows ? (int64_t)(m / e.remap_rows) * e.remap_stride + e.remap_offset + m % e.remap_rows
                      : (int64_t)m;
}

// One element (m < M, n < N).
__device__ __forceinline__ void epi_apply1(const EpiParams& e, int m, int n, float acc) {
  const int64_t cr = epi_crow(e, m);
  switch (e.epi) {
    case EPI_STORE: {
      float v = acc + (e.bias ? ldv(e.bias, e.bias_m ? m : n, e.bias_bf16) : 0.f);
      stv(e.C, e.c_trans ? (int64_t)n * e.ldc + cr : cr * e.ldc + n, e.c_bf16, v);
    } break;
    case EPI_GELU: {
      float g, dg;
      gelu_tanh_both(acc + (e.bias ? ldv(e.bias, n, e.bias_bf16) : 0.f), g, dg);
      if (e.C) stv(e.C, cr * e.ldc + n, e.c_bf16, dg);
      stv(e.C2, cr * e.ldc2 + n, e.c_bf16, g);
    } break;
    case EPI_GATE_RESID: {
      float y = acc + (e.bias ? ldv(e.bias, n, e.bias_bf16) : 0.f);
      stv(e.C, cr * e.ldc + n, e.c_bf16, y);
      float g = e.gate[(int64_t)(m / e.rows_per_seq) * e.gate_stride + n];
      const float* hin = static_cast<const float*>(e.aux);
      static_cast<float*>(e.C2)[(int64_t)m * e.ldc2 + n] = hin[(int64_t)m * e.ld_aux + n] + g * y;
    } break;
    case EPI_MUL_AUX:
      stv(e.C, cr * e.ldc + n, e.c_bf16, acc * ldv(e.aux, (int64_t)m * e.ld_aux + n, e.c_bf16));
      break;
    case EPI_ACCUM:
      atomicAdd(static_cast<float*>(e.C) + (e.c_trans ? (int64_t)n * e.ldc + cr : cr * e.ldc + n), acc);
      break;
  }
}

// Eight consecutive columns n .. n+7 of row m (m < M).  Vector path when aligned.
__device__ __forceinline__ void epi_apply8(const EpiParams& e, int m, int n, const float (&a)[8]) {
  if (!e.vec_ok || n + 8 > e.N) {
#pragma unroll
    for (int i = 0; i < 8; ++i)
      if (n + i < e.N) epi_apply1(e, m, n + i, a[i]);
    return;
  }
  const int64_t cr = epi_crow(e, m);
  float v[8];
  if (e.epi != EPI_MUL_AUX && e.epi != EPI_ACCUM && e.bias) {
    if (e.bias_bf16) {
      uint4 raw = *reinterpret_cast<const uint4*>(static_cast<const bf16*>(e.bias) + n);
      const bf16* b = reinterpret_cast<const bf16*>(&raw);
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = a[i] + __bfloat162float(b[i]);
    } else {
      const float4* b4 = reinterpret_cast<const float4*>(static_cast<const float*>(e.bias) + n);
      float4 b0 = b4[0], b1 = b4[1];
      v[0] = a[0] + b0.x; v[1] = a[1] + b0.y; v[2] = a[2] + b0.z; v[3] = a[3] + b0.w;
      v[4] = a[4] + b1.x; v[5] = a[5] + b1.y; v[6] = a[6] + b1.z; v[7] = a[7] + b1.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = a[i];
  }
  auto store8 = [&](void* base, int64_t idx, int is_bf16, const float (&x)[8]) {
    if (is_bf16) {
      uint4 raw;
      bf16* h = reinterpret_cast<bf16*>(&raw);
#pragma unroll
      for (int i = 0; i < 8; ++i) h[i] = __float2bfloat16_rn(x[i]);
      *reinterpret_cast<uint4*>(static_cast<bf16*>(base) + idx) = raw;
    } else {
      float4* p = reinterpret_cast<float4*>(static_cast<float*>(base) + idx);
      p[0] = make_float4(x[0], x[1], x[2], x[3]);
      p[1] = make_float4(x[4], x[5], x[6], x[7]);
    }
  };
  switch (e.epi) {
    case EPI_STORE:
      store8(e.C, cr * e.ldc + n, e.c_bf16, v);
      break;
    case EPI_GELU: {
      float gv[8], dv[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) gelu_tanh_both(v[i], gv[i], dv[i]);
      if (e.C) store8(e.C, cr * e.ldc + n, e.c_bf16, dv);
      store8(e.C2, cr * e.ldc2 + n, e.c_bf16, gv);
    } break;
    case EPI_GATE_RESID: {
      store8(e.C, cr * e.ldc + n, e.c_bf16, v);
      const float* g = e.gate + (int64_t)(m / e.rows_per_seq) * e.gate_stride + n;
      const float4* h4 = reinterpret_cast<const float4*>(static_cast<const float*>(e.aux) + (int64_t)m * e.ld_aux + n);
      float4 h0 = h4[0], h1 = h4[1];
      float o[8] = {h0.x + g[0] * v[0], h0.y + g[1] * v[1], h0.z + g[2] * v[2], h0.w + g[3] * v[3],
                    h1.x + g[4] * v[4], h1.y + g[5] * v[5], h1.z + g[6] * v[6], h1.w + g[7] * v[7]};
      store8(e.C2, (int64_t)m * e.ldc2 + n, 0, o);
    } break;
    case EPI_MUL_AUX: {
      float u[8];
      if (e.c_bf16) {
        uint4 raw = *reinterpret_cast<const uint4*>(static_cast<const bf16*>(e.aux) + (int64_t)m * e.ld_aux + n);
        const bf16* h = reinterpret_cast<const bf16*>(&raw);
#pragma unroll
        for (int i = 0; i < 8; ++i) u[i] = __bfloat162float(h[i]);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) u[i] = static_cast<const float*>(e.aux)[(int64_t)m * e.ld_aux + n + i];
      }
      float o[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) o[i] = a[i] * u[i];
      store8(e.C, cr * e.ldc + n, e.c_bf16, o);
    } break;
    case EPI_ACCUM: {
      float* p = static_cast<float*>(e.C) + cr * e.ldc + n;
      ptx::red_add_v4(p, a[0], a[1], a[2], a[3]);
      ptx::red_add_v4(p + 4, a[4], a[5], a[6], a[7]);
    } break;
  }
}

// ------------------------------------------------------------------ tcgen05 kernel
// Staged epilogues: the output tile goes through swizzled shared memory and leaves with
// TMA stores (or TMA f32 reduce-adds), and the multiplier of EPI_MUL_AUX arrives in
// shared memory by TMA before the accumulator is ready.
// STAGED_ROWS: the other row-major epilogues (GELU, gated residual, row-remapped stores):
// each 32 x 32 chunk goes through swizzled shared memory and back so that a lane holds 4
// consecutive columns of one row, and every global load / store of the epilogue covers
// contiguous 128-byte row segments.
enum : int { STAGED_NONE = 0, STAGED_STORE = 1, STAGED_MUL_AUX = 2, STAGED_ACCUM = 3, STAGED_ROWS = 4, STAGED_GELU = 5 };

struct TcParams {
  int tiles_m, tiles_n, splits, k_blocks;
  int raster_n;  // 1: consecutive tile indices walk N first (see tile_order)
  int staged;  // STAGED_*
  EpiParams e;
};

constexpr int TC_BM = 128;
constexpr int TC_BK = 64;
// Epilogue warps EW: 4 (one per TMEM lane quarter, two staging chunks each: the TMA-staged
// epilogues, whose stores overlap the next chunk) or 8 (two per quarter, alternate
// chunks, one staging chunk each: the arithmetic-heavy row-coalesced epilogues).
constexpr int TC_MAX_EPI_WARPS = 8;
__host__ __device__ constexpr int tc_threads(int ew) { return 64 + 32 * ew; }

// AUX: the instance can run EPI_MUL_AUX (the input-gradient products, K-major A and
// MN-major B): 1 = every multiplier chunk of a warp's tile loaded at once (tiles of at most
// 128 columns), 2 = a two-slot ring per epilogue warp refilled chunk by chunk (256-column
// tiles: for long K, where the main loop of the next tile covers the epilogue's loads);
// 0 = no shared memory for a multiplier.
template <int BN, int AUX, int EW>
struct TcCfg {
  static constexpr int SPLIT = EW / 4;           // chunk stride of an epilogue warp
  static constexpr int NSTG = EW == 4 ? 2 : 1;   // staging chunks per epilogue warp
  static constexpr int A_BYTES = TC_BM * TC_BK * 2;
  static constexpr int B_BYTES = BN * TC_BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  // Per epilogue warp (32 rows, every other 32-column chunk of the tile): one staging
  // chunk of 32 x 32 outputs (4 KB as f32; the bf16 output of EPI_MUL_AUX uses 2 KB), and
  // for EPI_MUL_AUX this warp's multiplier chunks (BN / 64 of 32 x 32 bf16) after it.
  static constexpr int CHUNK_BF16 = 32 * 32 * 2;
  static constexpr int AUX_SLOTS = AUX == 2 ? 2 : (BN / 32 + SPLIT - 1) / SPLIT;
  static constexpr int AUX_WARP_BYTES = NSTG * CHUNK_BF16 + AUX_SLOTS * CHUNK_BF16;
  static constexpr int EPI_WARP_BYTES =
      AUX && AUX_WARP_BYTES > NSTG * 2 * CHUNK_BF16 ? AUX_WARP_BYTES : NSTG * 2 * CHUNK_BF16;
  static constexpr int EPI_BYTES = EW * EPI_WARP_BYTES;
  static constexpr int FIXED = 1024 /*align*/ + 256 /*barriers*/;
  static constexpr int MAX_SMEM = 232448;
  static constexpr int FIT = (MAX_SMEM - FIXED - EPI_BYTES) / STAGE_BYTES;
  static constexpr int STAGES = FIT > 8 ? 8 : FIT;
  static constexpr int TMEM_COLS = 2 * BN < 32 ? 32 : 2 * BN;
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + EPI_BYTES + FIXED;
  static_assert(STAGES >= 4, "pipeline too shallow");
  static_assert((2 * STAGES + 4 + TC_MAX_EPI_WARPS + 1) * 8 + 4 <= 256, "barrier region");
  static_assert(SMEM_BYTES <= MAX_SMEM, "shared memory budget");
};

template <int BN, bool A_MN, bool B_MN, int AUX, int EW>
__global__ void __launch_bounds__(tc_threads(EW), 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmX, TcParams p) {
  using Cfg = TcCfg<BN, AUX, EW>;
  constexpr int STAGES = Cfg::STAGES;
  constexpr int SPLIT = Cfg::SPLIT;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* epi_smem = smem + STAGES * Cfg::STAGE_BYTES;  // 1024-byte aligned
  uint64_t* full = reinterpret_cast<uint64_t*>(epi_smem + Cfg::EPI_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* auxbar = tempty + 2;  // one per epilogue warp (two, one per ring slot, when AUX == 2)
  uint64_t* drainbar = auxbar + TC_MAX_EPI_WARPS;  // the MMA thread's drain after a give-up
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drainbar + 1);
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < STAGES; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      ptx::mbar_init(&tfull[a], 1);
      ptx::mbar_init(&tempty[a], EW);
    }
    for (int q = 0; q < (AUX == 2 ? 2 * EW : EW); ++q) ptx::mbar_init(&auxbar[q], 1);
    ptx::mbar_init(drainbar, 1);
    ptx::fence_mbar_init();
    ptx::prefetch_tmap(&tmA);
    ptx::prefetch_tmap(&tmB);
    if (p.staged != STAGED_NONE && p.staged != STAGED_ROWS) ptx::prefetch_tmap(&tmC);
    if (p.staged == STAGED_MUL_AUX || p.staged == STAGED_GELU) ptx::prefetch_tmap(&tmX);
  }
  if (warp == 1) {
    ptx::tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
    ptx::tmem_relinquish();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int total = p.tiles_m * p.tiles_n * p.splits;
  // tile index -> (m tile, n tile, split), the faster of m and n chosen by the host.
  auto decode = [&](int t, int& tm, int& tn, int& ks) {
    if (p.raster_n) {
      tn = t % p.tiles_n;
      const int r = t / p.tiles_n;
      tm = r % p.tiles_m;
      ks = r / p.tiles_m;
    } else {
      tm = t % p.tiles_m;
      const int r = t / p.tiles_m;
      tn = r % p.tiles_n;
      ks = r / p.tiles_n;
    }
  };
  auto krange = [&](int ks, int& kb0, int& kb1) {
    kb0 = (int)((long long)p.k_blocks * ks / p.splits);
    kb1 = (int)((long long)p.k_blocks * (ks + 1) / p.splits);
  };

  if (warp == 0) {
    if (ptx::elect_one()) {
      // ---------------- TMA producer
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0, issued_parity = 0;  // per stage: a load was issued, and its phase
      for (int t = blockIdx.x; t < total && !abort_flag; t += gridDim.x) {
        int tm, tn, ks, kb0, kb1;
        decode(t, tm, tn, ks);
        krange(ks, kb0, kb1);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!ptx::mbar_wait(&empty[stage], phase ^ 1)) { abort_flag = 1; break; }
          uint8_t* sA = smem + stage * Cfg::STAGE_BYTES;
          uint8_t* sB = sA + Cfg::A_BYTES;
          ptx::mbar_arrive_expect_tx(&full[stage], Cfg::STAGE_BYTES);
          if (!A_MN) {
            ptx::tma_load_2d(sA, &tmA, &full[stage], kb * TC_BK, tm * TC_BM);
          } else {
#pragma unroll
            for (int c = 0; c < TC_BM / 64; ++c)
              ptx::tma_load_2d(sA + c * (64 * TC_BK * 2), &tmA, &full[stage], tm * TC_BM + c * 64, kb * TC_BK);
          }
          if (!B_MN) {
            ptx::tma_load_2d(sB, &tmB, &full[stage], kb * TC_BK, tn * BN);
          } else {
#pragma unroll
            for (int c = 0; c < BN / 64; ++c)
              ptx::tma_load_2d(sB + c * (64 * TC_BK * 2), &tmB, &full[stage], tn * BN + c * 64, kb * TC_BK);
          }
          issued |= 1u << stage;
          issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
      }
      // After a give-up anywhere in the CTA, the loads already issued may still be landing
      // in shared memory: wait (bounded) for the last phase of every stage before exiting.
      if (abort_flag)
        for (int s = 0; s < STAGES; ++s)
          if (issued & (1u << s)) ptx::mbar_wait(&full[s], (issued_parity >> s) & 1u);
    }
  } else if (warp == 1) {
    if (ptx::elect_one()) {
      // ---------------- MMA issuer
      constexpr uint32_t idesc = ptx::idesc_bf16(TC_BM, BN, A_MN, B_MN);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      for (int t = blockIdx.x; t < total && !abort_flag; t += gridDim.x) {
        int tm, tn, ks, kb0, kb1;
        decode(t, tm, tn, ks);
        krange(ks, kb0, kb1);
        if (!ptx::mbar_wait(&tempty[acc], acc_phase ^ 1)) { abort_flag = 1; break; }
        ptx::tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!ptx::mbar_wait(&full[stage], phase)) { ok = false; break; }
          ptx::tc_fence_after();
          const uint32_t a_addr = ptx::smem_u32(smem + stage * Cfg::STAGE_BYTES);
          const uint32_t b_addr = a_addr + Cfg::A_BYTES;
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k) {
            // K-major: step 16 elements = 32 bytes inside the swizzled 128-byte row.
            // MN-major: step 16 k-rows = two 1024-byte atoms.
            const uint64_t ad = A_MN ? ptx::sdesc_sw128(a_addr + k * 2048, 64 * TC_BK * 2, 1024)
                                     : ptx::sdesc_sw128(a_addr + k * 32, 16, 1024);
            const uint64_t bd = B_MN ? ptx::sdesc_sw128(b_addr + k * 2048, 64 * TC_BK * 2, 1024)
                                     : ptx::sdesc_sw128(b_addr + k * 32, 16, 1024);
            ptx::umma_bf16(d_tmem, ad, bd, idesc, (kb > kb0 || k > 0) ? 1u : 0u);
          }
          ptx::umma_commit(&empty[stage]);
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
        if (!ok) { abort_flag = 1; break; }
        ptx::umma_commit(&tfull[acc]);
        if (++acc == 2) { acc = 0; acc_phase ^= 1; }
      }
      // After a give-up, MMAs of this thread may still be running on TMEM and shared
      // memory: commit them to the drain barrier and wait (bounded) before the CTA frees TMEM.
      if (abort_flag) {
        ptx::umma_commit(drainbar);
        ptx::mbar_wait(drainbar, 0);
      }
    }
  } else if constexpr (EW == 8) {
    // ---------------- row-coalesced epilogue (the only epilogue of the 8-warp instances), warps 2..9: TMEM lanes 32*(warp%4) .. +31, alternate chunks
    const int q = warp & 3, half = (warp - 2) >> 2, ew = warp - 2;  // half < SPLIT
    float* xch = reinterpret_cast<float*>(epi_smem + ew * Cfg::EPI_WARP_BYTES);  // one 32 x 32 f32 chunk
    const EpiParams& e = p.e;
    int acc = 0;
    uint32_t acc_phase = 0;
    const int sub = lane >> 3, c4 = lane & 7;  // read-back: rows sub, sub + 4, ...; columns 4 c4 .. +3
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
      int tm, tn, ks;
      decode(t, tm, tn, ks);
      bool ok = ptx::mbar_wait(&tfull[acc], acc_phase);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) { abort_flag = 1; break; }
      ptx::tc_fence_after();
      const int m0 = tm * TC_BM + q * 32;
      const int live_chunks = (m0 < e.M) ? min(BN / 32, (e.N - tn * BN + 31) / 32) : 0;
#pragma unroll 1
      for (int c = half; c < live_chunks; c += SPLIT) {
        uint32_t r[32];
        ptx::tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(q * 32) << 16) + acc * BN + c * 32, r);
        ptx::tmem_ld_wait();
        __syncwarp();  // the previous chunk's read-back is done
        uint8_t* row = reinterpret_cast<uint8_t*>(xch) + lane * 128;
#pragma unroll
        for (int u = 0; u < 8; ++u)
          *reinterpret_cast<uint4*>(row + ((u ^ (lane & 7)) << 4)) =
              make_uint4(r[4 * u], r[4 * u + 1], r[4 * u + 2], r[4 * u + 3]);
        __syncwarp();
        const int n = tn * BN + c * 32 + 4 * c4;
        float b4[4] = {0.f, 0.f, 0.f, 0.f};
        if (e.bias && e.epi != EPI_MUL_AUX && n < e.N) {
          if (e.bias_bf16) {
            const uint2 raw = *reinterpret_cast<const uint2*>(static_cast<const bf16*>(e.bias) + n);
            const bf16* hb = reinterpret_cast<const bf16*>(&raw);
#pragma unroll
            for (int i = 0; i < 4; ++i) b4[i] = __bfloat162float(hb[i]);
          } else {
            const float4 f = *reinterpret_cast<const float4*>(static_cast<const float*>(e.bias) + n);
            b4[0] = f.x; b4[1] = f.y; b4[2] = f.z; b4[3] = f.w;
          }
        }
        // every global operand of the chunk first (8 rows per lane), then the stores
        float4 av[8], xa[8], xg[8];
#pragma unroll
        for (int it = 0; it < 8; ++it) {
          const int rr = it * 4 + sub;
          const int m = m0 + rr;
          av[it] = *reinterpret_cast<const float4*>(reinterpret_cast<uint8_t*>(xch) + rr * 128 + ((c4 ^ (rr & 7)) << 4));
          xa[it] = make_float4(0.f, 0.f, 0.f, 0.f);
          xg[it] = xa[it];
          if (m < e.M && n < e.N) {
            if (e.epi == EPI_GATE_RESID) {
              xg[it] = *reinterpret_cast<const float4*>(e.gate + (int64_t)(m / e.rows_per_seq) * e.gate_stride + n);
              xa[it] = *reinterpret_cast<const float4*>(static_cast<const float*>(e.aux) + (int64_t)m * e.ld_aux + n);
            } else if (e.epi == EPI_MUL_AUX) {
              if (e.c_bf16) {
                const uint2 raw =
                    *reinterpret_cast<const uint2*>(static_cast<const bf16*>(e.aux) + (int64_t)m * e.ld_aux + n);
                const bf16* hb = reinterpret_cast<const bf16*>(&raw);
                xa[it] = make_float4(__bfloat162float(hb[0]), __bfloat162float(hb[1]), __bfloat162float(hb[2]),
                                     __bfloat162float(hb[3]));
              } else {
                xa[it] = *reinterpret_cast<const float4*>(static_cast<const float*>(e.aux) + (int64_t)m * e.ld_aux + n);
              }
            }
          }
        }
        __syncwarp();  // the chunk buffer is free for the next chunk
        auto st4 = [&](void* base, int64_t idx, int is_bf16, const float (&x)[4]) {
          if (is_bf16) {
            __nv_bfloat162 lo = __floats2bfloat162_rn(x[0], x[1]), hi = __floats2bfloat162_rn(x[2], x[3]);
            uint2 raw;
            raw.x = *reinterpret_cast<uint32_t*>(&lo);
            raw.y = *reinterpret_cast<uint32_t*>(&hi);
            *reinterpret_cast<uint2*>(static_cast<bf16*>(base) + idx) = raw;
          } else {
            *reinterpret_cast<float4*>(static_cast<float*>(base) + idx) = make_float4(x[0], x[1], x[2], x[3]);
          }
        };
#pragma unroll
        for (int it = 0; it < 8; ++it) {
          const int m = m0 + it * 4 + sub;
          if (m >= e.M || n >= e.N) continue;
          const float4 a4 = av[it];
          float v[4] = {a4.x + b4[0], a4.y + b4[1], a4.z + b4[2], a4.w + b4[3]};
          const int64_t cr = epi_crow(e, m);
          switch (e.epi) {
            case EPI_STORE:
              st4(e.C, cr * e.ldc + n, e.c_bf16, v);
              break;
            case EPI_GELU: {
              float g[4], dg[4];
#pragma unroll
              for (int i = 0; i < 4; ++i) gelu_tanh_both_approx(v[i], g[i], dg[i]);
              if (e.C) st4(e.C, cr * e.ldc + n, e.c_bf16, dg);
              st4(e.C2, cr * e.ldc2 + n, e.c_bf16, g);
            } break;
            case EPI_GATE_RESID: {
              st4(e.C, cr * e.ldc + n, e.c_bf16, v);
              const float4 g4 = xg[it], h4 = xa[it];
              const float o[4] = {h4.x + g4.x * v[0], h4.y + g4.y * v[1], h4.z + g4.z * v[2], h4.w + g4.w * v[3]};
              st4(e.C2, (int64_t)m * e.ldc2 + n, 0, o);
            } break;
            case EPI_MUL_AUX: {
              const float4 u4 = xa[it];
              const float o[4] = {a4.x * u4.x, a4.y * u4.y, a4.z * u4.z, a4.w * u4.w};
              st4(e.C, cr * e.ldc + n, e.c_bf16, o);
            } break;
            case EPI_ACCUM:
              ptx::red_add_v4(static_cast<float*>(e.C) + cr * e.ldc + n, a4.x, a4.y, a4.z, a4.w);
              break;
          }
        }
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(&tempty[acc]);
      if (++acc == 2) { acc = 0; acc_phase ^= 1; }
    }
  } else if (p.staged != STAGED_NONE) {
    // ---------------- staged epilogue (4-warp instances), warps 2..5: TMEM lanes 32*(warp%4) .. +31.
    // Thread = output row; per 32-column chunk: tcgen05.ld, the element-wise op, a write
    // into a swizzled staging chunk (64-byte rows for bf16, 128-byte rows for f32, so the
    // 16-byte writes of a warp hit distinct banks), then one TMA store / reduce-add of the
    // 32 x 32 box by lane 0.  The two warps of a lane quarter take alternate chunks.
    const int q = warp & 3, half = (warp - 2) >> 2, ew = warp - 2;  // half < SPLIT
    const bool mul = p.staged == STAGED_MUL_AUX;
    // STAGED_GELU: two bf16 outputs per chunk, GELU'(u) to C (when given, tmC) and GELU(u)
    // to C2 (tmX), both staged in one slot (a slot holds a 32 x 32 f32 box)
    // (the forward-only GELU epilogue is compiled into the forward-layout instances alone, so
    // the backward products keep their register budget)
    constexpr bool FWD = !A_MN && !B_MN;
    const bool gelu = FWD && p.staged == STAGED_GELU;
    const bool gelu_d = gelu && p.e.C != nullptr;
    const bool out_f32 = !p.e.c_bf16 && !gelu;
    const int chunk_bytes = out_f32 ? 4096 : Cfg::CHUNK_BF16;
    uint8_t* stg = epi_smem + ew * Cfg::EPI_WARP_BYTES;
    uint8_t* auxs = stg + Cfg::NSTG * Cfg::CHUNK_BF16;  // EPI_MUL_AUX only (bf16 output)
    int acc = 0, sbuf = 0;
    uint32_t acc_phase = 0, aux_phase = 0;
    uint32_t ring_phase[2] = {0u, 0u};  // AUX == 2: the phase each ring slot waits for next
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
      int tm, tn, ks;
      decode(t, tm, tn, ks);
      const int m0 = tm * TC_BM + q * 32;
      // boxes wholly outside the output (rows past M, column chunks past N) are skipped
      const bool rows_live = m0 < p.e.M;
      const int live_chunks = min(BN / 32, (p.e.N - tn * BN + 31) / 32);
      const int my_chunks = live_chunks > half ? (live_chunks - half + SPLIT - 1) / SPLIT : 0;
      const bool aux_load = mul && rows_live && my_chunks > 0;
      // AUX == 2: multiplier chunk i of the tile into ring slot i % 2 (this warp's chunks
      // i < 2 now, chunk i + 2 once chunk i has been used)
      auto ring_load = [&](int i) {
        ptx::mbar_arrive_expect_tx(&auxbar[2 * ew + (i & 1)], Cfg::CHUNK_BF16);
        ptx::tma_load_2d(auxs + (i & 1) * Cfg::CHUNK_BF16, &tmX, &auxbar[2 * ew + (i & 1)],
                         tn * BN + (half + SPLIT * i) * 32, m0);
      };
      if (aux_load) {
        // this warp's multiplier chunks of the tile; it finished reading the previous tile's
        __syncwarp();
        if (lane == 0) {
          if constexpr (AUX == 2) {
            for (int i = 0; i < 2 && i < my_chunks; ++i) ring_load(i);
          } else {
            ptx::mbar_arrive_expect_tx(&auxbar[ew], my_chunks * Cfg::CHUNK_BF16);
            for (int i = 0; i < my_chunks; ++i)
              ptx::tma_load_2d(auxs + i * Cfg::CHUNK_BF16, &tmX, &auxbar[ew], tn * BN + (half + SPLIT * i) * 32,
                               m0);
          }
        }
      }
      bool ok = ptx::mbar_wait(&tfull[acc], acc_phase);
      if (aux_load && AUX != 2) {  // waited for even after a give-up: the multiplier load is in flight
        ok = ptx::mbar_wait(&auxbar[ew], aux_phase) && ok;
        aux_phase ^= 1u;
      }
      if (aux_load && AUX == 2 && !ok) {  // a give-up: wait for the ring loads in flight
        for (int i = 0; i < 2 && i < my_chunks; ++i) {
          ptx::mbar_wait(&auxbar[2 * ew + i], ring_phase[i]);
          ring_phase[i] ^= 1u;
        }
      }
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) { abort_flag = 1; break; }
      ptx::tc_fence_after();
#pragma unroll 1
      for (int c = half; c < (rows_live ? live_chunks : 0); c += SPLIT) {
        uint32_t r[32];
        ptx::tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(q * 32) << 16) + acc * BN + c * 32, r);
        ptx::tmem_ld_wait();
        const int n0 = tn * BN + c * 32;
        float v[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
        if ((p.staged == STAGED_STORE || gelu) && p.e.bias) {
          if (n0 + 32 <= p.e.N) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] += ldv(p.e.bias, n0 + i, p.e.bias_bf16);
          } else {
            for (int i = 0; i < 32; ++i)
              if (n0 + i < p.e.N) v[i] += ldv(p.e.bias, n0 + i, p.e.bias_bf16);
          }
        }
        if (mul) {
          const int ci = (c - half) / SPLIT;  // this warp's chunk index within the tile
          if constexpr (AUX == 2) {
            // a give-up leaves the slot's load waited for; the chunk is then not stored
            const bool got = __all_sync(0xffffffffu, ptx::mbar_wait(&auxbar[2 * ew + (ci & 1)], ring_phase[ci & 1]));
            ring_phase[ci & 1] ^= 1u;
            if (!got) {
              abort_flag = 1;
              if (ci + 1 < my_chunks) {  // the other slot's load is in flight
                ptx::mbar_wait(&auxbar[2 * ew + ((ci + 1) & 1)], ring_phase[(ci + 1) & 1]);
                ring_phase[(ci + 1) & 1] ^= 1u;
              }
              break;
            }
          }
          const uint8_t* ar = auxs + (AUX == 2 ? (ci & 1) : ci) * Cfg::CHUNK_BF16 + lane * 64;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint4 raw = *reinterpret_cast<const uint4*>(ar + ((j ^ ((lane >> 1) & 3)) << 4));
            const bf16* h = reinterpret_cast<const bf16*>(&raw);
#pragma unroll
            for (int i = 0; i < 8; ++i) v[j * 8 + i] *= __bfloat162float(h[i]);
          }
          if constexpr (AUX == 2) {
            __syncwarp();  // every lane has read the slot: refill it with chunk ci + 2
            if (lane == 0 && ci + 2 < my_chunks) ring_load(ci + 2);
          }
        }
        // the staging chunk's previous TMA has read it
        if (lane == 0) {
          if constexpr (Cfg::NSTG == 2)
            ptx::bulk_wait_read<1>();
          else
            ptx::bulk_wait_read<0>();
        }
        __syncwarp();
        uint8_t* sb = stg + sbuf * (gelu ? 2 * Cfg::CHUNK_BF16 : chunk_bytes);
        if (gelu) {
          uint8_t* row_d = sb + lane * 64;
          uint8_t* row_g = sb + Cfg::CHUNK_BF16 + lane * 64;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            uint4 rd, rg;
            __nv_bfloat162* hd = reinterpret_cast<__nv_bfloat162*>(&rd);
            __nv_bfloat162* hg = reinterpret_cast<__nv_bfloat162*>(&rg);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              float g0, d0, g1, d1;
              gelu_tanh_both_approx(v[8 * j + 2 * i], g0, d0);
              gelu_tanh_both_approx(v[8 * j + 2 * i + 1], g1, d1);
              hd[i] = __floats2bfloat162_rn(d0, d1);
              hg[i] = __floats2bfloat162_rn(g0, g1);
            }
            const int off = (j ^ ((lane >> 1) & 3)) << 4;
            if (gelu_d) *reinterpret_cast<uint4*>(row_d + off) = rd;
            *reinterpret_cast<uint4*>(row_g + off) = rg;
          }
        } else if (out_f32) {
          uint8_t* row = sb + lane * 128;
#pragma unroll
          for (int j = 0; j < 8; ++j)
            *reinterpret_cast<float4*>(row + ((j ^ (lane & 7)) << 4)) =
                make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
        } else {
          uint8_t* row = sb + lane * 64;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            uint4 raw;
            __nv_bfloat162* h2 = reinterpret_cast<__nv_bfloat162*>(&raw);
#pragma unroll
            for (int i = 0; i < 4; ++i) h2[i] = __floats2bfloat162_rn(v[8 * j + 2 * i], v[8 * j + 2 * i + 1]);
            *reinterpret_cast<uint4*>(row + ((j ^ ((lane >> 1) & 3)) << 4)) = raw;
          }
        }
        ptx::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          if (p.staged == STAGED_ACCUM) {
            ptx::tma_reduce_add_2d(&tmC, sb, n0, m0);
          } else if (gelu) {
            if (gelu_d) ptx::tma_store_2d(&tmC, sb, n0, m0);
            ptx::tma_store_2d(&tmX, sb + Cfg::CHUNK_BF16, n0, m0);
          } else {
            ptx::tma_store_2d(&tmC, sb, n0, m0);
          }
          ptx::bulk_commit();
        }
        sbuf = (sbuf + 1) % Cfg::NSTG;
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(&tempty[acc]);
      if (++acc == 2) { acc = 0; acc_phase ^= 1; }
    }
    if (lane == 0) ptx::bulk_wait<0>();
    __syncwarp();
  } else {
    // ---------------- epilogue warps 2..9: TMEM lanes 32*(warp%4) .. +31, alternate chunks
    const int q = warp & 3, half = (warp - 2) >> 2;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
      int tm, tn, ks;
      decode(t, tm, tn, ks);
      bool ok = ptx::mbar_wait(&tfull[acc], acc_phase);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) { abort_flag = 1; break; }
      ptx::tc_fence_after();
      const int m = tm * TC_BM + q * 32 + lane;
#pragma unroll 1
      for (int c = half; c < BN / 32; c += SPLIT) {
        uint32_t r[32];
        ptx::tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(q * 32) << 16) + acc * BN + c * 32, r);
        ptx::tmem_ld_wait();
        const int n0 = tn * BN + c * 32;
        if (m < p.e.M && n0 < p.e.N) {
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            float v[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[j * 8 + i]);
            epi_apply8(p.e, m, n0 + j * 8, v);
          }
        }
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(&tempty[acc]);
      if (++acc == 2) { acc = 0; acc_phase ^= 1; }
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
  }
}

// ------------------------------------------------------------------ SIMT kernel
struct SimtParams {
  int M, N, K, splits, kb_total;
  const void* A;
  int64_t lda;
  int a_mn, a_bf16;
  const void* B;
  int64_t ldb;
  int b_mn, b_bf16;
  EpiParams e;
};

template <int BM, int BN>
__global__ void __launch_bounds__(256) gemm_simt_kernel(SimtParams p) {
  constexpr int BK = 16;
  constexpr int TM = BM / 16, TN = BN / 16;
  __shared__ float As[BK][BM + 1];
  __shared__ float Bs[BK][BN + 1];
  const int tid = threadIdx.x;
  const int tx = tid % 16, ty = tid / 16;
  const int tiles_m = (p.M + BM - 1) / BM;
  const int tm = blockIdx.x % tiles_m, tn = blockIdx.x / tiles_m;
  const int m0 = tm * BM, n0 = tn * BN;
  const int ks = blockIdx.y;
  const int kb0 = (int)((long long)p.kb_total * ks / p.splits);
  const int kb1 = (int)((long long)p.kb_total * (ks + 1) / p.splits);
  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;

  for (int kb = kb0; kb < kb1; ++kb) {
    const int k0 = kb * BK;
    for (int idx = tid; idx < BM * BK; idx += 256) {
      int mm, kk;
      if (p.a_mn) { mm = idx % BM; kk = idx / BM; } else { kk = idx % BK; mm = idx / BK; }
      const int m = m0 + mm, k = k0 + kk;
      float v = 0.f;
      if (m < p.M && k < p.K)
        v = ldv(p.A, p.a_mn ? (int64_t)k * p.lda + m : (int64_t)m * p.lda + k, p.a_bf16);
      As[kk][mm] = v;
    }
    for (int idx = tid; idx < BN * BK; idx += 256) {
      int nn, kk;
      if (p.b_mn) { nn = idx % BN; kk = idx / BN; } else { kk = idx % BK; nn = idx / BK; }
      const int n = n0 + nn, k = k0 + kk;
      float v = 0.f;
      if (n < p.N && k < p.K)
        v = ldv(p.B, p.b_mn ? (int64_t)k * p.ldb + n : (int64_t)n * p.ldb + k, p.b_bf16);
      Bs[kk][nn] = v;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      float a[TM], b[TN];
#pragma unroll
      for (int i = 0; i < TM; ++i) a[i] = As[kk][ty + 16 * i];
#pragma unroll
      for (int j = 0; j < TN; ++j) b[j] = Bs[kk][tx + 16 * j];
#pragma unroll
      for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int m = m0 + ty + 16 * i, n = n0 + tx + 16 * j;
      if (m < p.M && n < p.N) epi_apply1(p.e, m, n, acc[i][j]);
    }
}

// ------------------------------------------------------------------ host side
namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    // the entry point as introduced in CUDA 12.0
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

// 2D tensor map over a row-major [rows, cols] matrix with row pitch `ld` elements (bf16,
// or f32 when `f32`), boxes of box_rows x box_cols, the given shared-memory swizzle.
int make_tmap(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, int64_t ld, int box_cols, int box_rows,
              bool f32 = false, CUtensorMapSwizzle swz = CU_TENSOR_MAP_SWIZZLE_128B) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) {
    set_last_error("cuTensorMapEncodeTiled is not available from the driver");
    return JAGG_ERR_CUDA;
  }
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)(ld * (f32 ? 4 : 2))};
  cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                  const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_last_error("cuTensorMapEncodeTiled failed (%d) rows=%lld cols=%lld ld=%lld box=%dx%d", (int)r,
                   (long long)rows, (long long)cols, (long long)ld, box_rows, box_cols);
    return JAGG_ERR_CUDA;
  }
  return JAGG_OK;
}

EpiParams make_epi(const GemmArgs& g) {
  EpiParams e;
  e.M = g.M;
  e.N = g.N;
  e.epi = g.epi;
  e.bias = g.bias;
  e.bias_bf16 = g.bias_dtype == JAGG_DTYPE_BF16;
  e.C = g.C;
  e.ldc = g.ldc;
  e.c_bf16 = g.c_dtype == JAGG_DTYPE_BF16;
  e.C2 = g.C2;
  e.ldc2 = g.ldc2;
  e.aux = g.aux;
  e.ld_aux = g.ld_aux;
  e.gate = g.gate;
  e.gate_stride = g.gate_stride;
  e.rows_per_seq = g.rows_per_seq > 0 ? g.rows_per_seq : 1;
  e.remap_rows = g.remap_rows;
  e.remap_offset = g.remap_offset;
  e.remap_stride = g.remap_stride;
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
  bool ok = (g.N % 8 == 0) && (g.ldc % 8 == 0) && al16(g.C);
  if (g.bias) ok = ok && al16(g.bias);
  if (g.epi == EPI_GELU || g.epi == EPI_GATE_RESID) ok = ok && (g.ldc2 % 8 == 0) && al16(g.C2);
  if (g.epi == EPI_GATE_RESID || g.epi == EPI_MUL_AUX) ok = ok && (g.ld_aux % 8 == 0) && al16(g.aux);
  e.c_trans = g.c_trans ? 1 : 0;
  e.bias_m = g.bias_m ? 1 : 0;
  if (g.c_trans || g.bias_m) ok = false;  // per-element path for transposed outputs
  e.vec_ok = ok ? 1 : 0;
  return e;
}

// Split-K factor of an accumulating product (the partial sums meet in the f32 output through
// reduce-adds): the split count with the fewest waves of units times k-blocks per unit, each
// unit charged two k-blocks for its pipeline fill and epilogue.  Products with few tiles and a
// long K (the weight gradients, K = rows) split so that their units fill whole waves.
int choose_splits(const GemmArgs& g, int BN, int nsm) {
  if (g.epi != EPI_ACCUM) return 1;
  const int k_blocks = ceil_div(g.K, TC_BK);
  if (g.split_k > 0) return g.split_k < k_blocks ? g.split_k : k_blocks;
  const long long tiles = (long long)ceil_div(g.M, TC_BM) * ceil_div(g.N, BN);
  int best = 1;
  double best_cost = 0.0;
  for (int s = 1; s <= k_blocks && s <= 32; ++s) {
    const double waves = (double)((tiles * s + nsm - 1) / nsm);
    const double cost = waves * (ceil_div(k_blocks, s) + 2.0);
    if (s == 1 || cost < 0.999 * best_cost) {
      best = s;
      best_cost = cost;
    }
  }
  return best;
}

// Relative duration of the product with BN-wide tiles: waves of work units times the
// work per unit, over the tile's relative efficiency (FLOP per byte of operand traffic).
double tile_cost(const GemmArgs& g, int BN, int nsm) {
  const int splits = choose_splits(g, BN, nsm);
  const long long units = (long long)ceil_div(g.M, TC_BM) * ceil_div(g.N, BN) * splits;
  const double waves = (double)((units + nsm - 1) / nsm);
  const double eff = BN >= 256 ? 1.33 : 1.0;
  return waves * BN * ((double)ceil_div(g.K, TC_BK) / splits) / eff;
}

// Tile order.  The CTAs resident at one time work on consecutive tile indices, so the
// operand panel that those tiles share is read from DRAM once and from L2 after that.  With
// N fastest, tiles_n neighbours share one 128-row panel of A; with M fastest, tiles_m
// neighbours share one panel of B.  Sharing the panel of the larger operand saves the
// more DRAM traffic: the tall products (rows x d outputs, A = activations) walk N first.
int tile_order_n_first(const GemmArgs& g) { return (long long)g.M > (long long)g.N ? 1 : 0; }

// Which staged epilogue (if any) serves the product: row-major outputs without row remap,
// 16-byte aligned with 16-byte row pitches.
int staged_mode(const GemmArgs& g) {
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
  if (g.c_trans || g.bias_m || (g.C && !al16(g.C))) return STAGED_NONE;
  if (g.epi == EPI_GELU && !g.remap_rows && g.c_dtype == JAGG_DTYPE_BF16 && g.C2 && al16(g.C2) &&
      g.ldc2 % 8 == 0 && (!g.C || g.ldc % 8 == 0) && (!g.bias || al16(g.bias)))
    return STAGED_GELU;
  if (!g.C) return STAGED_NONE;
  if (g.remap_rows || g.epi == EPI_GELU || g.epi == EPI_GATE_RESID) {
    // row-coalesced path: 4-column groups, 16-byte aligned rows of every operand
    bool ok = g.N % 4 == 0 && g.ldc % 4 == 0 && (!g.bias || al16(g.bias));
    if (g.epi == EPI_GELU || g.epi == EPI_GATE_RESID) ok = ok && g.C2 && al16(g.C2) && g.ldc2 % 4 == 0;
    if (g.epi == EPI_GATE_RESID || g.epi == EPI_MUL_AUX) ok = ok && al16(g.aux) && g.ld_aux % 4 == 0;
    if (g.epi == EPI_GATE_RESID) ok = ok && g.gate_stride % 4 == 0 && al16(g.gate);
    return ok ? STAGED_ROWS : STAGED_NONE;
  }
  const bool c_f32 = g.c_dtype == JAGG_DTYPE_F32;
  if ((g.ldc * (c_f32 ? 4 : 2)) % 16) return STAGED_NONE;
  switch (g.epi) {
    case EPI_STORE:
      return (!g.bias || al16(g.bias)) ? STAGED_STORE : STAGED_NONE;
    case EPI_MUL_AUX:
      return (!c_f32 && al16(g.aux) && g.ld_aux % 8 == 0) ? STAGED_MUL_AUX : STAGED_NONE;
    case EPI_ACCUM:
      return c_f32 ? STAGED_ACCUM : STAGED_NONE;
  }
  return STAGED_NONE;
}

int validate(const GemmArgs& g) {
  JAGG_CHECK_ARG(g.M > 0 && g.N > 0 && g.K > 0, "gemm: empty shape %dx%dx%d", g.M, g.N, g.K);
  JAGG_CHECK_ARG(g.A && g.B && (g.C || (g.epi == EPI_GELU && g.C2)), "gemm: null operand");
  JAGG_CHECK_ARG(g.epi >= EPI_STORE && g.epi <= EPI_ACCUM, "gemm: bad epilogue %d", g.epi);
  JAGG_CHECK_ARG(g.epi != EPI_ACCUM || g.c_dtype == JAGG_DTYPE_F32, "gemm: accumulation needs an f32 output");
  JAGG_CHECK_ARG(g.epi != EPI_GELU || g.C2, "gemm: GELU epilogue needs C2");
  JAGG_CHECK_ARG(g.epi != EPI_GATE_RESID || (g.C2 && g.aux && g.gate), "gemm: gate epilogue needs C2/aux/gate");
  JAGG_CHECK_ARG(g.epi != EPI_MUL_AUX || g.aux, "gemm: multiply epilogue needs aux");
  return JAGG_OK;
}

template <int BN, bool A_MN, bool B_MN, int AUX, int EW = 4>
int launch_tc(const GemmArgs& g, cudaStream_t stream) {
  using Cfg = TcCfg<BN, AUX, EW>;
  CUtensorMap ta, tb;
  if (!A_MN)
    JAGG_TRY(make_tmap(&ta, g.A, g.M, g.K, g.lda, TC_BK, TC_BM));
  else
    JAGG_TRY(make_tmap(&ta, g.A, g.K, g.M, g.lda, 64, TC_BK));
  if (!B_MN)
    JAGG_TRY(make_tmap(&tb, g.B, g.N, g.K, g.ldb, TC_BK, BN));
  else
    JAGG_TRY(make_tmap(&tb, g.B, g.K, g.N, g.ldb, 64, TC_BK));
  TcParams p;
  p.staged = staged_mode(g);
  // the row-coalesced epilogue exists in the 8-warp instances only; elsewhere the
  // per-thread epilogue serves those requests
  if ((p.staged == STAGED_ROWS) != (EW == 8)) p.staged = EW == 8 ? STAGED_ROWS : STAGED_NONE;
  CUtensorMap tc = ta, tx = ta;  // unused unless staged through TMA
  if (p.staged != STAGED_NONE && p.staged != STAGED_ROWS && g.C) {
    const bool c_f32 = g.c_dtype == JAGG_DTYPE_F32;
    JAGG_TRY(make_tmap(&tc, g.C, g.M, g.N, g.ldc, 32, 32, c_f32,
                       c_f32 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B));
  }
  if (p.staged == STAGED_GELU)
    JAGG_TRY(make_tmap(&tx, g.C2, g.M, g.N, g.ldc2, 32, 32, false, CU_TENSOR_MAP_SWIZZLE_64B));
  if (p.staged == STAGED_MUL_AUX && !AUX) p.staged = STAGED_NONE;  // no multiplier space
  if (p.staged == STAGED_MUL_AUX)
    JAGG_TRY(make_tmap(&tx, g.aux, g.M, g.N, g.ld_aux, 32, 32, false, CU_TENSOR_MAP_SWIZZLE_64B));
  p.tiles_m = ceil_div(g.M, TC_BM);
  p.tiles_n = ceil_div(g.N, BN);
  p.k_blocks = ceil_div(g.K, TC_BK);
  p.raster_n = tile_order_n_first(g);
  const int nsm = sm_count();
  p.splits = choose_splits(g, BN, nsm);
  p.e = make_epi(g);
  const int total = p.tiles_m * p.tiles_n * p.splits;
  const int grid = total < nsm ? total : nsm;
  static bool attr_set = false;  // one per template instance
  if (!attr_set) {
    JAGG_CUDA_TRY(cudaFuncSetAttribute(gemm_tc_kernel<BN, A_MN, B_MN, AUX, EW>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg::SMEM_BYTES));
    attr_set = true;
  }
  const int tok = prof_start(stream);
  gemm_tc_kernel<BN, A_MN, B_MN, AUX, EW><<<grid, tc_threads(EW), Cfg::SMEM_BYTES, stream>>>(ta, tb, tc, tx, p);
  JAGG_LAUNCHED();
  prof_stop(tok, stream, PROF_GEMM_TC, 2.0 * g.M * g.N * g.K,
            2.0 * ((double)g.M * g.K + (double)g.N * g.K) + (double)g.M * g.N * (g.c_dtype == JAGG_DTYPE_F32 ? 4 : 2),
            g.M, g.N, g.K);
  return JAGG_OK;
}

template <bool A_MN, bool B_MN>
int dispatch_bn(const GemmArgs& g, cudaStream_t stream) {
  // The multiplier epilogue needs its own shared memory: the input-gradient instance
  // (K-major A, MN-major B), with every chunk of a warp's tile (BN <= 128) or a two-slot
  // ring (BN = 256).
  JAGG_CHECK_ARG(g.tile_n == 0 || g.tile_n == 64 || g.tile_n == 128 || g.tile_n == 256, "gemm: tile width %d",
                 g.tile_n);
  if constexpr (!A_MN && B_MN) {
    if (staged_mode(g) == STAGED_MUL_AUX) {
      if (g.tile_n == 64 || (g.tile_n == 0 && g.N < 128)) return launch_tc<64, A_MN, B_MN, 1>(g, stream);
      // 256-column tiles with the multiplier ring when K is long enough for the next tile's
      // main loop (K / 64 k-blocks) to cover the epilogue's chunk loads
      if (g.tile_n == 256 || (g.tile_n == 0 && g.N >= 256 && g.K >= 2048)) return launch_tc<256, A_MN, B_MN, 2>(g, stream);
      return launch_tc<128, A_MN, B_MN, 1>(g, stream);
    }
  }
  if constexpr (!A_MN && !B_MN) {
    // the forward products' arithmetic-heavy epilogues (GELU, gated residual) on 8 warps
    if (staged_mode(g) == STAGED_ROWS) {
      const int nsm = sm_count();
      if (g.tile_n == 64 || (g.tile_n == 0 && g.N < 128)) return launch_tc<64, false, false, 0, 8>(g, stream);
      if (g.tile_n == 128) return launch_tc<128, false, false, 0, 8>(g, stream);
      if (g.tile_n == 256 || (g.tile_n == 0 && g.N >= 256 && tile_cost(g, 256, nsm) < tile_cost(g, 128, nsm)))
        return launch_tc<256, false, false, 0, 8>(g, stream);
      return launch_tc<128, false, false, 0, 8>(g, stream);
    }
  }
  if (g.tile_n == 64 || (g.tile_n == 0 && g.N < 128)) return launch_tc<64, A_MN, B_MN, 0>(g, stream);
  if (g.tile_n == 128) return launch_tc<128, A_MN, B_MN, 0>(g, stream);
  if (g.tile_n == 256) return launch_tc<256, A_MN, B_MN, 0>(g, stream);
  // Wider tiles halve the B-operand traffic per FLOP (the products are bound by L2
  // bandwidth at 128 x 128), at the price of coarser waves over the SMs.
  const int nsm = sm_count();
  if (g.N >= 256 && tile_cost(g, 256, nsm) < tile_cost(g, 128, nsm)) return launch_tc<256, A_MN, B_MN, 0>(g, stream);
  return launch_tc<128, A_MN, B_MN, 0>(g, stream);
}

bool tc_eligible(const GemmArgs& g) {
  if (g.a_dtype != JAGG_DTYPE_BF16 || g.b_dtype != JAGG_DTYPE_BF16) return false;
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
  if (!al16(g.A) || !al16(g.B)) return false;
  // Row pitches must be multiples of 16 bytes.  Extents smaller than a tile are fine:
  // TMA fills the part of a box outside the tensor with zeros.
  if (g.lda % 8 || g.ldb % 8) return false;
  return true;
}

}  // namespace

int encode_tmap(CUtensorMap* m, bool f32, int rank, const void* base, const uint64_t* dims, const uint64_t* strides,
                const uint32_t* box, CUtensorMapSwizzle swz) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) {
    set_last_error("cuTensorMapEncodeTiled is not available from the driver");
    return JAGG_ERR_CUDA;
  }
  cuuint64_t d[5], st[4];
  cuuint32_t bx[5], estr[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    bx[i] = box[i];
    estr[i] = 1;
    if (i + 1 < rank) st[i] = strides[i];
  }
  CUresult r = fn(m, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank,
                  const_cast<void*>(base), d, st, bx, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_last_error("cuTensorMapEncodeTiled failed (%d): rank %d, dims %llu x %llu", (int)r, rank,
                   (unsigned long long)dims[0], (unsigned long long)(rank > 1 ? dims[1] : 1));
    return JAGG_ERR_CUDA;
  }
  return JAGG_OK;
}

int gemm_simt(const GemmArgs& g, cudaStream_t stream) {
  JAGG_TRY(validate(g));
  SimtParams p;
  p.M = g.M; p.N = g.N; p.K = g.K;
  p.A = g.A; p.lda = g.lda; p.a_mn = g.a_mn; p.a_bf16 = g.a_dtype == JAGG_DTYPE_BF16;
  p.B = g.B; p.ldb = g.ldb; p.b_mn = g.b_mn; p.b_bf16 = g.b_dtype == JAGG_DTYPE_BF16;
  p.e = make_epi(g);
  p.e.vec_ok = 0;
  const bool skinny = g.M <= 16;
  const int BM = skinny ? 16 : 64, BN = 64;
  const int tiles = ceil_div(g.M, BM) * ceil_div(g.N, BN);
  p.kb_total = ceil_div(g.K, 16);
  int splits = 1;
  if (g.epi == EPI_ACCUM) {
    const int nsm = sm_count();
    if (g.split_k > 0)
      splits = g.split_k;
    else if (tiles < 2 * nsm)
      splits = (2 * nsm + tiles - 1) / tiles;
    if (splits > p.kb_total) splits = p.kb_total;
    if (splits > 65535) splits = 65535;
  }
  p.splits = splits;
  dim3 grid(tiles, splits);
  const int tok = prof_start(stream);
  if (skinny)
    gemm_simt_kernel<16, 64><<<grid, 256, 0, stream>>>(p);
  else
    gemm_simt_kernel<64, 64><<<grid, 256, 0, stream>>>(p);
  JAGG_LAUNCHED();
  prof_stop(tok, stream, PROF_GEMM_SIMT, 2.0 * g.M * g.N * g.K, 0.0, g.M, g.N, g.K);
  return JAGG_OK;
}

int gemm(const GemmArgs& g, cudaStream_t stream) {
  JAGG_TRY(validate(g));
  if (!tc_eligible(g)) return gemm_simt(g, stream);
  if (!g.a_mn && !g.b_mn) return dispatch_bn<false, false>(g, stream);
  if (!g.a_mn && g.b_mn) return dispatch_bn<false, true>(g, stream);
  if (g.a_mn && g.b_mn) return dispatch_bn<true, true>(g, stream);
  return dispatch_bn<true, false>(g, stream);
}

}  // namespace jagg
