// The backbone's forward (Phase 1) and parameter VJP (Phase 4) as sequences of the
// library's kernels, the parameter table, the saved-activation arena and the C ABI of
// the model entry points.
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "attention.cuh"
#include "elementwise.cuh"
#include "gemm.cuh"

namespace jagg {

// ------------------------------------------------------------------ host errors
namespace {
thread_local char g_err[512] = "";
}
void set_last_error(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
}
int cuda_status(cudaError_t e, const char* where) {
  set_last_error("CUDA error %d (%s) at %s", (int)e, cudaGetErrorString(e), where);
  return JAGG_ERR_CUDA;
}
int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 148;
  return n;
}

// ------------------------------------------------------------------ parameter table
struct TensorInfo {
  std::string name;
  int64_t off, rows, cols;
};

struct DitBlockW {
  int64_t qkv_w, qkv_b, proj_w, proj_b, fc1_w, fc1_b, fc2_w, fc2_b;
  int64_t mod_col;  // offset of this block's segment inside the stacked modulation output
};

// One stream (text or image) of an MMDiT double block.
struct StreamW {
  int64_t qkv_w, qkv_b, qn, kn, proj_w, proj_b, fc1_w, fc1_b, fc2_w, fc2_b;
  int64_t mod_col;
};
struct DoubleW {
  StreamW s[2];  // 0 = text, 1 = image
};
// Flux-style single block: lin1 -> [qkv | u], lin2 on [o | GELU(u)].
struct SingleW {
  int64_t lin1_w, lin1_b, qn, kn, lin2_w, lin2_b;
  int64_t mod_col;
};

struct ParamTable {
  std::vector<TensorInfo> t;
  int64_t total = 0;
  int64_t x_w, x_b, txt_w, txt_b, t_w1, t_b1, t_w2, t_b2;
  int64_t mod_w, mod_b;  // stacked modulation weights [Lmod, d] and biases [Lmod]
  int64_t Lmod = 0;
  int64_t final_mod_col;
  int64_t out_w, out_b;
  std::vector<DitBlockW> blocks;
  std::vector<DoubleW> doubles;
  std::vector<SingleW> singles;
};

static int64_t align64(int64_t x) { return (x + 63) / 64 * 64; }

static bool build_table(const jagg_config& c, ParamTable& T) {
  const int64_t d = c.hidden, dm = c.mlp, pd = (int64_t)c.in_channels * c.patch * c.patch;
  T = ParamTable();
  auto add = [&](const std::string& n, int64_t rows, int64_t cols) {
    T.total = align64(T.total);
    T.t.push_back({n, T.total, rows, cols});
    T.total += rows * cols;
    return T.t.back().off;
  };
  T.x_w = add("x_embed.w", d, pd);
  T.x_b = add("x_embed.b", d, 1);
  T.txt_w = add("txt_embed.w", d, c.txt_dim);
  T.txt_b = add("txt_embed.b", d, 1);
  T.t_w1 = add("t_embed.w1", d, c.freq_dim);
  T.t_b1 = add("t_embed.b1", d, 1);
  T.t_w2 = add("t_embed.w2", d, d);
  T.t_b2 = add("t_embed.b2", d, 1);
  const bool mm = c.arch == JAGG_ARCH_MMDIT;
  const int64_t dh = c.hidden / c.heads;
  // stacked modulation: every block's rows (DiT: [6d, d]; MMDiT: [6d, d] per stream of a
  // double block, [3d, d] per single block), then the final layer's [2d, d]
  std::vector<std::string> mods;
  std::vector<int64_t> mrows;
  if (!mm) {
    for (int i = 0; i < c.depth; ++i) {
      mods.push_back("blocks." + std::to_string(i) + ".mod");
      mrows.push_back(6 * d);
    }
  } else {
    for (int i = 0; i < c.depth_double; ++i)
      for (const char* s : {"txt", "img"}) {
        mods.push_back("double." + std::to_string(i) + "." + s + ".mod");
        mrows.push_back(6 * d);
      }
    for (int i = 0; i < c.depth; ++i) {
      mods.push_back("single." + std::to_string(i) + ".mod");
      mrows.push_back(3 * d);
    }
  }
  mods.push_back("final.mod");
  mrows.push_back(2 * d);
  int64_t col = 0;
  std::vector<int64_t> mcol;
  for (size_t i = 0; i < mods.size(); ++i) {
    const int64_t o = add(mods[i] + ".w", mrows[i], d);
    if (i == 0) T.mod_w = o;
    mcol.push_back(col);
    col += mrows[i];
  }
  T.Lmod = col;
  for (size_t i = 0; i < mods.size(); ++i) {
    const int64_t o = add(mods[i] + ".b", mrows[i], 1);
    if (i == 0) T.mod_b = o;
  }
  T.final_mod_col = mcol.back();
  if (mm) {
    size_t mi = 0;
    for (int i = 0; i < c.depth_double; ++i) {
      DoubleW w;
      for (int si = 0; si < 2; ++si) {
        const std::string p = "double." + std::to_string(i) + (si == 0 ? ".txt." : ".img.");
        StreamW& s = w.s[si];
        s.mod_col = mcol[mi++];
        s.qkv_w = add(p + "qkv.w", 3 * d, d);
        s.qkv_b = add(p + "qkv.b", 3 * d, 1);
        s.qn = add(p + "q_norm", dh, 1);
        s.kn = add(p + "k_norm", dh, 1);
        s.proj_w = add(p + "proj.w", d, d);
        s.proj_b = add(p + "proj.b", d, 1);
        s.fc1_w = add(p + "fc1.w", dm, d);
        s.fc1_b = add(p + "fc1.b", dm, 1);
        s.fc2_w = add(p + "fc2.w", d, dm);
        s.fc2_b = add(p + "fc2.b", d, 1);
      }
      T.doubles.push_back(w);
    }
    for (int i = 0; i < c.depth; ++i) {
      const std::string p = "single." + std::to_string(i) + ".";
      SingleW w;
      w.mod_col = mcol[mi++];
      w.lin1_w = add(p + "lin1.w", 3 * d + dm, d);
      w.lin1_b = add(p + "lin1.b", 3 * d + dm, 1);
      w.qn = add(p + "q_norm", dh, 1);
      w.kn = add(p + "k_norm", dh, 1);
      w.lin2_w = add(p + "lin2.w", d, d + dm);
      w.lin2_b = add(p + "lin2.b", d, 1);
      T.singles.push_back(w);
    }
  }
  for (int i = 0; i < (mm ? 0 : c.depth); ++i) {
    const std::string p = "blocks." + std::to_string(i) + ".";
    DitBlockW w;
    w.mod_col = mcol[i];
    w.qkv_w = add(p + "qkv.w", 3 * d, d);
    w.qkv_b = add(p + "qkv.b", 3 * d, 1);
    w.proj_w = add(p + "proj.w", d, d);
    w.proj_b = add(p + "proj.b", d, 1);
    w.fc1_w = add(p + "fc1.w", dm, d);
    w.fc1_b = add(p + "fc1.b", dm, 1);
    w.fc2_w = add(p + "fc2.w", d, dm);
    w.fc2_b = add(p + "fc2.b", d, 1);
    T.blocks.push_back(w);
  }
  T.out_w = add("final.out.w", pd, d);
  T.out_b = add("final.out.b", pd, 1);
  T.total = align64(T.total);
  return true;
}

static int check_config(const jagg_config* c) {
  JAGG_CHECK_ARG(c, "null config");
  JAGG_CHECK_ARG(c->dtype == JAGG_DTYPE_F32 || c->dtype == JAGG_DTYPE_BF16, "bad dtype %d", c->dtype);
  JAGG_CHECK_ARG(c->hidden > 0 && c->heads > 0 && c->hidden % c->heads == 0, "hidden %d / heads %d", c->hidden,
                 c->heads);
  JAGG_CHECK_ARG(c->hidden % 64 == 0 && c->mlp % 64 == 0, "hidden and mlp must be multiples of 64");
  JAGG_CHECK_ARG(c->hidden <= 3072, "hidden %d above 3072", c->hidden);
  JAGG_CHECK_ARG(c->patch > 0 && c->latent_h % c->patch == 0 && c->latent_w % c->patch == 0,
                 "latent %dx%d not divisible by patch %d", c->latent_h, c->latent_w, c->patch);
  JAGG_CHECK_ARG(c->in_channels > 0 && c->txt_len > 0 && c->txt_dim > 0 && c->txt_dim % 8 == 0,
                 "bad channels / text shape");
  JAGG_CHECK_ARG(c->freq_dim > 0 && c->freq_dim % 2 == 0, "bad freq_dim");
  JAGG_CHECK_ARG(c->depth >= 0 && c->depth_double >= 0, "negative depth");
  const int dh = c->hidden / c->heads;
  JAGG_CHECK_ARG(dh == 16 || dh == 32 || dh == 64 || dh == 128, "head dim %d unsupported", dh);
  JAGG_CHECK_ARG(c->dtype == JAGG_DTYPE_F32 || dh >= 64, "bf16 needs head dim 64 or 128");
  if (c->arch != JAGG_ARCH_DIT) {
    set_last_error("arch %d not implemented in this build", c->arch);
    return JAGG_ERR_UNSUPPORTED;
  }
  return JAGG_OK;
}

}  // namespace jagg

using namespace jagg;

struct jagg_model {
  jagg_config cfg;
  const void* w;
  ParamTable T;
  int d, dm, heads, dh, pd, Ni, Nt, N, gh, gw;
  size_t esz;  // bytes per storage element
};

namespace jagg {
namespace {

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct Carver {
  uint8_t* base;
  size_t off = 0;
  explicit Carver(void* b) : base(static_cast<uint8_t*>(b)) {}
  void* take(size_t bytes) {
    off = align256(off);
    void* p = base ? base + off : nullptr;
    off += bytes;
    return p;
  }
  float* f32(int64_t n) { return static_cast<float*>(take((size_t)n * 4)); }
};

// Per-block saved activations (single-stream DiT block).
struct DitSaved {
  float* h_in;   // [M, d] block input (residual stream)
  void* a;       // [M, d] LN1 + modulation
  void* qkv;     // [M, 3d]
  void* o;       // [M, d] attention output
  float* lse;    // [B, heads, N]
  void* y1;      // [M, d] proj output (before the gate)
  float* h_mid;  // [M, d]
  void* m;       // [M, d] LN2 + modulation
  void* gp;      // [M, dm] GELU'(u) at the fc1 output u (all the backward needs of u)
  void* gu;      // [M, dm] GELU(u)
  void* y2;      // [M, d] fc2 output (before the gate)
  float* st1;    // [2, M] mean, rstd of LN1
  float* st2;
};

struct Saved {
  void* xp;      // [B*Ni, pd]
  void* txt;     // [B*Nt, txt_dim]
  float* phi;    // [B, freq]
  void* phi_b;   // [B, freq] storage type
  void* se1_b;   // [B, d] silu(e1), storage type
  float* e1;     // [B, d]
  float* se1;    // [B, d] silu(e1)
  float* c;      // [B, d]
  float* sc;     // [B, d] silu(c)
  void* sc_b;    // [B, d] silu(c) in the storage type (operand of the modulation products)
  float* mod;    // [B, Lmod]
  std::vector<DitSaved> blk;
  float* h_fin;  // [M, d]
  float* st_f;   // [2, B*Ni]
  void* mf;      // [B*Ni, d]
};

void carve_block(Carver& cv, const jagg_model& m, int B, DitSaved& s) {
  const int64_t M = (int64_t)B * m.N;
  const size_t e = m.esz;
  s.h_in = cv.f32(M * m.d);
  s.a = cv.take(M * m.d * e);
  s.qkv = cv.take(M * 3 * m.d * e);
  s.o = cv.take(M * m.d * e);
  s.lse = cv.f32((int64_t)B * m.heads * m.N);
  s.y1 = cv.take(M * m.d * e);
  s.h_mid = cv.f32(M * m.d);
  s.m = cv.take(M * m.d * e);
  s.gp = cv.take(M * m.dm * e);
  s.gu = cv.take(M * m.dm * e);
  s.y2 = cv.take(M * m.d * e);
  s.st1 = cv.f32(2 * M);
  s.st2 = cv.f32(2 * M);
}

// save == true: every block gets its own slots (the saved arena).  save == false: one set
// of block slots reused by every block (a forward that keeps nothing).
size_t carve_saved(const jagg_model& m, int B, void* base, bool save, Saved& s) {
  Carver cv(base);
  const int64_t M = (int64_t)B * m.N, Mi = (int64_t)B * m.Ni, Mt = (int64_t)B * m.Nt;
  s.xp = cv.take(Mi * m.pd * m.esz);
  s.txt = cv.take(Mt * m.cfg.txt_dim * m.esz);
  s.phi = cv.f32((int64_t)B * m.cfg.freq_dim);
  s.phi_b = cv.take((size_t)B * m.cfg.freq_dim * m.esz);
  s.se1_b = cv.take((size_t)B * m.d * m.esz);
  s.e1 = cv.f32((int64_t)B * m.d);
  s.se1 = cv.f32((int64_t)B * m.d);
  s.c = cv.f32((int64_t)B * m.d);
  s.sc = cv.f32((int64_t)B * m.d);
  s.sc_b = cv.take((size_t)B * m.d * m.esz);
  s.mod = cv.f32((int64_t)B * m.T.Lmod);
  const int L = m.cfg.depth;
  s.blk.assign(L, DitSaved());
  if (save) {
    for (int l = 0; l < L; ++l) carve_block(cv, m, B, s.blk[l]);
    s.h_fin = cv.f32(M * m.d);
  } else {
    DitSaved one;
    carve_block(cv, m, B, one);
    float* h_other = cv.f32(M * m.d);
    for (int l = 0; l < L; ++l) {
      s.blk[l] = one;
      // ping-pong the residual stream between two buffers
      s.blk[l].h_in = (l % 2 == 0) ? one.h_in : h_other;
    }
    s.h_fin = (L % 2 == 0) ? one.h_in : h_other;
  }
  s.st_f = cv.f32(2 * Mi);
  s.mf = cv.take(Mi * m.d * m.esz);
  return align256(cv.off);
}

// Workspace of the VJP.
struct VjpWs {
  float* dh;    // [M, d]
  void* dy;     // [M, d]
  void* du;     // [M, dm]
  float* dx32;  // [M, d] f32 input-gradients feeding LayerNorm backward
  void* dO;     // [M, d]
  void* dqkv;   // [M, 3d]
  float* attn;  // attention scratch
  float* dmod;  // [B, Lmod]
  void* dmod_b;  // [B, Lmod] in the storage type
  void* dvt;    // [B*Ni, pd]
  float* dsc;   // [B, d]
  float* de1;   // [B, d]
  void* dc_b;   // [B, d] storage-type copy of dc, then of de1
  void* dxe;    // [max(Mi, Mt), d] embedding-input gradients in storage type
};

size_t carve_vjp_ws(const jagg_model& m, int B, void* base, VjpWs& w) {
  Carver cv(base);
  const int64_t M = (int64_t)B * m.N, Mi = (int64_t)B * m.Ni, Mt = (int64_t)B * m.Nt;
  const size_t e = m.esz;
  w.dh = cv.f32(M * m.d);
  w.dy = cv.take(M * m.d * e);
  w.du = cv.take(M * m.dm * e);
  w.dx32 = cv.f32(M * m.d);
  w.dO = cv.take(M * m.d * e);
  w.dqkv = cv.take(M * 3 * m.d * e);
  w.attn = cv.f32(attention_bwd_scratch_floats(B, m.N, m.heads, m.dh));
  w.dmod = cv.f32((int64_t)B * m.T.Lmod);
  w.dmod_b = cv.take((size_t)B * m.T.Lmod * m.esz);
  w.dvt = cv.take(Mi * m.pd * e);
  w.dsc = cv.f32((int64_t)B * m.d);
  w.de1 = cv.f32((int64_t)B * m.d);
  w.dc_b = cv.take((size_t)B * m.d * m.esz);
  w.dxe = cv.take((Mi > Mt ? Mi : Mt) * m.d * e);
  return align256(cv.off);
}

// Workspace of the forward: the final layer's token output.
size_t carve_fwd_ws(const jagg_model& m, int B, void* base, void** vt) {
  Carver cv(base);
  *vt = cv.take((int64_t)B * m.Ni * m.pd * m.esz);
  return align256(cv.off);
}

const void* W(const jagg_model& m, int64_t off) { return static_cast<const uint8_t*>(m.w) + off * m.esz; }

// Product helpers ------------------------------------------------------------------
// Y[M, N] = X[M, K] Wt[N, K]^T (+ bias), X K-major in storage type.
GemmArgs fwd_gemm(const jagg_model& m, int M, int N, int K, const void* X, int64_t ldx, int64_t w_off,
                  int64_t b_off) {
  GemmArgs g;
  g.M = M; g.N = N; g.K = K;
  g.A = X; g.lda = ldx; g.a_mn = false; g.a_dtype = m.cfg.dtype;
  g.B = W(m, w_off); g.ldb = K; g.b_mn = false; g.b_dtype = m.cfg.dtype;
  g.bias = b_off >= 0 ? W(m, b_off) : nullptr;
  g.bias_dtype = m.cfg.dtype;
  g.c_dtype = m.cfg.dtype;
  return g;
}
// dX[M, K] = dY[M, N] Wt[N, K]  (Wt stored [N, K] row-major: MN-major operand).
GemmArgs dx_gemm(const jagg_model& m, int M, int N, int K, const void* dY, int64_t ldy, int64_t w_off) {
  GemmArgs g;
  g.M = M; g.N = K; g.K = N;
  g.A = dY; g.lda = ldy; g.a_mn = false; g.a_dtype = m.cfg.dtype;
  g.B = W(m, w_off); g.ldb = K; g.b_mn = true; g.b_dtype = m.cfg.dtype;
  g.c_dtype = m.cfg.dtype;
  return g;
}
// grad[N, K] += dY[M, N]^T X[M, K]  (both MN-major).
GemmArgs dw_gemm(const jagg_model& m, int M, int N, int K, const void* dY, int64_t ldy, const void* X, int64_t ldx,
                 float* grad, int64_t w_off) {
  GemmArgs g;
  g.M = N; g.N = K; g.K = M;
  g.A = dY; g.lda = ldy; g.a_mn = true; g.a_dtype = m.cfg.dtype;
  g.B = X; g.ldb = ldx; g.b_mn = true; g.b_dtype = m.cfg.dtype;
  g.epi = EPI_ACCUM;
  g.C = grad + w_off; g.ldc = K; g.c_dtype = JAGG_DTYPE_F32;
  return g;
}

// Products over the B per-sequence rows (t-embedding MLP, stacked modulation), in the
// transposed form whose M is a feature dimension:
//   rows_gemm: C[B, out] (f32) = X[B, in] W[out, in]^T + b   as  C^T = W X^T
//   rows_dw:   grad[out, in] += dY[B, out]^T X[B, in]        (K = B)
//   rows_dx:   dX[B, in] += dY[B, out] W[out, in]             as  dX^T = W^T dY^T
// X / dY are in the storage type; dX accumulates in f32 (split over out).
GemmArgs rows_gemm(const jagg_model& m, int out, int in, int B, const void* X, int64_t w_off, int64_t b_off,
                   float* C) {
  GemmArgs g;
  g.M = out; g.N = B; g.K = in;
  g.A = W(m, w_off); g.lda = in; g.a_dtype = m.cfg.dtype;
  g.B = X; g.ldb = in; g.b_dtype = m.cfg.dtype;
  g.bias = W(m, b_off); g.bias_dtype = m.cfg.dtype; g.bias_m = true;
  g.C = C; g.ldc = out; g.c_dtype = JAGG_DTYPE_F32; g.c_trans = true;
  return g;
}
GemmArgs rows_dw(const jagg_model& m, int out, int in, int B, const void* dY, const void* X, float* grad,
                 int64_t w_off) {
  GemmArgs g;
  g.M = out; g.N = in; g.K = B;
  g.A = dY; g.lda = out; g.a_mn = true; g.a_dtype = m.cfg.dtype;
  g.B = X; g.ldb = in; g.b_mn = true; g.b_dtype = m.cfg.dtype;
  g.epi = EPI_ACCUM; g.C = grad + w_off; g.ldc = in; g.c_dtype = JAGG_DTYPE_F32;
  return g;
}
GemmArgs rows_dx(const jagg_model& m, int out, int in, int B, const void* dY, int64_t w_off, float* dX) {
  GemmArgs g;
  g.M = in; g.N = B; g.K = out;
  g.A = W(m, w_off); g.lda = in; g.a_mn = true; g.a_dtype = m.cfg.dtype;
  g.B = dY; g.ldb = out; g.b_mn = false; g.b_dtype = m.cfg.dtype;
  g.epi = EPI_ACCUM; g.C = dX; g.ldc = in; g.c_dtype = JAGG_DTYPE_F32; g.c_trans = true;
  return g;
}

int forward_impl(const jagg_model& m, const void* z, const float* t, const void* txt, int B, void* v_out,
                 void* saved, void* ws, cudaStream_t s) {
  const jagg_config& c = m.cfg;
  const int dt = c.dtype;
  const int d = m.d, N = m.N, Ni = m.Ni, Nt = m.Nt;
  const int M = B * N, Mi = B * Ni, Mt = B * Nt;
  const int64_t Lm = m.T.Lmod;
  // With a saved arena every activation goes there; otherwise one block's worth of slots
  // at the start of the workspace is reused by every block.
  Saved S;
  const size_t used = carve_saved(m, B, saved ? saved : ws, saved != nullptr, S);
  void* vt = nullptr;
  carve_fwd_ws(m, B, static_cast<uint8_t*>(ws) + (saved ? 0 : used), &vt);
  float* hstart = S.blk.empty() ? S.h_fin : S.blk[0].h_in;

  // embeddings into the joint [txt; img] residual stream
  JAGG_TRY(launch_patchify(z, dt == JAGG_DTYPE_F32, S.xp, dt == JAGG_DTYPE_F32, dt, B, c.in_channels, c.latent_h,
                           c.latent_w, c.patch, s));
  JAGG_CUDA_TRY(cudaMemcpyAsync(S.txt, txt, (size_t)Mt * c.txt_dim * m.esz, cudaMemcpyDeviceToDevice, s));
  {
    GemmArgs g = fwd_gemm(m, Mi, d, m.pd, S.xp, m.pd, m.T.x_w, m.T.x_b);
    g.C = hstart; g.ldc = d; g.c_dtype = JAGG_DTYPE_F32;
    g.remap_rows = Ni; g.remap_offset = Nt; g.remap_stride = N;
    JAGG_TRY(gemm(g, s));
    GemmArgs gt = fwd_gemm(m, Mt, d, c.txt_dim, S.txt, c.txt_dim, m.T.txt_w, m.T.txt_b);
    gt.C = hstart; gt.ldc = d; gt.c_dtype = JAGG_DTYPE_F32;
    gt.remap_rows = Nt; gt.remap_offset = 0; gt.remap_stride = N;
    JAGG_TRY(gemm(gt, s));
  }
  JAGG_TRY(launch_add_pos_embed(hstart, B, N, Nt, m.gh, m.gw, d, s));
  // t-embedding MLP and every block's modulation (per-sequence rows, f32 activations)
  JAGG_TRY(launch_timestep_embedding(t, S.phi, B, c.freq_dim, s));
  // t-embedding MLP and every block's modulation at once (stacked weights): products
  // with B per-sequence rows, each run as Y^T = W X^T so that the long dimension is M
  JAGG_TRY(launch_gather_rows(S.phi, c.freq_dim, 0, 0, 0, S.phi_b, dt, B, c.freq_dim, s));
  JAGG_TRY(gemm(rows_gemm(m, d, c.freq_dim, B, S.phi_b, m.T.t_w1, m.T.t_b1, S.e1), s));
  JAGG_TRY(launch_silu(S.e1, S.se1, (int64_t)B * d, s));
  JAGG_TRY(launch_gather_rows(S.se1, d, 0, 0, 0, S.se1_b, dt, B, d, s));
  JAGG_TRY(gemm(rows_gemm(m, d, d, B, S.se1_b, m.T.t_w2, m.T.t_b2, S.c), s));
  JAGG_TRY(launch_silu(S.c, S.sc, (int64_t)B * d, s));
  JAGG_TRY(launch_gather_rows(S.sc, d, 0, 0, 0, S.sc_b, dt, B, d, s));
  JAGG_TRY(gemm(rows_gemm(m, (int)Lm, d, B, S.sc_b, m.T.mod_w, m.T.mod_b, S.mod), s));
  // blocks
  for (int l = 0; l < c.depth; ++l) {
    const DitBlockW& bw = m.T.blocks[l];
    const DitSaved& k = S.blk[l];
    float* h_out = (l + 1 < c.depth) ? S.blk[l + 1].h_in : S.h_fin;
    const float* mod = S.mod + bw.mod_col;
    LnModFwd ln{k.h_in, 0, 0, 0, M, d, N, mod, mod + d, Lm, k.a, dt, k.st1, k.st1 + M};
    JAGG_TRY(launch_ln_mod_fwd(ln, s));
    GemmArgs g = fwd_gemm(m, M, 3 * d, d, k.a, d, bw.qkv_w, bw.qkv_b);
    g.C = k.qkv; g.ldc = 3 * d;
    JAGG_TRY(gemm(g, s));
    AttnArgs at;
    at.B = B; at.N = N; at.heads = m.heads; at.dh = m.dh; at.scale = 1.f / sqrtf((float)m.dh);
    at.q = at.k = at.v = seg_single(k.qkv, 3 * d, N);
    at.q_col0 = 0; at.k_col0 = d; at.v_col0 = 2 * d;
    at.o = seg_single(k.o, d, N);
    at.lse = k.lse;
    at.dtype = dt;
    JAGG_TRY(attention_fwd(at, s));
    g = fwd_gemm(m, M, d, d, k.o, d, bw.proj_w, bw.proj_b);
    g.epi = EPI_GATE_RESID; g.C = k.y1; g.ldc = d;
    g.C2 = k.h_mid; g.ldc2 = d; g.aux = k.h_in; g.ld_aux = d;
    g.gate = mod + 2 * d; g.gate_stride = Lm; g.rows_per_seq = N;
    JAGG_TRY(gemm(g, s));
    LnModFwd ln2{k.h_mid, 0, 0, 0, M, d, N, mod + 3 * d, mod + 4 * d, Lm, k.m, dt, k.st2, k.st2 + M};
    JAGG_TRY(launch_ln_mod_fwd(ln2, s));
    g = fwd_gemm(m, M, m.dm, d, k.m, d, bw.fc1_w, bw.fc1_b);
    g.epi = EPI_GELU; g.C = k.gp; g.ldc = m.dm; g.C2 = k.gu; g.ldc2 = m.dm;
    JAGG_TRY(gemm(g, s));
    g = fwd_gemm(m, M, d, m.dm, k.gu, m.dm, bw.fc2_w, bw.fc2_b);
    g.epi = EPI_GATE_RESID; g.C = k.y2; g.ldc = d;
    g.C2 = h_out; g.ldc2 = d; g.aux = k.h_mid; g.ld_aux = d;
    g.gate = mod + 5 * d; g.gate_stride = Lm; g.rows_per_seq = N;
    JAGG_TRY(gemm(g, s));
  }
  // final layer on the image tokens
  const float* fm = S.mod + m.T.final_mod_col;
  LnModFwd lf{S.h_fin, Ni, Nt, N, Mi, d, Ni, fm, fm + d, Lm, S.mf, dt, S.st_f, S.st_f + Mi};
  JAGG_TRY(launch_ln_mod_fwd(lf, s));
  GemmArgs g = fwd_gemm(m, Mi, m.pd, d, S.mf, d, m.T.out_w, m.T.out_b);
  g.C = vt; g.ldc = m.pd;
  JAGG_TRY(gemm(g, s));
  JAGG_TRY(launch_unpatchify(vt, v_out, dt, B, c.in_channels, c.latent_h, c.latent_w, c.patch, s));
  return JAGG_OK;
}

int vjp_impl(const jagg_model& m, const void* saved, int B, const float* cot, float* grad, void* ws,
             cudaStream_t s) {
  const jagg_config& c = m.cfg;
  const int dt = c.dtype;
  const int d = m.d, dmw = m.dm, N = m.N, Ni = m.Ni, Nt = m.Nt;
  const int M = B * N, Mi = B * Ni, Mt = B * Nt;
  const int64_t Lm = m.T.Lmod;
  Saved S;
  carve_saved(m, B, const_cast<void*>(saved), true, S);
  VjpWs w;
  carve_vjp_ws(m, B, ws, w);
  JAGG_CUDA_TRY(cudaMemsetAsync(w.dmod, 0, sizeof(float) * (size_t)B * Lm, s));
  JAGG_CUDA_TRY(cudaMemsetAsync(w.dh, 0, sizeof(float) * (size_t)M * d, s));
  JAGG_CUDA_TRY(cudaMemsetAsync(w.dsc, 0, sizeof(float) * (size_t)B * d, s));
  JAGG_CUDA_TRY(cudaMemsetAsync(w.de1, 0, sizeof(float) * (size_t)B * d, s));

  // final layer
  JAGG_TRY(launch_patchify(cot, 1, w.dvt, dt == JAGG_DTYPE_F32, dt, B, c.in_channels, c.latent_h, c.latent_w,
                           c.patch, s));
  JAGG_TRY(launch_colsum(w.dvt, dt == JAGG_DTYPE_F32, dt, Mi, m.pd, m.pd, grad + m.T.out_b, s));
  JAGG_TRY(gemm(dw_gemm(m, Mi, m.pd, d, w.dvt, m.pd, S.mf, d, grad, m.T.out_w), s));
  {
    GemmArgs g = dx_gemm(m, Mi, m.pd, d, w.dvt, m.pd, m.T.out_w);
    g.C = w.dx32; g.ldc = d; g.c_dtype = JAGG_DTYPE_F32;
    JAGG_TRY(gemm(g, s));
  }
  const float* fm = S.mod + m.T.final_mod_col;
  float* dfm = w.dmod + m.T.final_mod_col;
  {
    LnGateBwd a{};
    a.M = Mi; a.d = d; a.rows_per_seq = Ni;
    a.seg = Ni; a.seg_off = Nt; a.seg_stride = N;
    a.do_ln = 1; a.dm = w.dx32; a.dm_f32 = 1; a.h = S.h_fin; a.mean = S.st_f; a.rstd = S.st_f + Mi;
    a.scale = fm + d; a.mod_stride = Lm; a.dshift = dfm; a.dscale = dfm + d; a.dmod_stride = Lm;
    a.dh_in = w.dh; a.dh_out = w.dh;
    a.dtype = dt;
    JAGG_TRY(launch_ln_gate_bwd(a, s));
  }
  // Gate of block l's MLP branch (dg2, dy2 = g2 dh, db_fc2): for the last block a pass of
  // its own; for the others fused into the LayerNorm-1 backward of block l + 1, which
  // produces exactly that gradient.
  auto mlp_gate = [&](LnGateBwd& a, int l) {
    const DitBlockW& bw = m.T.blocks[l];
    a.do_gate = 1; a.y = S.blk[l].y2; a.gate = S.mod + bw.mod_col + 5 * d; a.mod_stride = Lm;
    a.dgate = w.dmod + bw.mod_col + 5 * d; a.dmod_stride = Lm; a.dy = w.dy; a.dbias = grad + bw.fc2_b;
  };
  if (c.depth > 0) {
    LnGateBwd a{};
    a.M = M; a.d = d; a.rows_per_seq = N;
    a.do_ln = 0; a.dh_in = w.dh; a.dh_out = w.dh; a.dtype = dt;
    mlp_gate(a, c.depth - 1);
    JAGG_TRY(launch_ln_gate_bwd(a, s));
  }
  // blocks, last to first
  for (int l = c.depth - 1; l >= 0; --l) {
    const DitBlockW& bw = m.T.blocks[l];
    const DitSaved& k = S.blk[l];
    const float* mod = S.mod + bw.mod_col;
    float* dmod = w.dmod + bw.mod_col;
    JAGG_TRY(gemm(dw_gemm(m, M, d, dmw, w.dy, d, k.gu, dmw, grad, bw.fc2_w), s));
    {
      GemmArgs g = dx_gemm(m, M, d, dmw, w.dy, d, bw.fc2_w);
      g.epi = EPI_MUL_AUX; g.C = w.du; g.ldc = dmw; g.aux = k.gp; g.ld_aux = dmw;
      JAGG_TRY(gemm(g, s));
    }
    JAGG_TRY(launch_colsum(w.du, dt == JAGG_DTYPE_F32, dt, M, dmw, dmw, grad + bw.fc1_b, s));
    JAGG_TRY(gemm(dw_gemm(m, M, dmw, d, w.du, dmw, k.m, d, grad, bw.fc1_w), s));
    {
      GemmArgs g = dx_gemm(m, M, dmw, d, w.du, dmw, bw.fc1_w);
      g.C = w.dx32; g.ldc = d; g.c_dtype = JAGG_DTYPE_F32;
      JAGG_TRY(gemm(g, s));
    }
    {  // LN2 + modulation backward, then the attention branch's gate
      LnGateBwd a{};
      a.M = M; a.d = d; a.rows_per_seq = N;
      a.do_ln = 1; a.dm = w.dx32; a.dm_f32 = 1; a.h = k.h_mid; a.mean = k.st2; a.rstd = k.st2 + M;
      a.scale = mod + 4 * d; a.mod_stride = Lm; a.dshift = dmod + 3 * d; a.dscale = dmod + 4 * d;
      a.dmod_stride = Lm; a.dh_in = w.dh; a.dh_out = w.dh;
      a.do_gate = 1; a.y = k.y1; a.gate = mod + 2 * d; a.dgate = dmod + 2 * d; a.dy = w.dy;
      a.dbias = grad + bw.proj_b; a.dtype = dt;
      JAGG_TRY(launch_ln_gate_bwd(a, s));
    }
    JAGG_TRY(gemm(dw_gemm(m, M, d, d, w.dy, d, k.o, d, grad, bw.proj_w), s));
    {
      GemmArgs g = dx_gemm(m, M, d, d, w.dy, d, bw.proj_w);
      g.C = w.dO; g.ldc = d;
      JAGG_TRY(gemm(g, s));
    }
    {
      AttnBwdArgs ab;
      AttnArgs& at = ab.f;
      at.B = B; at.N = N; at.heads = m.heads; at.dh = m.dh; at.scale = 1.f / sqrtf((float)m.dh);
      at.q = at.k = at.v = seg_single(k.qkv, 3 * d, N);
      at.q_col0 = 0; at.k_col0 = d; at.v_col0 = 2 * d;
      at.o = seg_single(k.o, d, N);
      at.lse = k.lse; at.dtype = dt;
      ab.dO = seg_single(w.dO, d, N);
      attention_bwd_scratch(w.attn, B, N, m.heads, &ab.Dv, &ab.dq_acc);
      ab.dq = ab.dk = ab.dv = seg_single(w.dqkv, 3 * d, N);
      ab.dq_col0 = 0; ab.dk_col0 = d; ab.dv_col0 = 2 * d;
      JAGG_TRY(attention_bwd(ab, s));
    }
    JAGG_TRY(launch_colsum(w.dqkv, dt == JAGG_DTYPE_F32, dt, M, 3 * d, 3 * d, grad + bw.qkv_b, s));
    JAGG_TRY(gemm(dw_gemm(m, M, 3 * d, d, w.dqkv, 3 * d, k.a, d, grad, bw.qkv_w), s));
    {
      GemmArgs g = dx_gemm(m, M, 3 * d, d, w.dqkv, 3 * d, bw.qkv_w);
      g.C = w.dx32; g.ldc = d; g.c_dtype = JAGG_DTYPE_F32;
      JAGG_TRY(gemm(g, s));
    }
    {  // LN1 + modulation backward, then the previous block's MLP gate
      LnGateBwd a{};
      a.M = M; a.d = d; a.rows_per_seq = N;
      a.do_ln = 1; a.dm = w.dx32; a.dm_f32 = 1; a.h = k.h_in; a.mean = k.st1; a.rstd = k.st1 + M;
      a.scale = mod + d; a.mod_stride = Lm; a.dshift = dmod; a.dscale = dmod + d; a.dmod_stride = Lm;
      a.dh_in = w.dh; a.dh_out = w.dh; a.dtype = dt;
      if (l > 0) mlp_gate(a, l - 1);
      JAGG_TRY(launch_ln_gate_bwd(a, s));
    }
  }
  // input projections (no gradient to z or txt)
  JAGG_TRY(launch_gather_rows(w.dh, d, Ni, Nt, N, w.dxe, dt, Mi, d, s));
  JAGG_TRY(launch_colsum(w.dxe, dt == JAGG_DTYPE_F32, dt, Mi, d, d, grad + m.T.x_b, s));
  JAGG_TRY(gemm(dw_gemm(m, Mi, d, m.pd, w.dxe, d, S.xp, m.pd, grad, m.T.x_w), s));
  JAGG_TRY(launch_gather_rows(w.dh, d, Nt, 0, N, w.dxe, dt, Mt, d, s));
  JAGG_TRY(launch_colsum(w.dxe, dt == JAGG_DTYPE_F32, dt, Mt, d, d, grad + m.T.txt_b, s));
  JAGG_TRY(gemm(dw_gemm(m, Mt, d, c.txt_dim, w.dxe, d, S.txt, c.txt_dim, grad, m.T.txt_w), s));
  // stacked modulation: dW += dmod^T silu(c), db += sum_b dmod, d silu(c) = dmod W
  JAGG_TRY(launch_colsum(w.dmod, 1, dt, B, (int)Lm, Lm, grad + m.T.mod_b, s));
  JAGG_TRY(launch_gather_rows(w.dmod, Lm, 0, 0, 0, w.dmod_b, dt, B, (int)Lm, s));
  JAGG_TRY(gemm(rows_dw(m, (int)Lm, d, B, w.dmod_b, S.sc_b, grad, m.T.mod_w), s));
  JAGG_TRY(gemm(rows_dx(m, (int)Lm, d, B, w.dmod_b, m.T.mod_w, w.dsc), s));  // d silu(c)
  // t-embedding MLP
  JAGG_TRY(launch_mul_silu_grad(w.dsc, S.c, (int64_t)B * d, s));  // dc
  JAGG_TRY(launch_colsum(w.dsc, 1, dt, B, d, d, grad + m.T.t_b2, s));
  JAGG_TRY(launch_gather_rows(w.dsc, d, 0, 0, 0, w.dc_b, dt, B, d, s));
  JAGG_TRY(gemm(rows_dw(m, d, d, B, w.dc_b, S.se1_b, grad, m.T.t_w2), s));
  JAGG_TRY(gemm(rows_dx(m, d, d, B, w.dc_b, m.T.t_w2, w.de1), s));  // d silu(e1)
  JAGG_TRY(launch_mul_silu_grad(w.de1, S.e1, (int64_t)B * d, s));
  JAGG_TRY(launch_colsum(w.de1, 1, dt, B, d, d, grad + m.T.t_b1, s));
  JAGG_TRY(launch_gather_rows(w.de1, d, 0, 0, 0, w.dc_b, dt, B, d, s));
  JAGG_TRY(gemm(rows_dw(m, d, c.freq_dim, B, w.dc_b, S.phi_b, grad, m.T.t_w1), s));
  return JAGG_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

}  // namespace
}  // namespace jagg

// ------------------------------------------------------------------ C ABI
namespace jagg {
const char* last_error_text() { return g_err; }
}  // namespace jagg

extern "C" const char* jagg_last_error(void) { return jagg::last_error_text(); }

extern "C" int jagg_device_status(unsigned* status_out, int clear) {
  JAGG_CHECK_ARG(status_out, "jagg_device_status: null output");
  JAGG_CUDA_TRY(cudaDeviceSynchronize());
  unsigned a = 0, b = 0;
  if (jagg::unit_status_gemm(&a, clear) || jagg::unit_status_signals(&b, clear)) {
    set_last_error("jagg_device_status: reading the status word failed");
    return JAGG_ERR_CUDA;
  }
  *status_out = a | b;
  return JAGG_OK;
}

extern "C" int64_t jagg_param_count(const jagg_config* cfg) {
  if (check_config(cfg) != JAGG_OK) return -1;
  ParamTable T;
  build_table(*cfg, T);
  return T.total;
}

extern "C" int jagg_param_tensor_count(const jagg_config* cfg) {
  if (check_config(cfg) != JAGG_OK) return -1;
  ParamTable T;
  build_table(*cfg, T);
  return (int)T.t.size();
}

extern "C" int jagg_param_info(const jagg_config* cfg, int index, char* name, size_t name_cap, int64_t* offset,
                               int64_t* rows, int64_t* cols) {
  JAGG_TRY(check_config(cfg));
  ParamTable T;
  build_table(*cfg, T);
  JAGG_CHECK_ARG(index >= 0 && index < (int)T.t.size(), "jagg_param_info: index %d out of range", index);
  const TensorInfo& ti = T.t[index];
  if (name && name_cap) {
    strncpy(name, ti.name.c_str(), name_cap - 1);
    name[name_cap - 1] = '\0';
  }
  if (offset) *offset = ti.off;
  if (rows) *rows = ti.rows;
  if (cols) *cols = ti.cols;
  return JAGG_OK;
}

extern "C" int jagg_model_create(const jagg_config* cfg, const void* weights, jagg_model_t* model_out) {
  JAGG_TRY(check_config(cfg));
  JAGG_CHECK_ARG(weights && model_out, "jagg_model_create: null weights or output");
  JAGG_CHECK_ARG(aligned16(weights), "jagg_model_create: weights not 16-byte aligned");
  jagg_model* m = new jagg_model();
  m->cfg = *cfg;
  m->w = weights;
  build_table(*cfg, m->T);
  m->d = cfg->hidden;
  m->dm = cfg->mlp;
  m->heads = cfg->heads;
  m->dh = cfg->hidden / cfg->heads;
  m->pd = cfg->in_channels * cfg->patch * cfg->patch;
  m->gh = cfg->latent_h / cfg->patch;
  m->gw = cfg->latent_w / cfg->patch;
  m->Ni = m->gh * m->gw;
  m->Nt = cfg->txt_len;
  m->N = m->Ni + m->Nt;
  m->esz = cfg->dtype == JAGG_DTYPE_BF16 ? 2 : 4;
  *model_out = m;
  return JAGG_OK;
}

extern "C" int jagg_model_destroy(jagg_model_t model) {
  delete model;
  return JAGG_OK;
}

extern "C" int64_t jagg_saved_bytes(jagg_model_t m, int B) {
  if (!m || B <= 0) return -1;
  Saved S;
  return (int64_t)carve_saved(*m, B, nullptr, true, S);
}

extern "C" int64_t jagg_workspace_bytes(jagg_model_t m, int B) {
  if (!m || B <= 0) return -1;
  Saved S;
  void* vt;
  const size_t fwd = carve_saved(*m, B, nullptr, false, S) + carve_fwd_ws(*m, B, nullptr, &vt);
  VjpWs w;
  const size_t vjp = carve_vjp_ws(*m, B, nullptr, w);
  return (int64_t)(fwd > vjp ? fwd : vjp);
}

static int check_rows(jagg_model_t m, int B) {
  JAGG_CHECK_ARG(m, "null model");
  JAGG_CHECK_ARG(B > 0, "B=%d must be positive", B);
  JAGG_CHECK_ARG((int64_t)B * m->N < (1ll << 31) / 4, "B=%d too large", B);
  return JAGG_OK;
}

extern "C" int dit_forward_save(jagg_model_t m, const void* z, const float* t, const void* txt, int B, void* v_out,
                                void* saved, size_t saved_bytes, void* ws, size_t ws_bytes, cudaStream_t stream) {
  JAGG_TRY(check_rows(m, B));
  JAGG_CHECK_ARG(z && t && txt && v_out && ws, "dit_forward_save: null pointer");
  JAGG_CHECK_ARG(aligned16(z) && aligned16(txt) && aligned16(v_out) && aligned16(ws) && (!saved || aligned16(saved)),
                 "dit_forward_save: buffers must be 16-byte aligned");
  if (saved && (int64_t)saved_bytes < jagg_saved_bytes(m, B)) {
    set_last_error("dit_forward_save: saved arena %zu < %lld bytes", saved_bytes, (long long)jagg_saved_bytes(m, B));
    return JAGG_ERR_WORKSPACE;
  }
  if ((int64_t)ws_bytes < jagg_workspace_bytes(m, B)) {
    set_last_error("dit_forward_save: workspace %zu < %lld bytes", ws_bytes, (long long)jagg_workspace_bytes(m, B));
    return JAGG_ERR_WORKSPACE;
  }
  return forward_impl(*m, z, t, txt, B, v_out, saved, ws, stream);
}

extern "C" int dit_joint_vjp(jagg_model_t m, const void* saved, size_t saved_bytes, int B, const float* cot,
                             float* grad, void* ws, size_t ws_bytes, cudaStream_t stream) {
  JAGG_TRY(check_rows(m, B));
  JAGG_CHECK_ARG(saved && cot && grad && ws, "dit_joint_vjp: null pointer");
  JAGG_CHECK_ARG(aligned16(saved) && aligned16(cot) && aligned16(grad) && aligned16(ws),
                 "dit_joint_vjp: buffers must be 16-byte aligned");
  if ((int64_t)saved_bytes < jagg_saved_bytes(m, B)) {
    set_last_error("dit_joint_vjp: saved arena %zu < %lld bytes for B=%d", saved_bytes,
                   (long long)jagg_saved_bytes(m, B), B);
    return JAGG_ERR_WORKSPACE;
  }
  if ((int64_t)ws_bytes < jagg_workspace_bytes(m, B)) {
    set_last_error("dit_joint_vjp: workspace %zu < %lld bytes", ws_bytes, (long long)jagg_workspace_bytes(m, B));
    return JAGG_ERR_WORKSPACE;
  }
  return vjp_impl(*m, saved, B, cot, grad, ws, stream);
}
