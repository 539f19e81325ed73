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
  JAGG_CHECK_ARG(c->arch == JAGG_ARCH_DIT || c->arch == JAGG_ARCH_MMDIT, "unknown arch %d", c->arch);
  JAGG_CHECK_ARG(c->arch == JAGG_ARCH_MMDIT || c->depth_double == 0, "a DiT has no double blocks");
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
  // MMDiT double-block streams only: q/k after RMSNorm + RoPE and the saved 1/rms
  void* qk = nullptr;    // [M, 2d]
  float* rq = nullptr;   // [M, heads]
  float* rk = nullptr;
};

// An MMDiT double block: the text (0) and image (1) streams, each laid out as a DiT block
// over its own rows, and the joint attention's log-sum-exp.
struct DoubleSaved {
  DitSaved s[2];
  float* lse;  // [B, heads, N]
};

// A Flux-style single block.
struct SingleSaved {
  float* h_in;  // [M, d]
  void* a;      // [M, d] LN + modulation
  float* st1;   // [2, M]
  void* qkv;    // [M, 3d] first 3d outputs of lin1
  void* gp;     // [M, dm] GELU'(u) for the last dm outputs u of lin1
  void* cat;    // [M, d + dm] [attention output | GELU(u)], the input of lin2
  void* qk;     // [M, 2d]
  float* rq;    // [M, heads]
  float* rk;
  float* lse;   // [B, heads, N]
  void* y;      // [M, d] lin2 output (before the gate)
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
  std::vector<DoubleSaved> dbl;
  std::vector<SingleSaved> sgl;
  float* hD[2] = {nullptr, nullptr};  // outputs of the last double block per stream
  float* h_fin;  // [M, d]
  bool keep = true;  // a saving forward; false: nothing is kept, so GELU'(u) is not formed
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

void carve_stream(Carver& cv, const jagg_model& m, int B, int Ns, DitSaved& q) {
  const int64_t Ms = (int64_t)B * Ns;
  const size_t e = m.esz;
  q.h_in = cv.f32(Ms * m.d);
  q.a = cv.take(Ms * m.d * e);
  q.qkv = cv.take(Ms * 3 * m.d * e);
  q.qk = cv.take(Ms * 2 * m.d * e);
  q.rq = cv.f32(Ms * m.heads);
  q.rk = cv.f32(Ms * m.heads);
  q.o = cv.take(Ms * m.d * e);
  q.lse = nullptr;
  q.y1 = cv.take(Ms * m.d * e);
  q.h_mid = cv.f32(Ms * m.d);
  q.m = cv.take(Ms * m.d * e);
  q.gp = cv.take(Ms * m.dm * e);
  q.gu = cv.take(Ms * m.dm * e);
  q.y2 = cv.take(Ms * m.d * e);
  q.st1 = cv.f32(2 * Ms);
  q.st2 = cv.f32(2 * Ms);
}

void carve_double(Carver& cv, const jagg_model& m, int B, DoubleSaved& k) {
  carve_stream(cv, m, B, m.Nt, k.s[0]);
  carve_stream(cv, m, B, m.Ni, k.s[1]);
  k.lse = cv.f32((int64_t)B * m.heads * m.N);
}

void carve_single(Carver& cv, const jagg_model& m, int B, SingleSaved& k) {
  const int64_t M = (int64_t)B * m.N;
  const size_t e = m.esz;
  k.h_in = cv.f32(M * m.d);
  k.a = cv.take(M * m.d * e);
  k.st1 = cv.f32(2 * M);
  k.qkv = cv.take(M * 3 * m.d * e);
  k.gp = cv.take(M * m.dm * e);
  k.cat = cv.take(M * (m.d + m.dm) * e);
  k.qk = cv.take(M * 2 * m.d * e);
  k.rq = cv.f32(M * m.heads);
  k.rk = cv.f32(M * m.heads);
  k.lse = cv.f32((int64_t)B * m.heads * m.N);
  k.y = cv.take(M * m.d * e);
}

// save == true: every block gets its own slots (the saved arena).  save == false: one set
// of block slots reused by every block (a forward that keeps nothing).
size_t carve_saved(const jagg_model& m, int B, void* base, bool save, Saved& s) {
  Carver cv(base);
  const int64_t M = (int64_t)B * m.N, Mi = (int64_t)B * m.Ni, Mt = (int64_t)B * m.Nt;
  s.keep = save;
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
  if (m.cfg.arch == JAGG_ARCH_MMDIT) {
    const int Ld = m.cfg.depth_double, Ls = m.cfg.depth;
    s.blk.clear();
    s.dbl.assign(Ld, DoubleSaved());
    s.sgl.assign(Ls, SingleSaved());
    if (save) {
      for (int l = 0; l < Ld; ++l) carve_double(cv, m, B, s.dbl[l]);
      if (Ld > 0) {
        s.hD[0] = cv.f32(Mt * m.d);
        s.hD[1] = cv.f32(Mi * m.d);
      }
      for (int l = 0; l < Ls; ++l) carve_single(cv, m, B, s.sgl[l]);
      s.h_fin = cv.f32(M * m.d);
    } else {
      // one set of slots per block type; residual streams ping-pong between two buffers
      if (Ld > 0) {
        DoubleSaved one;
        carve_double(cv, m, B, one);
        float* other[2] = {cv.f32(Mt * m.d), cv.f32(Mi * m.d)};
        for (int l = 0; l < Ld; ++l) {
          s.dbl[l] = one;
          for (int si = 0; si < 2; ++si) s.dbl[l].s[si].h_in = (l % 2 == 0) ? one.s[si].h_in : other[si];
        }
        for (int si = 0; si < 2; ++si) s.hD[si] = (Ld % 2 == 0) ? one.s[si].h_in : other[si];
      }
      if (Ls > 0) {
        SingleSaved one;
        carve_single(cv, m, B, one);
        float* other = cv.f32(M * m.d);
        for (int l = 0; l < Ls; ++l) {
          s.sgl[l] = one;
          s.sgl[l].h_in = (l % 2 == 0) ? one.h_in : other;
        }
        s.h_fin = (Ls % 2 == 0) ? one.h_in : other;
      } else {
        s.h_fin = cv.f32(M * m.d);
      }
    }
    s.st_f = cv.f32(2 * Mi);
    s.mf = cv.take(Mi * m.d * m.esz);
    return align256(cv.off);
  }
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
  void* dqkv;   // [M, 3d] (MMDiT: [M, 3d + dm], the gradient of a single block's lin1 output)
  float* dhs[2] = {nullptr, nullptr};  // MMDiT double blocks: per-stream residual gradients
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
  const bool mm = m.cfg.arch == JAGG_ARCH_MMDIT;
  w.dqkv = cv.take(M * (3 * m.d + (mm ? m.dm : 0)) * e);
  if (mm && m.cfg.depth_double > 0) {
    w.dhs[0] = cv.f32(Mt * m.d);
    w.dhs[1] = cv.f32(Mi * m.d);
  }
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
// ldw: row pitch of Wt when the K columns are a slice of a wider matrix (0 = K).
GemmArgs dx_gemm(const jagg_model& m, int M, int N, int K, const void* dY, int64_t ldy, int64_t w_off,
                 int64_t ldw = 0) {
  GemmArgs g;
  g.M = M; g.N = K; g.K = N;
  g.A = dY; g.lda = ldy; g.a_mn = false; g.a_dtype = m.cfg.dtype;
  g.B = W(m, w_off); g.ldb = ldw ? ldw : K; g.b_mn = true; g.b_dtype = m.cfg.dtype;
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

// Products over the B per-sequence rows (t-embedding MLP, stacked modulation).  B is small
// (a few dozen rows: one 128-row tile, the rest of it zero-filled by TMA), and the products
// are bound by reading W, so they keep the plain row-major output with the staged
// epilogues:
//   rows_gemm: C[B, out] (f32) = X[B, in] W[out, in]^T + b
//   rows_dw:   grad[out, in] += dY[B, out]^T X[B, in]        (K = B)
//   rows_dx:   dX[B, in] += dY[B, out] W[out, in]             (split over out)
// X / dY are in the storage type; dX accumulates in f32.
GemmArgs rows_gemm(const jagg_model& m, int out, int in, int B, const void* X, int64_t w_off, int64_t b_off,
                   float* C) {
  GemmArgs g;
  g.M = B; g.N = out; g.K = in;
  g.A = X; g.lda = in; g.a_dtype = m.cfg.dtype;
  g.B = W(m, w_off); g.ldb = in; g.b_dtype = m.cfg.dtype;
  g.bias = W(m, b_off); g.bias_dtype = m.cfg.dtype;
  g.C = C; g.ldc = out; g.c_dtype = JAGG_DTYPE_F32;
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
  g.M = B; g.N = in; g.K = out;
  g.A = dY; g.lda = out; g.a_mn = false; g.a_dtype = m.cfg.dtype;
  g.B = W(m, w_off); g.ldb = in; g.b_mn = true; g.b_dtype = m.cfg.dtype;
  g.epi = EPI_ACCUM; g.C = dX; g.ldc = in; g.c_dtype = JAGG_DTYPE_F32;
  return g;
}

// Row map of a token range inside the joint [txt; img] layout of B sequences of N rows:
// row r of the range is (r / seg) * stride + off + r % seg (seg = 0: the identity).
struct RowMap {
  int seg, off;
  int64_t stride;
};
RowMap img_rows_of(const jagg_model& m) { return RowMap{m.Ni, m.Nt, m.N}; }
RowMap txt_rows_of(const jagg_model& m) { return RowMap{m.Nt, 0, m.N}; }
constexpr RowMap kContiguous{0, 0, 0};

// Phase 1 prologue: patch and text embeddings into the residual stream(s) (image rows at
// h_img through mi, text rows at h_txt through mt), the t-embedding MLP and every block's
// modulation at once from the stacked weights.
int prologue_fwd(const jagg_model& m, const void* z, const float* t, const void* txt, int B, const Saved& S,
                 float* h_img, RowMap mi, float* h_txt, RowMap mt, cudaStream_t s) {
  const jagg_config& c = m.cfg;
  const int dt = c.dtype, d = m.d;
  const int Mi = B * m.Ni, Mt = B * m.Nt;
  JAGG_TRY(launch_patchify(z, dt == JAGG_DTYPE_F32, S.xp, dt == JAGG_DTYPE_F32, dt, B, c.in_channels, c.latent_h,
                           c.latent_w, c.patch, s));
  JAGG_CUDA_TRY(cudaMemcpyAsync(S.txt, txt, (size_t)Mt * c.txt_dim * m.esz, cudaMemcpyDeviceToDevice, s));
  GemmArgs g = fwd_gemm(m, Mi, d, m.pd, S.xp, m.pd, m.T.x_w, m.T.x_b);
  g.C = h_img; g.ldc = d; g.c_dtype = JAGG_DTYPE_F32;
  g.remap_rows = mi.seg; g.remap_offset = mi.off; g.remap_stride = mi.stride;
  JAGG_TRY(gemm(g, s));
  GemmArgs gt = fwd_gemm(m, Mt, d, c.txt_dim, S.txt, c.txt_dim, m.T.txt_w, m.T.txt_b);
  gt.C = h_txt; gt.ldc = d; gt.c_dtype = JAGG_DTYPE_F32;
  gt.remap_rows = mt.seg; gt.remap_offset = mt.off; gt.remap_stride = mt.stride;
  JAGG_TRY(gemm(gt, s));
  // the single-stream DiT adds the fixed 2D sin-cos table; the MMDiT rotates q/k instead
  if (c.arch == JAGG_ARCH_DIT) JAGG_TRY(launch_add_pos_embed(h_img, B, m.N, m.Nt, m.gh, m.gw, d, s));
  // t-embedding MLP and every block's modulation (stacked weights): products with B
  // per-sequence rows, each run as Y^T = W X^T so that the long dimension is M
  JAGG_TRY(launch_timestep_embedding(t, S.phi, B, c.freq_dim, s));
  JAGG_TRY(launch_gather_rows(S.phi, c.freq_dim, 0, 0, 0, S.phi_b, dt, B, c.freq_dim, s));
  JAGG_TRY(gemm(rows_gemm(m, d, c.freq_dim, B, S.phi_b, m.T.t_w1, m.T.t_b1, S.e1), s));
  JAGG_TRY(launch_silu(S.e1, S.se1, (int64_t)B * d, s));
  JAGG_TRY(launch_gather_rows(S.se1, d, 0, 0, 0, S.se1_b, dt, B, d, s));
  JAGG_TRY(gemm(rows_gemm(m, d, d, B, S.se1_b, m.T.t_w2, m.T.t_b2, S.c), s));
  JAGG_TRY(launch_silu(S.c, S.sc, (int64_t)B * d, s));
  JAGG_TRY(launch_gather_rows(S.sc, d, 0, 0, 0, S.sc_b, dt, B, d, s));
  JAGG_TRY(gemm(rows_gemm(m, (int)m.T.Lmod, d, B, S.sc_b, m.T.mod_w, m.T.mod_b, S.mod), s));
  return JAGG_OK;
}

// Final layer on the image rows of the joint stream S.h_fin, then unpatchify.
int final_fwd(const jagg_model& m, int B, const Saved& S, void* vt, void* v_out, cudaStream_t s) {
  const jagg_config& c = m.cfg;
  const int d = m.d, Mi = B * m.Ni;
  const float* fm = S.mod + m.T.final_mod_col;
  LnModFwd lf{S.h_fin, m.Ni, m.Nt, m.N, Mi, d, m.Ni, fm, fm + d, m.T.Lmod, S.mf, c.dtype, S.st_f, S.st_f + Mi};
  JAGG_TRY(launch_ln_mod_fwd(lf, s));
  GemmArgs g = fwd_gemm(m, Mi, m.pd, d, S.mf, d, m.T.out_w, m.T.out_b);
  g.C = vt; g.ldc = m.pd;
  JAGG_TRY(gemm(g, s));
  JAGG_TRY(launch_unpatchify(vt, v_out, c.dtype, B, c.in_channels, c.latent_h, c.latent_w, c.patch, s));
  return JAGG_OK;
}

// Backward of the final layer: parameter gradients, and dh (joint layout, zeroed by the
// caller) += the gradient reaching the image rows.
int final_bwd(const jagg_model& m, int B, const Saved& S, const VjpWs& w, const float* cot, float* grad,
              cudaStream_t s) {
  const jagg_config& c = m.cfg;
  const int dt = c.dtype, d = m.d, Mi = B * m.Ni;
  const int64_t Lm = m.T.Lmod;
  JAGG_TRY(launch_patchify(cot, 1, w.dvt, dt == JAGG_DTYPE_F32, dt, B, c.in_channels, c.latent_h, c.latent_w,
                           c.patch, s));
  JAGG_TRY(launch_colsum(w.dvt, dt == JAGG_DTYPE_F32, dt, Mi, m.pd, m.pd, grad + m.T.out_b, s));
  JAGG_TRY(gemm(dw_gemm(m, Mi, m.pd, d, w.dvt, m.pd, S.mf, d, grad, m.T.out_w), s));
  GemmArgs g = dx_gemm(m, Mi, m.pd, d, w.dvt, m.pd, m.T.out_w);
  g.C = w.dx32; g.ldc = d; g.c_dtype = JAGG_DTYPE_F32;
  JAGG_TRY(gemm(g, s));
  const float* fm = S.mod + m.T.final_mod_col;
  float* dfm = w.dmod + m.T.final_mod_col;
  LnGateBwd a{};
  a.M = Mi; a.d = d; a.rows_per_seq = m.Ni;
  a.seg = m.Ni; a.seg_off = m.Nt; a.seg_stride = m.N;
  a.do_ln = 1; a.dm = w.dx32; a.dm_f32 = 1; a.h = S.h_fin; a.mean = S.st_f; a.rstd = S.st_f + Mi;
  a.scale = fm + d; a.mod_stride = Lm; a.dshift = dfm; a.dscale = dfm + d; a.dmod_stride = Lm;
  a.dh_in = w.dh; a.dh_out = w.dh;
  a.dtype = dt;
  return launch_ln_gate_bwd(a, s);
}

// Backward of the embeddings (no gradient to z or txt) and of the stacked modulation and
// the t-embedding MLP, from the residual gradients at the embedding outputs.
int epilogue_bwd(const jagg_model& m, int B, const Saved& S, const VjpWs& w, const float* dh_img, RowMap mi,
                 const float* dh_txt, RowMap mt, float* grad, cudaStream_t s) {
  const jagg_config& c = m.cfg;
  const int dt = c.dtype, d = m.d, Mi = B * m.Ni, Mt = B * m.Nt;
  const int64_t Lm = m.T.Lmod;
  JAGG_TRY(launch_gather_rows(dh_img, d, mi.seg, mi.off, mi.stride, w.dxe, dt, Mi, d, s));
  JAGG_TRY(launch_colsum(w.dxe, dt == JAGG_DTYPE_F32, dt, Mi, d, d, grad + m.T.x_b, s));
  JAGG_TRY(gemm(dw_gemm(m, Mi, d, m.pd, w.dxe, d, S.xp, m.pd, grad, m.T.x_w), s));
  JAGG_TRY(launch_gather_rows(dh_txt, d, mt.seg, mt.off, mt.stride, w.dxe, dt, Mt, d, s));
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

int zero_vjp_accumulators(const jagg_model& m, int B, const VjpWs& w, cudaStream_t s) {
  JAGG_CUDA_TRY(cudaMemsetAsync(w.dmod, 0, sizeof(float) * (size_t)B * m.T.Lmod, s));
  JAGG_CUDA_TRY(cudaMemsetAsync(w.dh, 0, sizeof(float) * (size_t)B * m.N * m.d, s));
  JAGG_CUDA_TRY(cudaMemsetAsync(w.dsc, 0, sizeof(float) * (size_t)B * m.d, s));
  JAGG_CUDA_TRY(cudaMemsetAsync(w.de1, 0, sizeof(float) * (size_t)B * m.d, s));
  return JAGG_OK;
}

// The MLP half of a block's backward, shared by DiT blocks and the streams of MMDiT
// double blocks (Ms rows of Ns tokens per sequence): from dy = g2 dh (already formed)
// through fc2, GELU, fc1 and LN2 + modulation, then the attention branch's gate, ending
// with dO = dy1 Wproj.  dh accumulates in place.
struct BranchW {
  int64_t proj_w, proj_b, fc1_w, fc1_b, fc2_w, fc2_b, mod_col;
};
int mlp_and_proj_bwd(const jagg_model& m, int Ms, int Ns, const DitSaved& k, const BranchW& bw, const float* mod,
                     float* dmod, float* dh, void* dy, void* dO, const VjpWs& w, float* grad, cudaStream_t s) {
  const int dt = m.cfg.dtype, d = m.d, dmw = m.dm;
  const int64_t Lm = m.T.Lmod;
  JAGG_TRY(gemm(dw_gemm(m, Ms, d, dmw, dy, d, k.gu, dmw, grad, bw.fc2_w), s));
  {
    GemmArgs g = dx_gemm(m, Ms, d, dmw, dy, d, bw.fc2_w);
    g.epi = EPI_MUL_AUX; g.C = w.du; g.ldc = dmw; g.aux = k.gp; g.ld_aux = dmw;
    JAGG_TRY(gemm(g, s));
  }
  JAGG_TRY(launch_colsum(w.du, dt == JAGG_DTYPE_F32, dt, Ms, dmw, dmw, grad + bw.fc1_b, s));
  JAGG_TRY(gemm(dw_gemm(m, Ms, dmw, d, w.du, dmw, k.m, d, grad, bw.fc1_w), s));
  {
    GemmArgs g = dx_gemm(m, Ms, dmw, d, w.du, dmw, bw.fc1_w);
    g.C = w.dx32; g.ldc = d; g.c_dtype = JAGG_DTYPE_F32;
    JAGG_TRY(gemm(g, s));
  }
  {  // LN2 + modulation backward, then the attention branch's gate
    LnGateBwd a{};
    a.M = Ms; a.d = d; a.rows_per_seq = Ns;
    a.do_ln = 1; a.dm = w.dx32; a.dm_f32 = 1; a.h = k.h_mid; a.mean = k.st2; a.rstd = k.st2 + Ms;
    a.scale = mod + 4 * d; a.mod_stride = Lm; a.dshift = dmod + 3 * d; a.dscale = dmod + 4 * d;
    a.dmod_stride = Lm; a.dh_in = dh; a.dh_out = dh;
    a.do_gate = 1; a.y = k.y1; a.gate = mod + 2 * d; a.dgate = dmod + 2 * d; a.dy = dy;
    a.dbias = grad + bw.proj_b; a.dtype = dt;
    JAGG_TRY(launch_ln_gate_bwd(a, s));
  }
  JAGG_TRY(gemm(dw_gemm(m, Ms, d, d, dy, d, k.o, d, grad, bw.proj_w), s));
  GemmArgs g = dx_gemm(m, Ms, d, d, dy, d, bw.proj_w);
  g.C = dO; g.ldc = d;
  return gemm(g, s);
}

// The qkv half of a block's backward after attention: qkv bias / weight gradients, the
// gradient into the LN1 input, and LN1 + modulation backward (dh accumulates in place).
// `gate`, when given, fuses the gate backward of the previous block's last branch.
int qkv_and_ln1_bwd(const jagg_model& m, int Ms, int Ns, const void* dqkv, int64_t ld_dqkv, int n_out,
                    int64_t w_off, int64_t b_off, const void* a_in, const float* h_in, const float* st1,
                    const float* mod, float* dmod, float* dh, const LnGateBwd* gate, const VjpWs& w, float* grad,
                    cudaStream_t s) {
  const int dt = m.cfg.dtype, d = m.d;
  const int64_t Lm = m.T.Lmod;
  JAGG_TRY(launch_colsum(dqkv, dt == JAGG_DTYPE_F32, dt, Ms, n_out, ld_dqkv, grad + b_off, s));
  JAGG_TRY(gemm(dw_gemm(m, Ms, n_out, d, dqkv, ld_dqkv, a_in, d, grad, w_off), s));
  {
    GemmArgs g = dx_gemm(m, Ms, n_out, d, dqkv, ld_dqkv, w_off);
    g.C = w.dx32; g.ldc = d; g.c_dtype = JAGG_DTYPE_F32;
    JAGG_TRY(gemm(g, s));
  }
  LnGateBwd a = gate ? *gate : LnGateBwd{};
  a.M = Ms; a.d = d; a.rows_per_seq = Ns;
  a.do_ln = 1; a.dm = w.dx32; a.dm_f32 = 1; a.h = h_in; a.mean = st1; a.rstd = st1 + Ms;
  a.scale = mod + d; a.mod_stride = Lm; a.dshift = dmod; a.dscale = dmod + d; a.dmod_stride = Lm;
  a.dh_in = dh; a.dh_out = dh; a.dtype = dt;
  return launch_ln_gate_bwd(a, s);
}

// Gate backward of a branch y with gate mod[gcol]: dgate += sum dh y; dy = gate dh; dbias.
LnGateBwd gate_args(const jagg_model& m, int Ms, int Ns, float* dh, const void* y, const float* gate,
                    float* dgate, void* dy, float* dbias) {
  LnGateBwd a{};
  a.M = Ms; a.d = m.d; a.rows_per_seq = Ns;
  a.do_ln = 0; a.dh_in = dh; a.dh_out = dh;
  a.do_gate = 1; a.y = y; a.gate = gate; a.mod_stride = m.T.Lmod; a.dgate = dgate; a.dmod_stride = m.T.Lmod;
  a.dy = dy; a.dbias = dbias; a.dtype = m.cfg.dtype;
  return a;
}

AttnArgs attn_args(const jagg_model& m, int B, SegRows qk, SegRows v, SegRows o, float* lse) {
  AttnArgs at;
  at.B = B; at.N = m.N; at.heads = m.heads; at.dh = m.dh; at.scale = 1.f / sqrtf((float)m.dh);
  at.q = at.k = qk;
  at.v = v;
  at.o = o;
  at.lse = lse;
  at.dtype = m.cfg.dtype;
  return at;
}

QkNormRope qk_args(const jagg_model& m, const void* qkv, int Ms, int Ns, int n_txt, int64_t qn, int64_t kn, void* qk,
                   float* rq, float* rk) {
  QkNormRope q{};
  q.qkv = qkv; q.ld_qkv = 3 * m.d;
  q.M = Ms; q.N = Ns; q.d = m.d; q.heads = m.heads; q.n_txt = n_txt; q.gw = m.gw;
  q.qscale_txt = q.qscale_img = W(m, qn);
  q.kscale_txt = q.kscale_img = W(m, kn);
  q.rope = 1;
  q.qk_out = qk; q.rq = rq; q.rk = rk;
  q.dtype = m.cfg.dtype;
  return q;
}

// ---------------------------------------------------------------- single-stream DiT
int forward_dit(const jagg_model& m, const Saved& S, int B, cudaStream_t s) {
  const jagg_config& c = m.cfg;
  const int dt = c.dtype, d = m.d, N = m.N, M = B * N;
  const int64_t Lm = m.T.Lmod;
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
    AttnArgs at = attn_args(m, B, seg_single(k.qkv, 3 * d, N), seg_single(k.qkv, 3 * d, N), seg_single(k.o, d, N),
                            k.lse);
    at.q_col0 = 0; at.k_col0 = d; at.v_col0 = 2 * d;
    JAGG_TRY(attention_fwd(at, s));
    g = fwd_gemm(m, M, d, d, k.o, d, bw.proj_w, bw.proj_b);
    g.epi = EPI_GATE_RESID; g.C = k.y1; g.ldc = d;
    g.C2 = k.h_mid; g.ldc2 = d; g.aux = k.h_in; g.ld_aux = d;
    g.gate = mod + 2 * d; g.gate_stride = Lm; g.rows_per_seq = N;
    JAGG_TRY(gemm(g, s));
    LnModFwd ln2{k.h_mid, 0, 0, 0, M, d, N, mod + 3 * d, mod + 4 * d, Lm, k.m, dt, k.st2, k.st2 + M};
    JAGG_TRY(launch_ln_mod_fwd(ln2, s));
    g = fwd_gemm(m, M, m.dm, d, k.m, d, bw.fc1_w, bw.fc1_b);
    g.epi = EPI_GELU; g.C = S.keep ? k.gp : nullptr; g.ldc = m.dm; g.C2 = k.gu; g.ldc2 = m.dm;
    JAGG_TRY(gemm(g, s));
    g = fwd_gemm(m, M, d, m.dm, k.gu, m.dm, bw.fc2_w, bw.fc2_b);
    g.epi = EPI_GATE_RESID; g.C = k.y2; g.ldc = d;
    g.C2 = h_out; g.ldc2 = d; g.aux = k.h_mid; g.ld_aux = d;
    g.gate = mod + 5 * d; g.gate_stride = Lm; g.rows_per_seq = N;
    JAGG_TRY(gemm(g, s));
  }
  return JAGG_OK;
}

BranchW branch_of(const DitBlockW& b) {
  return BranchW{b.proj_w, b.proj_b, b.fc1_w, b.fc1_b, b.fc2_w, b.fc2_b, b.mod_col};
}
BranchW branch_of(const StreamW& b) {
  return BranchW{b.proj_w, b.proj_b, b.fc1_w, b.fc1_b, b.fc2_w, b.fc2_b, b.mod_col};
}

int vjp_dit(const jagg_model& m, const Saved& S, int B, const VjpWs& w, float* grad, cudaStream_t s) {
  const jagg_config& c = m.cfg;
  const int d = m.d, N = m.N, M = B * N;
  // Gate of block l's MLP branch (dg2, dy2 = g2 dh, db_fc2): for the last block a pass of
  // its own; for the others fused into the LayerNorm-1 backward of block l + 1, which
  // produces exactly that gradient.
  auto mlp_gate = [&](int l) {
    const DitBlockW& bw = m.T.blocks[l];
    return gate_args(m, M, N, w.dh, S.blk[l].y2, S.mod + bw.mod_col + 5 * d, w.dmod + bw.mod_col + 5 * d, w.dy,
                     grad + bw.fc2_b);
  };
  if (c.depth > 0) JAGG_TRY(launch_ln_gate_bwd(mlp_gate(c.depth - 1), s));
  for (int l = c.depth - 1; l >= 0; --l) {
    const DitBlockW& bw = m.T.blocks[l];
    const DitSaved& k = S.blk[l];
    const float* mod = S.mod + bw.mod_col;
    float* dmod = w.dmod + bw.mod_col;
    JAGG_TRY(mlp_and_proj_bwd(m, M, N, k, branch_of(bw), mod, dmod, w.dh, w.dy, w.dO, w, grad, s));
    AttnBwdArgs ab;
    ab.f = attn_args(m, B, seg_single(k.qkv, 3 * d, N), seg_single(k.qkv, 3 * d, N), seg_single(k.o, d, N), k.lse);
    ab.f.q_col0 = 0; ab.f.k_col0 = d; ab.f.v_col0 = 2 * d;
    ab.dO = seg_single(w.dO, d, N);
    attention_bwd_scratch(w.attn, B, N, m.heads, &ab.Dv, &ab.dq_acc);
    ab.dq = ab.dk = ab.dv = seg_single(w.dqkv, 3 * d, N);
    ab.dq_col0 = 0; ab.dk_col0 = d; ab.dv_col0 = 2 * d;
    JAGG_TRY(attention_bwd(ab, s));
    LnGateBwd prev{};
    if (l > 0) prev = mlp_gate(l - 1);
    JAGG_TRY(qkv_and_ln1_bwd(m, M, N, w.dqkv, 3 * d, 3 * d, bw.qkv_w, bw.qkv_b, k.a, k.h_in, k.st1, mod, dmod, w.dh,
                             l > 0 ? &prev : nullptr, w, grad, s));
  }
  return JAGG_OK;
}

// ---------------------------------------------------------------- MMDiT
// Double blocks run each stream as its own rows (Ms = B Ns, Ns = Nt or Ni tokens per
// sequence) and meet only in the joint attention, which addresses the two streams'
// buffers as one [txt; img] sequence.  Single blocks run on the joint layout.
int forward_mmdit(const jagg_model& m, const Saved& S, int B, cudaStream_t s) {
  const jagg_config& c = m.cfg;
  const int dt = c.dtype, d = m.d, dm = m.dm, N = m.N, Nt = m.Nt, Ni = m.Ni, M = B * N;
  const int Ld = c.depth_double, Ls = c.depth;
  const int64_t Lm = m.T.Lmod;
  for (int l = 0; l < Ld; ++l) {
    const DoubleW& bw = m.T.doubles[l];
    const DoubleSaved& k = S.dbl[l];
    for (int si = 0; si < 2; ++si) {
      const StreamW& sw = bw.s[si];
      const DitSaved& q = k.s[si];
      const int Ns = si ? Ni : Nt, Ms = B * Ns;
      const float* mod = S.mod + sw.mod_col;
      LnModFwd ln{q.h_in, 0, 0, 0, Ms, d, Ns, mod, mod + d, Lm, q.a, dt, q.st1, q.st1 + Ms};
      JAGG_TRY(launch_ln_mod_fwd(ln, s));
      GemmArgs g = fwd_gemm(m, Ms, 3 * d, d, q.a, d, sw.qkv_w, sw.qkv_b);
      g.C = q.qkv; g.ldc = 3 * d;
      JAGG_TRY(gemm(g, s));
      // text tokens sit at RoPE position (0, 0): the whole text stream is unrotated
      JAGG_TRY(launch_qk_norm_rope_fwd(qk_args(m, q.qkv, Ms, Ns, si ? 0 : Ns, sw.qn, sw.kn, q.qk, q.rq, q.rk), s));
    }
    AttnArgs at = attn_args(m, B, SegRows{k.s[0].qk, k.s[1].qk, 2 * d, 2 * d, Nt},
                            SegRows{k.s[0].qkv, k.s[1].qkv, 3 * d, 3 * d, Nt},
                            SegRows{k.s[0].o, k.s[1].o, d, d, Nt}, k.lse);
    at.q_col0 = 0; at.k_col0 = d; at.v_col0 = 2 * d;
    JAGG_TRY(attention_fwd(at, s));
    for (int si = 0; si < 2; ++si) {
      const StreamW& sw = bw.s[si];
      const DitSaved& q = k.s[si];
      const int Ns = si ? Ni : Nt, Ms = B * Ns;
      const float* mod = S.mod + sw.mod_col;
      float* h_out = (l + 1 < Ld) ? S.dbl[l + 1].s[si].h_in : S.hD[si];
      GemmArgs g = fwd_gemm(m, Ms, d, d, q.o, d, sw.proj_w, sw.proj_b);
      g.epi = EPI_GATE_RESID; g.C = q.y1; g.ldc = d;
      g.C2 = q.h_mid; g.ldc2 = d; g.aux = q.h_in; g.ld_aux = d;
      g.gate = mod + 2 * d; g.gate_stride = Lm; g.rows_per_seq = Ns;
      JAGG_TRY(gemm(g, s));
      LnModFwd ln2{q.h_mid, 0, 0, 0, Ms, d, Ns, mod + 3 * d, mod + 4 * d, Lm, q.m, dt, q.st2, q.st2 + Ms};
      JAGG_TRY(launch_ln_mod_fwd(ln2, s));
      g = fwd_gemm(m, Ms, dm, d, q.m, d, sw.fc1_w, sw.fc1_b);
      g.epi = EPI_GELU; g.C = S.keep ? q.gp : nullptr; g.ldc = dm; g.C2 = q.gu; g.ldc2 = dm;
      JAGG_TRY(gemm(g, s));
      g = fwd_gemm(m, Ms, d, dm, q.gu, dm, sw.fc2_w, sw.fc2_b);
      g.epi = EPI_GATE_RESID; g.C = q.y2; g.ldc = d;
      g.C2 = h_out; g.ldc2 = d; g.aux = q.h_mid; g.ld_aux = d;
      g.gate = mod + 5 * d; g.gate_stride = Lm; g.rows_per_seq = Ns;
      JAGG_TRY(gemm(g, s));
    }
  }
  float* hj = Ls > 0 ? S.sgl[0].h_in : S.h_fin;
  if (Ld > 0) {  // the two streams join into the [txt; img] layout
    JAGG_TRY(launch_copy_rows(S.hD[0], d, 0, 0, 0, hj, d, Nt, 0, N, B * Nt, d, 4, s));
    JAGG_TRY(launch_copy_rows(S.hD[1], d, 0, 0, 0, hj, d, Ni, Nt, N, B * Ni, d, 4, s));
  }
  const size_t e = m.esz;
  for (int l = 0; l < Ls; ++l) {
    const SingleW& sw = m.T.singles[l];
    const SingleSaved& k = S.sgl[l];
    float* h_out = (l + 1 < Ls) ? S.sgl[l + 1].h_in : S.h_fin;
    const float* mod = S.mod + sw.mod_col;
    LnModFwd ln{k.h_in, 0, 0, 0, M, d, N, mod, mod + d, Lm, k.a, dt, k.st1, k.st1 + M};
    JAGG_TRY(launch_ln_mod_fwd(ln, s));
    // lin1 = [qkv | u]: two products over the row blocks of its weight
    GemmArgs g = fwd_gemm(m, M, 3 * d, d, k.a, d, sw.lin1_w, sw.lin1_b);
    g.C = k.qkv; g.ldc = 3 * d;
    JAGG_TRY(gemm(g, s));
    g = fwd_gemm(m, M, dm, d, k.a, d, sw.lin1_w + (int64_t)3 * d * d, sw.lin1_b + 3 * d);
    g.epi = EPI_GELU; g.C = S.keep ? k.gp : nullptr; g.ldc = dm;
    g.C2 = static_cast<uint8_t*>(k.cat) + (size_t)d * e; g.ldc2 = d + dm;
    JAGG_TRY(gemm(g, s));
    JAGG_TRY(launch_qk_norm_rope_fwd(qk_args(m, k.qkv, M, N, Nt, sw.qn, sw.kn, k.qk, k.rq, k.rk), s));
    AttnArgs at = attn_args(m, B, seg_single(k.qk, 2 * d, N), seg_single(k.qkv, 3 * d, N),
                            seg_single(k.cat, d + dm, N), k.lse);
    at.q_col0 = 0; at.k_col0 = d; at.v_col0 = 2 * d;
    JAGG_TRY(attention_fwd(at, s));
    g = fwd_gemm(m, M, d, d + dm, k.cat, d + dm, sw.lin2_w, sw.lin2_b);
    g.epi = EPI_GATE_RESID; g.C = k.y; g.ldc = d;
    g.C2 = h_out; g.ldc2 = d; g.aux = k.h_in; g.ld_aux = d;
    g.gate = mod + 2 * d; g.gate_stride = Lm; g.rows_per_seq = N;
    JAGG_TRY(gemm(g, s));
  }
  return JAGG_OK;
}

int vjp_mmdit(const jagg_model& m, const Saved& S, int B, const VjpWs& w, float* grad, cudaStream_t s) {
  const jagg_config& c = m.cfg;
  const int d = m.d, dm = m.dm, N = m.N, Nt = m.Nt, Ni = m.Ni, M = B * N, Mt = B * Nt;
  const int Ld = c.depth_double, Ls = c.depth;
  const size_t e = m.esz;
  auto at_byte = [](void* p, size_t off) { return static_cast<void*>(static_cast<uint8_t*>(p) + off); };
  // single blocks, last to first, on the joint gradient w.dh
  auto single_gate = [&](int l) {
    const SingleW& sw = m.T.singles[l];
    return gate_args(m, M, N, w.dh, S.sgl[l].y, S.mod + sw.mod_col + 2 * d, w.dmod + sw.mod_col + 2 * d, w.dy,
                     grad + sw.lin2_b);
  };
  if (Ls > 0) JAGG_TRY(launch_ln_gate_bwd(single_gate(Ls - 1), s));
  const int64_t ld1 = 3 * d + dm;  // w.dqkv holds d(lin1 output) = [dqkv | du]
  for (int l = Ls - 1; l >= 0; --l) {
    const SingleW& sw = m.T.singles[l];
    const SingleSaved& k = S.sgl[l];
    const float* mod = S.mod + sw.mod_col;
    float* dmod = w.dmod + sw.mod_col;
    JAGG_TRY(gemm(dw_gemm(m, M, d, d + dm, w.dy, d, k.cat, d + dm, grad, sw.lin2_w), s));
    {  // d(cat) = dy Wlin2: the attention-output columns, then GELU's columns times GELU'
      GemmArgs g = dx_gemm(m, M, d, d, w.dy, d, sw.lin2_w, d + dm);
      g.C = w.dO; g.ldc = d;
      JAGG_TRY(gemm(g, s));
      g = dx_gemm(m, M, d, dm, w.dy, d, sw.lin2_w + d, d + dm);
      g.epi = EPI_MUL_AUX; g.C = at_byte(w.dqkv, (size_t)3 * d * e); g.ldc = ld1; g.aux = k.gp; g.ld_aux = dm;
      JAGG_TRY(gemm(g, s));
    }
    AttnBwdArgs ab;
    ab.f = attn_args(m, B, seg_single(k.qk, 2 * d, N), seg_single(k.qkv, 3 * d, N), seg_single(k.cat, d + dm, N),
                     k.lse);
    ab.f.q_col0 = 0; ab.f.k_col0 = d; ab.f.v_col0 = 2 * d;
    ab.dO = seg_single(w.dO, d, N);
    attention_bwd_scratch(w.attn, B, N, m.heads, &ab.Dv, &ab.dq_acc);
    ab.dq = ab.dk = ab.dv = seg_single(w.dqkv, ld1, N);
    ab.dq_col0 = 0; ab.dk_col0 = d; ab.dv_col0 = 2 * d;
    JAGG_TRY(attention_bwd(ab, s));
    QkNormRopeBwd qb;
    qb.f = qk_args(m, k.qkv, M, N, Nt, sw.qn, sw.kn, k.qk, k.rq, k.rk);
    qb.dqk = w.dqkv; qb.ld_dqk = ld1;
    qb.dqs_txt = qb.dqs_img = grad + sw.qn;
    qb.dks_txt = qb.dks_img = grad + sw.kn;
    JAGG_TRY(launch_qk_norm_rope_bwd(qb, s));
    LnGateBwd prev{};
    if (l > 0) prev = single_gate(l - 1);
    JAGG_TRY(qkv_and_ln1_bwd(m, M, N, w.dqkv, ld1, (int)ld1, sw.lin1_w, sw.lin1_b, k.a, k.h_in, k.st1, mod, dmod,
                             w.dh, l > 0 ? &prev : nullptr, w, grad, s));
  }
  if (Ld == 0) return JAGG_OK;
  // the joint gradient splits into the two streams
  JAGG_TRY(launch_copy_rows(w.dh, d, Nt, 0, N, w.dhs[0], d, 0, 0, 0, B * Nt, d, 4, s));
  JAGG_TRY(launch_copy_rows(w.dh, d, Ni, Nt, N, w.dhs[1], d, 0, 0, 0, B * Ni, d, 4, s));
  // per-stream regions of the gradient buffers: text rows first, image rows after
  void* dy_s[2] = {w.dy, at_byte(w.dy, (size_t)Mt * d * e)};
  void* dO_s[2] = {w.dO, at_byte(w.dO, (size_t)Mt * d * e)};
  void* dqkv_s[2] = {w.dqkv, at_byte(w.dqkv, (size_t)Mt * 3 * d * e)};
  auto mlp_gate = [&](int l, int si) {
    const StreamW& sw = m.T.doubles[l].s[si];
    const int Ns = si ? Ni : Nt;
    return gate_args(m, B * Ns, Ns, w.dhs[si], S.dbl[l].s[si].y2, S.mod + sw.mod_col + 5 * d,
                     w.dmod + sw.mod_col + 5 * d, dy_s[si], grad + sw.fc2_b);
  };
  for (int si = 0; si < 2; ++si) JAGG_TRY(launch_ln_gate_bwd(mlp_gate(Ld - 1, si), s));
  for (int l = Ld - 1; l >= 0; --l) {
    const DoubleW& bw = m.T.doubles[l];
    const DoubleSaved& k = S.dbl[l];
    for (int si = 0; si < 2; ++si) {
      const int Ns = si ? Ni : Nt;
      JAGG_TRY(mlp_and_proj_bwd(m, B * Ns, Ns, k.s[si], branch_of(bw.s[si]), S.mod + bw.s[si].mod_col,
                                w.dmod + bw.s[si].mod_col, w.dhs[si], dy_s[si], dO_s[si], w, grad, s));
    }
    AttnBwdArgs ab;
    ab.f = attn_args(m, B, SegRows{k.s[0].qk, k.s[1].qk, 2 * d, 2 * d, Nt},
                     SegRows{k.s[0].qkv, k.s[1].qkv, 3 * d, 3 * d, Nt}, SegRows{k.s[0].o, k.s[1].o, d, d, Nt}, k.lse);
    ab.f.q_col0 = 0; ab.f.k_col0 = d; ab.f.v_col0 = 2 * d;
    ab.dO = SegRows{dO_s[0], dO_s[1], d, d, Nt};
    attention_bwd_scratch(w.attn, B, N, m.heads, &ab.Dv, &ab.dq_acc);
    ab.dq = ab.dk = ab.dv = SegRows{dqkv_s[0], dqkv_s[1], 3 * d, 3 * d, Nt};
    ab.dq_col0 = 0; ab.dk_col0 = d; ab.dv_col0 = 2 * d;
    JAGG_TRY(attention_bwd(ab, s));
    for (int si = 0; si < 2; ++si) {
      const StreamW& sw = bw.s[si];
      const DitSaved& q = k.s[si];
      const int Ns = si ? Ni : Nt, Ms = B * Ns;
      QkNormRopeBwd qb;
      qb.f = qk_args(m, q.qkv, Ms, Ns, si ? 0 : Ns, sw.qn, sw.kn, q.qk, q.rq, q.rk);
      qb.dqk = dqkv_s[si]; qb.ld_dqk = 3 * d;
      qb.dqs_txt = qb.dqs_img = grad + sw.qn;
      qb.dks_txt = qb.dks_img = grad + sw.kn;
      JAGG_TRY(launch_qk_norm_rope_bwd(qb, s));
      LnGateBwd prev{};
      if (l > 0) prev = mlp_gate(l - 1, si);
      JAGG_TRY(qkv_and_ln1_bwd(m, Ms, Ns, dqkv_s[si], 3 * d, 3 * d, sw.qkv_w, sw.qkv_b, q.a, q.h_in, q.st1,
                               S.mod + sw.mod_col, w.dmod + sw.mod_col, w.dhs[si], l > 0 ? &prev : nullptr, w, grad,
                               s));
    }
  }
  return JAGG_OK;
}

int forward_impl(const jagg_model& m, const void* z, const float* t, const void* txt, int B, void* v_out,
                 void* saved, void* ws, cudaStream_t s) {
  const jagg_config& c = m.cfg;
  // With a saved arena every activation goes there; otherwise one block's worth of slots
  // at the start of the workspace is reused by every block.
  Saved S;
  const size_t used = carve_saved(m, B, saved ? saved : ws, saved != nullptr, S);
  void* vt = nullptr;
  carve_fwd_ws(m, B, static_cast<uint8_t*>(ws) + (saved ? 0 : used), &vt);
  if (c.arch == JAGG_ARCH_DIT) {
    float* h0 = S.blk.empty() ? S.h_fin : S.blk[0].h_in;
    JAGG_TRY(prologue_fwd(m, z, t, txt, B, S, h0, img_rows_of(m), h0, txt_rows_of(m), s));
    JAGG_TRY(forward_dit(m, S, B, s));
  } else {
    if (c.depth_double > 0) {
      JAGG_TRY(prologue_fwd(m, z, t, txt, B, S, S.dbl[0].s[1].h_in, kContiguous, S.dbl[0].s[0].h_in, kContiguous,
                            s));
    } else {
      float* h0 = S.sgl.empty() ? S.h_fin : S.sgl[0].h_in;
      JAGG_TRY(prologue_fwd(m, z, t, txt, B, S, h0, img_rows_of(m), h0, txt_rows_of(m), s));
    }
    JAGG_TRY(forward_mmdit(m, S, B, s));
  }
  return final_fwd(m, B, S, vt, v_out, s);
}

int vjp_impl(const jagg_model& m, const void* saved, int B, const float* cot, float* grad, void* ws,
             cudaStream_t s) {
  const jagg_config& c = m.cfg;
  Saved S;
  carve_saved(m, B, const_cast<void*>(saved), true, S);
  VjpWs w;
  carve_vjp_ws(m, B, ws, w);
  JAGG_TRY(zero_vjp_accumulators(m, B, w, s));
  JAGG_TRY(final_bwd(m, B, S, w, cot, grad, s));
  if (c.arch == JAGG_ARCH_DIT) {
    JAGG_TRY(vjp_dit(m, S, B, w, grad, s));
  } else {
    JAGG_TRY(vjp_mmdit(m, S, B, w, grad, s));
    if (c.depth_double > 0)
      return epilogue_bwd(m, B, S, w, w.dhs[1], kContiguous, w.dhs[0], kContiguous, grad, s);
  }
  return epilogue_bwd(m, B, S, w, w.dh, img_rows_of(m), w.dh, txt_rows_of(m), grad, s);
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
  unsigned a = 0, b = 0, c = 0, d = 0;
  if (jagg::unit_status_gemm(&a, clear) || jagg::unit_status_signals(&b, clear) ||
      jagg::unit_status_attention_tc(&c, clear) || jagg::unit_status_testing(&d, clear)) {
    set_last_error("jagg_device_status: reading the status word failed");
    return JAGG_ERR_CUDA;
  }
  *status_out = a | b | c | d;
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
