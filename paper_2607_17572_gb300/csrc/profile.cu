// Launch counting and event-based per-family kernel timing (host side).
#include <atomic>
#include <cstring>
#include <mutex>
#include <vector>

#include "common.cuh"

namespace jagg {
namespace {

std::atomic<long long> g_launches{0};
std::atomic<bool> g_prof_on{false};
std::mutex g_mu;

struct Rec {
  cudaEvent_t a = nullptr, b = nullptr;
  int family = -1;
  double flops = 0, bytes = 0;
  int m = 0, n = 0, k = 0;
};
std::vector<Rec> g_recs;
std::vector<cudaEvent_t> g_pool;

cudaEvent_t get_event() {
  if (!g_pool.empty()) {
    cudaEvent_t e = g_pool.back();
    g_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

const char* kFamilyNames[PROF_FAMILIES] = {"gemm_tcgen05",     "gemm_simt",   "attention_fwd", "attention_bwd",
                                           "ln_gate_bwd",      "attention_bwd_aux", "qk_norm_rope_bwd",
                                           "colsum",           "copy_rows",   "step_signals",  "grad_reduce",
                                           "ln_mod_fwd",       "qk_norm_rope_fwd"};

}  // namespace

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

int prof_start(cudaStream_t s) {
  if (!g_prof_on.load(std::memory_order_relaxed)) return -1;
  std::lock_guard<std::mutex> lk(g_mu);
  Rec r;
  r.a = get_event();
  r.b = get_event();
  if (!r.a || !r.b) return -1;
  cudaEventRecord(r.a, s);
  g_recs.push_back(r);
  return (int)g_recs.size() - 1;
}

void prof_stop(int token, cudaStream_t s, int family, double flops, double bytes, int m, int n, int k) {
  if (token < 0) return;
  std::lock_guard<std::mutex> lk(g_mu);
  if (token >= (int)g_recs.size()) return;
  Rec& r = g_recs[token];
  cudaEventRecord(r.b, s);
  r.family = family;
  r.flops = flops;
  r.bytes = bytes;
  r.m = m;
  r.n = n;
  r.k = k;
}

}  // namespace jagg

using namespace jagg;

extern "C" int64_t jagg_launch_count(void) { return g_launches.load(); }

extern "C" int jagg_profile_enable(int on) {
  std::lock_guard<std::mutex> lk(g_mu);
  for (Rec& r : g_recs) {
    g_pool.push_back(r.a);
    g_pool.push_back(r.b);
  }
  g_recs.clear();
  g_prof_on.store(on != 0);
  return JAGG_OK;
}

extern "C" int jagg_profile_read(jagg_profile_stat* out, int cap, int* n_out) {
  JAGG_CHECK_ARG(out && n_out && cap >= 0, "jagg_profile_read: null output");
  JAGG_CUDA_TRY(cudaDeviceSynchronize());
  std::lock_guard<std::mutex> lk(g_mu);
  jagg_profile_stat acc[PROF_FAMILIES];
  std::memset(acc, 0, sizeof(acc));
  for (int f = 0; f < PROF_FAMILIES; ++f) std::strncpy(acc[f].family, kFamilyNames[f], sizeof(acc[f].family) - 1);
  for (const Rec& r : g_recs) {
    if (r.family < 0 || r.family >= PROF_FAMILIES) continue;
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) continue;
    acc[r.family].launches += 1;
    acc[r.family].ms += ms;
    acc[r.family].flops += r.flops;
    acc[r.family].bytes += r.bytes;
  }
  int n = 0;
  for (int f = 0; f < PROF_FAMILIES && n < cap; ++f) out[n++] = acc[f];
  *n_out = n;
  return JAGG_OK;
}

extern "C" int jagg_profile_launches(jagg_profile_launch* out, int cap, int* n_out) {
  JAGG_CHECK_ARG(out && n_out && cap >= 0, "jagg_profile_launches: null output");
  JAGG_CUDA_TRY(cudaDeviceSynchronize());
  std::lock_guard<std::mutex> lk(g_mu);
  int n = 0;
  for (const Rec& r : g_recs) {
    if (n >= cap) break;
    if (r.family < 0 || r.family >= PROF_FAMILIES) continue;
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) continue;
    jagg_profile_launch& o = out[n++];
    std::memset(&o, 0, sizeof(o));
    std::strncpy(o.family, kFamilyNames[r.family], sizeof(o.family) - 1);
    o.m = r.m;
    o.n = r.n;
    o.k = r.k;
    o.ms = ms;
    o.flops = r.flops;
    o.bytes = r.bytes;
  }
  *n_out = n;
  return JAGG_OK;
}
