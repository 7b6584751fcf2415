// The extern "C" entry points declared in include/moe.h: argument
// validation, workspace carving, per-device state and the call sequence of
// each layer stage.  No entry point allocates or synchronises (except
// moe_check_device_status / moe_device_status_word / moe_prof_get).
#include <atomic>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "common.cuh"
#include "launch.h"

namespace moe {

// Device status word (one per device that loads the library).
__device__ uint32_t g_status_word;

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mu;
uint32_t* g_status_ptr[kMaxDevices] = {};
int g_num_sms[kMaxDevices] = {};
thread_local int g_last_cuda = 0;
std::atomic<uint64_t> g_launches{0};

// ---- profiling ------------------------------------------------------------
struct ProfRec {
  std::string name;
  int launches = 0;
  double total_ms = 0.0;
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> pending;
};
std::atomic<bool> g_prof_on{false};
std::mutex g_prof_mu;
std::vector<ProfRec> g_prof;
std::vector<cudaEvent_t> g_event_pool;
struct Open {
  cudaStream_t s;
  cudaEvent_t ev;
};
thread_local std::vector<Open> g_open;

cudaEvent_t pool_get() {
  if (g_event_pool.empty()) {
    for (int i = 0; i < 256; ++i) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) break;
      g_event_pool.push_back(e);
    }
    if (g_event_pool.empty()) return nullptr;
  }
  cudaEvent_t e = g_event_pool.back();
  g_event_pool.pop_back();
  return e;
}

ProfRec& prof_rec(const char* name) {
  for (auto& r : g_prof)
    if (r.name == name) return r;
  g_prof.push_back(ProfRec{});
  g_prof.back().name = name;
  return g_prof.back();
}

void prof_harvest() {
  for (auto& r : g_prof) {
    for (auto& pr : r.pending) {
      float ms = 0.f;
      cudaEventSynchronize(pr.second);
      if (cudaEventElapsedTime(&ms, pr.first, pr.second) == cudaSuccess) r.total_ms += ms;
      g_event_pool.push_back(pr.first);
      g_event_pool.push_back(pr.second);
    }
    r.pending.clear();
  }
}

// ---- per-device context ---------------------------------------------------
int get_ctx(void* stream, Ctx* c) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    g_last_cuda = (int)e;
    return MOE_ERR_CUDA;
  }
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_status_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_status_word);
    if (e != cudaSuccess) {
      g_last_cuda = (int)e;
      return MOE_ERR_CUDA;
    }
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) {
      g_last_cuda = (int)e;
      return MOE_ERR_CUDA;
    }
    g_status_ptr[dev] = (uint32_t*)p;
    g_num_sms[dev] = sms;
  }
  c->stream = (cudaStream_t)stream;
  c->err = g_status_ptr[dev];
  c->num_sms = g_num_sms[dev];
  c->device = dev;
  return MOE_OK;
}

int cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return MOE_OK;
  g_last_cuda = (int)e;
  return MOE_ERR_CUDA;
}

// ---- validation -----------------------------------------------------------
struct Dims {
  int64_t S, GBS, T, TK;
  int K, D, E, F, H, Din;
  DType dt;
  size_t bx;
};

int check_shape(const moe_shape_t* s, Dims* d) {
  if (!s) return MOE_ERR_NULL;
  if (s->x_dtype != MOE_BF16 && s->x_dtype != MOE_F32) return MOE_ERR_DTYPE;
  if (s->S <= 0 || s->GBS <= 0 || s->K <= 0 || s->D <= 0 || s->E <= 0 || s->F <= 0 || s->H < 0)
    return MOE_ERR_SHAPE;
  if (s->K > s->E || s->E > kMaxE || s->K > kMaxK) return MOE_ERR_SHAPE;
  if (s->D % 64 || s->F % 64 || s->H % 64) return MOE_ERR_SHAPE;
  if (s->S > (int64_t(1) << 31) || s->GBS > (int64_t(1) << 31)) return MOE_ERR_SHAPE;
  const int64_t T = s->S * s->GBS;
  const int64_t TK = T * s->K;
  if (TK >= (int64_t(1) << 31)) return MOE_ERR_SHAPE;
  d->S = s->S;
  d->GBS = s->GBS;
  d->T = T;
  d->TK = TK;
  d->K = s->K;
  d->D = s->D;
  d->E = s->E;
  d->F = s->F;
  d->H = s->H;
  d->Din = s->H ? s->H : s->D;
  d->dt = s->x_dtype == MOE_BF16 ? DType::BF16 : DType::F32;
  d->bx = dsize(d->dt);
  return MOE_OK;
}

bool aligned(const void* p) { return ((uintptr_t)p & 15u) == 0; }

#define REQUIRE_PTR(p)                     \
  do {                                     \
    if (!(p)) return MOE_ERR_NULL;         \
    if (!aligned(p)) return MOE_ERR_ALIGN; \
  } while (0)
#define OPTIONAL_PTR(p)                          \
  do {                                           \
    if ((p) && !aligned(p)) return MOE_ERR_ALIGN; \
  } while (0)
#define TRY(expr)                    \
  do {                               \
    int _st = (expr);                \
    if (_st != MOE_OK) return _st;   \
  } while (0)
#define TRY_CUDA(expr) TRY(cuda_status(expr))

size_t align_up(size_t v) { return (v + 255) & ~size_t(255); }

// Workspace carve-up.  Calls are ordered on one stream, so the regions used by
// different calls may overlap.
size_t ws_perm(const Dims& d) { return align_up(perm_workspace_bytes(d.TK, d.E)); }
// dH [TK, 2F], dA [TK, F], then the two wgrad GEMMs' per-expert tail tensor
// maps (one region each: one launch builds both)
size_t ws_ffn_bwd_maps_offset(const Dims& d) { return align_up((size_t)d.TK * 3 * d.F * d.bx); }
size_t ws_ffn_bwd_maps_bytes(const Dims& d) { return align_up(gemm_tc_group_scratch_bytes(d.E)); }
size_t ws_ffn_bwd(const Dims& d) { return ws_ffn_bwd_maps_offset(d) + 2 * ws_ffn_bwd_maps_bytes(d); }
// Router weight gradient: split-K over the T tokens into at most kRouterSplits
// fp32 partial products, summed in order afterwards.
constexpr int kRouterSplits = 16;
size_t ws_route_dz(const Dims& d) { return align_up((size_t)d.T * d.E * 2); }
size_t ws_route_parts(const Dims& d) { return align_up((size_t)kRouterSplits * d.E * d.Din * 4); }
size_t ws_route_bwd(const Dims& d) {
  return ws_route_dz(d) + ws_route_parts(d) + align_up(gemm_tc_group_scratch_bytes(kRouterSplits));
}
// Splits that fill the GPU: the output has ceil(E / tile rows) x ceil(Din / 256) tiles.
int router_splits(const Dims& d, int num_sms) {
  const bool pair = d.E > 128;
  const int64_t tiles = ((d.E + (pair ? 255 : 127)) / (pair ? 256 : 128)) * ((d.Din + 255) / 256);
  const int64_t slots = pair ? num_sms / 2 : num_sms;
  int64_t s = slots / (tiles > 0 ? tiles : 1);
  if (s > kRouterSplits) s = kRouterSplits;
  if (s > d.T / 256) s = d.T / 256;
  return s < 1 ? 1 : (int)s;
}
// Sigmoid router forward: per-token score sums and the balance statistics'
// per-chunk partial sums.
size_t ws_route_sigmoid(const Dims& d) { return align_up(route_sigmoid_fwd_ws_bytes(d.T, d.S, d.GBS, d.E)); }
size_t ws_total(const Dims& d) {
  size_t m = ws_perm(d);
  m = std::max(m, ws_route_sigmoid(d));
  m = std::max(m, ws_ffn_bwd(d));
  m = std::max(m, ws_route_bwd(d));
  return m + 256;
}

// Runs one GEMM on the tensor-core engine when it supports the descriptor,
// else on the CUDA-core engine.
cudaError_t gemm(const Ctx& c, const GemmDesc& g, const char* tc_name, const char* simt_name) {
  if (gemm_tc_supports(g)) return launch_gemm_tc(c, g, tc_name);
  return launch_gemm_simt(c, g, simt_name);
}

}  // namespace

void prof_begin(const char* name, cudaStream_t s) {
  (void)name;
  if (!g_prof_on.load(std::memory_order_relaxed)) return;
  std::lock_guard<std::mutex> lk(g_prof_mu);
  cudaEvent_t e = pool_get();
  if (!e) return;
  cudaEventRecord(e, s);
  g_open.push_back(Open{s, e});
}

void prof_end(const char* name, cudaStream_t s) {
  if (!g_prof_on.load(std::memory_order_relaxed)) return;
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (g_open.empty()) return;
  Open o = g_open.back();
  g_open.pop_back();
  cudaEvent_t e = pool_get();
  if (!e) {
    g_event_pool.push_back(o.ev);
    return;
  }
  cudaEventRecord(e, s);
  ProfRec& r = prof_rec(name);
  r.launches += 1;
  r.pending.emplace_back(o.ev, e);
}

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

int abi_check_shape(const moe_shape_t* s, ShapeInfo* out) {
  Dims d;
  const int st = check_shape(s, &d);
  if (st != MOE_OK) return st;
  out->T = d.T;
  out->TK = d.TK;
  out->K = d.K;
  out->D = d.D;
  out->E = d.E;
  out->F = d.F;
  out->H = d.H;
  out->Din = d.Din;
  out->dt = d.dt;
  out->bx = d.bx;
  return MOE_OK;
}

int abi_device_ctx(void* stream, Ctx* c) { return get_ctx(stream, c); }

int abi_cuda_status(cudaError_t e) { return cuda_status(e); }

}  // namespace moe

using namespace moe;

extern "C" {

int moe_version(void) { return 100; }

const char* moe_strerror(int status) {
  switch (status) {
    case MOE_OK: return "ok";
    case MOE_ERR_SHAPE: return "invalid shape (non-positive size, K > E, E > 256, K > 16, D/F/H not a multiple of 64, or T*K >= 2^31)";
    case MOE_ERR_DTYPE: return "unknown dtype";
    case MOE_ERR_ALIGN: return "pointer not 16-byte aligned";
    case MOE_ERR_NULL: return "required pointer is NULL";
    case MOE_ERR_WORKSPACE: return "workspace smaller than moe_workspace_size()";
    case MOE_ERR_CUDA: return "CUDA runtime error (see moe_last_cuda_error)";
    case MOE_ERR_DEVICE: return "device status word set (out-of-range expert index or expired bounded wait)";
    case MOE_ERR_UNSUPPORTED: return "unsupported request";
    case MOE_ERR_TOO_LARGE: return "shape exceeds the fixed scratch of moe_dispatch_noalloc (E * ceil(T*K/2048) > 262144)";
    default: return "unknown status";
  }
}

int moe_last_cuda_error(void) { return g_last_cuda; }

uint64_t moe_launch_count(void) { return g_launches.load(); }

int moe_workspace_size(const moe_shape_t* shape, size_t* bytes) {
  Dims d;
  TRY(check_shape(shape, &d));
  if (!bytes) return MOE_ERR_NULL;
  *bytes = ws_total(d);
  return MOE_OK;
}

uint64_t moe_eq1_bytes(const moe_shape_t* shape) {
  Dims d;
  if (check_shape(shape, &d) != MOE_OK) return 0;
  return (uint64_t)shape->S * (uint64_t)shape->GBS * (uint64_t)shape->K *
         (4ull * (uint64_t)shape->D * (uint64_t)d.bx + 2ull * 4ull);
}

int moe_topk(const moe_shape_t* shape, const float* logits, int32_t* topk_idx, float* topk_prob, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(logits);
  REQUIRE_PTR(topk_idx);
  REQUIRE_PTR(topk_prob);
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(launch_topk(c, logits, d.T, d.E, d.K, topk_idx, topk_prob));
  return MOE_OK;
}

int moe_route(const moe_shape_t* shape, const void* x, const void* w_router, const float* bias, float* logits,
              int32_t* topk_idx, float* topk_prob, void* ws, size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(x);
  REQUIRE_PTR(w_router);
  OPTIONAL_PTR(bias);
  REQUIRE_PTR(logits);
  REQUIRE_PTR(topk_idx);
  REQUIRE_PTR(topk_prob);
  (void)ws;
  (void)ws_bytes;
  Ctx c;
  TRY(get_ctx(stream, &c));
  GemmDesc g;
  g.group = Group::Dense;
  g.epi = Epi::StoreBias;
  g.M = d.T;
  g.N = d.E;
  g.K = d.Din;
  g.A = x;
  g.a_type = d.dt;
  g.sa_m = d.Din;
  g.sa_k = 1;
  g.B = w_router;
  g.b_type = d.dt;
  g.sb_n = d.Din;
  g.sb_k = 1;
  g.C = logits;
  g.c_type = DType::F32;
  g.ldc = d.E;
  g.bias = bias;
  if (d.T > 0) TRY_CUDA(gemm(c, g, "router_gemm_tc", "router_gemm_simt"));
  TRY_CUDA(launch_topk(c, logits, d.T, d.E, d.K, topk_idx, topk_prob));
  return MOE_OK;
}

int moe_dispatch(const moe_shape_t* shape, const void* x, const int32_t* topk_idx, const float* topk_prob,
                 int32_t* expert_offsets, int32_t* row_of_slot, int32_t* token_of_row, void* x_perm,
                 float* prob_perm, void* ws, size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(topk_idx);
  REQUIRE_PTR(topk_prob);
  REQUIRE_PTR(expert_offsets);
  REQUIRE_PTR(row_of_slot);
  REQUIRE_PTR(token_of_row);
  REQUIRE_PTR(prob_perm);
  REQUIRE_PTR(ws);
  OPTIONAL_PTR(x_perm);
  if (x_perm) REQUIRE_PTR(x);
  if (ws_bytes < ws_perm(d)) return MOE_ERR_WORKSPACE;
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(launch_permutation(c, topk_idx, topk_prob, d.T, d.K, d.E, expert_offsets, row_of_slot, token_of_row,
                              prob_perm, ws));
  if (x_perm) TRY_CUDA(launch_dispatch_rows(c, x, row_of_slot, d.T, d.K, (int64_t)d.D * d.bx, x_perm));
  return MOE_OK;
}

int moe_dispatch_fp8(const moe_shape_t* shape, const void* x, const int32_t* topk_idx, const float* topk_prob,
                     int32_t* expert_offsets, int32_t* row_of_slot, int32_t* token_of_row, void* x_perm_q,
                     float* x_scale_perm, float* prob_perm, void* ws, size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  if (d.dt != DType::BF16) return MOE_ERR_UNSUPPORTED;
  REQUIRE_PTR(x);
  REQUIRE_PTR(topk_idx);
  REQUIRE_PTR(topk_prob);
  REQUIRE_PTR(expert_offsets);
  REQUIRE_PTR(row_of_slot);
  REQUIRE_PTR(token_of_row);
  REQUIRE_PTR(x_perm_q);
  REQUIRE_PTR(x_scale_perm);
  REQUIRE_PTR(prob_perm);
  REQUIRE_PTR(ws);
  if (ws_bytes < ws_perm(d)) return MOE_ERR_WORKSPACE;
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(launch_permutation(c, topk_idx, topk_prob, d.T, d.K, d.E, expert_offsets, row_of_slot, token_of_row,
                              prob_perm, ws));
  TRY_CUDA(launch_dispatch_fp8(c, x, row_of_slot, d.T, d.K, d.D, x_perm_q, x_scale_perm));
  return MOE_OK;
}

int moe_dequant_rows(const moe_shape_t* shape, const void* x_perm_q, const float* x_scale_perm, void* x_perm,
                     void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  if (d.dt != DType::BF16) return MOE_ERR_UNSUPPORTED;
  REQUIRE_PTR(x_perm_q);
  REQUIRE_PTR(x_scale_perm);
  REQUIRE_PTR(x_perm);
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(launch_dequant_rows(c, x_perm_q, x_scale_perm, d.TK, d.D, x_perm));
  return MOE_OK;
}

int moe_dispatch_nvfp4(const moe_shape_t* shape, const void* x, const int32_t* topk_idx, const float* topk_prob,
                       int32_t* expert_offsets, int32_t* row_of_slot, int32_t* token_of_row, void* x_perm_q,
                       uint8_t* x_bscale_perm, float* x_rscale_perm, float* prob_perm, void* ws, size_t ws_bytes,
                       void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  if (d.dt != DType::BF16) return MOE_ERR_UNSUPPORTED;
  REQUIRE_PTR(x);
  REQUIRE_PTR(topk_idx);
  REQUIRE_PTR(topk_prob);
  REQUIRE_PTR(expert_offsets);
  REQUIRE_PTR(row_of_slot);
  REQUIRE_PTR(token_of_row);
  REQUIRE_PTR(x_perm_q);
  REQUIRE_PTR(x_bscale_perm);
  REQUIRE_PTR(x_rscale_perm);
  REQUIRE_PTR(prob_perm);
  REQUIRE_PTR(ws);
  if (ws_bytes < ws_perm(d)) return MOE_ERR_WORKSPACE;
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(launch_permutation(c, topk_idx, topk_prob, d.T, d.K, d.E, expert_offsets, row_of_slot, token_of_row,
                              prob_perm, ws));
  TRY_CUDA(launch_dispatch_nvfp4(c, x, row_of_slot, d.T, d.K, d.D, x_perm_q, x_bscale_perm, x_rscale_perm));
  return MOE_OK;
}

int moe_dequant_nvfp4(const moe_shape_t* shape, const void* x_perm_q, const uint8_t* x_bscale_perm,
                      const float* x_rscale_perm, void* x_perm, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  if (d.dt != DType::BF16) return MOE_ERR_UNSUPPORTED;
  REQUIRE_PTR(x_perm_q);
  REQUIRE_PTR(x_bscale_perm);
  REQUIRE_PTR(x_rscale_perm);
  REQUIRE_PTR(x_perm);
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(launch_dequant_nvfp4(c, x_perm_q, x_bscale_perm, x_rscale_perm, d.TK, d.D, x_perm));
  return MOE_OK;
}

// The expert FFN with GEMM-1's A rows either read in order (x_rows = x_perm,
// gather = NULL) or gathered from the dispatch input (x_rows = x [T, D],
// gather = token_of_row).
static int expert_ffn_impl(const Ctx& c, const Dims& d, const void* x_rows, const int32_t* gather,
                           const int32_t* expert_offsets, const void* w1, const void* w2, void* h_save,
                           void* act_save, void* y_perm) {
  if (d.TK == 0) return MOE_OK;
  // GEMM-1 + fused SwiGLU: h = x_perm . w1_e^T, a = silu(g) * u
  GemmDesc g1;
  g1.group = Group::M;
  g1.epi = Epi::SwigluFwd;
  g1.N = 2 * d.F;
  g1.K = d.D;
  g1.num_groups = d.E;
  g1.offsets = expert_offsets;
  g1.max_rows = d.TK;
  g1.A = x_rows;
  g1.a_type = d.dt;
  g1.sa_m = d.D;
  g1.sa_k = 1;
  g1.gather = gather;
  g1.gather_rows = d.T;
  g1.B = w1;
  g1.b_type = d.dt;
  g1.sb_n = d.D;
  g1.sb_k = 1;
  g1.sb_g = (int64_t)2 * d.F * d.D;
  g1.C = h_save;
  g1.c_type = d.dt;
  g1.ldc = 2 * d.F;
  g1.aux = act_save;
  TRY_CUDA(gemm(c, g1, "ffn1_swiglu_tc", "ffn1_swiglu_simt"));
  // GEMM-2: y_perm = a . w2_e^T
  GemmDesc g2;
  g2.group = Group::M;
  g2.epi = Epi::Store;
  g2.N = d.D;
  g2.K = d.F;
  g2.num_groups = d.E;
  g2.offsets = expert_offsets;
  g2.max_rows = d.TK;
  g2.A = act_save;
  g2.a_type = d.dt;
  g2.sa_m = d.F;
  g2.sa_k = 1;
  g2.B = w2;
  g2.b_type = d.dt;
  g2.sb_n = d.F;
  g2.sb_k = 1;
  g2.sb_g = (int64_t)d.D * d.F;
  g2.C = y_perm;
  g2.c_type = d.dt;
  g2.ldc = d.D;
  TRY_CUDA(gemm(c, g2, "ffn2_tc", "ffn2_simt"));
  return MOE_OK;
}

int moe_expert_ffn(const moe_shape_t* shape, const void* x_perm, const int32_t* expert_offsets, const void* w1,
                   const void* w2, void* h_save, void* act_save, void* y_perm, void* ws, size_t ws_bytes,
                   void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(x_perm);
  REQUIRE_PTR(expert_offsets);
  REQUIRE_PTR(w1);
  REQUIRE_PTR(w2);
  REQUIRE_PTR(h_save);
  REQUIRE_PTR(act_save);
  REQUIRE_PTR(y_perm);
  (void)ws;
  (void)ws_bytes;
  Ctx c;
  TRY(get_ctx(stream, &c));
  return expert_ffn_impl(c, d, x_perm, nullptr, expert_offsets, w1, w2, h_save, act_save, y_perm);
}

int moe_expert_ffn_gather(const moe_shape_t* shape, const void* x, const int32_t* token_of_row,
                          const int32_t* expert_offsets, const void* w1, const void* w2, void* h_save,
                          void* act_save, void* y_perm, void* ws, size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(x);
  REQUIRE_PTR(token_of_row);
  REQUIRE_PTR(expert_offsets);
  REQUIRE_PTR(w1);
  REQUIRE_PTR(w2);
  REQUIRE_PTR(h_save);
  REQUIRE_PTR(act_save);
  REQUIRE_PTR(y_perm);
  (void)ws;
  (void)ws_bytes;
  Ctx c;
  TRY(get_ctx(stream, &c));
  return expert_ffn_impl(c, d, x, token_of_row, expert_offsets, w1, w2, h_save, act_save, y_perm);
}

int moe_combine(const moe_shape_t* shape, const void* y_perm, const float* prob_perm, const int32_t* row_of_slot,
                void* y, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(y_perm);
  REQUIRE_PTR(prob_perm);
  REQUIRE_PTR(row_of_slot);
  REQUIRE_PTR(y);
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(launch_combine(c, d.dt, y_perm, prob_perm, row_of_slot, d.T, d.K, d.D, y));
  return MOE_OK;
}

int moe_combine_bwd(const moe_shape_t* shape, const void* dy, const void* y_perm, const float* prob_perm,
                    const int32_t* row_of_slot, void* dy_perm, float* dprob_perm, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(dy);
  REQUIRE_PTR(y_perm);
  REQUIRE_PTR(prob_perm);
  REQUIRE_PTR(row_of_slot);
  REQUIRE_PTR(dy_perm);
  REQUIRE_PTR(dprob_perm);
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(launch_combine_bwd(c, d.dt, dy, y_perm, prob_perm, row_of_slot, d.T, d.K, d.D, dy_perm, dprob_perm));
  return MOE_OK;
}

// Expert FFN backward; the weight gradient of GEMM-1 reads x_rows in order
// (x_perm, gather = NULL) or gathers them from x [T, D] by token_of_row.
static int expert_ffn_bwd_impl(const Ctx& c, const Dims& d, const void* dy_perm, const void* x_rows,
                               const int32_t* gather, const void* h_save, const void* act_save,
                               const int32_t* expert_offsets, const void* w1, const void* w2, void* dx_perm,
                               float* dw1, float* dw2, void* ws) {
  void* dH = ws;
  void* dA = static_cast<char*>(ws) + (size_t)d.TK * 2 * d.F * d.bx;
  void* maps = static_cast<char*>(ws) + ws_ffn_bwd_maps_offset(d);
  void* maps1 = static_cast<char*>(maps) + ws_ffn_bwd_maps_bytes(d);
  // dgrad-2: dA = dy_perm . w2_e, then the SwiGLU backward dA, h -> dH
  GemmDesc a;
  a.group = Group::M;
  a.epi = Epi::Store;
  a.N = d.F;
  a.K = d.D;
  a.num_groups = d.E;
  a.offsets = expert_offsets;
  a.max_rows = d.TK;
  a.A = dy_perm;
  a.a_type = d.dt;
  a.sa_m = d.D;
  a.sa_k = 1;
  a.B = w2;
  a.b_type = d.dt;
  a.sb_n = 1;
  a.sb_k = d.F;
  a.sb_g = (int64_t)d.D * d.F;
  a.C = dA;
  a.c_type = d.dt;
  a.ldc = d.F;
  // wgrad-2: dw2_e[d, f] = sum_rows dy_perm[r, d] a[r, f]
  GemmDesc b;
  b.group = Group::K;
  b.epi = Epi::Store;
  b.M = d.D;
  b.N = d.F;
  b.num_groups = d.E;
  b.offsets = expert_offsets;
  b.A = dy_perm;
  b.a_type = d.dt;
  b.sa_m = 1;
  b.sa_k = d.D;
  b.B = act_save;
  b.b_type = d.dt;
  b.sb_n = 1;
  b.sb_k = d.F;
  b.max_rows = d.TK;
  b.scratch = maps;
  b.C = dw2;
  b.c_type = DType::F32;
  b.ldc = d.F;
  b.sc_g = (int64_t)d.D * d.F;
  // dgrad-1: dx_perm = dH . w1_e
  GemmDesc cg;
  cg.group = Group::M;
  cg.epi = Epi::Store;
  cg.N = d.D;
  cg.K = 2 * d.F;
  cg.num_groups = d.E;
  cg.offsets = expert_offsets;
  cg.max_rows = d.TK;
  cg.A = dH;
  cg.a_type = d.dt;
  cg.sa_m = 2 * d.F;
  cg.sa_k = 1;
  cg.B = w1;
  cg.b_type = d.dt;
  cg.sb_n = 1;
  cg.sb_k = d.D;
  cg.sb_g = (int64_t)2 * d.F * d.D;
  cg.C = dx_perm;
  cg.c_type = d.dt;
  cg.ldc = d.D;
  // wgrad-1: dw1_e[j, d] = sum_rows dH[r, j] x_perm[r, d]
  GemmDesc w;
  w.group = Group::K;
  w.epi = Epi::Store;
  w.M = 2 * d.F;
  w.N = d.D;
  w.num_groups = d.E;
  w.offsets = expert_offsets;
  w.A = dH;
  w.a_type = d.dt;
  w.sa_m = 1;
  w.sa_k = 2 * d.F;
  w.B = x_rows;
  w.b_type = d.dt;
  w.sb_n = 1;
  w.sb_k = d.D;
  w.gather = gather;
  w.gather_rows = d.T;
  w.max_rows = d.TK;
  w.scratch = maps1;
  w.C = dw1;
  w.c_type = DType::F32;
  w.ldc = d.D;
  w.sc_g = (int64_t)2 * d.F * d.D;
  if (d.TK > 0) {
    // on the tensor-core engine the SwiGLU backward runs in dgrad-2's epilogue
    // (dA stays in TMEM: h in, dH out); otherwise as a separate pass over dA
    GemmDesc af = a;
    af.epi = Epi::SwigluBwd;
    af.aux = const_cast<void*>(h_save);
    af.C = dH;
    af.ldc = 2 * d.F;
    if (gemm_tc_supports(af)) {
      TRY_CUDA(launch_gemm_tc(c, af, "ffn2_dgrad_swiglu_tc"));
    } else {
      TRY_CUDA(gemm(c, a, "ffn2_dgrad_tc", "ffn2_dgrad_simt"));
      TRY_CUDA(launch_swiglu_bwd(c, d.dt, dA, h_save, d.TK, d.F, dH));
    }
  }
  // both weight gradients' tail maps in one launch (each GEMM builds its own
  // if they are not both on the tensor-core engine)
  cudaError_t maps_st = cudaSuccess;
  if (gemm_tc_group_maps_pair(c, b, w, &maps_st)) {
    TRY_CUDA(maps_st);
    b.maps_ready = w.maps_ready = true;
  }
  TRY_CUDA(gemm(c, b, "ffn2_wgrad_tc", "ffn2_wgrad_simt"));
  TRY_CUDA(gemm(c, w, "ffn1_wgrad_tc", "ffn1_wgrad_simt"));
  // dgrad-1 last: the dispatch backward that follows reads its output while
  // part of it is still in L2 (the weight gradients' fp32 writes would flush it)
  if (d.TK > 0) TRY_CUDA(gemm(c, cg, "ffn1_dgrad_tc", "ffn1_dgrad_simt"));
  return MOE_OK;
}

int moe_expert_ffn_bwd(const moe_shape_t* shape, const void* dy_perm, const void* x_perm, const void* h_save,
                       const void* act_save, const int32_t* expert_offsets, const void* w1, const void* w2,
                       void* dx_perm, float* dw1, float* dw2, void* ws, size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(dy_perm);
  REQUIRE_PTR(x_perm);
  REQUIRE_PTR(h_save);
  REQUIRE_PTR(act_save);
  REQUIRE_PTR(expert_offsets);
  REQUIRE_PTR(w1);
  REQUIRE_PTR(w2);
  REQUIRE_PTR(dx_perm);
  REQUIRE_PTR(dw1);
  REQUIRE_PTR(dw2);
  REQUIRE_PTR(ws);
  if (ws_bytes < ws_ffn_bwd(d)) return MOE_ERR_WORKSPACE;
  Ctx c;
  TRY(get_ctx(stream, &c));
  return expert_ffn_bwd_impl(c, d, dy_perm, x_perm, nullptr, h_save, act_save, expert_offsets, w1, w2, dx_perm,
                             dw1, dw2, ws);
}

int moe_expert_ffn_bwd_gather(const moe_shape_t* shape, const void* dy_perm, const void* x,
                              const int32_t* token_of_row, const void* h_save, const void* act_save,
                              const int32_t* expert_offsets, const void* w1, const void* w2, void* dx_perm,
                              float* dw1, float* dw2, void* ws, size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(dy_perm);
  REQUIRE_PTR(x);
  REQUIRE_PTR(token_of_row);
  REQUIRE_PTR(h_save);
  REQUIRE_PTR(act_save);
  REQUIRE_PTR(expert_offsets);
  REQUIRE_PTR(w1);
  REQUIRE_PTR(w2);
  REQUIRE_PTR(dx_perm);
  REQUIRE_PTR(dw1);
  REQUIRE_PTR(dw2);
  REQUIRE_PTR(ws);
  if (ws_bytes < ws_ffn_bwd(d)) return MOE_ERR_WORKSPACE;
  Ctx c;
  TRY(get_ctx(stream, &c));
  return expert_ffn_bwd_impl(c, d, dy_perm, x, token_of_row, h_save, act_save, expert_offsets, w1, w2, dx_perm,
                             dw1, dw2, ws);
}

int moe_dispatch_bwd(const moe_shape_t* shape, const void* dx_perm, const float* dprob_perm,
                     const int32_t* row_of_slot, void* dx, float* dtopk_prob, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(dx_perm);
  REQUIRE_PTR(dprob_perm);
  REQUIRE_PTR(row_of_slot);
  REQUIRE_PTR(dx);
  REQUIRE_PTR(dtopk_prob);
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(launch_dispatch_bwd(c, d.dt, dx_perm, dprob_perm, row_of_slot, d.T, d.K, d.D, dx, dtopk_prob));
  return MOE_OK;
}

static GemmDesc dense_desc(Epi epi, int64_t M, int64_t N, int64_t K, const void* A, DType at, int64_t sa_m,
                           int64_t sa_k, const void* B, DType bt, int64_t sb_n, int64_t sb_k, void* C, DType ct,
                           int64_t ldc) {
  GemmDesc g;
  g.group = Group::Dense;
  g.epi = epi;
  g.M = M;
  g.N = N;
  g.K = K;
  g.A = A;
  g.a_type = at;
  g.sa_m = sa_m;
  g.sa_k = sa_k;
  g.B = B;
  g.b_type = bt;
  g.sb_n = sb_n;
  g.sb_k = sb_k;
  g.C = C;
  g.c_type = ct;
  g.ldc = ldc;
  return g;
}

// dx[T, Din] += dz . w_router and dw_router = dz^T . x, from dz [T, E] fp32 and
// (bf16 inputs) its bf16 copy dz16 (rows dz16_ld elements apart); scratch
// holds the weight gradient's split-K partials and tail maps.
static int router_grad_gemms(const Ctx& c, const Dims& d, const void* x, const void* w_router, const float* dlogits,
                             void* dx, float* dw_router, const void* dz16, int64_t dz16_ld, void* scratch,
                             bool dgrad = true) {
  // dx += dz . w_router   (M = T, N = Din, K = E)
  GemmDesc a;
  a.group = Group::Dense;
  a.epi = Epi::Accum;
  a.M = d.T;
  a.N = d.Din;
  a.K = d.E;
  a.A = dlogits;
  a.a_type = DType::F32;
  a.sa_m = d.E;
  a.sa_k = 1;
  a.B = w_router;
  a.b_type = d.dt;
  a.sb_n = 1;
  a.sb_k = d.Din;
  a.C = dx;
  a.c_type = d.dt;
  a.ldc = d.Din;
  // dw_router = dz^T . x   (M = E, N = Din, K = T)
  GemmDesc b;
  b.group = Group::Dense;
  b.epi = Epi::Store;
  b.M = d.E;
  b.N = d.Din;
  b.K = d.T;
  b.A = dlogits;
  b.a_type = DType::F32;
  b.sa_m = 1;
  b.sa_k = d.E;
  b.B = x;
  b.b_type = d.dt;
  b.sb_n = 1;
  b.sb_k = d.Din;
  b.C = dw_router;
  b.c_type = DType::F32;
  b.ldc = d.Din;
  if (d.dt == DType::BF16) {
    // tensor-core path reads the bf16 copy of dz
    GemmDesc a16 = a, b16 = b;
    a16.A = dz16;
    a16.a_type = DType::BF16;
    a16.sa_m = dz16_ld;
    b16.A = dz16;
    b16.a_type = DType::BF16;
    b16.sa_k = dz16_ld;
    if (gemm_tc_supports(a16)) a = a16;
    if (gemm_tc_supports(b16)) b = b16;
  }
  if (dgrad && d.T > 0) TRY_CUDA(gemm(c, a, "router_dgrad_tc", "router_dgrad_simt"));
  const int splits = d.dt == DType::BF16 ? router_splits(d, c.num_sms) : 1;
  if (splits > 1) {
    // split-K: partial products of token ranges of near-equal size that start
    // on 64-row boundaries, then their in-order sum
    GemmDesc bs = b;
    bs.group = Group::K;
    bs.num_groups = splits;
    bs.offsets = nullptr;
    bs.split_rows = d.T;
    bs.max_rows = d.T;
    bs.A = dz16;
    bs.a_type = DType::BF16;
    bs.C = scratch;
    bs.sc_g = (int64_t)d.E * d.Din;
    bs.scratch = static_cast<char*>(scratch) + ws_route_parts(d);
    if (gemm_tc_supports(bs)) {
      TRY_CUDA(launch_gemm_tc(c, bs, "router_wgrad_tc"));
      TRY_CUDA(launch_sum_splits(c, static_cast<const float*>(bs.C), splits, (int64_t)d.E * d.Din, dw_router));
      return MOE_OK;
    }
  }
  TRY_CUDA(gemm(c, b, "router_wgrad_tc", "router_wgrad_simt"));
  return MOE_OK;
}


int moe_route_bwd(const moe_shape_t* shape, const void* x, const void* w_router, const int32_t* topk_idx,
                  const float* topk_prob, const float* dtopk_prob, void* dx, float* dw_router, float* dlogits,
                  void* ws, size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(x);
  REQUIRE_PTR(w_router);
  REQUIRE_PTR(topk_idx);
  REQUIRE_PTR(topk_prob);
  REQUIRE_PTR(dtopk_prob);
  REQUIRE_PTR(dx);
  REQUIRE_PTR(dw_router);
  REQUIRE_PTR(dlogits);
  REQUIRE_PTR(ws);
  if (ws_bytes < ws_route_bwd(d)) return MOE_ERR_WORKSPACE;
  Ctx c;
  TRY(get_ctx(stream, &c));
  void* dz16 = d.dt == DType::BF16 ? ws : nullptr;
  TRY_CUDA(launch_route_dz(c, topk_idx, topk_prob, dtopk_prob, d.T, d.E, d.K, dlogits, dz16));
  return router_grad_gemms(c, d, x, w_router, dlogits, dx, dw_router, ws, d.E,
                           static_cast<char*>(ws) + ws_route_dz(d));
}

int moe_dispatch_route_bwd(const moe_shape_t* shape, const void* dx_perm, const float* dprob_perm,
                           const int32_t* row_of_slot, const void* x, const void* w_router, const int32_t* topk_idx,
                           const float* topk_prob, void* dx, float* dtopk_prob, float* dlogits, float* dw_router,
                           void* ws, size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  if (d.H) return MOE_ERR_UNSUPPORTED;  // the router reads x [T, H], the dispatch x_lat [T, D]
  REQUIRE_PTR(dx_perm);
  REQUIRE_PTR(dprob_perm);
  REQUIRE_PTR(row_of_slot);
  REQUIRE_PTR(x);
  REQUIRE_PTR(w_router);
  REQUIRE_PTR(topk_idx);
  REQUIRE_PTR(topk_prob);
  REQUIRE_PTR(dx);
  REQUIRE_PTR(dtopk_prob);
  REQUIRE_PTR(dlogits);
  REQUIRE_PTR(dw_router);
  REQUIRE_PTR(ws);
  if (ws_bytes < ws_route_bwd(d)) return MOE_ERR_WORKSPACE;
  Ctx c;
  TRY(get_ctx(stream, &c));
  void* dz16 = d.dt == DType::BF16 ? ws : nullptr;
  TRY_CUDA(launch_dispatch_route_bwd(c, d.dt, dx_perm, dprob_perm, row_of_slot, topk_idx, topk_prob, w_router, d.T,
                                     d.K, d.E, d.D, dx, dtopk_prob, dlogits, dz16));
  return router_grad_gemms(c, d, x, w_router, dlogits, dx, dw_router, ws, d.E,
                           static_cast<char*>(ws) + ws_route_dz(d), /*dgrad=*/false);
}

int moe_latent_route_bwd(const moe_shape_t* shape, const void* dx_perm, const float* dprob_perm,
                         const int32_t* row_of_slot, const void* x, const void* w_down_router,
                         const int32_t* topk_idx, const float* topk_prob, void* dx_cat, void* dx,
                         float* dtopk_prob, float* dlogits, float* dw_down, float* dw_router, void* ws,
                         size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  if (!d.H || d.dt != DType::BF16 || (d.D + d.E) % 8) return MOE_ERR_UNSUPPORTED;
  REQUIRE_PTR(dx_perm);
  REQUIRE_PTR(dprob_perm);
  REQUIRE_PTR(row_of_slot);
  REQUIRE_PTR(x);
  REQUIRE_PTR(w_down_router);
  REQUIRE_PTR(topk_idx);
  REQUIRE_PTR(topk_prob);
  REQUIRE_PTR(dx_cat);
  REQUIRE_PTR(dx);
  REQUIRE_PTR(dtopk_prob);
  REQUIRE_PTR(dlogits);
  REQUIRE_PTR(dw_down);
  REQUIRE_PTR(dw_router);
  REQUIRE_PTR(ws);
  if (ws_bytes < ws_route_bwd(d)) return MOE_ERR_WORKSPACE;
  Ctx c;
  TRY(get_ctx(stream, &c));
  const int64_t ldk = d.D + d.E;                   // row length of [dx_lat | dz16]
  bf16* cat = static_cast<bf16*>(dx_cat);
  void* scratch = ws;
  const bf16* w_router = static_cast<const bf16*>(w_down_router) + (int64_t)d.D * d.H;
  TRY_CUDA(launch_dispatch_bwd(c, d.dt, dx_perm, dprob_perm, row_of_slot, d.T, d.K, d.D, cat, dtopk_prob, ldk));
  TRY_CUDA(launch_route_dz(c, topk_idx, topk_prob, dtopk_prob, d.T, d.E, d.K, dlogits, cat + d.D, ldk));
  if (d.T > 0) {
    // dx = dx_lat . w_down + dz . w_router   (M = T, N = H, K = D + E, one rounding)
    GemmDesc a = dense_desc(Epi::Store, d.T, d.H, ldk, cat, d.dt, ldk, 1, w_down_router, d.dt, 1, d.H, dx, d.dt,
                            d.H);
    TRY_CUDA(gemm(c, a, "latent_dgrad_tc", "latent_dgrad_simt"));
  }
  // dw_down = dx_lat^T . x   (M = D, N = H, K = T)
  GemmDesc b = dense_desc(Epi::Store, d.D, d.H, d.T, cat, d.dt, 1, ldk, x, d.dt, 1, d.H, dw_down, DType::F32, d.H);
  TRY_CUDA(gemm(c, b, "latent_wgrad_tc", "latent_wgrad_simt"));
  return router_grad_gemms(c, d, x, w_router, dlogits, dx, dw_router, cat + d.D, ldk, scratch, /*dgrad=*/false);
}

int moe_route_sigmoid(const moe_shape_t* shape, const void* x, const void* w_router, const float* expert_bias,
                      float aux_coef, float* logits, int32_t* topk_idx, float* topk_prob, float* aux_f,
                      float* aux_loss, void* ws, size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(x);
  REQUIRE_PTR(w_router);
  OPTIONAL_PTR(expert_bias);
  REQUIRE_PTR(logits);
  REQUIRE_PTR(topk_idx);
  REQUIRE_PTR(topk_prob);
  REQUIRE_PTR(aux_f);
  REQUIRE_PTR(aux_loss);
  REQUIRE_PTR(ws);
  if (ws_bytes < ws_route_sigmoid(d)) return MOE_ERR_WORKSPACE;
  if (!(aux_coef == aux_coef)) return MOE_ERR_SHAPE;
  Ctx c;
  TRY(get_ctx(stream, &c));
  GemmDesc g;
  g.group = Group::Dense;
  g.epi = Epi::StoreBias;  // with no bias: the instantiated fp32-output router GEMM
  g.M = d.T;
  g.N = d.E;
  g.K = d.Din;
  g.A = x;
  g.a_type = d.dt;
  g.sa_m = d.Din;
  g.sa_k = 1;
  g.B = w_router;
  g.b_type = d.dt;
  g.sb_n = d.Din;
  g.sb_k = 1;
  g.C = logits;
  g.c_type = DType::F32;
  g.ldc = d.E;
  TRY_CUDA(gemm(c, g, "router_gemm_tc", "router_gemm_simt"));
  TRY_CUDA(launch_route_sigmoid_select(c, logits, expert_bias, d.T, d.S, d.GBS, d.E, d.K, aux_coef, topk_idx,
                                       topk_prob, aux_f, aux_loss, ws));
  return MOE_OK;
}

int moe_topk_sigmoid(const moe_shape_t* shape, const float* logits, const float* expert_bias, float aux_coef,
                     float* select_keys, int32_t* topk_idx, float* topk_prob, float* aux_f, float* aux_loss, void* ws,
                     size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(logits);
  OPTIONAL_PTR(expert_bias);
  OPTIONAL_PTR(select_keys);
  REQUIRE_PTR(topk_idx);
  REQUIRE_PTR(topk_prob);
  REQUIRE_PTR(aux_f);
  REQUIRE_PTR(aux_loss);
  REQUIRE_PTR(ws);
  if (ws_bytes < ws_route_sigmoid(d)) return MOE_ERR_WORKSPACE;
  if (!(aux_coef == aux_coef)) return MOE_ERR_SHAPE;
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(launch_route_sigmoid_select(c, logits, expert_bias, d.T, d.S, d.GBS, d.E, d.K, aux_coef, topk_idx,
                                       topk_prob, aux_f, aux_loss, ws, select_keys));
  return MOE_OK;
}

int moe_route_sigmoid_bwd(const moe_shape_t* shape, const void* x, const void* w_router, const float* logits,
                          const int32_t* topk_idx, const float* topk_prob, const float* dtopk_prob,
                          const float* aux_f, float aux_coef, float aux_grad, void* dx, float* dw_router,
                          float* dlogits, void* ws, size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(x);
  REQUIRE_PTR(w_router);
  REQUIRE_PTR(logits);
  REQUIRE_PTR(topk_idx);
  REQUIRE_PTR(topk_prob);
  REQUIRE_PTR(dtopk_prob);
  REQUIRE_PTR(aux_f);
  REQUIRE_PTR(dx);
  REQUIRE_PTR(dw_router);
  REQUIRE_PTR(dlogits);
  REQUIRE_PTR(ws);
  if (ws_bytes < ws_route_bwd(d)) return MOE_ERR_WORKSPACE;
  if (!(aux_coef == aux_coef) || !(aux_grad == aux_grad)) return MOE_ERR_SHAPE;
  Ctx c;
  TRY(get_ctx(stream, &c));
  void* dz16 = d.dt == DType::BF16 ? ws : nullptr;
  TRY_CUDA(launch_route_dz_sigmoid(c, logits, topk_idx, topk_prob, dtopk_prob, aux_f, d.T, d.S, d.GBS, d.E, d.K,
                                   aux_coef, aux_grad, dlogits, dz16));
  return router_grad_gemms(c, d, x, w_router, dlogits, dx, dw_router, ws, d.E,
                           static_cast<char*>(ws) + ws_route_dz(d));
}

int moe_latent_proj(const moe_shape_t* shape, int32_t n_in, int32_t n_out, const void* in, const void* w,
                    void* out, void* ws, size_t ws_bytes, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  if (n_in <= 0 || n_out <= 0 || n_in % 64 || n_out % 64) return MOE_ERR_SHAPE;
  REQUIRE_PTR(in);
  REQUIRE_PTR(w);
  REQUIRE_PTR(out);
  (void)ws;
  (void)ws_bytes;
  Ctx c;
  TRY(get_ctx(stream, &c));
  GemmDesc g;
  g.group = Group::Dense;
  g.epi = Epi::Store;
  g.M = d.T;
  g.N = n_out;
  g.K = n_in;
  g.A = in;
  g.a_type = d.dt;
  g.sa_m = n_in;
  g.sa_k = 1;
  g.B = w;
  g.b_type = d.dt;
  g.sb_n = n_in;
  g.sb_k = 1;
  g.C = out;
  g.c_type = d.dt;
  g.ldc = n_out;
  if (d.T > 0) TRY_CUDA(gemm(c, g, "latent_fwd_tc", "latent_fwd_simt"));
  return MOE_OK;
}

int moe_latent_proj_bwd(const moe_shape_t* shape, int32_t n_in, int32_t n_out, const void* dout, const void* in,
                        const void* w, void* din, int32_t accumulate, float* dw, void* ws, size_t ws_bytes,
                        void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  if (n_in <= 0 || n_out <= 0 || n_in % 64 || n_out % 64) return MOE_ERR_SHAPE;
  REQUIRE_PTR(dout);
  REQUIRE_PTR(in);
  REQUIRE_PTR(w);
  REQUIRE_PTR(dw);
  OPTIONAL_PTR(din);
  (void)ws;
  (void)ws_bytes;
  Ctx c;
  TRY(get_ctx(stream, &c));
  if (din && d.T > 0) {
    // din = dout . w   (M = T, N = n_in, K = n_out)
    GemmDesc a;
    a.group = Group::Dense;
    a.epi = accumulate ? Epi::Accum : Epi::Store;
    a.M = d.T;
    a.N = n_in;
    a.K = n_out;
    a.A = dout;
    a.a_type = d.dt;
    a.sa_m = n_out;
    a.sa_k = 1;
    a.B = w;
    a.b_type = d.dt;
    a.sb_n = 1;
    a.sb_k = n_in;
    a.C = din;
    a.c_type = d.dt;
    a.ldc = n_in;
    TRY_CUDA(gemm(c, a, "latent_dgrad_tc", "latent_dgrad_simt"));
  }
  // dw = dout^T . in   (M = n_out, N = n_in, K = T)
  GemmDesc b;
  b.group = Group::Dense;
  b.epi = Epi::Store;
  b.M = n_out;
  b.N = n_in;
  b.K = d.T;
  b.A = dout;
  b.a_type = d.dt;
  b.sa_m = 1;
  b.sa_k = n_out;
  b.B = in;
  b.b_type = d.dt;
  b.sb_n = 1;
  b.sb_k = n_in;
  b.C = dw;
  b.c_type = DType::F32;
  b.ldc = n_in;
  TRY_CUDA(gemm(c, b, "latent_wgrad_tc", "latent_wgrad_simt"));
  return MOE_OK;
}

// A dense C(m, n) = sum_k A(m, k) B(n, k) descriptor (element strides).

int moe_shared_expert(const moe_shape_t* shape, int32_t F_s, const void* x, const void* w_s1, const void* w_s2,
                      void* h_save, void* act_save, void* y, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  if (F_s <= 0 || F_s % 64) return MOE_ERR_SHAPE;
  REQUIRE_PTR(x);
  REQUIRE_PTR(w_s1);
  REQUIRE_PTR(w_s2);
  REQUIRE_PTR(h_save);
  REQUIRE_PTR(act_save);
  REQUIRE_PTR(y);
  Ctx c;
  TRY(get_ctx(stream, &c));
  // h = x . w_s1^T, a = relu(h)^2   (M = T, N = F_s, K = Din)
  GemmDesc g1 = dense_desc(Epi::ReluSqFwd, d.T, F_s, d.Din, x, d.dt, d.Din, 1, w_s1, d.dt, d.Din, 1, h_save, d.dt,
                           F_s);
  g1.aux = act_save;
  TRY_CUDA(gemm(c, g1, "shared_fc1_tc", "shared_fc1_simt"));
  // y += a . w_s2^T   (M = T, N = Din, K = F_s)
  GemmDesc g2 = dense_desc(Epi::Accum, d.T, d.Din, F_s, act_save, d.dt, F_s, 1, w_s2, d.dt, F_s, 1, y, d.dt, d.Din);
  TRY_CUDA(gemm(c, g2, "shared_fc2_tc", "shared_fc2_simt"));
  return MOE_OK;
}

int moe_shared_expert_bwd(const moe_shape_t* shape, int32_t F_s, const void* dy, const void* x, const void* h_save,
                          const void* act_save, const void* w_s1, const void* w_s2, void* dh, void* dx, float* dw_s1,
                          float* dw_s2, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  if (F_s <= 0 || F_s % 64) return MOE_ERR_SHAPE;
  REQUIRE_PTR(dy);
  REQUIRE_PTR(x);
  REQUIRE_PTR(h_save);
  REQUIRE_PTR(act_save);
  REQUIRE_PTR(w_s1);
  REQUIRE_PTR(w_s2);
  REQUIRE_PTR(dh);
  REQUIRE_PTR(dx);
  REQUIRE_PTR(dw_s1);
  REQUIRE_PTR(dw_s2);
  Ctx c;
  TRY(get_ctx(stream, &c));
  // dA = dy . w_s2   (M = T, N = F_s, K = Din), into dh
  GemmDesc a = dense_desc(Epi::Store, d.T, F_s, d.Din, dy, d.dt, d.Din, 1, w_s2, d.dt, 1, F_s, dh, d.dt, F_s);
  TRY_CUDA(gemm(c, a, "shared_fc2_dgrad_tc", "shared_fc2_dgrad_simt"));
  // dh = 2 relu(h) dA, in place
  TRY_CUDA(launch_relusq_bwd(c, d.dt, dh, h_save, d.T * (int64_t)F_s, dh));
  // dx += dh . w_s1   (M = T, N = Din, K = F_s)
  GemmDesc b = dense_desc(Epi::Accum, d.T, d.Din, F_s, dh, d.dt, F_s, 1, w_s1, d.dt, 1, d.Din, dx, d.dt, d.Din);
  TRY_CUDA(gemm(c, b, "shared_fc1_dgrad_tc", "shared_fc1_dgrad_simt"));
  // dw_s2 = dy^T . a   (M = Din, N = F_s, K = T)
  GemmDesc w2 = dense_desc(Epi::Store, d.Din, F_s, d.T, dy, d.dt, 1, d.Din, act_save, d.dt, 1, F_s, dw_s2,
                           DType::F32, F_s);
  TRY_CUDA(gemm(c, w2, "shared_fc2_wgrad_tc", "shared_fc2_wgrad_simt"));
  // dw_s1 = dh^T . x   (M = F_s, N = Din, K = T)
  GemmDesc w1 = dense_desc(Epi::Store, F_s, d.Din, d.T, dh, d.dt, 1, F_s, x, d.dt, 1, d.Din, dw_s1, DType::F32,
                           d.Din);
  TRY_CUDA(gemm(c, w1, "shared_fc1_wgrad_tc", "shared_fc1_wgrad_simt"));
  return MOE_OK;
}

int moe_pack_w1(const moe_shape_t* shape, const void* w_gate, const void* w_up, void* w1, void* stream) {
  Dims d;
  TRY(check_shape(shape, &d));
  REQUIRE_PTR(w_gate);
  REQUIRE_PTR(w_up);
  REQUIRE_PTR(w1);
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(launch_pack_w1(c, d.dt, w_gate, w_up, d.E, d.F, d.D, w1));
  return MOE_OK;
}

int moe_device_status_word(void* stream, uint32_t* word) {
  if (!word) return MOE_ERR_NULL;
  Ctx c;
  TRY(get_ctx(stream, &c));
  TRY_CUDA(cudaStreamSynchronize(c.stream));
  TRY_CUDA(cudaMemcpy(word, c.err, sizeof(uint32_t), cudaMemcpyDeviceToHost));
  return MOE_OK;
}

int moe_check_device_status(void* stream) {
  uint32_t w = 0;
  TRY(moe_device_status_word(stream, &w));
  if (w) {
    Ctx c;
    TRY(get_ctx(stream, &c));
    TRY_CUDA(cudaMemsetAsync(c.err, 0, sizeof(uint32_t), c.stream));
    TRY_CUDA(cudaStreamSynchronize(c.stream));
    return MOE_ERR_DEVICE;
  }
  return MOE_OK;
}

int moe_prof_enable(int on) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (on && g_event_pool.empty()) {
    for (int i = 0; i < 1024; ++i) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) break;
      g_event_pool.push_back(e);
    }
  }
  g_prof_on.store(on != 0);
  return MOE_OK;
}

int moe_prof_reset(void) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  prof_harvest();
  g_prof.clear();
  return MOE_OK;
}

int moe_prof_count(void) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  return (int)g_prof.size();
}

int moe_prof_get(int i, const char** name, int* launches, double* total_ms) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  prof_harvest();
  if (i < 0 || i >= (int)g_prof.size()) return MOE_ERR_SHAPE;
  if (name) *name = g_prof[i].name.c_str();
  if (launches) *launches = g_prof[i].launches;
  if (total_ms) *total_ms = g_prof[i].total_ms;
  return MOE_OK;
}

}  // extern "C"
