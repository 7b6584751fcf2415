// Host side of the tcgen05 engine: which GemmDesc shapes it takes, tensor-map
// encoding (cuTensorMapEncodeTiled through the runtime's driver entry point)
// and the launch of the matching kernel instantiation.
#include <array>
#include <cstring>
#include <map>
#include <memory>
#include <mutex>

#include "gemm_tc.cuh"

namespace moe {

using tc::BM;
using tc::Cfg;
using tc::Params;

namespace {

using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn encode_fn() {
  static EncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(ptr);
  });
  return fn;
}

// 2-D bf16 tensor map: `inner` contiguous elements per row, `outer` rows of
// `stride_bytes`, box {box_inner, box_outer}, 128-byte swizzle, zero fill.
bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t stride_bytes,
              uint32_t box_inner, uint32_t box_outer) {
  EncodeFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {stride_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool al16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

// Group::K tail templates, one per row count r = 1 .. BK - 1, for MN-major A
// (and B unless B is gathered) with {64, 64} boxes.  They depend only on the
// operands' row length and stride (the device replaces the base address), so
// each combination is encoded once and kept for the life of the process.
const tc::TailTemplates* tail_templates(const void* a, int64_t a_inner, int64_t a_stride, const void* b,
                                        int64_t b_inner, int64_t b_stride) {
  static std::mutex mu;
  static std::map<std::array<int64_t, 5>, std::unique_ptr<tc::TailTemplates>> cache;
  const std::array<int64_t, 5> key = {a_inner, a_stride, b ? b_inner : -1, b ? b_stride : -1, 0};
  std::lock_guard<std::mutex> lk(mu);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second.get();
  auto t = std::make_unique<tc::TailTemplates>();
  memset(t.get(), 0, sizeof(tc::TailTemplates));
  for (int r = 1; r < tc::BK; ++r) {
    if (!make_map(&t->a[r], a, a_inner, r, a_stride, 64, 64)) return nullptr;
    if (b && !make_map(&t->b[r], b, b_inner, r, b_stride, 64, 64)) return nullptr;
  }
  const tc::TailTemplates* out = t.get();
  cache.emplace(key, std::move(t));
  return out;
}

struct Plan {
  int bn;
  int cg;  // CTAs per tile: 2 (a cluster pair, 256-row tiles) or 1 (128-row tiles)
  bool a_mn, b_mn;
  int64_t lda, ldb;
};

bool make_plan(const GemmDesc& d, Plan* pl) {
  if (d.a_type != DType::BF16 || d.b_type != DType::BF16) return false;
  if (d.N <= 0 || (d.group != Group::M && d.M <= 0) || (d.group != Group::K && d.K <= 0)) return false;
  if (d.sa_k == 1 && d.sa_m > 1) { pl->a_mn = false; pl->lda = d.sa_m; }
  else if (d.sa_m == 1 && d.sa_k > 1) { pl->a_mn = true; pl->lda = d.sa_k; }
  else return false;
  if (d.sb_k == 1 && d.sb_n > 1) { pl->b_mn = false; pl->ldb = d.sb_n; }
  else if (d.sb_n == 1 && d.sb_k > 1) { pl->b_mn = true; pl->ldb = d.sb_k; }
  else return false;
  if ((pl->lda * 2) % 16 || (pl->ldb * 2) % 16) return false;
  if (!al16(d.A) || !al16(d.B) || !al16(d.C)) return false;
  if (d.group == Group::K && !(pl->a_mn && pl->b_mn)) return false;
  if (d.group == Group::K && (!d.scratch || ((uintptr_t)d.scratch & 127u) || d.max_rows <= 0)) return false;
  if (d.group == Group::K && !d.offsets && d.split_rows <= 0) return false;
  if (d.group == Group::M && pl->a_mn) return false;
  if (d.group == Group::M && (d.sb_g % pl->ldb)) return false;
  if (d.group != Group::Dense && (d.num_groups <= 0 || d.num_groups > kMaxE)) return false;
  if (d.group == Group::M && !d.offsets) return false;
  if (d.gather) {
    // gathered operand: K-major A of Group::M or MN-major B of Group::K
    if (d.gather_rows <= 0 || d.group == Group::Dense) return false;
    if (d.group == Group::M && pl->a_mn) return false;
  }
  const size_t cs = dsize(d.c_type);
  if ((d.ldc * cs) % 16) return false;
  switch (d.epi) {
    case Epi::Store: break;
    case Epi::StoreBias: if (d.c_type != DType::F32) return false; break;
    case Epi::Accum: if (d.c_type != DType::BF16 || d.N % 64) return false; break;
    case Epi::SwigluFwd:
      if (d.c_type != DType::BF16 || d.N % 128 || !d.aux || !al16(d.aux)) return false;
      break;
    case Epi::ReluSqFwd:
      if (d.c_type != DType::BF16 || d.N % 64 || !d.aux || !al16(d.aux)) return false;
      break;
    case Epi::SwigluBwd:
      if (d.c_type != DType::BF16 || d.N % 64 || !d.aux || !al16(d.aux) || d.ldc != 2 * d.N) return false;
      break;
  }
  pl->bn = 256;
  pl->cg = 1;
  if (d.group == Group::Dense && d.epi == Epi::StoreBias) {
    pl->bn = d.N <= 64 ? 64 : (d.N <= 128 ? 128 : 256);  // router logits: N = E
  } else if (d.group == Group::M || d.M > BM) {
    pl->cg = 2;
  }
  return true;
}

// Co-resident 2-CTA clusters of an instantiation (0 if the query fails).
template <typename KernelT>
int max_pair_clusters(KernelT k, int smem, int threads) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2, 1, 1);
  cfg.blockDim = dim3(threads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, k, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

// ub = upper bound on the number of tiles (each tile is one CTA, or one pair for CG 2).
template <int BN, bool A_MN, bool B_MN, int GROUP, int EPI, typename TC, int CG, int GATHER = 0>
cudaError_t launch_inst(const Ctx& c, const Params& p, int64_t ub) {
  auto k = tc::gemm_tc_kernel<BN, A_MN, B_MN, GROUP, EPI, TC, CG, GATHER>;
  constexpr int kZW = (GROUP == 2 && sizeof(TC) == 4 && GATHER == 0) ? 1 : 0;
  constexpr int kSmem = Cfg<BN, CG, sizeof(TC), EPI, kZW>::kSmem;
  constexpr int kThreads = Cfg<BN, CG, sizeof(TC), EPI, kZW>::kThreads;
  static bool configured = false;
  static int pairs = 0;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
    if (e != cudaSuccess) return e;
    if (CG == 2) {
      e = cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 0);
      (void)e;
      cudaGetLastError();
      pairs = max_pair_clusters(k, kSmem, kThreads);
    }
    configured = true;
  }
  if (CG == 1) {
    const int grid = (int)(ub < c.num_sms ? ub : c.num_sms);
    k<<<grid, kThreads, kSmem, c.stream>>>(p);
    return cudaGetLastError();
  }
  int np = pairs > 0 ? pairs : c.num_sms / 2;
  if (ub < np) np = (int)ub;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * np, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = kSmem;
  cfg.stream = c.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k, p);
}

}  // namespace

// {A, B} map per group, then (for equal splits) the group offsets.
size_t gemm_tc_group_scratch_bytes(int num_groups) {
  return (size_t)num_groups * 2 * sizeof(CUtensorMap) + (((size_t)num_groups + 1) * 4 + 127) / 128 * 128;
}

bool gemm_tc_supports(const GemmDesc& d) {
  Plan pl;
  if (!make_plan(d, &pl)) return false;
  const int g = (int)d.group, e = (int)d.epi;
  const bool f32 = d.c_type == DType::F32;
  if (d.gather) {
    if (g == 1 && !pl.b_mn && e == 3 && !f32 && pl.cg == 2) return true;  // GEMM-1 + SwiGLU from x
    if (g == 2 && e == 0 && f32) return true;                            // GEMM-1 weight gradient from x
    return false;
  }
  // the instantiated combinations
  if (g == 1 && !pl.a_mn && !pl.b_mn && e == 3 && !f32) return true;
  if (g == 1 && !pl.a_mn && !pl.b_mn && e == 0 && !f32) return true;
  if (g == 1 && !pl.a_mn && pl.b_mn && e == 0 && !f32) return true;
  if (g == 1 && !pl.a_mn && pl.b_mn && e == 5 && !f32) return true;
  if (g == 2 && pl.a_mn && pl.b_mn && e == 0 && f32) return true;
  if (g == 0 && !pl.a_mn && !pl.b_mn && e == 1 && f32) return true;
  if (g == 0 && !pl.a_mn && !pl.b_mn && (e == 0 || e == 2 || e == 4) && !f32) return true;
  if (g == 0 && !pl.a_mn && pl.b_mn && (e == 0 || e == 2) && !f32) return true;
  if (g == 0 && pl.a_mn && pl.b_mn && e == 0 && f32) return true;
  return false;
}

cudaError_t launch_gemm_tc(const Ctx& c, const GemmDesc& d, const char* name) {
  Plan pl;
  if (!make_plan(d, &pl) || !gemm_tc_supports(d)) return cudaErrorNotSupported;
  Params p;
  memset(&p, 0, sizeof(p));
  const int bn = pl.bn, bmp = BM * pl.cg, bnc = bn / pl.cg;
  // A: K-major box {64 k, 128 m}; MN-major box {64 m, 64 k}
  const bool ga = d.gather && d.group == Group::M;  // A's rows gathered (cp.async row copies; its map unused)
  const bool gb = d.gather && d.group == Group::K;  // B's k rows gathered (cp.async row copies; its map unused)
  int64_t a_rows = pl.a_mn ? (d.group == Group::K ? d.max_rows : d.K) : (d.group == Group::M ? d.max_rows : d.M);
  if (ga) a_rows = d.gather_rows;
  const int64_t a_inner = pl.a_mn ? d.M : d.K;
  if (!make_map(&p.ta, d.A, a_inner, a_rows, pl.lda * 2, 64, ga ? 1 : (pl.a_mn ? 64 : BM)))
    return cudaErrorInvalidValue;
  // B: K-major box {64 k, BN / CG n}; MN-major box {64 n, 64 k}
  const int64_t grows = d.group == Group::M ? d.sb_g / pl.ldb : 0;
  int64_t b_rows;
  if (pl.b_mn) b_rows = d.group == Group::M ? grows * d.num_groups : (d.group == Group::K ? d.max_rows : d.K);
  else b_rows = d.group == Group::M ? grows * d.num_groups : d.N;
  if (gb) b_rows = d.gather_rows;
  const int64_t b_inner = pl.b_mn ? d.N : d.K;
  if (!make_map(&p.tb, d.B, b_inner, b_rows, pl.ldb * 2, 64, gb ? 1 : (pl.b_mn ? 64 : bnc)))
    return cudaErrorInvalidValue;
  p.M = d.M;
  p.N = d.N;
  p.K = d.K;
  p.b_group_rows = grows;
  p.num_groups = d.group == Group::Dense ? 1 : d.num_groups;
  p.tiles_m = (int)((d.M + bmp - 1) / bmp);
  p.tiles_n = (int)((d.N + bn - 1) / bn);
  p.offsets = d.offsets;
  p.C = d.C;
  p.ldc = d.ldc;
  p.sc_g = d.sc_g;
  p.bias = d.bias;
  p.aux = d.aux;
  p.err = c.err;
  p.gather = d.gather;
  if (ga) {
    p.gsrc = static_cast<const uint8_t*>(d.A);
    p.gsrc_ld = pl.lda * 2;
    p.gsrc_rows = d.gather_rows;
  } else if (gb) {
    p.gsrc = static_cast<const uint8_t*>(d.B);
    p.gsrc_ld = pl.ldb * 2;
    p.gsrc_rows = d.gather_rows;
  }
  int64_t ub;
  if (d.group == Group::Dense) ub = (int64_t)p.tiles_m * p.tiles_n;
  else if (d.group == Group::M) ub = ((d.max_rows + bmp - 1) / bmp + d.num_groups) * p.tiles_n;
  else ub = (int64_t)d.num_groups * p.tiles_m * p.tiles_n;
  if (ub <= 0) return cudaSuccess;
  const int g = (int)d.group, e = (int)d.epi;
  if (d.group == Group::K) {
    // tail maps: host-encoded templates of 1 .. BK - 1 rows, the base moved per group
    const tc::TailTemplates* tails = tail_templates(d.A, a_inner, pl.lda * 2, gb ? nullptr : d.B, b_inner, pl.ldb * 2);
    if (!tails) return cudaErrorInvalidValue;
    CUtensorMap* maps = static_cast<CUtensorMap*>(d.scratch);
    p.split_rows = d.offsets ? 0 : d.split_rows;
    // splits of a dense product start on k-block boundaries, so they need
    // tail maps only when the whole range ends inside a k-block
    if (!d.maps_ready && (d.offsets || d.split_rows % tc::BK != 0)) {
      KernelScope ks("group_maps", c.stream);
      tc::build_group_maps<<<(d.num_groups + tc::kMapWarps - 1) / tc::kMapWarps, 32 * tc::kMapWarps, 0, c.stream>>>(
          *tails, d.offsets, d.num_groups, d.split_rows, static_cast<const uint8_t*>(d.A), pl.lda * 2,
          gb ? nullptr : static_cast<const uint8_t*>(d.B), pl.ldb * 2, maps);
      cudaError_t st = cudaGetLastError();
      if (st != cudaSuccess) return st;
    }
    p.gmaps = maps;
  }
  KernelScope ks(name, c.stream);
  if (ga) return launch_inst<256, false, false, 1, 3, bf16, 2, 1>(c, p, ub);
  if (gb && pl.cg == 2) return launch_inst<256, true, true, 2, 0, float, 2, 2>(c, p, ub);
  if (gb) return launch_inst<256, true, true, 2, 0, float, 1, 2>(c, p, ub);
  if (pl.cg == 2) {
    if (g == 2) return launch_inst<256, true, true, 2, 0, float, 2>(c, p, ub);
    if (g == 1 && !pl.b_mn && e == 3) return launch_inst<256, false, false, 1, 3, bf16, 2>(c, p, ub);
    if (g == 1 && !pl.b_mn && e == 0) return launch_inst<256, false, false, 1, 0, bf16, 2>(c, p, ub);
    if (g == 1 && pl.b_mn && e == 0) return launch_inst<256, false, true, 1, 0, bf16, 2>(c, p, ub);
    if (g == 1 && pl.b_mn && e == 5) return launch_inst<256, false, true, 1, 5, bf16, 2>(c, p, ub);
    if (g == 0 && !pl.a_mn && !pl.b_mn && e == 0) return launch_inst<256, false, false, 0, 0, bf16, 2>(c, p, ub);
    if (g == 0 && !pl.a_mn && !pl.b_mn && e == 2) return launch_inst<256, false, false, 0, 2, bf16, 2>(c, p, ub);
    if (g == 0 && !pl.a_mn && !pl.b_mn && e == 4) return launch_inst<256, false, false, 0, 4, bf16, 2>(c, p, ub);
    if (g == 0 && !pl.a_mn && pl.b_mn && e == 0) return launch_inst<256, false, true, 0, 0, bf16, 2>(c, p, ub);
    if (g == 0 && !pl.a_mn && pl.b_mn && e == 2) return launch_inst<256, false, true, 0, 2, bf16, 2>(c, p, ub);
    if (g == 0 && pl.a_mn && pl.b_mn) return launch_inst<256, true, true, 0, 0, float, 2>(c, p, ub);
    return cudaErrorNotSupported;
  }
  if (g == 2) return launch_inst<256, true, true, 2, 0, float, 1>(c, p, ub);
  if (g == 0 && e == 1) {
    if (bn == 64) return launch_inst<64, false, false, 0, 1, float, 1>(c, p, ub);
    if (bn == 128) return launch_inst<128, false, false, 0, 1, float, 1>(c, p, ub);
    return launch_inst<256, false, false, 0, 1, float, 1>(c, p, ub);
  }
  if (g == 0 && !pl.a_mn && !pl.b_mn && e == 0) return launch_inst<256, false, false, 0, 0, bf16, 1>(c, p, ub);
  if (g == 0 && !pl.a_mn && !pl.b_mn && e == 2) return launch_inst<256, false, false, 0, 2, bf16, 1>(c, p, ub);
  if (g == 0 && !pl.a_mn && !pl.b_mn && e == 4) return launch_inst<256, false, false, 0, 4, bf16, 1>(c, p, ub);
  if (g == 0 && !pl.a_mn && pl.b_mn && e == 0) return launch_inst<256, false, true, 0, 0, bf16, 1>(c, p, ub);
  if (g == 0 && !pl.a_mn && pl.b_mn && e == 2) return launch_inst<256, false, true, 0, 2, bf16, 1>(c, p, ub);
  if (g == 0 && pl.a_mn && pl.b_mn) return launch_inst<256, true, true, 0, 0, float, 1>(c, p, ub);
  return cudaErrorNotSupported;
}

bool gemm_tc_group_maps_pair(const Ctx& c, const GemmDesc& d0, const GemmDesc& d1, cudaError_t* err) {
  *err = cudaSuccess;
  const GemmDesc* ds[2] = {&d0, &d1};
  Plan pl[2];
  const tc::TailTemplates* tails[2];
  for (int k = 0; k < 2; ++k) {
    const GemmDesc& d = *ds[k];
    if (d.group != Group::K || !d.offsets || !d.scratch || !make_plan(d, &pl[k]) || !gemm_tc_supports(d))
      return false;
    const bool gb = d.gather != nullptr;
    tails[k] = tail_templates(d.A, pl[k].a_mn ? d.M : d.K, pl[k].lda * 2, gb ? nullptr : d.B,
                              pl[k].b_mn ? d.N : d.K, pl[k].ldb * 2);
    if (!tails[k]) return false;
  }
  if (d0.offsets != d1.offsets || d0.num_groups != d1.num_groups || d0.num_groups <= 0) return false;
  static thread_local tc::TailTemplatesPair tt;  // 32 KB: not on the stack
  for (int k = 0; k < 2; ++k) {
    memcpy(tt.a[k], &tails[k]->a[1], sizeof(tt.a[k]));
    memcpy(tt.b[k], &tails[k]->b[1], sizeof(tt.b[k]));
  }
  const int G = d0.num_groups;
  auto bbase = [&](int k) {
    return ds[k]->gather ? nullptr : static_cast<const uint8_t*>(ds[k]->B);
  };
  KernelScope ks("group_maps", c.stream);
  tc::build_group_maps_pair<<<(2 * G + tc::kMapWarps - 1) / tc::kMapWarps, 32 * tc::kMapWarps, 0, c.stream>>>(
      tt, d0.offsets, G, static_cast<const uint8_t*>(d0.A), pl[0].lda * 2, bbase(0), pl[0].ldb * 2,
      static_cast<CUtensorMap*>(d0.scratch), static_cast<const uint8_t*>(d1.A), pl[1].lda * 2, bbase(1),
      pl[1].ldb * 2, static_cast<CUtensorMap*>(d1.scratch));
  *err = cudaGetLastError();
  return true;
}

}  // namespace moe
