// moe_dispatch_noalloc: the dispatch entry point for callers that cannot
// allocate device memory when they call it.
//
// Some callers have no way to hand the library a workspace: a host framework
// that has already reserved all device memory for its own pool, a step loop
// that forbids allocation, or a runtime that cannot afford cudaMalloc's
// implicit device-wide synchronisation.  For them the counting sort's scratch
// (the per-chunk expert histogram table) lives in a fixed array compiled into
// the library: every GPU that loads the library holds one copy of it until the
// process exits.  After the first call on a device (which loads this module
// there and looks up the array's address) the call allocates nothing.
#include <mutex>

#include "common.cuh"
#include "launch.h"

namespace moe {

// Scratch of the counting sort: E * ceil(T*K / 2048) int32 per-chunk counts
// (counts[e * nchunks + chunk]).
static __device__ __align__(256) int32_t g_dispatch_scratch[MOE_DISPATCH_NOALLOC_SCRATCH_INTS];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
int32_t* g_scratch_ptr[kMaxDevices] = {};

// Device address of this device's copy of the array.  In host code the name
// g_dispatch_scratch is only a host-side stand-in, so the address is looked up
// once per device, with that device current, and passed to the kernels.
int scratch_for_device(int dev, int32_t** out) {
  if (dev < 0 || dev >= kMaxDevices) return abi_cuda_status(cudaErrorInvalidDevice);
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_dispatch_scratch);
    if (e != cudaSuccess) return abi_cuda_status(e);
    g_scratch_ptr[dev] = static_cast<int32_t*>(p);
  }
  *out = g_scratch_ptr[dev];
  return MOE_OK;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

}  // namespace

}  // namespace moe

using namespace moe;

extern "C" int moe_dispatch_noalloc(const moe_shape_t* shape, const void* x, const int32_t* topk_idx,
                                    const float* topk_prob, int32_t* expert_offsets, int32_t* row_of_slot,
                                    int32_t* token_of_row, void* x_perm, float* prob_perm, void* stream) {
  ShapeInfo d;
  int st = abi_check_shape(shape, &d);
  if (st != MOE_OK) return st;
  const void* need[] = {topk_idx, topk_prob, expert_offsets, row_of_slot, token_of_row, prob_perm};
  for (const void* p : need) {
    if (!p) return MOE_ERR_NULL;
    if (!aligned16(p)) return MOE_ERR_ALIGN;
  }
  if (x_perm) {
    if (!x) return MOE_ERR_NULL;
    if (!aligned16(x_perm) || !aligned16(x)) return MOE_ERR_ALIGN;
  }
  // the counting sort's tables must fit the fixed array
  if (perm_workspace_bytes(d.TK, d.E) > sizeof(int32_t) * (size_t)MOE_DISPATCH_NOALLOC_SCRATCH_INTS)
    return MOE_ERR_TOO_LARGE;
  Ctx c;
  st = abi_device_ctx(stream, &c);
  if (st != MOE_OK) return st;
  int32_t* scratch = nullptr;
  st = scratch_for_device(c.device, &scratch);
  if (st != MOE_OK) return st;
  // Every table entry the kernels read is written earlier in the same call
  // (the histogram writes all E x chunks counts), so no clearing is needed.
  st = abi_cuda_status(launch_permutation(c, topk_idx, topk_prob, d.T, d.K, d.E, expert_offsets, row_of_slot,
                                          token_of_row, prob_perm, scratch));
  if (st != MOE_OK) return st;
  if (x_perm)
    st = abi_cuda_status(launch_dispatch_rows(c, x, row_of_slot, d.T, d.K, (int64_t)d.D * d.bx, x_perm));
  return st;
}
