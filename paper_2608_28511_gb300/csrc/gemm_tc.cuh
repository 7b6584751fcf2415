// Tensor-core grouped GEMM engine for sm_103a: TMA -> shared memory ->
// tcgen05.mma (bf16 x bf16 -> fp32 in TMEM) -> tcgen05.ld -> fused epilogue.
//
// C(m, n) = sum_k A(m, k) B(n, k) over 128 x BN x 64 tiles.  One persistent
// CTA per SM walks a static tile sequence decoded on the device from the
// expert offsets (no host synchronisation).  Warp roles:
//   warp 0      TMA producer (one lane) filling a kStages-deep smem ring;
//   warp 1      TMEM allocator and MMA issuer (one lane issues, all wait);
//   warps 2..   epilogue (4, or 8 for bf16 outputs): TMEM -> registers ->
//               global, one accumulator row per thread, double-buffered
//               accumulators (2 x BN columns);
//   last warp   Group::K with fp32 gradients only: writes the empty groups'
//               zero gradients, paced by the producer.
// Operands are staged with 128-byte swizzle; A and B may each be K-major
// (rows of K contiguous) or MN-major (rows of M / N contiguous).
//
// Grouping: Group::M tiles never mix experts in an output row range (rows
// past an expert's end are computed and dropped); Group::K reduces each
// expert over its own row range: whole 64-row k-blocks through the full
// tensor maps, the last rows through a per-expert tail map (a host-encoded
// template of exactly that many rows whose base build_group_maps moves), so
// the copy engine zero-fills past the expert's end.
//
// Every mbarrier wait is bounded (kWaitLimitNs); on expiry the CTA sets the
// device status word, drains its own copies and MMAs, frees TMEM and exits.
#pragma once

#include <cuda.h>

#include "common.cuh"
#include "launch.h"

namespace moe {
namespace tc {

constexpr int BM = 128;
constexpr int BK = 64;                  // bf16: 128 bytes, one swizzle row
constexpr uint64_t kWaitLimitNs = 4000000000ull;

struct Params {
  CUtensorMap ta;
  CUtensorMap tb;
  int64_t M, N, K;
  int64_t b_group_rows;   // rows of B's tensor map per group (Group::M)
  int num_groups;
  int tiles_m, tiles_n;
  const int32_t* offsets;
  void* C;
  int64_t ldc, sc_g;
  const float* bias;
  void* aux;
  uint32_t* err;
  const CUtensorMap* gmaps;  // Group::K: per group {A, B} maps of its last rows (fewer than BK)
  int64_t split_rows;        // Group::K with offsets == nullptr: split g is rows
                             // [lo(g), lo(g + 1)), lo(g) = split_rows g / G rounded down to a
                             // multiple of BK (lo(G) = split_rows): only the last split can
                             // end inside a k-block
  const int32_t* gather;     // GATHER: source row of each gathered row (the permutation's token_of_row)
  const uint8_t* gsrc;       // GATHER: the source matrix (bf16, row-major), its row pitch in bytes
  int64_t gsrc_ld;           //   and its row count (source rows are checked against it)
  int64_t gsrc_rows;
};

// ---------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
// Waits on barriers that the other CTA of a pair signals (the leader's full and
// accumulator-empty barriers) use the default CTA scope too.  What crosses CTAs
// there is either asynchronous-proxy completion (TMA complete_tx, tcgen05.commit),
// whose mbarrier completion already makes the data visible to the waiter, or a
// pure write-after-read hand-off of TMEM: an epilogue thread arrives only after
// tcgen05.wait::ld has returned its loads into registers and
// tcgen05.fence::before_thread_sync has ordered them before the arrive, so the
// MMA that then overwrites the accumulator cannot change what was read.  The
// one exception is the gathering producer, whose row copies are ordinary
// (generic-proxy) writes: the other CTA of a pair forwards them with a proxy
// fence and a cluster-scope release, and the MMA issuer waits on those full
// barriers with mbar_try_wait_cluster and fences again before its MMAs.
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// The same wait with acquire at cluster scope: for barriers on which the other
// CTA of a pair publishes data written through the generic proxy (the row
// copies of the gathering producer).
__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Wait for phase `parity` of `bar`; false if the CTA aborted or the limit
// expired.  cluster: acquire at cluster scope (mbar_try_wait_cluster).
__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                             uint32_t* err, bool cluster = false) {
  auto try_wait = [&]() { return cluster ? mbar_try_wait_cluster(bar, parity) : mbar_try_wait(bar, parity); };
  if (try_wait()) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t i = 1;; ++i) {
    if (try_wait()) return true;
    if ((i & 63u) == 0) {
      if (*abort_flag) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        *abort_flag = 1;
        set_error(err, kErrTimeout);
        return false;
      }
    }
  }
}
// Same, ignoring the abort flag (used while draining).
__device__ __forceinline__ bool wait_drain(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > limit_ns) return false;
  }
  return true;
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y)
      : "memory");
}
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}
// A tensor map written in global memory by an earlier kernel: order its
// generic-proxy writes before this thread's TMA reads of it.
__device__ __forceinline__ void tmap_acquire(const CUtensorMap* map) {
  asm volatile("fence.proxy.tensormap::generic.acquire.gpu [%0], 128;" ::"l"(reinterpret_cast<uint64_t>(map))
               : "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}
// ---- CTA-pair (cta_group::2) forms: one leader CTA issues the MMAs of a
// 256-row tile whose halves live in the two CTAs of a cluster of 2.
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// The shared::cluster address of `saddr`'s counterpart in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_to_rank(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// TMA load into this CTA's shared memory that completes on an mbarrier of
// either CTA of the pair (here: the leader's).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, uint32_t bar_cluster, int x,
                                                 int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, "
      "%4}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(x), "r"(y)
      : "memory");
}
// ---- row gathers by the producer warp's lanes (cp.async, 16 bytes each)
// 16 bytes from global memory into shared memory, through L2 only; with
// nbytes = 0 nothing is read and the 16 bytes are zero-filled.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t nbytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(nbytes) : "memory");
}
// An arrival on `bar` (this CTA) once all of this thread's earlier cp.async
// copies have landed; the arrival counts toward the barrier's expected count.
__device__ __forceinline__ void cp_async_arrive(uint32_t bar) {
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait_group() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ uint4 lds128(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a) : "memory");
  return v;
}
__device__ __forceinline__ void sts128(uint32_t a, const uint4& v) {
  asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w) : "memory");
}
// EPI 5 slots: a 32-row x 32-byte block (16 bf16 columns) at byte
// r * 32 + 16 (piece ^ (r / 4 mod 2)): conflict-free for a lane reading its own
// row and for 4 rows x 2 pieces per quarter of a copy instruction.
__device__ __forceinline__ uint32_t hs_off(int r, int pc) { return r * 32 + ((pc ^ ((r >> 2) & 1)) << 4); }
// cp.async of the gate block (columns gcol .. gcol + 15) and the up block
// (gcol + 64 ..) of rows 0 .. nrows - 1 into a slot (gate at +0, up at +1024);
// one commit group.
__device__ __forceinline__ void h_fetch(uint32_t slot, const uint8_t* rows, int64_t ld_b, int64_t gcol, int lane,
                                        int nrows) {
#pragma unroll
  for (int it = 0; it < 2; ++it) {
    const int r = it * 16 + lane / 2, pc = lane % 2;
    if (r < nrows) {
      const uint8_t* src = rows + r * ld_b + gcol * 2 + pc * 16;
      cp_async16(slot + hs_off(r, pc), src, 16u);
      cp_async16(slot + 1024 + hs_off(r, pc), src + 128, 16u);
    }
  }
  cp_async_commit();
}

// Arrival on an mbarrier of either CTA of the cluster, releasing this
// thread's earlier writes at cluster scope.
__device__ __forceinline__ void mbar_arrive_release_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
template <int CG>
__device__ __forceinline__ void tmem_alloc_cg(uint32_t dst_smem, uint32_t ncols) {
  if (CG == 2)
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
                 : "memory");
  else
    tmem_alloc(dst_smem, ncols);
}
template <int CG>
__device__ __forceinline__ void tmem_relinquish_cg() {
  if (CG == 2) asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  else tmem_relinquish();
}
template <int CG>
__device__ __forceinline__ void tmem_dealloc_cg(uint32_t taddr, uint32_t ncols) {
  if (CG == 2)
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
  else
    tmem_dealloc(taddr, ncols);
}
template <int CG>
__device__ __forceinline__ void mma_bf16_cg(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
  if (CG == 2)
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
  else
    mma_bf16(d_tmem, adesc, bdesc, idesc, accumulate);
}
// Arrive on `bar` (same offset) in every CTA of `mask` once this thread's
// earlier MMAs complete.
template <int CG>
__device__ __forceinline__ void mma_commit_cg(uint32_t bar, uint16_t mask) {
  if (CG == 2)
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
            bar),
        "h"(mask)
        : "memory");
  else
    mma_commit(bar);
}

// 32 consecutive fp32 columns of this warp's 32 TMEM lanes (one row per
// thread), issued without waiting: the registers hold the values only after
// tmem_ld_wait(r), which every use must follow.
__device__ __forceinline__ void tmem_ld32_issue(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}
// Waits for every tcgen05.ld this thread issued; the registers of r are tied
// to the wait so that no use of them is scheduled before it.
__device__ __forceinline__ void tmem_ld_wait(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                 "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                 "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                 "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
  uint32_t r[32];
  tmem_ld32_issue(taddr, r);
  tmem_ld_wait(r);
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor, 128-byte swizzle, tcgen05 version bits.
//  K-major : LBO unused, SBO = 1024 (8 rows x 128 B); a 16-element k step is +32 B.
//  MN-major: LBO = byte stride between 64-element MN chunks, SBO = 1024
//            (8 k rows x 128 B); a 16-element k step is +2048 B.
__device__ __forceinline__ uint64_t make_sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Instruction descriptor for kind::f16: fp32 accumulator, bf16 A and B,
// operand majorness, N >> 3 at bit 17, M >> 4 at bit 24 (M = 128 per CTA,
// 256 for a CTA pair).
__host__ __device__ constexpr uint32_t make_idesc(int bn, int bm, bool a_mn, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) |
         ((uint32_t)(bn >> 3) << 17) | ((uint32_t)(bm >> 4) << 24);
}

// CG = 1: one CTA computes a 128 x BN tile.  CG = 2: a cluster of two CTAs
// computes a 256 x BN tile; each CTA stages its 128 rows of A and BN / 2 rows
// of B, and holds its 128 accumulator rows in its own TMEM.
template <int BN, int CG = 1, int TCB = 2, int EPI = 0, int ZW = 0>  // TCB: bytes per element of C
struct Cfg {
  static constexpr int kBRows = BN / CG;
  static constexpr int kABytes = BM * BK * 2;
  static constexpr int kBBytes = kBRows * BK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  // EPI 5 (SwiGLU backward) gives one stage to its h slots
  static constexpr int kStages = EPI == 5 ? 5 : ((196608 / kStageBytes) < 8 ? (196608 / kStageBytes) : 8);
  static constexpr int kCols = 2 * BN;  // double-buffered fp32 accumulator
  // Epilogue warps: 8 (two per TMEM lane quarter, each taking half the
  // columns) for bf16 outputs, whose epilogues are latency-bound; 4 for fp32
  // outputs, which are bound by their store bandwidth.
  static constexpr int kEpiWarps = TCB == 2 ? 8 : 4;
  // ZW: one more warp that writes the empty groups' zero gradients (Group::K, fp32)
  static constexpr int kThreads = 64 + 32 * kEpiWarps + 32 * ZW;
  // per epilogue warp: 32 rows x 32 columns of C staging, rows padded by 16 B
  // (conflict-free both ways)
  static constexpr int kRowBytes = 32 * TCB;
  static constexpr int kPitch = kRowBytes + 16;
  // EPI 5: a ring of three 2 KB slots per warp, each the gate and up blocks of
  // h (in) and of dH (out) for 16 columns of dA, 32 rows x 32 bytes apiece
  static constexpr int kStageBufBytes = EPI == 5 ? 6144 : 32 * kPitch;
  static constexpr int kStagingBytes = kEpiWarps * kStageBufBytes;
  static constexpr int kSmem = kStages * kStageBytes + kStagingBytes + 1024 /*align*/ + 512 /*barriers*/;
};

// ---------------------------------------------------------------------------
// Epilogue staging: each epilogue warp owns 32 accumulator rows (one per
// lane) of its share of the columns.  A lane writes its row into the warp's staging buffer, then the warp
// copies the 32 rows to global memory with lanes covering consecutive 16-byte
// pieces of a row, so every store instruction writes whole 128-byte lines
// instead of 32 scattered half-sectors.  Loads of epilogue inputs (the saved
// h, an accumulation target) take the reverse path.
// ---------------------------------------------------------------------------
template <int NB>  // bytes per row: 64 or 128
__device__ __forceinline__ void stage_put(uint8_t* buf, int lane, const uint4* row) {
#pragma unroll
  for (int j = 0; j < NB / 16; ++j) *reinterpret_cast<uint4*>(buf + lane * (NB + 16) + j * 16) = row[j];
}
template <int NB>
__device__ __forceinline__ void stage_get(const uint8_t* buf, int lane, uint4* row) {
#pragma unroll
  for (int j = 0; j < NB / 16; ++j) row[j] = *reinterpret_cast<const uint4*>(buf + lane * (NB + 16) + j * 16);
}
// buf rows 0..31 -> gbase + r * ld_bytes (rows r >= nrows are skipped).
template <int NB>
__device__ __forceinline__ void stage_store(const uint8_t* buf, int lane, uint8_t* gbase, int64_t ld_bytes,
                                            int nrows) {
  constexpr int CPR = NB / 16, RPI = 32 / CPR;
#pragma unroll
  for (int it = 0; it < 32 / RPI; ++it) {
    const int r = it * RPI + lane / CPR, c = lane % CPR;
    const uint4 v = *reinterpret_cast<const uint4*>(buf + r * (NB + 16) + c * 16);
    if (r < nrows) *reinterpret_cast<uint4*>(gbase + r * ld_bytes + c * 16) = v;
  }
}
// The 32 x 32 bf16 block of C an accumulating chunk adds to, fetched into
// registers as 16-byte pieces (4 per lane; rows >= nrows as zero), and put
// into the staging buffer in row order (64-byte rows, 80-byte pitch).
__device__ __forceinline__ void acc_fetch(const uint8_t* rows, int64_t ld_b, int64_t col0, int lane, int nrows,
                                          uint4* dst) {
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int r = it * 8 + lane / 4, pc = lane % 4;
    dst[it] = r < nrows ? *reinterpret_cast<const uint4*>(rows + r * ld_b + col0 * 2 + pc * 16)
                        : make_uint4(0, 0, 0, 0);
  }
}
__device__ __forceinline__ void acc_put(uint8_t* buf, int lane, const uint4* src) {
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int r = it * 8 + lane / 4, pc = lane % 4;
    *reinterpret_cast<uint4*>(buf + r * 80 + pc * 16) = src[it];
  }
}
// gbase + r * ld_bytes -> buf rows 0..31 (rows r >= nrows read as zero).
template <int NB>
__device__ __forceinline__ void stage_load(uint8_t* buf, int lane, const uint8_t* gbase, int64_t ld_bytes,
                                           int nrows) {
  constexpr int CPR = NB / 16, RPI = 32 / CPR;
#pragma unroll
  for (int it = 0; it < 32 / RPI; ++it) {
    const int r = it * RPI + lane / CPR, c = lane % CPR;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (r < nrows) v = *reinterpret_cast<const uint4*>(gbase + r * ld_bytes + c * 16);
    *reinterpret_cast<uint4*>(buf + r * (NB + 16) + c * 16) = v;
  }
}

struct Tile {
  int g;
  int64_t row0, row_end, n0, kbeg, kend;
  int nkb;
};

// Tile t of the static sequence.  GROUP: 0 dense, 1 by M, 2 by K.  Tiles
// are BM * CG rows high; row0 is this CTA's first row (rank * BM into the tile).
template <int GROUP, int CG = 1>
__device__ __forceinline__ void decode_tile(const Params& p, int t, const int* s_off, const int* s_pref,
                                            uint32_t rank, Tile& ti) {
  constexpr int BMP = BM * CG;
  if (GROUP == 0) {
    const int mt = t / p.tiles_n, nt = t % p.tiles_n;
    ti.g = 0;
    ti.row0 = (int64_t)mt * BMP + rank * BM;
    ti.row_end = p.M;
    ti.n0 = nt;
    ti.kbeg = 0;
    ti.kend = p.K;
  } else if (GROUP == 1) {
    const int mb = t / p.tiles_n, nt = t % p.tiles_n;
    int lo = 0, hi = p.num_groups - 1;  // last g with s_pref[g] <= mb
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (s_pref[mid] <= mb) lo = mid;
      else hi = mid - 1;
    }
    ti.g = lo;
    ti.row0 = (int64_t)s_off[lo] + (int64_t)(mb - s_pref[lo]) * BMP + rank * BM;
    ti.row_end = s_off[lo + 1];
    ti.n0 = nt;
    ti.kbeg = 0;
    ti.kend = p.K;
  } else {
    const int per = p.tiles_m * p.tiles_n;
    const int g = t / per, rem = t % per;
    ti.g = g;
    ti.row0 = (int64_t)(rem / p.tiles_n) * BMP + rank * BM;
    ti.row_end = p.M;
    ti.n0 = rem % p.tiles_n;
    ti.kbeg = s_off[g];
    ti.kend = s_off[g + 1];
  }
  ti.nkb = (int)((ti.kend - ti.kbeg + BK - 1) / BK);
}

// The tiles one walker (a CTA, or a CTA pair) takes, in order.  Dense and
// Group::M GEMMs: tiles cta0, cta0 + ncta, ...  Group::K GEMMs (per-expert
// weight gradients) cost in proportion to the group's rows, and a group
// without rows only writes zeros, which needs no MMA and no accumulator.
// There the prologue partitions the groups, stably, into the non-empty ones
// and the empty ones, and every walker takes:
//   * the non-empty groups' tiles round-robin over the walkers (round r takes
//     tiles r * ncta .. r * ncta + ncta - 1, walker p the p-th), or, when the
//     groups' k-block counts differ by more than a factor of two, in snake
//     order (walker p the (ncta - 1 - p)-th of an odd round), which evens out
//     the k-blocks per walker;
//   * the empty groups' tiles p, p + ncta, ..., interleaved with its
//     non-empty ones in proportion to the k-blocks done so far, so that the
//     epilogue writes the zero tiles while the MMA works on the next tiles
//     instead of in a write-only phase at the end.
// On the skewed workload (94 of 128 experts empty, the largest ones at 32768
// rows) this took the GEMM-1 weight gradient from 1.68 to 1.43 ms; on
// balanced workloads the snake order measured 3-4 % slower than round-robin.
// Where the empty groups' gradients are contiguous (every expert weight
// gradient) a dedicated warp writes them instead (the zero warp below), and
// the walk leaves their tiles out: 1.43 to 1.36 ms.
// Producer, MMA issuer and epilogue warps of both CTAs of a pair walk the
// same sequence.
struct Walker {
  int t, total, ncta, p;           // Dense / Group::M
  int r, zi, nz, nc, nce, per;     // Group::K: next round, zero tiles taken / owned, non-empty tiles and groups
  bool snake;                      // Group::K: snake order
  int64_t cum, tot;                // Group::K: k-blocks taken / owned
};

__device__ __forceinline__ int kblocks(const int* s_off, int g) { return (s_off[g + 1] - s_off[g] + BK - 1) / BK; }
__device__ __forceinline__ int walk_index(int r, int p, int ncta, bool snake) {
  return r * ncta + ((snake && (r & 1)) ? ncta - 1 - p : p);
}

template <int GROUP>
__device__ __forceinline__ Walker make_walker(int cta0, int ncta, int total, int per, int nce, int nz,
                                              int64_t tot, bool snake) {
  Walker w;
  w.t = cta0 - ncta;
  w.total = total;
  w.ncta = ncta;
  w.p = cta0;
  w.r = 0;
  w.zi = 0;
  w.nz = nz;
  w.nce = nce;
  w.per = per;
  w.nc = nce * per;
  w.snake = snake;
  w.cum = 0;
  w.tot = tot;
  return w;
}

// The walker's next tile (the index decode_tile takes); false when done.
// s_ord (Group::K): the non-empty groups by index, then the empty ones.
template <int GROUP>
__device__ __forceinline__ bool next_tile(Walker& w, const int* s_off, const int* s_ord, int& t) {
  if (GROUP != 2 || (!w.snake && w.nce * w.per == w.total)) {
    // Dense, Group::M, or Group::K without empty groups in round-robin order
    // (the partition is then the identity): tiles cta0, cta0 + ncta, ...
    w.t += w.ncta;
    t = w.t;
    return w.t < w.total;
  }
  bool zero = w.zi < w.nz && (int64_t)w.zi * w.tot <= w.cum * w.nz;
  if (!zero) {
    const int c = walk_index(w.r, w.p, w.ncta, w.snake);
    if (c < w.nc) {
      const int g = s_ord[c / w.per];
      t = g * w.per + c % w.per;
      w.cum += kblocks(s_off, g);
      ++w.r;
      return true;
    }
    zero = w.zi < w.nz;
  }
  if (!zero) return false;
  const int z = w.p + w.zi * w.ncta;
  t = s_ord[w.nce + z / w.per] * w.per + z % w.per;
  ++w.zi;
  return true;
}

__device__ __forceinline__ int64_t imin64(int64_t a, int64_t b) { return a < b ? a : b; }
__device__ __forceinline__ int64_t imax64(int64_t a, int64_t b) { return a > b ? a : b; }

// silu(v) = v sigmoid(v) with sigmoid(v) = (1 + tanh(v / 2)) / 2 on the
// hardware tanh approximation (one MUFU op; its ~5e-4 error is far below
// the bf16 rounding of the stored activation).
__device__ __forceinline__ float tanh_approx(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float sigmoid_f(float v) { return fmaf(0.5f, tanh_approx(0.5f * v), 0.5f); }
__device__ __forceinline__ float silu_f(float v) { return v * sigmoid_f(v); }

template <typename T>
__device__ __forceinline__ void store_row32(T* dst, const float* v, int valid) {
  constexpr int NV = Vec<T>::N;
  if (valid >= 32) {
#pragma unroll
    for (int i = 0; i < 32; i += NV) *reinterpret_cast<uint4*>(dst + i) = pack16<T>(v + i);
  } else {
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (i < valid) dst[i] = from_f32<T>(v[i]);
  }
}
template <typename T>
__device__ __forceinline__ void load_row32(const T* src, float* v) {
  constexpr int NV = Vec<T>::N;
#pragma unroll
  for (int i = 0; i < 32; i += NV) unpack16<T>(*reinterpret_cast<const uint4*>(src + i), v + i);
}

// EPI: 0 Store, 1 StoreBias, 2 Accum, 3 SwigluFwd, 4 ReluSqFwd, 5 SwigluBwd (values of moe::Epi).
// CG: 1 = one CTA per 128 x BN tile; 2 = a cluster of two CTAs per 256 x BN
// tile (the even CTA issues the MMAs; both stage their halves and drain
// their own accumulator rows).
// GATHER: 0 tiled copies; 1 A's rows (K-major, Group::M) and 2 B's k rows
// (MN-major, Group::K) are gathered from a source matrix through p.gather
// (row -> source row), four rows per copy, by the 32 lanes of the producer warp.
template <int BN, bool A_MN, bool B_MN, int GROUP, int EPI, typename TC, int CG, int GATHER = 0>
__global__ void __launch_bounds__(
    Cfg<BN, CG, sizeof(TC), 0, (GROUP == 2 && sizeof(TC) == 4 && GATHER == 0) ? 1 : 0>::kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ Params p) {
  constexpr int kZW = (GROUP == 2 && sizeof(TC) == 4 && GATHER == 0) ? 1 : 0;  // the zero-gradient warp
  using C = Cfg<BN, CG, sizeof(TC), EPI, kZW>;
  constexpr int EW = C::kEpiWarps;
  constexpr int CSTEP = EW / 4;  // epilogue warps sharing a lane quarter
  constexpr int BMP = BM * CG;
  constexpr int BNC = C::kBRows;
  constexpr uint32_t kIdesc = make_idesc(BN, BMP, A_MN, B_MN);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::kStages * C::kStageBytes + C::kStagingBytes);
  uint64_t* full = bars;                       // [kStages]
  uint64_t* empty = bars + C::kStages;         // [kStages]
  uint64_t* tfull = bars + 2 * C::kStages;     // [2]
  uint64_t* tempty = tfull + 2;                // [2]
  uint64_t* done = tempty + 2;                 // [1]
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(done + 1);
  __shared__ int s_off[kMaxE + 1];
  __shared__ int s_pref[kMaxE + 1];
  __shared__ int s_total;
  __shared__ volatile int s_abort;
  __shared__ int s_knce, s_knz;      // Group::K: non-empty groups; this walker's zero tiles
  __shared__ int s_ksnake;           // Group::K: snake order
  __shared__ long long s_ktot;       // Group::K: this walker's k-blocks
  __shared__ volatile int s_kprog;   // zero warp: k-blocks the producer has issued so far
  __shared__ int s_zmode;            // zero warp: on (the empty groups' gradients are its job)
  __shared__ long long s_zbeg, s_zend;  // zero warp: this CTA's share of the empty groups' bytes

  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = CG == 2 ? cluster_ctarank() : 0u;
  const bool leader = rank == 0;
  const int cta0 = blockIdx.x / CG, ncta = gridDim.x / CG;  // tile-walker index and count

  if (warp == 0 && lane == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      // gathering: the leader's expect_tx arrival, one arrival per producer
      // lane of this CTA once its row copies into the stage have landed, and
      // in a pair the other CTA's forwarded arrival; the other CTA of a pair
      // counts only its own lanes' arrivals on its full barriers
      const uint32_t cnt = GATHER == 0 ? 1u : CG == 1 ? 33u : (leader ? 34u : 32u);
      mbar_init(smem_u32(&full[s]), cnt);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), EW * CG);
    }
    mbar_init(smem_u32(done), 1);
    fence_barrier_init();
    s_abort = 0;
    tma_prefetch_desc(&p.ta);
    tma_prefetch_desc(&p.tb);
  }
  if (warp == 1) {
    tmem_alloc_cg<CG>(smem_u32(s_tmem), C::kCols);
    tmem_relinquish_cg<CG>();
  }
  if (GROUP != 0) {
    if (p.offsets) {
      for (int i = tid; i <= p.num_groups; i += C::kThreads) s_off[i] = p.offsets[i];
    } else {
      for (int i = tid; i <= p.num_groups; i += C::kThreads)
        s_off[i] = i < p.num_groups ? (int)((p.split_rows * i / p.num_groups) & ~(int64_t)(BK - 1))
                                    : (int)p.split_rows;
    }
  }
  __syncthreads();
  if (GROUP == 2 && warp == 0) {
    // s_pref: the non-empty groups by index, then the empty ones (a stable
    // partition); the walker's share of the non-empty tiles' k-blocks and of
    // the empty tiles; snake order when the k-block counts spread widely
    const int G = p.num_groups;
    const int per = p.tiles_m * p.tiles_n;
    int nce = 0, kmin = 0x7fffffff, kmax = 0;
    for (int j = lane; j < G; j += 32) {
      const int kj = kblocks(s_off, j);
      if (kj > 0) {
        ++nce;
        kmin = min(kmin, kj);
        kmax = max(kmax, kj);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      nce += __shfl_xor_sync(0xffffffffu, nce, o);
      kmin = min(kmin, __shfl_xor_sync(0xffffffffu, kmin, o));
      kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, o));
    }
    int before_ne = 0, before_e = 0;
    for (int j0 = 0; j0 < G; j0 += 32) {
      const int j = j0 + lane;
      const bool ne = j < G && kblocks(s_off, j) > 0;
      const unsigned bne = __ballot_sync(0xffffffffu, ne), be = __ballot_sync(0xffffffffu, j < G && !ne);
      const unsigned below = (1u << lane) - 1u;
      if (j < G) s_pref[ne ? before_ne + __popc(bne & below) : nce + before_e + __popc(be & below)] = j;
      before_ne += __popc(bne);
      before_e += __popc(be);
    }
    __syncwarp();
    const bool snake = nce > 0 && kmax > 2 * kmin;
    const int nc = nce * per, nzt = (G - nce) * per;
    long long tot = 0;
    if (nzt > 0) {  // the walker's k-blocks pace its zero tiles
      for (int r = lane;; r += 32) {
        const int c = walk_index(r, cta0, ncta, snake);
        if (c >= nc) break;
        tot += kblocks(s_off, s_pref[c / per]);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    }
    if (lane == 0) {
      s_knce = nce;
      s_ktot = tot;
      s_knz = cta0 < nzt ? (nzt - cta0 + ncta - 1) / ncta : 0;
      s_ksnake = snake ? 1 : 0;
      s_kprog = 0;
      s_zmode = 0;
      // the empty groups' gradients are contiguous blocks of M x N fp32: the zero
      // warps write them, each CTA an equal share of the bytes, and the walk
      // leaves their tiles out
      if (kZW && nzt > 0 && p.ldc == p.N && p.sc_g == p.M * p.N && (p.M * p.N) % 4 == 0) {
        const int64_t zbytes = (int64_t)(G - nce) * p.M * p.N * 4;
        const int64_t b = blockIdx.x, nbk = gridDim.x;
        s_zbeg = (zbytes * b / nbk) & ~(int64_t)15;
        s_zend = b + 1 == nbk ? zbytes : ((zbytes * (b + 1) / nbk) & ~(int64_t)15);
        s_zmode = 1;
        s_knz = 0;
      }
    }
  }
  if (tid == 0) {
    if (GROUP == 0) {
      s_total = p.tiles_m * p.tiles_n;
    } else if (GROUP == 1) {
      int acc = 0;
      for (int g = 0; g < p.num_groups; ++g) {
        s_pref[g] = acc;
        acc += (s_off[g + 1] - s_off[g] + BMP - 1) / BMP;
      }
      s_pref[p.num_groups] = acc;
      s_total = acc * p.tiles_n;
    } else {
      s_total = p.num_groups * p.tiles_m * p.tiles_n;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (CG == 2) cluster_sync();  // both CTAs' barriers exist before any cross-CTA signal
  tc_fence_after();
  const uint32_t tmem_base = *s_tmem;
  const int total = s_total;
  const int kper = p.tiles_m * p.tiles_n;
  const int knce = GROUP == 2 ? s_knce : 0, knz = GROUP == 2 ? s_knz : 0;
  const int64_t ktot = GROUP == 2 ? (int64_t)s_ktot : 0;
  const bool ksnake = GROUP == 2 && s_ksnake != 0;

  if (warp == 0 && GATHER != 0) {
    // ------------------------------------------------------------ producer (gathering, warp-wide)
    // The gathered operand's rows come from p.gsrc through p.gather, as 16-byte
    // cp.async copies by the 32 lanes into the stage's 128-byte-swizzled
    // layout (chunk c of row r at r * 128 + ((c ^ (r & 7)) << 4), the layout a
    // tiled 128-byte-swizzle copy writes); lane 0 issues the other operand's
    // tiled copies, which complete on the leader's full barrier as usual.
    // Every lane then arrives on its CTA's full barrier of the stage once its
    // copies have landed (cp.async.mbarrier.arrive), so the producer never
    // waits for its own copies; in a pair the other CTA's MMA warp forwards
    // its completed stages to the leader.
    int stage = 0;
    uint32_t phase = 0;
    int issued = 0;
    uint32_t last_phase = 0;
    bool ok = true;
    const int q = lane >> 3, c = lane & 7;  // a warp instruction covers 4 rows of 8 chunks
    auto src_row = [&](int64_t r) -> const uint8_t* {
      int64_t src = r >= 0 ? (int64_t)__ldg(p.gather + r) : 0;
      if (src < 0 || src >= p.gsrc_rows) {  // a bad row index: recorded, row 0 read instead
        set_error(p.err, kErrIndex);
        src = 0;
      }
      return p.gsrc + src * p.gsrc_ld;
    };
    Walker wk = make_walker<GROUP>(cta0, ncta, total, kper, knce, knz, ktot, ksnake);
    for (int t; ok && next_tile<GROUP>(wk, s_off, s_pref, t);) {
      Tile ti;
      decode_tile<GROUP, CG>(p, t, s_off, s_pref, rank, ti);
      const int64_t nb = ti.n0 * BN + (int64_t)rank * BNC;
      // GATHER 1: source rows of this CTA's A rows lane, lane + 32, lane + 64,
      // lane + 96 (rows past the expert's end read row 0; their outputs are dropped)
      const uint8_t* ra[4];
      if (GATHER == 1) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int64_t r = ti.row0 + lane + 32 * i;
          ra[i] = src_row(r < ti.row_end ? r : -1);
        }
      }
      for (int kb = 0; kb < ti.nkb; ++kb) {
        // every lane observes the stage's release before its copies overwrite it
        const bool okw = wait_bounded(smem_u32(&empty[stage]), phase ^ 1u, &s_abort, p.err);
        if (!__all_sync(0xffffffffu, okw)) { ok = false; break; }
        const uint32_t fb_local = smem_u32(&full[stage]);
        const uint32_t fb = CG == 2 ? map_to_rank(fb_local, 0) : fb_local;
        // the leader expects the tiled operand's bytes of both CTAs
        if (leader && lane == 0) mbar_expect_tx(fb_local, CG * (GATHER == 1 ? C::kBBytes : C::kABytes));
        const uint32_t sa = smem_u32(smem + stage * C::kStageBytes);
        const uint32_t sb = sa + C::kABytes;
        const int k0 = (int)(ti.kbeg + (int64_t)kb * BK);
        auto load = [&](uint32_t dst, const CUtensorMap* m, int x, int y) {
          if (CG == 2) tma_load_2d_pair(dst, m, fb, x, y);
          else tma_load_2d(dst, m, fb, x, y);
        };
        if (GATHER == 1) {
          if (lane == 0) {
            if (B_MN) {
              const int ky = (int)(ti.g * p.b_group_rows) + k0;
#pragma unroll
              for (int j = 0; j < BNC / 64; ++j) load(sb + j * 8192, &p.tb, (int)nb + 64 * j, ky);
            } else {
              load(sb, &p.tb, k0, (int)(ti.g * p.b_group_rows + nb));
            }
          }
          // A: 128 rows x 64 k (128 bytes) of the source rows, K-major
#pragma unroll
          for (int it = 0; it < BM / 4; ++it) {
            const int r = 4 * it + q;
            const uint8_t* base = reinterpret_cast<const uint8_t*>(
                __shfl_sync(0xffffffffu, reinterpret_cast<uintptr_t>(ra[it >> 3]), r & 31));
            cp_async16(sa + r * 128 + ((c ^ (r & 7)) << 4), base + (int64_t)k0 * 2 + c * 16, 16u);
          }
        } else {
          // A: whole k-blocks from the full map, the group's last rows from
          // its tail map (zero past the group's rows)
          if (lane == 0) {
            if (kb < (int)((ti.kend - ti.kbeg) / BK)) {
              load(sa, &p.ta, (int)ti.row0, k0);
              load(sa + 8192, &p.ta, (int)ti.row0 + 64, k0);
            } else {
              const CUtensorMap* ma = p.gmaps + 2 * ti.g;
              tmap_acquire(ma);
              load(sa, ma, (int)ti.row0, 0);
              load(sa + 8192, ma, (int)ti.row0 + 64, 0);
            }
          }
          // B: the block's 64 k rows (source rows through p.gather) x this
          // CTA's BNC columns, MN-major in 64-column boxes of 8 KB; past the
          // group's rows A is zero, so any valid source row will do; columns
          // past N are zero-filled
          const uint8_t* rb[2];
#pragma unroll
          for (int i = 0; i < 2; ++i) {
            const int64_t kr = (int64_t)k0 + lane + 32 * i;
            rb[i] = src_row(kr < ti.kend ? kr : -1);
          }
#pragma unroll
          for (int it = 0; it < (BNC / 64) * 16; ++it) {
            const int j = it >> 4, r = (4 * it + q) & 63;
            const uint8_t* base = reinterpret_cast<const uint8_t*>(
                __shfl_sync(0xffffffffu, reinterpret_cast<uintptr_t>(rb[(it >> 3) & 1]), r & 31));
            const int64_t col = nb + 64 * j + 8 * c;
            const bool in = col < p.N;
            cp_async16(sb + j * 8192 + r * 128 + ((c ^ (r & 7)) << 4), in ? base + col * 2 : p.gsrc, in ? 16u : 0u);
          }
        }
        cp_async_arrive(fb_local);
        last_phase = (last_phase & ~(1u << stage)) | (phase << stage);
        ++issued;
        if (++stage == C::kStages) { stage = 0; phase ^= 1u; }
      }
    }
    cp_async_wait_all();  // every copy lands before the CTA goes on
    // tail: wait until the MMA warp has released every stage this CTA filled.
    // Its releases are asynchronous arrivals (multicast to both CTAs of a pair)
    // that may still be in flight when the MMAs are done; waiting here keeps
    // either CTA from exiting before they land in its shared memory.  Stages
    // never filled pass at once.
    if (lane == 0 && ok) {
      int s = stage;
      uint32_t ph = phase;
      for (int i = 0; i < C::kStages; ++i) {
        wait_drain(smem_u32(&empty[s]), ph ^ 1u, 1000000000ull);
        if (++s == C::kStages) { s = 0; ph ^= 1u; }
      }
    }
    if (leader && lane == 0) {
      const int pending = issued < C::kStages ? issued : C::kStages;
      for (int i = 0; i < pending; ++i) {
        stage = (stage + C::kStages - 1) % C::kStages;
        wait_drain(smem_u32(&full[stage]), (last_phase >> stage) & 1u, 1000000000ull);
      }
    }
  } else if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      uint32_t last_phase = 0;  // bit s: phase of the last copy issued into stage s
      bool ok = true;
      Walker wk = make_walker<GROUP>(cta0, ncta, total, kper, knce, knz, ktot, ksnake);
      for (int t; ok && next_tile<GROUP>(wk, s_off, s_pref, t);) {
        Tile ti;
        decode_tile<GROUP, CG>(p, t, s_off, s_pref, rank, ti);
        const int64_t nb = ti.n0 * BN + (int64_t)rank * BNC;  // this CTA's first B row / column
        for (int kb = 0; kb < ti.nkb; ++kb) {
          if (!wait_bounded(smem_u32(&empty[stage]), phase ^ 1u, &s_abort, p.err)) { ok = false; break; }
          const uint32_t fb_local = smem_u32(&full[stage]);
          // CG 2: both CTAs' copies complete on the leader's barrier, which expects both
          const uint32_t fb = CG == 2 ? map_to_rank(fb_local, 0) : fb_local;
          if (leader) mbar_expect_tx(fb_local, CG * C::kStageBytes);
          const uint32_t sa = smem_u32(smem + stage * C::kStageBytes);
          const uint32_t sb = sa + C::kABytes;
          const int k0 = (int)(ti.kbeg + (int64_t)kb * BK);
          auto load = [&](uint32_t dst, const CUtensorMap* m, int x, int y) {
            if (CG == 2) tma_load_2d_pair(dst, m, fb, x, y);
            else tma_load_2d(dst, m, fb, x, y);
          };
          if (GROUP == 2) {
            // whole k-blocks of the group from the full-tensor maps at absolute
            // rows; its last n % BK rows from the group's tail maps, whose row
            // extent ends at the group's end, so the copy engine zero-fills the
            // rest of the block (the next group's rows never enter the reduction)
            const CUtensorMap* ma = &p.ta;
            const CUtensorMap* mb = &p.tb;
            int ky = k0;
            if (kb >= (int)((ti.kend - ti.kbeg) / BK)) {
              ma = p.gmaps + 2 * ti.g;
              mb = ma + 1;
              tmap_acquire(ma);
              tmap_acquire(mb);
              ky = 0;
            }
            load(sa, ma, (int)ti.row0, ky);
            load(sa + 8192, ma, (int)ti.row0 + 64, ky);
#pragma unroll
            for (int j = 0; j < BNC / 64; ++j) load(sb + j * 8192, mb, (int)nb + 64 * j, ky);
          } else {
            if (A_MN) {
              load(sa, &p.ta, (int)ti.row0, k0);
              load(sa + 8192, &p.ta, (int)ti.row0 + 64, k0);
            } else {
              load(sa, &p.ta, k0, (int)ti.row0);
            }
            if (B_MN) {
              const int ky = (int)(ti.g * p.b_group_rows) + k0;
#pragma unroll
              for (int j = 0; j < BNC / 64; ++j) load(sb + j * 8192, &p.tb, (int)nb + 64 * j, ky);
            } else {
              load(sb, &p.tb, k0, (int)(ti.g * p.b_group_rows + nb));
            }
          }
          last_phase = (last_phase & ~(1u << stage)) | (phase << stage);
          ++issued;
          if (kZW) s_kprog = issued;
          if (++stage == C::kStages) { stage = 0; phase ^= 1u; }
        }
      }
      // tail: wait until the MMA warp has released every stage this CTA
      // filled (see the gathering producer above)
      if (ok) {
        int s = stage;
        uint32_t ph = phase;
        for (int i = 0; i < C::kStages; ++i) {
          wait_drain(smem_u32(&empty[s]), ph ^ 1u, 1000000000ull);
          if (++s == C::kStages) { s = 0; ph ^= 1u; }
        }
      }
      // drain: every issued copy must land before the CTA exits (the leader's
      // barriers also count the other CTA's copies)
      if (leader) {
        const int pending = issued < C::kStages ? issued : C::kStages;
        for (int i = 0; i < pending; ++i) {
          stage = (stage + C::kStages - 1) % C::kStages;
          wait_drain(smem_u32(&full[stage]), (last_phase >> stage) & 1u, 1000000000ull);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (the leader CTA)
    int stage = 0;
    uint32_t phase = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    bool ok = true;
    bool issued_any = false;
    constexpr uint16_t kBoth = 0x3;
    Walker wk = make_walker<GROUP>(cta0, ncta, total, kper, knce, knz, ktot, ksnake);
    for (int t; ok && leader && next_tile<GROUP>(wk, s_off, s_pref, t);) {
      Tile ti;
      decode_tile<GROUP, CG>(p, t, s_off, s_pref, rank, ti);
      if (ti.nkb == 0) continue;
      issued_any = true;
      if (!wait_bounded(smem_u32(&tempty[acc]), acc_phase ^ 1u, &s_abort, p.err)) { ok = false; break; }
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
      for (int kb = 0; kb < ti.nkb; ++kb) {
        if (!wait_bounded(smem_u32(&full[stage]), phase, &s_abort, p.err, GATHER != 0 && CG == 2)) {
          ok = false;
          break;
        }
        if (GATHER != 0) fence_proxy_async_smem();  // the row copies, before the tensor core reads them
        tc_fence_after();
        const uint32_t sa = smem_u32(smem + stage * C::kStageBytes);
        const uint32_t sb = sa + C::kABytes;
        if (lane == 0) {
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            uint64_t ad, bd;
            if (A_MN) ad = make_sdesc(sa + k * 2048, 8192, 1024);
            else ad = make_sdesc(sa + k * 32, 16, 1024);
            if (B_MN) bd = make_sdesc(sb + k * 2048, 8192, 1024);
            else bd = make_sdesc(sb + k * 32, 16, 1024);
            mma_bf16_cg<CG>(d_tmem, ad, bd, kIdesc, (kb > 0 || k > 0) ? 1u : 0u);
          }
          mma_commit_cg<CG>(smem_u32(&empty[stage]), kBoth);
        }
        __syncwarp();
        if (++stage == C::kStages) { stage = 0; phase ^= 1u; }
      }
      if (!ok) break;
      if (lane == 0) mma_commit_cg<CG>(smem_u32(&tfull[acc]), kBoth);
      __syncwarp();
      if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
    }
    if (GATHER != 0 && CG == 2 && !leader && lane == 0) {
      // the other CTA of a pair: forward each stage whose row copies have all
      // landed here (this CTA's full barrier) to the leader's full barrier
      int fs = 0;
      uint32_t fph = 0;
      Walker fw = make_walker<GROUP>(cta0, ncta, total, kper, knce, knz, ktot, ksnake);
      bool fok = true;
      for (int t; fok && next_tile<GROUP>(fw, s_off, s_pref, t);) {
        Tile ti;
        decode_tile<GROUP, CG>(p, t, s_off, s_pref, rank, ti);
        for (int kb = 0; kb < ti.nkb; ++kb) {
          if (!wait_bounded(smem_u32(&full[fs]), fph, &s_abort, p.err)) { fok = false; break; }
          fence_proxy_async_smem();
          mbar_arrive_release_cluster(map_to_rank(smem_u32(&full[fs]), 0));
          if (++fs == C::kStages) { fs = 0; fph ^= 1u; }
        }
      }
    }
    // drain: all MMAs issued by this warp have completed before TMEM is freed
    if (lane == 0 && issued_any) {
      mma_commit_cg<CG>(smem_u32(done), 0x1);
      wait_drain(smem_u32(done), 0, 1000000000ull);
    }
    __syncwarp();
  } else if (kZW && warp == 2 + EW) {
    // ------------------------------------------------------------ zero gradients
    // This CTA's share of the empty groups' bytes, paced by the producer's
    // k-blocks so that the writes spread over the main loop (512 bytes per
    // warp store, every 16-byte piece inside one group's block).
    if (s_zmode) {
      const int64_t zb = s_zbeg, ze = s_zend, gbytes = p.M * p.N * 4;
      const int64_t kall = s_ktot;
      const int nce0 = s_knce;
      uint8_t* cbase = static_cast<uint8_t*>(p.C);
      const uint4 z = make_uint4(0, 0, 0, 0);
      int64_t done = zb;
      int64_t j = zb / gbytes, w = zb - j * gbytes;  // group and offset of `done`
      uint64_t t0 = global_timer_ns();  // the last time the producer was seen to move
      int last = -1;
      while (done < ze) {
        const int prog = s_kprog;
        if (prog != last) {
          last = prog;
          t0 = global_timer_ns();
        }
        int64_t target = (kall > 0 && prog < kall) ? (zb + (ze - zb) * (int64_t)prog / kall) & ~(int64_t)15 : ze;
        if (target - done >= 8192 || target == ze) {
          while (done < target) {
            // one group's contiguous piece: plain 16-byte stores, 512 bytes per warp store
            const int64_t seg = imin64(target - done, gbytes - w);
            uint4* ptr = reinterpret_cast<uint4*>(cbase + (int64_t)s_pref[nce0 + j] * p.sc_g * 4 + w);
            const int n16 = (int)(seg >> 4);
#pragma unroll 4
            for (int i = lane; i < n16; i += 32) ptr[i] = z;
            done += seg;
            w += seg;
            if (w == gbytes) { w = 0; ++j; }
          }
        }
        if (done < ze) {
          if (s_abort) break;
          if (global_timer_ns() - t0 > kWaitLimitNs) {
            s_abort = 1;
            set_error(p.err, kErrTimeout);
            break;
          }
          __nanosleep(256);
        }
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;            // TMEM lane quarter
    const int ew = warp - 2;
    const int ch = ew >> 2;            // which of the CSTEP column interleaves this warp takes
    uint8_t* stg = smem + C::kStages * C::kStageBytes + ew * C::kStageBufBytes;
    constexpr int RB = C::kRowBytes;               // bytes per staged row (32 columns)
    constexpr int NP = RB / 16;                    // 16-byte pieces per staged row
    constexpr int RPC = (int)sizeof(TC) * 32 / RB; // rounds per 32-column chunk (1)
    constexpr int CPR = RB / (int)sizeof(TC);      // columns per round
    const int64_t ldc_b = p.ldc * (int64_t)sizeof(TC);
    int acc = 0;
    uint32_t acc_phase = 0;
    int hq = 0;  // EPI 5: ring slot of the current tile's first half
    Walker wk = make_walker<GROUP>(cta0, ncta, total, kper, knce, knz, ktot, ksnake);
    for (int t; next_tile<GROUP>(wk, s_off, s_pref, t);) {
      Tile ti;
      decode_tile<GROUP, CG>(p, t, s_off, s_pref, rank, ti);
      const int64_t n0 = ti.n0 * BN;
      const int64_t rbase = ti.row0 + q * 32;  // this warp's first row
      const int nrows = (int)imax64(0, imin64(32, ti.row_end - rbase));
      const int64_t grow = rbase + lane;
      const bool vrow = lane < nrows;
      TC* Cb = static_cast<TC*>(p.C) + (GROUP == 2 ? (int64_t)ti.g * p.sc_g : 0);
      uint8_t* c_rows = reinterpret_cast<uint8_t*>(Cb) + rbase * ldc_b;
      if (ti.nkb == 0) {
        // an expert with no rows: its weight-gradient tile is zero
        uint4 z[NP];
#pragma unroll
        for (int i = 0; i < NP; ++i) z[i] = make_uint4(0, 0, 0, 0);
        for (int c = ch; c < BN / 32; c += CSTEP) {
          const int64_t col0 = n0 + c * 32;
          if (col0 >= p.N) break;
          if (p.N - col0 >= 32) {
#pragma unroll
            for (int r = 0; r < RPC; ++r) {
              __syncwarp();
              stage_put<RB>(stg, lane, z);
              __syncwarp();
              stage_store<RB>(stg, lane, c_rows + (col0 + r * CPR) * sizeof(TC), ldc_b, nrows);
            }
          } else if (vrow) {
            float zf[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) zf[i] = 0.f;
            store_row32<TC>(Cb + grow * p.ldc + col0, zf, (int)(p.N - col0));
          }
        }
        continue;
      }
      // EPI 2: every chunk's C block is fetched before the accumulator wait, so
      // the reads overlap the MMA and each other
      constexpr int kPre = EPI == 2 ? BN / 32 / CSTEP : 1;  // this warp's chunks: ch, ch + CSTEP, ...
      uint4 pre[kPre][4];
      const int nch_acc = (int)imin64(BN / 32, (p.N - n0) / 32);
      if (EPI == 2) {
#pragma unroll
        for (int i = 0; i < kPre; ++i)
          if (ch + i * CSTEP < nch_acc) acc_fetch(c_rows, ldc_b, n0 + (ch + i * CSTEP) * 32, lane, nrows, pre[i]);
      }
      // EPI 5: this warp's columns of dA go in halves of 16 (half k of the tile:
      // chunk k / 2, i.e. columns 32 (ch + CSTEP k / 2) + 16 (k mod 2)) through a
      // ring of three slots.  The gate and up blocks of h for halves 0 and 1 are
      // copied in before the accumulator wait; half k + 2's when half k starts,
      // into the slot that half k - 1 has just written out.  Every half commits
      // one cp.async group (empty past the tile's last column).
      const uint8_t* h_rows = EPI == 5 ? static_cast<const uint8_t*>(p.aux) + rbase * ldc_b : nullptr;
      const uint32_t hs = smem_u32(stg);
      auto hcol = [&](int k) -> int64_t {  // column of h's gate block for half k
        const int64_t f = n0 + (ch + (k >> 1) * CSTEP) * 32 + (k & 1) * 16;
        return (f >> 6) * 128 + (f & 63);
      };
      auto hvalid = [&](int k) { return ch + (k >> 1) * CSTEP < nch_acc; };
      if (EPI == 5) {
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          if (hvalid(k)) h_fetch(hs + ((hq + k) % 3) * 2048, h_rows, ldc_b, hcol(k), lane, nrows);
          else cp_async_commit();
        }
      }
      if (!wait_bounded(smem_u32(&tfull[acc]), acc_phase, &s_abort, p.err)) break;
      tc_fence_after();
      const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
      float v[32];
      uint4 pk[NP];
      if (EPI == 3) {
        // packed [gate 64 | up 64] blocks: h = [g | u] stored as computed, a = silu(g) * u
        uint8_t* a_rows = reinterpret_cast<uint8_t*>(static_cast<TC*>(p.aux) + rbase * (p.N / 2));
        const int64_t lda_b = (p.N / 2) * (int64_t)sizeof(TC);
#pragma unroll 1
        for (int hb = ch; hb < BN / 64; hb += CSTEP) {  // half-blocks: 32 gate + 32 up columns
          const int blk = hb >> 1, half = hb & 1;
          const int64_t cb = n0 + blk * 128;
          if (cb >= p.N) break;
          {
            // g (in v) and u are stored first; a = silu(g) * u then overwrites v,
            // so only two 32-value rows are live at a time
            float u[32];
            tmem_ld32(tbase + blk * 128 + half * 32, v);
            tmem_ld32(tbase + blk * 128 + 64 + half * 32, u);
#pragma unroll
            for (int i = 0; i < NP; ++i) pk[i] = pack16<TC>(v + i * Vec<TC>::N);
            __syncwarp();
            stage_put<RB>(stg, lane, pk);
            __syncwarp();
            stage_store<RB>(stg, lane, c_rows + (cb + half * 32) * sizeof(TC), ldc_b, nrows);
#pragma unroll
            for (int i = 0; i < NP; ++i) pk[i] = pack16<TC>(u + i * Vec<TC>::N);
            __syncwarp();
            stage_put<RB>(stg, lane, pk);
            __syncwarp();
            stage_store<RB>(stg, lane, c_rows + (cb + 64 + half * 32) * sizeof(TC), ldc_b, nrows);
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = silu_f(v[i]) * u[i];
#pragma unroll
            for (int i = 0; i < NP; ++i) pk[i] = pack16<TC>(v + i * Vec<TC>::N);
            __syncwarp();
            stage_put<RB>(stg, lane, pk);
            __syncwarp();
            stage_store<RB>(stg, lane, a_rows + (cb / 2 + half * 32) * sizeof(TC), lda_b, nrows);
          }
        }
      } else if (EPI == 5) {
        // the SwiGLU backward on the accumulator dA: per 16 columns of dA, the
        // 16 gate and 16 up columns of h in, the same columns of dH out, each
        // lane on its own row of the slot
        constexpr int NH = 2 * (BN / 32 / CSTEP);  // halves per tile
        uint32_t ra[32];
#pragma unroll
        for (int k = 0; k < NH; ++k) {
          const uint32_t slot = hs + ((hq + k) % 3) * 2048;
          if (k + 2 < NH && hvalid(k + 2))
            h_fetch(hs + ((hq + k + 2) % 3) * 2048, h_rows, ldc_b, hcol(k + 2), lane, nrows);
          else
            cp_async_commit();
          cp_async_wait_group<2>();  // half k's group: only halves k + 1 and k + 2 may still be in flight
          __syncwarp();
          if (hvalid(k)) {
            const int c = ch + (k >> 1) * CSTEP;
            if ((k & 1) == 0) tmem_ld32_issue(tbase + c * 32, ra);
            float g[16], u[16];
#pragma unroll
            for (int j = 0; j < 2; ++j) {
              unpack16<TC>(lds128(slot + hs_off(lane, j)), g + j * Vec<TC>::N);
              unpack16<TC>(lds128(slot + 1024 + hs_off(lane, j)), u + j * Vec<TC>::N);
            }
            if ((k & 1) == 0) tmem_ld_wait(ra);
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const float a = __uint_as_float(ra[(k & 1) * 16 + j]);
              const float s = sigmoid_f(g[j]);
              const float dg = a * u[j] * s * (1.0f + g[j] * (1.0f - s));
              u[j] = a * g[j] * s;
              g[j] = dg;
            }
#pragma unroll
            for (int j = 0; j < 2; ++j) {
              sts128(slot + hs_off(lane, j), pack16<TC>(g + j * Vec<TC>::N));
              sts128(slot + 1024 + hs_off(lane, j), pack16<TC>(u + j * Vec<TC>::N));
            }
            __syncwarp();
            const int64_t gc = hcol(k);
#pragma unroll
            for (int it = 0; it < 2; ++it) {
              const int r = it * 16 + lane / 2, pc = lane % 2;
              if (r < nrows) {
                uint8_t* dst = c_rows + r * ldc_b + gc * 2 + pc * 16;
                *reinterpret_cast<uint4*>(dst) = lds128(slot + hs_off(r, pc));
                *reinterpret_cast<uint4*>(dst + 128) = lds128(slot + 1024 + hs_off(r, pc));
              }
            }
            __syncwarp();  // the slot is read out before it is refilled
          }
        }
        hq = (hq + NH) % 3;
      } else if (EPI == 2) {
        // C += acc, with the C blocks fetched above
#pragma unroll
        for (int i = 0; i < kPre; ++i) {
          const int c = ch + i * CSTEP;
          if (c < nch_acc) {
            const int64_t col0 = n0 + c * 32;
            tmem_ld32(tbase + c * 32, v);
            __syncwarp();
            acc_put(stg, lane, pre[i]);
            __syncwarp();
            stage_get<RB>(stg, lane, pk);
            float o[32];
#pragma unroll
            for (int i = 0; i < NP; ++i) unpack16<TC>(pk[i], o + i * Vec<TC>::N);
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] += v[i];
#pragma unroll
            for (int i = 0; i < NP; ++i) pk[i] = pack16<TC>(o + i * Vec<TC>::N);
            stage_put<RB>(stg, lane, pk);
            __syncwarp();
            stage_store<RB>(stg, lane, c_rows + col0 * sizeof(TC), ldc_b, nrows);
          }
        }
      } else if (EPI == 0 && n0 + BN <= p.N) {
        // every column of the tile exists: chunk i + 1's TMEM load is in
        // flight while chunk i is staged and stored
        constexpr int NC = BN / 32 / CSTEP;  // this warp's chunks: ch, ch + CSTEP, ...
        static_assert(RPC == 1 && NC % 2 == 0, "one staging round per chunk, chunks in pairs");
        uint32_t ra[32], rb[32];
        auto put = [&](const uint32_t(&r)[32], int i) {
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
#pragma unroll
          for (int j = 0; j < NP; ++j) pk[j] = pack16<TC>(v + j * Vec<TC>::N);
          __syncwarp();
          stage_put<RB>(stg, lane, pk);
          __syncwarp();
          stage_store<RB>(stg, lane, c_rows + (n0 + (ch + i * CSTEP) * 32) * sizeof(TC), ldc_b, nrows);
        };
        tmem_ld32_issue(tbase + ch * 32, ra);
#pragma unroll 1
        for (int i = 0; i < NC; i += 2) {
          tmem_ld_wait(ra);
          tmem_ld32_issue(tbase + (ch + (i + 1) * CSTEP) * 32, rb);
          put(ra, i);
          tmem_ld_wait(rb);
          if (i + 2 < NC) tmem_ld32_issue(tbase + (ch + (i + 2) * CSTEP) * 32, ra);
          put(rb, i + 1);
        }
      } else {
#pragma unroll 1
        for (int c = ch; c < BN / 32; c += CSTEP) {
          const int64_t col0 = n0 + c * 32;
          if (col0 >= p.N) break;
          tmem_ld32(tbase + c * 32, v);
          const int nvalid = (int)imin64(32, p.N - col0);
          if (EPI == 1 || nvalid < 32) {
            // router logits (E columns, possibly ragged): direct row stores
            if (!vrow) continue;
            TC* crow = Cb + grow * p.ldc;
            if (EPI == 1 && p.bias) {
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (i < nvalid) v[i] += p.bias[col0 + i];
            }
            if (EPI == 2) {
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (i < nvalid) v[i] += to_f32<TC>(crow[col0 + i]);
            }
            store_row32<TC>(crow + col0, v, nvalid);
            if (EPI == 4) {
#pragma unroll
              for (int i = 0; i < 32; ++i) v[i] = fmaxf(v[i], 0.f) * fmaxf(v[i], 0.f);
              store_row32<TC>(static_cast<TC*>(p.aux) + grow * p.ldc + col0, v, nvalid);
            }
          } else if (EPI == 0 || EPI == 4) {
#pragma unroll
            for (int r = 0; r < RPC; ++r) {
#pragma unroll
              for (int i = 0; i < NP; ++i) pk[i] = pack16<TC>(v + r * CPR + i * Vec<TC>::N);
              __syncwarp();
              stage_put<RB>(stg, lane, pk);
              __syncwarp();
              stage_store<RB>(stg, lane, c_rows + (col0 + r * CPR) * sizeof(TC), ldc_b, nrows);
            }
            if (EPI == 4) {
              // a = relu(h)^2 at the same positions of aux
              uint8_t* a_rows = reinterpret_cast<uint8_t*>(static_cast<TC*>(p.aux)) + rbase * ldc_b;
#pragma unroll
              for (int i = 0; i < 32; ++i) v[i] = fmaxf(v[i], 0.f) * fmaxf(v[i], 0.f);
#pragma unroll
              for (int r = 0; r < RPC; ++r) {
#pragma unroll
                for (int i = 0; i < NP; ++i) pk[i] = pack16<TC>(v + r * CPR + i * Vec<TC>::N);
                __syncwarp();
                stage_put<RB>(stg, lane, pk);
                __syncwarp();
                stage_store<RB>(stg, lane, a_rows + (col0 + r * CPR) * sizeof(TC), ldc_b, nrows);
              }
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        // the accumulator buffer is free once every epilogue warp of the tile drained it
        if (CG == 2) mbar_arrive_cluster(map_to_rank(smem_u32(&tempty[acc]), 0));
        else mbar_arrive(smem_u32(&tempty[acc]));
      }
      if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
    }
    if (EPI == 5) cp_async_wait_all();  // no h copy is still landing when the CTA exits
  }

  tc_fence_before();
  __syncthreads();
  if (CG == 2) cluster_sync();  // neither CTA frees TMEM or exits while the other may still signal it
  tc_fence_after();
  if (warp == 1) tmem_dealloc_cg<CG>(tmem_base, C::kCols);
}

// Tail maps for Group::K.  A group's whole k-blocks are read through the
// full-tensor maps; its last r = n % BK rows (0 < r < BK) through tail maps:
// host-encoded templates of exactly r rows (TailTemplates, one per r) whose
// base the device moves to the group's first tail row.  Only the address is
// replaced on the device, which leaves a map identical to a host encoding of
// the same tensor; the copy engine zero-fills the block's rows past the
// group's end, so the next group's rows never enter the reduction, and every
// map's base lies inside its tensor.  out[2g] = A, out[2g + 1] = B (none for
// a group whose row count is a multiple of BK).  With offsets == nullptr the
// groups are the G splits of [0, split_rows) that the GEMM forms itself
// (Params::split_rows), of which only the last can have a tail.
// One warp per group: the template is copied into shared memory, its address
// is replaced there (tensormap.replace on shared::cta), and the warp copies
// the finished map to global memory with tensormap.cp_fenceproxy, which
// releases it to the tensormap proxy; the GEMM's producer acquires it before
// its copy.
struct TailTemplates {
  CUtensorMap a[BK];  // [r]: r rows (r = 1 .. BK - 1)
  CUtensorMap b[BK];
};
// The tail templates of two Group::K GEMMs (index r - 1 for r rows), for one
// launch that builds the maps of both: 4 x 63 maps fit the 32764-byte kernel
// parameter limit with the launch's other arguments.
struct TailTemplatesPair {
  CUtensorMap a[2][BK - 1];
  CUtensorMap b[2][BK - 1];
};
static_assert(sizeof(TailTemplatesPair) + 256 <= 32764, "kernel parameter limit");
constexpr int kMapWarps = 4;

// One group's tail maps, by one warp: the templates for its r = (hi - lo) % BK
// rows (ta1[r - 1], tb1[r - 1]; tb1 unused without b_base) moved to the
// group's first tail row and copied to out2[0], out2[1].
__device__ __forceinline__ void build_tail_maps(CUtensorMap* sm, int lane, const CUtensorMap* ta1,
                                                const CUtensorMap* tb1, int64_t lo, int64_t hi,
                                                const uint8_t* a_base, int64_t a_row_bytes, const uint8_t* b_base,
                                                int64_t b_row_bytes, CUtensorMap* out2) {
  const int r = (int)((hi - lo) % BK);
  if (r == 0) return;  // no tail: every k-block of the group is whole
  const int64_t first = hi - r;
  const bool has_b = b_base != nullptr;  // NULL: B is gathered row by row (no tail B map)
  // 32 lanes x 4 bytes = one 128-byte map
  reinterpret_cast<uint32_t*>(&sm[0])[lane] = reinterpret_cast<const uint32_t*>(&ta1[r - 1])[lane];
  if (has_b) reinterpret_cast<uint32_t*>(&sm[1])[lane] = reinterpret_cast<const uint32_t*>(&tb1[r - 1])[lane];
  __syncwarp();
  const uint32_t sa = smem_u32(&sm[0]), sb = smem_u32(&sm[1]);
  if (lane == 0) {
    const uint64_t pa = reinterpret_cast<uint64_t>(a_base + first * a_row_bytes);
    asm volatile("tensormap.replace.tile.global_address.shared::cta.b1024.b64 [%0], %1;" ::"r"(sa), "l"(pa)
                 : "memory");
    if (has_b) {
      const uint64_t pb = reinterpret_cast<uint64_t>(b_base + first * b_row_bytes);
      asm volatile("tensormap.replace.tile.global_address.shared::cta.b1024.b64 [%0], %1;" ::"r"(sb), "l"(pb)
                   : "memory");
    }
  }
  __syncwarp();
  asm volatile(
      "tensormap.cp_fenceproxy.global.shared::cta.tensormap::generic.release.gpu.sync.aligned [%0], [%1], 128;" ::"l"(
          reinterpret_cast<uint64_t>(out2)),
      "r"(sa)
      : "memory");
  if (has_b)
    asm volatile(
        "tensormap.cp_fenceproxy.global.shared::cta.tensormap::generic.release.gpu.sync.aligned [%0], [%1], 128;" ::
            "l"(reinterpret_cast<uint64_t>(out2 + 1)),
        "r"(sb)
        : "memory");
}

__global__ void __launch_bounds__(32 * kMapWarps) build_group_maps(
    const __grid_constant__ TailTemplates tt, const int32_t* __restrict__ offsets, int G, int64_t split_rows,
    const uint8_t* a_base, int64_t a_row_bytes, const uint8_t* b_base, int64_t b_row_bytes, CUtensorMap* out) {
  __shared__ alignas(128) CUtensorMap sm[kMapWarps][2];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = blockIdx.x * kMapWarps + warp;
  if (g >= G) return;  // the whole warp
  int64_t lo, hi;
  if (offsets) {
    lo = offsets[g];
    hi = offsets[g + 1];
  } else {
    lo = (split_rows * g / G) & ~(int64_t)(BK - 1);
    hi = g + 1 < G ? (split_rows * (g + 1) / G) & ~(int64_t)(BK - 1) : split_rows;
  }
  build_tail_maps(sm[warp], lane, &tt.a[1], &tt.b[1], lo, hi, a_base, a_row_bytes, b_base, b_row_bytes,
                  out + 2 * g);
}

// The tail maps of two Group::K GEMMs over the same groups (the two expert
// weight gradients), in one launch: warp w builds GEMM w / G's maps of group
// w % G.
__global__ void __launch_bounds__(32 * kMapWarps) build_group_maps_pair(
    const __grid_constant__ TailTemplatesPair tt, const int32_t* __restrict__ offsets, int G,
    const uint8_t* a_base0, int64_t a_row_bytes0, const uint8_t* b_base0, int64_t b_row_bytes0, CUtensorMap* out0,
    const uint8_t* a_base1, int64_t a_row_bytes1, const uint8_t* b_base1, int64_t b_row_bytes1, CUtensorMap* out1) {
  __shared__ alignas(128) CUtensorMap sm[kMapWarps][2];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int w = blockIdx.x * kMapWarps + warp;
  if (w >= 2 * G) return;  // the whole warp
  const int k = w / G, g = w - k * G;
  const int64_t lo = offsets[g], hi = offsets[g + 1];
  if (k == 0)
    build_tail_maps(sm[warp], lane, tt.a[0], tt.b[0], lo, hi, a_base0, a_row_bytes0, b_base0, b_row_bytes0,
                    out0 + 2 * g);
  else
    build_tail_maps(sm[warp], lane, tt.a[1], tt.b[1], lo, hi, a_base1, a_row_bytes1, b_base1, b_row_bytes1,
                    out1 + 2 * g);
}

}  // namespace tc
}  // namespace moe
