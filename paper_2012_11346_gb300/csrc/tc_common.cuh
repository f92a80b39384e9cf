// Blackwell (sm_103a) tensor-core building blocks for libslim, in inline PTX:
// mbarriers with bounded waits, tcgen05 TMEM allocation / MMA / commit / load,
// 128-byte-swizzled shared-memory operand layouts and their descriptors.
//
// Operand tiles.  Every bf16 operand lives in shared memory as "row tiles":
// a row-major [R][64] block, 128 bytes per row, 1024-byte aligned, with the
// 16-byte chunk c of row r stored at chunk position c ^ (r % 8) (the 128B
// swizzle).  A matrix with more than 64 columns is a sequence of such blocks
// (columns 64b..64b+63 in block b, blocks R*128 bytes apart).  The same bytes
// serve as
//   * a K-major operand (rows = M or N index, columns = K), and
//   * an MN-major operand (columns = M or N index, rows = K),
// which only changes the descriptor:
//   K-major : start + 32 B per 16-element K step inside a block, next block
//             for the next 64 K; SBO = 1024 B (8 rows), LBO unused.
//   MN-major: start + 2048 B per 16-element K step (16 rows); LBO = byte
//             distance between 64-column blocks, SBO = 1024 B (8 K rows).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace slim {
namespace tc {

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ------------------------------------------------------------------ mbarrier
__device__ __forceinline__ void mbar_init(uint32_t addr, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(addr), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t addr, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(addr), "r"(parity)
      : "memory");
  return ok != 0;
}
// ------------------------------------------------------------------ bounded waits
// Every wait of a kernel is bounded by time: after kWaitLimitNs of the global
// timer (and, as a second bound, a fixed number of polls) it gives up.
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // 1 s
constexpr uint32_t kWaitMaxPolls = 1u << 24;
__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// The error word of a call sits at the start of its workspace.  Word 0 is set
// by a wait that gives up; the other CTAs of the call poll it and leave early.
// Bytes 8..15 hold the address of a host-visible report counter (or zero),
// stored by the call's first kernel, which a wait that gives up also
// increments, so that the next call on the workspace learns of it without
// synchronising the device.  The grid-dependency wait first makes that
// kernel's store visible (it returns at once where there is nothing to wait
// for, and a wait gives up only after a second anyway).
__device__ __forceinline__ void give_up(int* err) {
  atomicExch(err, 1);
  asm volatile("griddepcontrol.wait;" ::: "memory");
  unsigned* rep = reinterpret_cast<unsigned* const volatile*>(err)[1];
  if (rep) atomicAdd_system(rep, 1u);
}
// Stores a call's report-counter address beside its error word (thread 0 of
// the call's first kernel).
__device__ __forceinline__ void set_report(int* err, unsigned* rep) {
  reinterpret_cast<unsigned**>(err)[1] = rep;
}
// Bounded mbarrier wait: records a failure and returns false when it gives up.
// err is a workspace error word (see give_up), or, with workspace_word false,
// a plain int that is only set.
__device__ __forceinline__ bool mbar_wait(uint32_t addr, uint32_t parity, int* err,
                                          bool workspace_word = true) {
  if (mbar_try_wait(addr, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 0; i < kWaitMaxPolls; ++i) {
    if (mbar_try_wait(addr, parity)) return true;
    if (i > 16) __nanosleep(256);
    if ((i & 15) == 15 && globaltimer_ns() - t0 > kWaitLimitNs) break;
  }
  if (err) {
    if (workspace_word)
      give_up(err);
    else
      atomicExch(err, 1);
  }
  return false;
}

// ------------------------------------------------------------------ bulk copies
// Plain (non-tensor) bulk copies between global and shared memory: both
// addresses 16-byte aligned, the size a multiple of 16.  A load completes on
// an mbarrier that expects its bytes; stores complete per bulk group of the
// issuing thread.
__device__ __forceinline__ void mbar_expect_tx(uint32_t mbar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(mbar), "r"(bytes)
               : "memory");
}
// An L2 policy that marks the lines an access touches first to be evicted:
// for data read or written for the last time, so that it does not push out
// data that is read again later.
__device__ __forceinline__ uint64_t l2_evict_first() {
  uint64_t p;
  asm("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// ------------------------------------------------------------------ TMA tile loads
// Tensor-map loads into 128-byte-swizzled row tiles (the layout above): the
// map's box is {64 bf16, R rows[, 1]} with CU_TENSOR_MAP_SWIZZLE_128B, the
// shared destination is 1024-byte aligned, and the innermost coordinate is 0
// (16-byte aligned).  Elements outside the tensor read as zero.  The map is a
// __grid_constant__ kernel parameter (param space); completion is counted on
// mbar like a bulk copy.
__device__ __forceinline__ void tma_load_3d(uint32_t sdst, const CUtensorMap* map, int y, int z,
                                            uint32_t mbar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3, %4}], [%5];" ::"r"(sdst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(y), "r"(z), "r"(mbar)
      : "memory");
}
__device__ __forceinline__ void tma_load_2d(uint32_t sdst, const CUtensorMap* map, int y,
                                            uint32_t mbar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3}], [%4];" ::"r"(sdst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(y), "r"(mbar)
      : "memory");
}

// Brings `bytes` (a multiple of 16, 16-byte aligned) of global memory into L2
// ahead of a later load.
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
// The source is read for the last time (evict-first in L2).
__device__ __forceinline__ void bulk_load(uint32_t sdst, const void* gsrc, uint32_t bytes,
                                          uint32_t mbar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
      "[%0], [%1], %2, [%3], %4;" ::"r"(sdst),
      "l"(gsrc), "r"(bytes), "r"(mbar), "l"(l2_evict_first())
      : "memory");
}
__device__ __forceinline__ void bulk_store(void* gdst, uint32_t ssrc, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(gdst), "r"(ssrc),
               "r"(bytes)
               : "memory");
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// The shared source of this thread's bulk stores may be overwritten.
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// This thread's bulk stores are complete, and ordered before its later
// generic operations (a release that publishes them).
__device__ __forceinline__ void bulk_wait_done() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
  asm volatile("fence.proxy.async.global;" ::: "memory");
}
// Orders this thread's earlier generic accesses (an acquire) before its later
// async-proxy accesses to global memory (bulk loads of what was published).
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// ------------------------------------------------------------------ proxies / fences
__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// ------------------------------------------------------------------ TMEM
// Executed by one whole warp.  Writes the TMEM base address to smem.
__device__ __forceinline__ void tmem_alloc(uint32_t smem_dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_dst),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

// 32 consecutive fp32 columns of this thread's TMEM lane (warp w reads lanes
// 32w..32w+31; `taddr` carries the lane base in bits 31:16).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_ld1(uint32_t taddr, float& v) {
  uint32_t r;
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(r) : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
  v = __uint_as_float(r);
}

// ------------------------------------------------------------------ MMA
// Instruction descriptor, kind::f16 with bf16 A/B and fp32 accumulate.
// a_mn / b_mn = 1 selects the MN-major (transposed) operand layout.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, int a_mn, int b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)a_mn << 15) | ((uint32_t)b_mn << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// Shared-memory matrix descriptor, 128-byte swizzle.
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version of tcgen05
  d |= (uint64_t)2 << 61;  // 128-byte swizzle
  return d;
}
// The start-address field holds address >> 4 in the low 14 bits, and shared
// memory offsets stay below 256 KB, so the descriptor of a later position in
// the same operand is the base descriptor plus (byte offset >> 4).  Every
// offset below is a multiple of 16 bytes, and the base descriptor is loop
// invariant, so an MMA loop pays one 64-bit add per operand.
// K-major operand stored as row tiles of `rows` rows: element (row, k0..k0+15).
__device__ __forceinline__ uint64_t kmaj(uint32_t base, int rows, int k0) {
  return sdesc(base, 16, 1024) + (uint64_t)((k0 >> 6) * rows * 8 + (k0 & 63) / 8);
}
// MN-major operand stored as row tiles whose rows are K and columns MN:
// K rows k0..k0+15, MN blocks `block_bytes` apart.
__device__ __forceinline__ uint64_t mnmaj(uint32_t base, int k0, uint32_t block_bytes) {
  return sdesc(base, block_bytes, 1024) + (uint64_t)(k0 * 8);
}

// D[tmem] (+)= A * B, issued by a single thread.
__device__ __forceinline__ void mma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                    uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
      ::"r"(d_tmem), "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on the mbarrier once every MMA issued so far by this thread is done.
__device__ __forceinline__ void mma_commit(uint32_t mbar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(mbar)
      : "memory");
}

// ------------------------------------------------------------------ tile memory
// Byte offset of element (r, c) inside a row tile with R rows (c may exceed 63).
__device__ __forceinline__ uint32_t tile_off(int R, int r, int c) {
  return (uint32_t)((c >> 6) * R * 128 + r * 128 + ((((c & 63) >> 3) ^ (r & 7)) << 4) +
                    (c & 7) * 2);
}
// Stores 8 consecutive bf16 (one 16-byte chunk, c multiple of 8).
__device__ __forceinline__ void st_chunk(uint8_t* tile, int R, int r, int c, uint4 v) {
  *reinterpret_cast<uint4*>(tile + tile_off(R, r, c)) = v;
}
__device__ __forceinline__ uint4 ld_chunk(const uint8_t* tile, int R, int r, int c) {
  return *reinterpret_cast<const uint4*>(tile + tile_off(R, r, c));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ void unpack_bf16(uint32_t u, float& lo, float& hi) {
  __nv_bfloat162 h = *reinterpret_cast<__nv_bfloat162*>(&u);
  lo = __low2float(h);
  hi = __high2float(h);
}

// cp.async of one 16-byte chunk; src_bytes = 0 zero-fills the destination.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

// Loads rows [0, R) of a row-major [.][64] bf16 global matrix (row stride 64
// elements) into a row tile; rows >= valid are zero.  All `nthreads` threads
// of the CTA take part; completes with cp_async_wait_all().
__device__ __forceinline__ void load_rows64(uint8_t* tile, int R, const __nv_bfloat16* g,
                                            int valid, int tid, int nthreads) {
  const uint32_t base = smem_u32(tile);
  for (int e = tid; e < R * 8; e += nthreads) {
    const int r = e >> 3, c = (e & 7) * 8;
    const bool ok = r < valid;
    const __nv_bfloat16* src = g + (size_t)(ok ? r : 0) * 64 + c;
    cp_async16(base + tile_off(R, r, c), src, ok ? 16u : 0u);
  }
}

// Programmatic dependent launch: wait until the previous kernel in the stream
// has completed and its writes are visible (returns at once when the kernel
// was not launched as a dependent), then let the next kernel start launching.
// Work before grid_dependency_wait() may only touch data that no kernel of the
// same call writes (the caller's input tensors).
__device__ __forceinline__ void grid_dependency_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ex2 on the MUFU unit (approximate, ~2 ulp), used for the FAVOR+ features.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

}  // namespace tc
}  // namespace slim
