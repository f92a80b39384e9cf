// Tensor-core (tcgen05) path of libslim: bf16 inputs, d = 64, M in {128, 256}.
//
// Same slice algorithm as the fp32 path (Algorithm 1; App. B block form with
// masked tile products), on tiles of T = 128 rows with one CTA of 512 threads
// per (tile, chain).  Every tile product is a chain of tcgen05 MMAs on
// 128-byte-swizzled bf16 shared-memory operands with an fp32 accumulator in
// tensor memory.  In the row-wise epilogues warp w serves TMEM lanes
// 32(w%4)..32(w%4)+31 and column group w/4 of each row.
//
// State prefixes are chained from tile to tile.  The CTA of a tile computes
// its own delta Delta_t = phiK^T [V_t | 1], waits (bounded) for the prefix its
// neighbour tile left in a workspace slot, and leaves its own there for the
// next tile: inside a slice this is the prefix sum of eqs. 14-15, across a
// slice boundary it is the slice carry B^(n) (eq. 16).
//
//   forward, one launch, tiles in sequence order:
//     phiQ, phiK, Delta_t, A = tril(phiQ phiK^T);  S_t, z_t = prefix before
//     tile t;  num = phiQ S_t + A V_t,  den = phiQ z_t + rowsum A,  out = num/den
//   backward, one launch, slices in reverse (Algorithm 1's reverse sweep); one
//   CTA per tile runs the tile's dq part and then its dk/dv part:
//     dq part, tiles in reverse order: phiQ, phiK, Delta_t, A;
//       rollback P_t = P_{t+1} - Delta_t (eq. 17);  den, dnum = dout/den,
//       dden = -<dout,out>/den, dA = tril(dnum V^T + dden);
//       dphiQ = dnum S_t^T + dden z_t + dA phiK,  Gd_t = phiQ^T [dnum | dden];
//       state-gradient chain G_t = G_{t+1} + Gd_{t+1} (eq. 18);
//       dq = u Omega - q sum(u),  dOmega partial u^T q
//     dk/dv part of the same tile (phiQ still in shared memory):
//       dV = A^T dnum + phiK G_t(S),  dphiK = dA^T phiQ + V G_t(S)^T + g_t(z),
//       dk = u Omega - k sum(u),  dOmega partial u^T k (+ the dq part's u^T q)
//     the tile's dOmega partial goes onto one running sum per tile position
//     (slices in order N-1 .. 0), and the sums are reduced once, in a fixed
//     order, at the end of the launch
#include <math.h>

#include "common.cuh"
#include "profiler.h"
#include "tc_common.cuh"
#include "tc_path.h"

namespace slim {
namespace tc {

constexpr int T = 128;           // tile rows
constexpr int D = 64;            // head width handled here
constexpr int ROWT = T * 128;    // bytes of a [128][64] bf16 row tile
constexpr float kLog2e = 1.4426950408889634f;

template <int MF>
struct Cfg {
  static constexpr int MH = MF / 128;       // feature halves (MMA M = 128 each)
  static constexpr int FEATB = T * MF * 2;  // [128][MF] bf16 feature tile
  static constexpr int OMB = MF * 128;      // [MF][64] bf16 (Omega, state)
  static constexpr int E = MF * 64 + MF;    // state floats per tile
};

// ------------------------------------------------------------------ helpers
// NG warps share each TMEM lane quarter: warp w serves rows 32(w%4)..+31 and
// column group w/4 of every row-wise epilogue, so a row's element-wise work
// is spread over NG threads.
constexpr int NG = 4;
constexpr int NTHR = 128 * NG;

// Loads 16 bf16 of a feature-tile row (columns c..c+15) as floats.
__device__ __forceinline__ void ld_feat16(const uint8_t* tile, int r, int c, float* f) {
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    uint4 v = ld_chunk(tile, T, r, c + 8 * h);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) unpack_bf16(w[i], f[8 * h + 2 * i], f[8 * h + 2 * i + 1]);
  }
}

// Reads this thread's column group of the projection P = X Omega^T from TMEM,
// applies the feature map, stores phi (bf16) into the [128][MF] feature tile.
// Columns c0 = first, first + step, ... below last, 32 at a time.
template <int MF, int FEAT>
__device__ __forceinline__ void feature_cols(uint32_t trow, uint8_t* phi, int r, int first,
                                             int last, int step, float x2, bool valid) {
  // exp map: phi = 2^(p log2e - (|x|^2/2) log2e - log2 sqrt(M))
  const float bias = -0.5f * x2 * kLog2e - 0.5f * log2f((float)MF);
  const float relu_scale = rsqrtf((float)MF);
#pragma unroll 1
  for (int c0 = first; c0 < last; c0 += step) {
    float v[32];
    tmem_ld32(trow + c0, v);
    uint32_t pk[16];
#pragma unroll
    for (int i = 0; i < 32; i += 2) {
      float a, b;
      if (FEAT == SLIM_FEAT_EXP) {
        a = ex2_approx(fmaf(v[i], kLog2e, bias));
        b = ex2_approx(fmaf(v[i + 1], kLog2e, bias));
      } else {
        a = fmaxf(v[i], 0.f) * relu_scale;
        b = fmaxf(v[i + 1], 0.f) * relu_scale;
      }
      if (!valid) a = b = 0.f;
      pk[i / 2] = pack_bf16(a, b);
    }
#pragma unroll
    for (int q = 0; q < 4; ++q)
      st_chunk(phi, T, r, c0 + 8 * q, make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]));
  }
}
// This thread's column group cg (MF/NG contiguous columns).
template <int MF, int FEAT>
__device__ __forceinline__ void feature_epilogue(uint32_t trow, uint8_t* phi, int r, int cg,
                                                 float x2, bool valid) {
  constexpr int W = MF / NG;
  feature_cols<MF, FEAT>(trow, phi, r, cg * W, (cg + 1) * W, 32, x2, valid);
}

// Squared norm of columns 16cg..16cg+15 of row r of a [128][64] row tile.
__device__ __forceinline__ float row_norm2_part(const uint8_t* tile, int r, int cg) {
  float f[16];
  ld_feat16(tile, r, 16 * cg, f);
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < 16; ++i) s = fmaf(f[i], f[i], s);
  return s;
}

// Sum of the NG column-group partials of each row, through shared scratch
// red[NG][128] (the caller separates writes and reads with a barrier).
__device__ __forceinline__ float group_total(const float* red, int row) {
  float s = 0.f;
#pragma unroll
  for (int g = 0; g < NG; ++g) s += red[g * T + row];
  return s;
}

// 16 fp32 values -> 16 bf16 at global dst (32 bytes, 16-byte aligned).
// 16 values of an output row (out, dq, dk, dv: never read back here), so
// evict-first in L2.
__device__ __forceinline__ void st_row16(__nv_bfloat16* dst, const float* v) {
  const uint64_t pol = l2_evict_first();
#pragma unroll
  for (int h = 0; h < 2; ++h)
    asm volatile("st.global.L2::cache_hint.v4.u32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(dst + 8 * h),
                 "r"(pack_bf16(v[8 * h], v[8 * h + 1])), "r"(pack_bf16(v[8 * h + 2], v[8 * h + 3])),
                 "r"(pack_bf16(v[8 * h + 4], v[8 * h + 5])), "r"(pack_bf16(v[8 * h + 6], v[8 * h + 7])),
                 "l"(pol)
                 : "memory");
}
__device__ __forceinline__ void st_f32x16(float* dst, const float* v) {
  float4* o = reinterpret_cast<float4*>(dst);
#pragma unroll
  for (int i = 0; i < 4; ++i) o[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
}

// One single-use mbarrier per MMA commit, each waited on with parity 0.  A
// barrier reused across commits would let a warp that reaches its wait after
// two completions see the parity of a later, unfinished phase and wait for
// it; with one barrier per event a late warp simply finds its phase done.
struct Sync {
  uint64_t* mb;
  int next;  // barrier of the next wait()
  int* err;
  __device__ uint32_t bar(int i) const { return smem_u32(&mb[i]); }
  __device__ bool wait() {
    const bool ok = mbar_wait(smem_u32(&mb[next]), 0, err);
    ++next;
    tc_fence_after();
    return ok;
  }
};
constexpr int NBAR = 12;  // mbarriers per tile CTA (and per part of a backward tile)
// the ones for tensor-map loads: the row tiles, Omega, and a later reload
constexpr int MB_TILES = 9, MB_OMEGA = 10, MB_RELOAD = 11;

// Make generic-proxy smem writes visible to the tensor core and order them
// with the thread that issues the next MMAs.
__device__ __forceinline__ void publish() {
  fence_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
}

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// Abort after a failed wait: every thread leaves through the teardown.
#define TC_WAIT(sy)                  \
  do {                               \
    if (!(sy).wait()) abort_ = 1;    \
    __syncthreads();                 \
    if (abort_) goto teardown;       \
  } while (0)

#define TC_PROLOGUE()                                    \
  const int tid = threadIdx.x, warp = tid >> 5;         \
  const int row = 32 * (warp & 3) + (tid & 31);         \
  const int cg = warp >> 2;                             \
  (void)cg;                                             \
  if (tid == 0) {                                       \
    abort_ = 0;                                         \
    for (int i_ = 0; i_ < NBAR; ++i_) mbar_init(smem_u32(&mb[i_]), 1); \
    mbar_fence_init();                                  \
  }                                                     \
  if (warp == 0) tmem_alloc(smem_u32(&tmem_base), 512)

#define TC_TEARDOWN()                                   \
  teardown:                                             \
  cp_async_wait_all();                                  \
  bulk_wait_read();                                     \
  tc_fence_before();                                    \
  __syncthreads();                                      \
  if (warp == 0) tmem_dealloc(tmem_base, 512)

// The same, for a role that runs on TMEM its caller allocated and frees.
#define TC_TEARDOWN_KEEP()                              \
  teardown:                                             \
  cp_async_wait_all();                                  \
  bulk_wait_read();                                     \
  tc_fence_before();                                    \
  __syncthreads()

// ------------------------------------------------------------------ chained tile prefixes
// A slot holds one state (or state-gradient) prefix, [S (M x 64) | z (M)] in
// fp32; its flag holds n + 1 once slice n's prefix is in the slot.  The CTA
// that waits on a slot always has a higher block index than the CTA that
// fills it, so the filling CTA was dispatched first and is running or done.
__device__ __forceinline__ int ld_relaxed_gpu(const int* p) {
  int v;
  asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void fence_acq_rel_gpu() {
  asm volatile("fence.acq_rel.gpu;" ::: "memory");
}
__device__ __forceinline__ void st_release_gpu(int* p, int v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void red_release_gpu(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Drops the L2 lines of a buffer that nobody reads again before it is next
// written (discard.global.L2: the lines become undefined and are not written
// back to DRAM).  A discard is a weak write, so it is ordered before a later
// release like the thread's other writes.  p and bytes are multiples of 128;
// `nthr` threads share the lines.
__device__ __forceinline__ void discard_l2(const void* p, size_t bytes, int i, int nthr) {
  const char* b = static_cast<const char*>(p);
  for (size_t off = (size_t)i * 128; off < bytes; off += (size_t)nthr * 128)
    asm volatile("discard.global.L2 [%0], 128;" ::"l"(b + off) : "memory");
}

// Flags sit 128 bytes apart, so the CTAs polling different flags do not
// share a cache line.
constexpr int FLAG_STRIDE = 32;

// Buffers exchanged between tile CTAs (prefix slots, dOmega partials, G_t)
// are "lane-major": the 16 values a thread owns in an epilogue (row m = 128h +
// row, columns 16cg..16cg+15 of an [M][64] matrix) are spread over four float4
// at  q = ((h NG + cg) 4 + i) 128 + row,  so a warp's 32 rows are 512
// contiguous bytes and every warp access is coalesced.
__device__ __forceinline__ size_t lm4(int h, int cg, int i, int row) {
  return (size_t)((h * NG + cg) * 4 + i) * 128 + row;
}
// 16 floats of a chain prefix through L2 (the data is written by other CTAs
// of the same kernel, so L1 must not serve stale lines).  A prefix is read
// once, by the next tile of its chain: evict-first in L2.
__device__ __forceinline__ void ld_lm16(const float* base, int h, int cg, int row, float* v) {
  const float4* s = reinterpret_cast<const float4*>(base);
  const uint64_t pol = l2_evict_first();
#pragma unroll
  for (int i = 0; i < 4; ++i)
    asm volatile("ld.global.cg.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=f"(v[4 * i]), "=f"(v[4 * i + 1]), "=f"(v[4 * i + 2]), "=f"(v[4 * i + 3])
                 : "l"(s + lm4(h, cg, i, row)), "l"(pol)
                 : "memory");
}
__device__ __forceinline__ void st_lm16(float* base, int h, int cg, int row, const float* v) {
  float4* d = reinterpret_cast<float4*>(base);
#pragma unroll
  for (int i = 0; i < 4; ++i)
    __stcg(d + lm4(h, cg, i, row), make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]));
}
// Adds 16 floats to a lane-major buffer in L2 (one vector reduction per
// float4; the adds of one element are ordered by the flags around them).
__device__ __forceinline__ void red_lm16(float* base, int h, int cg, int row, const float* v) {
  float4* d = reinterpret_cast<float4*>(base);
#pragma unroll
  for (int i = 0; i < 4; ++i)
    asm volatile("red.relaxed.gpu.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(d + lm4(h, cg, i, row)),
                 "f"(v[4 * i]), "f"(v[4 * i + 1]), "f"(v[4 * i + 2]), "f"(v[4 * i + 3])
                 : "memory");
}
// Row-major [M][64] (the caller's state tensors): 16 floats at p.
__device__ __forceinline__ void ld_row16f(const float* p, float* v) {
  const float4* s = reinterpret_cast<const float4*>(p);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float4 x = __ldcg(s + i);
    v[4 * i] = x.x;
    v[4 * i + 1] = x.y;
    v[4 * i + 2] = x.z;
    v[4 * i + 3] = x.w;
  }
}
// bf16 lane-major: 16-byte chunk k = ((h NG + cg) 2 + half) 128 + row holds
// row 128h + row, columns 16cg + 8 half .. +7.
__device__ __forceinline__ void st_lm16_bf16(__nv_bfloat16* base, int h, int cg, int row, const float* v) {
  uint4* d = reinterpret_cast<uint4*>(base);
#pragma unroll
  for (int hf = 0; hf < 2; ++hf)
    d[(size_t)((h * NG + cg) * 2 + hf) * 128 + row] =
        make_uint4(pack_bf16(v[8 * hf], v[8 * hf + 1]), pack_bf16(v[8 * hf + 2], v[8 * hf + 3]),
                   pack_bf16(v[8 * hf + 4], v[8 * hf + 5]), pack_bf16(v[8 * hf + 6], v[8 * hf + 7]));
}
// Copies an [MF][64] bf16 lane-major matrix into an [MF][64] row tile
// (cp.async, coalesced reads; completes with cp_async_wait_all()).
__device__ __forceinline__ void load_lm_bf16(uint8_t* tile, int MF, const __nv_bfloat16* g, int tid) {
  const uint32_t base = smem_u32(tile);
  for (int k = tid; k < MF * 8; k += NTHR) {
    const int row = k & 127, rest = k >> 7, hf = rest & 1, cg = (rest >> 1) % NG, h = rest / (2 * NG);
    cp_async16(base + tile_off(MF, 128 * h + row, 16 * cg + 8 * hf), g + (size_t)k * 8, 16u);
  }
}
// 16 floats as bf16 into columns c..c+15 of row r of a [R][64] row tile.
__device__ __forceinline__ void st_tile16(uint8_t* tile, int R, int r, int c, const float* v) {
  st_chunk(tile, R, r, c, make_uint4(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]),
                                     pack_bf16(v[4], v[5]), pack_bf16(v[6], v[7])));
  st_chunk(tile, R, r, c + 8, make_uint4(pack_bf16(v[8], v[9]), pack_bf16(v[10], v[11]),
                                         pack_bf16(v[12], v[13]), pack_bf16(v[14], v[15])));
}

// One side of a chain link: where a prefix lives.  S rows are 64 floats
// apart; lo (optional) adds a low-order residual to every value.
struct StateRef {
  const float *S, *z, *S_lo, *z_lo;
};

__device__ __forceinline__ void fill_ones(uint8_t* tile, int tid) {
  for (int e = tid; e < 4096 / 16; e += NTHR)
    reinterpret_cast<uint4*>(tile)[e] = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
}

// ================================================================== forward
struct FwdJob {
  // tensor maps of q, k, v ([chains][L][64] bf16, box {64, 128, 1}) and of
  // Omega's bf16 hi/lo rows ([2 M][64], box {64, M})
  CUtensorMap tq, tk, tv, tom;
  const __nv_bfloat16 *Q, *K, *V, *om16;
  int L, Cs, N, nt, P, chains;  // slice length, slices, tiles of a full slice, tile positions
  float* slot;                  // [chains][nt][E] inclusive prefixes
  int* flag;                    // [chains][nt], FLAG_STRIDE ints apart
  int* ticket;                  // tile counter of this launch (starts at 0)
  __nv_bfloat16* out;
  StateOut st;                  // B^(N), written by the last tile of each chain
  StateInit init;               // B^(0), read by the first tile of each chain (null: zero)
  int* err;
};

// The forward splits its warps after the g(K) epilogue: warps 0-7 (column
// groups 0, 1) compute g(Q), A and the A epilogue, while warps 8-15 (column
// groups 2, 3) take the chain hop, which needs only Delta_t.  Each MMA
// completion has its own single-use mbarrier, so the two groups wait on
// different events without sharing a phase.
constexpr int GRP = NTHR / 2;
__device__ __forceinline__ void group_bar(int id) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(GRP) : "memory");
}
// publish() for one warp group.
__device__ __forceinline__ void group_publish(int id) {
  fence_async_smem();
  tc_fence_before();
  group_bar(id);
  tc_fence_after();
}
// Bounded poll of a flag by one thread: returns once *flag == want (then an
// acquire fence).  It gives up after kWaitLimitNs (or kWaitMaxPolls polls), or
// early once another CTA has reported an error (checked every 64 polls, so
// that waiting CTAs do not all hammer the error word); a wait that gives up
// records itself through give_up(err).
__device__ __forceinline__ bool flag_poll(const int* flag, int want, int* err) {
  uint64_t t0 = 0;
  for (uint32_t i = 0; i < kWaitMaxPolls; ++i) {
    if (ld_relaxed_gpu(flag) == want) {
      fence_acq_rel_gpu();
      return true;
    }
    if ((i & 63) == 63) {
      if (*reinterpret_cast<volatile int*>(err) != 0) return false;
      if (i == 63) t0 = globaltimer_ns();
      else if (globaltimer_ns() - t0 > kWaitLimitNs) break;
    }
    __nanosleep(i < 16 ? 32 : 256);
  }
  give_up(err);
  return false;
}
// Bounded wait by one thread for up to two flags at once (a null flag is not
// waited on): both are read in every round, so a satisfied pair costs one trip.
__device__ __forceinline__ bool flag_poll2(const int* f1, int w1, const int* f2, int w2, int* err) {
  uint64_t t0 = 0;
  for (uint32_t i = 0; i < kWaitMaxPolls; ++i) {
    const int v1 = f1 ? ld_relaxed_gpu(f1) : w1;
    const int v2 = f2 ? ld_relaxed_gpu(f2) : w2;
    if (v1 == w1 && v2 == w2) {
      fence_acq_rel_gpu();
      return true;
    }
    if ((i & 63) == 63) {
      if (*reinterpret_cast<volatile int*>(err) != 0) return false;
      if (i == 63) t0 = globaltimer_ns();
      else if (globaltimer_ns() - t0 > kWaitLimitNs) break;
    }
    __nanosleep(i < 16 ? 32 : 256);
  }
  give_up(err);
  return false;
}
// The thread that polls the flags a tile needs from other tiles: lane 0 of
// the last warp, which takes no part in the tile loads, so its fence waits on
// no copies of its own.
constexpr int POLL = NTHR - 32, LDT = NTHR - 32;
// Bounded wait by one thread for a counter to reach at least want.
__device__ __forceinline__ bool counter_poll(const int* ctr, int want, int* err) {
  uint64_t t0 = 0;
  for (uint32_t i = 0; i < kWaitMaxPolls; ++i) {
    if (ld_relaxed_gpu(ctr) - want >= 0) {
      fence_acq_rel_gpu();
      return true;
    }
    if ((i & 63) == 63) {
      if (*reinterpret_cast<volatile int*>(err) != 0) return false;
      if (i == 63) t0 = globaltimer_ns();
      else if (globaltimer_ns() - t0 > kWaitLimitNs) break;
    }
    __nanosleep(i < 16 ? 32 : 256);
  }
  give_up(err);
  return false;
}

template <int MF, int FEAT>
__device__ __forceinline__ void role_fwd(const FwdJob& J, int pos, int c, uint8_t* smem_raw,
                                         uint64_t* mb, uint32_t& tmem_base, int& abort_) {
  using C = Cfg<MF>;
  uint8_t* base = align1024(smem_raw);
  uint8_t* sPhiQ = base;
  uint8_t* sPhiK = sPhiQ + C::FEATB;
  uint8_t* sQ = sPhiK + C::FEATB;  // later: A tile (2 row tiles)
  uint8_t* sK = sQ + ROWT;
  uint8_t* sA = sQ;
  uint8_t* sOm = sK + ROWT;        // later: S_t (bf16)
  uint8_t* sS = sOm;
  uint8_t* sV = sOm + C::OMB;
  uint8_t* sOnes = sV + ROWT;      // [16][128] K-major, all ones (8 KB region)
  uint8_t* sZt = sOnes;            // later: [16][MF] K-major, rows z_hi, z_lo, then zeros
  float* redA = reinterpret_cast<float*>(sOnes + 8192);  // [2][128] row sums of A
  int* gfail = reinterpret_cast<int*>(redA + 2 * T);    // [2] per-group failure flags
  // tile t of slice n
  const int n = min(pos / J.nt, J.N - 1), t = pos - n * J.nt;
  const int a = n * J.Cs, slen = min(J.Cs, J.L - a);
  const int row0 = a + t * T;
  const int valid = min(T, slen - t * T);
  const size_t g0 = ((size_t)c * J.L + row0) * D;
  // the tile before in sequence order (none for the first) and this tile's slot
  const int tp = t > 0 ? t - 1 : J.nt - 1;
  const float* pred = pos > 0 ? J.slot + ((size_t)c * J.nt + tp) * C::E : nullptr;
  const int* pflag = J.flag + ((size_t)c * J.nt + tp) * FLAG_STRIDE;
  const int pwant = (t > 0 ? n : n - 1) + 1;
  float* own = J.slot + ((size_t)c * J.nt + t) * C::E;
  int* oflag = J.flag + ((size_t)c * J.nt + t) * FLAG_STRIDE;
  const bool last = pos == J.P - 1;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int row = 32 * (warp & 3) + (tid & 31);
  const int cg = warp >> 2;
  if (tid == 0) {
    abort_ = 0;
    for (int i = 0; i < NBAR; ++i) mbar_init(smem_u32(&mb[i]), 1);
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(smem_u32(&tmem_base), 512);
  // Omega lo in the upper half of the phiQ tile: that half is written only
  // by the g(Q) epilogue, after the Q projection (the last reader) is done,
  // while the phiK tile is overwritten as soon as the K projection is done
  uint8_t* sOl = sPhiQ + C::OMB;
  if (tid == 0) {
    // the three row tiles by TMA (rows past the chain's end read as zero)
    const uint32_t bar = smem_u32(&mb[MB_TILES]);
    mbar_expect_tx(bar, 3 * ROWT);
    tma_load_3d(smem_u32(sQ), &J.tq, row0, c, bar);
    tma_load_3d(smem_u32(sK), &J.tk, row0, c, bar);
    tma_load_3d(smem_u32(sV), &J.tv, row0, c, bar);
  }
  fill_ones(sOnes, tid);
  if (tid < 2) gfail[tid] = 0;
  grid_dependency_wait();  // Omega (bf16) and the slots belong to earlier kernels
  if (tid == 0) {
    const uint32_t bar = smem_u32(&mb[MB_OMEGA]);
    mbar_expect_tx(bar, 2 * C::OMB);
    tma_load_2d(smem_u32(sOm), &J.tom, 0, bar);   // hi: rows [0, M)
    tma_load_2d(smem_u32(sOl), &J.tom, MF, bar);  // lo: rows [M, 2M)
  }
  __syncthreads();  // the barriers' initialisation is seen by every thread
  if (!mbar_wait(smem_u32(&mb[MB_TILES]), 0, J.err)) abort_ = 1;
  if (!mbar_wait(smem_u32(&mb[MB_OMEGA]), 0, J.err)) abort_ = 1;
  __syncthreads();
  if (abort_) goto teardown;
  {
    const bool rv = row < valid;
    float* redN = reinterpret_cast<float*>(sPhiQ);  // 4 KB scratch below Omega lo
    redN[cg * T + row] = row_norm2_part(sQ, row, cg);
    redN[(NG + cg) * T + row] = row_norm2_part(sK, row, cg);
    publish();
    const float q2 = group_total(redN, row), k2 = group_total(redN + NG * T, row);
    const uint32_t tmem = tmem_base;
    const uint32_t trow = tmem + ((uint32_t)(32 * (warp & 3)) << 16);
    if (tid == 0) {
      // K first: the chain needs only Delta_t
      const uint32_t aQ = smem_u32(sQ), aK = smem_u32(sK), aOm = smem_u32(sOm);
      const uint32_t aOl = smem_u32(sOl);
      for (int k0 = 0; k0 < D; k0 += 16) {
        mma(tmem + 256, kmaj(aK, T, k0), kmaj(aOm, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
        mma(tmem + 256, kmaj(aK, T, k0), kmaj(aOl, MF, k0), idesc_bf16(T, MF, 0, 0), 1);
      }
      mma_commit(smem_u32(&mb[0]));
      for (int k0 = 0; k0 < D; k0 += 16) {
        mma(tmem, kmaj(aQ, T, k0), kmaj(aOm, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
        mma(tmem, kmaj(aQ, T, k0), kmaj(aOl, MF, k0), idesc_bf16(T, MF, 0, 0), 1);
      }
      mma_commit(smem_u32(&mb[1]));
    }
    if (!mbar_wait(smem_u32(&mb[0]), 0, J.err)) abort_ = 1;
    tc_fence_after();
    __syncthreads();
    if (abort_) goto teardown;
    feature_epilogue<MF, FEAT>(trow + 256, sPhiK, row, cg, k2, rv);
    publish();
    if (tid == 0 || (C::MH > 1 && tid == 32)) {
      // Delta_t = phiK^T [V | 1], one feature half per issuing thread: two
      // issuers keep the tensor pipe fed with these narrow products
      const int h = tid == 0 ? 0 : 1;
      const uint32_t aPK = smem_u32(sPhiK), aV = smem_u32(sV), aOnes = smem_u32(sOnes);
      for (int k0 = 0; k0 < T; k0 += 16) {
        const uint64_t ad = mnmaj(aPK + h * 2 * ROWT, k0, ROWT);
        mma(tmem + 256 + 64 * h, ad, mnmaj(aV, k0, ROWT), idesc_bf16(T, 64, 1, 1), k0 > 0);
        mma(tmem + 384 + 16 * h, ad, kmaj(aOnes, 16, k0), idesc_bf16(T, 16, 1, 0), k0 > 0);
      }
      mma_commit(smem_u32(&mb[h == 0 ? 2 : 5]));
    }
    if (warp < 8) {
      // ---- compute group: g(Q), A = tril(g(Q) g(K)^T), A's bf16 tile and row sums
      if (!mbar_wait(smem_u32(&mb[1]), 0, J.err)) gfail[0] = 1;
      tc_fence_after();
      group_bar(1);
      if (gfail[0]) goto join;
      feature_cols<MF, FEAT>(trow, sPhiQ, row, 32 * cg, MF, 64, q2, rv);
      group_publish(1);
      if (tid == 0) {
        const uint32_t aPQ = smem_u32(sPhiQ), aPK = smem_u32(sPhiK);
        for (int k0 = 0; k0 < MF; k0 += 16)
          mma(tmem, kmaj(aPQ, T, k0), kmaj(aPK, T, k0), idesc_bf16(T, T, 0, 0), k0 > 0);
        mma_commit(smem_u32(&mb[3]));
      }
      if (!mbar_wait(smem_u32(&mb[3]), 0, J.err)) gfail[0] = 1;
      tc_fence_after();
      group_bar(1);
      if (gfail[0]) goto join;
      float rs = 0.f;
#pragma unroll 1
      for (int c0 = 32 * cg; c0 < T; c0 += 64) {
        float v[32];
        tmem_ld32(trow + c0, v);
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          const float x0 = (c0 + i <= row) ? v[i] : 0.f;
          const float x1 = (c0 + i + 1 <= row) ? v[i + 1] : 0.f;
          pk[i / 2] = pack_bf16(x0, x1);
          float r0, r1;
          unpack_bf16(pk[i / 2], r0, r1);
          rs += r0 + r1;
        }
#pragma unroll
        for (int q = 0; q < 4; ++q)
          st_chunk(sA, T, row, c0 + 8 * q, make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]));
      }
      redA[cg * T + row] = rs;
    } else {
      // ---- chain group: S_t, z_t = the predecessor's inclusive prefix (zero
      // for the first tile); S_t + Delta_t goes to this tile's slot.  Thread
      // (row, cg) handles column groups 2(cg-2) and 2(cg-2)+1.
      const int gl = tid - GRP;  // 0..255
      if (!mbar_wait(smem_u32(&mb[2]), 0, J.err)) gfail[1] = 1;
      if (C::MH > 1 && !mbar_wait(smem_u32(&mb[5]), 0, J.err)) gfail[1] = 1;
      tc_fence_after();
      if (pred && gl == 0 && !gfail[1] && !flag_poll(pflag, pwant, J.err)) gfail[1] = 1;
      group_bar(2);
      if (gfail[1]) goto join;
      const int cq = 2 * (cg - 2);
      float pv[C::MH][2][16], pz[C::MH];
#pragma unroll
      for (int h = 0; h < C::MH; ++h) {
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          if (pred) {
            ld_lm16(pred, h, cq + j, row, pv[h][j]);
          } else if (J.init.S) {
            // the first tile of the sequence starts from the caller's B^(0)
            const size_t e = ((size_t)c * MF + 128 * h + row) * 64 + 16 * (cq + j);
            ld_row16f(J.init.S + e, pv[h][j]);
            if (J.init.S_lo) {
              float lo[16];
              ld_row16f(J.init.S_lo + e, lo);
#pragma unroll
              for (int i = 0; i < 16; ++i) pv[h][j][i] += lo[i];
            }
          } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) pv[h][j][i] = 0.f;
          }
        }
        pz[h] = 0.f;
        if (cq == 0) {
          const size_t e = (size_t)c * MF + 128 * h + row;
          if (pred)
            pz[h] = __ldcg(pred + MF * 64 + 128 * h + row);
          else if (J.init.z)
            pz[h] = __ldcg(J.init.z + e) + (J.init.z_lo ? __ldcg(J.init.z_lo + e) : 0.f);
        }
      }
#pragma unroll
      for (int h = 0; h < C::MH; ++h) {
        const int m = 128 * h + row;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          float inc[16];
          tmem_ld16(trow + 256 + 64 * h + 16 * (cq + j), inc);
#pragma unroll
          for (int i = 0; i < 16; ++i) inc[i] += pv[h][j][i];
          st_lm16(own, h, cq + j, row, inc);
          st_tile16(sS, MF, m, 16 * (cq + j), pv[h][j]);
          if (last) {
            st_f32x16(J.st.S + ((size_t)c * MF + m) * 64 + 16 * (cq + j), inc);
            if (J.st.S_lo) {
#pragma unroll
              for (int i = 0; i < 16; ++i) inc[i] = 0.f;
              st_f32x16(J.st.S_lo + ((size_t)c * MF + m) * 64 + 16 * (cq + j), inc);
            }
          }
        }
      }
      // z_t as the first two rows (hi, lo in bf16) of a K-major [16][MF]
      // operand, so that g(Q) z_t is a tensor-core product with ~16-bit z
      if (cq == 0) {
#pragma unroll
        for (int h = 0; h < C::MH; ++h) {
          const int m = 128 * h + row;
          float dz;
          tmem_ld1(trow + 384 + 16 * h, dz);
          __stcg(own + MF * 64 + m, pz[h] + dz);
          const __nv_bfloat16 zh = __float2bfloat16_rn(pz[h]);
          *reinterpret_cast<__nv_bfloat16*>(sZt + tile_off(16, 0, m)) = zh;
          *reinterpret_cast<__nv_bfloat16*>(sZt + tile_off(16, 1, m)) =
              __float2bfloat16_rn(pz[h] - __bfloat162float(zh));
          if (last) {
            J.st.z[(size_t)c * MF + m] = pz[h] + dz;
            if (J.st.z_lo) J.st.z_lo[(size_t)c * MF + m] = 0.f;
          }
        }
      } else {
        // rows 2..15 of the z operand are zero (the ones tile was there)
        for (int e = gl - 128; e < 14 * MF / 8; e += 128) {
          const int r16 = 2 + e / (MF / 8), k = (e % (MF / 8)) * 8;
          st_chunk(sZt, 16, r16, k, make_uint4(0u, 0u, 0u, 0u));
        }
      }
      group_bar(2);  // every slot write of the group is issued
      if (gl == 0) st_release_gpu(oflag, n + 1);
    }
  join:
    __syncthreads();
    if (gfail[0] | gfail[1]) goto teardown;
    publish();
    // three issuing threads: the narrow products are issue-bound
    if (tid == 0) {
      const uint32_t aPQ = smem_u32(sPhiQ), aS = smem_u32(sS);
      for (int k0 = 0; k0 < MF; k0 += 16)  // num = phiQ S_t
        mma(tmem + 128, kmaj(aPQ, T, k0), mnmaj(aS, k0, C::OMB), idesc_bf16(T, 64, 0, 1), k0 > 0);
      mma_commit(smem_u32(&mb[4]));
    } else if (tid == 64) {
      const uint32_t aA = smem_u32(sA), aV = smem_u32(sV);
      for (int k0 = 0; k0 < T; k0 += 16)  // + A V, in a second accumulator
        mma(tmem + 256, kmaj(aA, T, k0), mnmaj(aV, k0, ROWT), idesc_bf16(T, 64, 0, 1), k0 > 0);
      mma_commit(smem_u32(&mb[7]));
    } else if (tid == 32) {
      // phiQ [z_hi | z_lo], from a second issuing thread
      const uint32_t aPQ = smem_u32(sPhiQ), aZ = smem_u32(sZt);
      for (int k0 = 0; k0 < MF; k0 += 16)
        mma(tmem + 192, kmaj(aPQ, T, k0), kmaj(aZ, 16, k0), idesc_bf16(T, 16, 0, 0), k0 > 0);
      mma_commit(smem_u32(&mb[6]));
    }
    const float rsA = redA[row] + redA[T + row];
    if (!mbar_wait(smem_u32(&mb[4]), 0, J.err)) abort_ = 1;
    if (!mbar_wait(smem_u32(&mb[6]), 0, J.err)) abort_ = 1;
    if (!mbar_wait(smem_u32(&mb[7]), 0, J.err)) abort_ = 1;
    tc_fence_after();
    __syncthreads();
    if (abort_) goto teardown;
    {
      float zh, zl;
      tmem_ld1(trow + 192, zh);
      tmem_ld1(trow + 193, zl);
      const float den = rsA + (zh + zl);
      const float inv = den != 0.f ? 1.f / den : 0.f;
      float v[16], w[16];
      tmem_ld16(trow + 128 + 16 * cg, v);  // every lane loads (warp-aligned op)
      tmem_ld16(trow + 256 + 16 * cg, w);
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = (v[i] + w[i]) * inv;
      if (rv) st_row16(J.out + g0 + (size_t)row * D + 16 * cg, v);
    }
  }
  TC_TEARDOWN();
}

// ================================================================== backward, dq side
struct BwdQJob {
  // tensor maps (in the launch's parameters) of q, k, v, dout and Omega hi/lo
  const CUtensorMap *tq, *tk, *tv, *tdo, *tom;
  const __nv_bfloat16 *Q, *K, *V, *Out, *dOut, *om16;
  StateIn fin;            // B^(N), the state the forward returned
  int L, a, b, ntn, n, N, nt, chains;  // slice n = rows [a, a+b), ntn tiles; nt: full slice
  float *slot1, *slot2;   // [chains][nt][E]: state prefixes, state-gradient prefixes
  int *flag1, *flag2;     // [chains][nt], FLAG_STRIDE ints apart
  // Hand-off to the tile's dk/dv part, through the buffers of ring slot
  // n % R indexed by (chain, tile) of a full slice (written by this CTA and read
  // back by it, so they stay in L2; the dk/dv part discards them):
  __nv_bfloat16* gS;      // [chains][nt][MF][64] G_t(S)
  float* gz;              // [chains][nt][MF]     g_t(z)
  float* rowstat;         // [chains][nt][T][2]   (den, dden)
  float* domq;            // [chains][nt][MF][64] lane-major: the dOmega partial u^T q
  uint8_t* img;           // [chains][nt][FEATB + 32 KB]: phiK as its shared-memory tile
                          //   image (bf16, 128-byte swizzle), then tril(A) in bf16,
                          //   lane-major (chunk of 8 columns c/8, row r at 16-byte
                          //   unit (c/8) 128 + r)
  const int* kvread;      // [chains][nt]: n + R + 1 once slice n+R's dk/dv part has read them
  int ring;               // R, slots of the hand-off ring
  int nRtiles;            // tiles of slice n+R per chain (0: no such slice)
  __nv_bfloat16* dq;
  int* err;
  GradIO gio;             // G^(N) in (null: zero), G^(0) out (null: not returned)
};

// The dq part splits its warps twice, as the forward does: after the g(K)
// epilogue, warps 0-7 compute g(Q), A and dout V^T while warps 8-15 run the
// rollback chain (which needs only Delta_t); after dphiQ, warps 0-7 compute u
// and issue dq while warps 8-15 run the state-gradient chain.  The TMEM
// columns (all 512) are allocated by the caller for both parts of the tile.
template <int MF, int FEAT>
__device__ __forceinline__ void role_bwd_q(const BwdQJob& J, int b, uint8_t* smem_raw,
                                           uint64_t* mb, uint32_t& tmem_base, int& abort_,
                                           int& done_) {
  using C = Cfg<MF>;
  uint8_t* base = align1024(smem_raw);
  uint8_t* sPhiQ = base;              // first: norm scratch | Omega lo (upper half)
  uint8_t* sOl = sPhiQ + C::OMB;
  uint8_t* sPhiK = sPhiQ + C::FEATB;  // later: u
  uint8_t* sU = sPhiK;
  uint8_t* sX = sPhiK + C::FEATB;     // [Q | K | Omega] -> [Q | ones | S_t] -> [dA | S_t] -> [Q | red | Omega]
  uint8_t* sQ = sX;
  uint8_t* sK = sX + ROWT;
  uint8_t* sOnes = sK;                // written once the K projection is done
  uint8_t* sdA = sX;
  uint8_t* sOm = sX + 2 * ROWT;
  uint8_t* sS = sOm;
  float* redU = reinterpret_cast<float*>(sX + ROWT);  // [2][128], late phase
  uint8_t* sV = sOm + C::OMB;         // later: dden as a K-major [16][128] operand + row partials
  uint8_t* sDd = sV;
  float* redA = reinterpret_cast<float*>(sV + 8192);  // [2][128] row sums of A
  float* redZ = redA + 2 * T;                          // [NG][128] g(Q) . z_t partials
  uint8_t* sDo = sV + ROWT;           // dout, then dnum in place
  float* sZ = reinterpret_cast<float*>(sDo + ROWT);
  int* gfail = reinterpret_cast<int*>(sZ + MF);       // [2] per-group failure flags
  // tiles in reverse order: CTA b takes tile ntn-1-b/chains of chain b%chains
  const int c = b % J.chains, t = J.ntn - 1 - b / J.chains, n = J.n;
  const int row0 = J.a + t * T;
  const int valid = min(T, J.b - t * T);
  const size_t g0 = ((size_t)c * J.L + row0) * D;
  const size_t tf = (size_t)c * J.nt + t;   // hand-off buffers, flags
  // The prefixes after this tile: the next tile's slots, the first tile of
  // slice n+1, or (at the end of the sequence) B^(N) and G = 0.
  const bool inner = t + 1 < J.ntn, next_slice = n + 1 < J.N;
  const int snext = inner ? t + 1 : 0;
  const int wnext = inner ? n + 1 : n + 2;
  const bool linked = inner || next_slice;
  StateRef s1, s2;
  bool s2_rowmajor = false;  // the caller's G^(N) is row-major, the slots lane-major
  if (linked) {
    const float* p1 = J.slot1 + ((size_t)c * J.nt + snext) * C::E;
    const float* p2 = J.slot2 + ((size_t)c * J.nt + snext) * C::E;
    s1 = StateRef{p1, p1 + MF * 64, nullptr, nullptr};
    s2 = StateRef{p2, p2 + MF * 64, nullptr, nullptr};
  } else {
    s1 = StateRef{J.fin.S + (size_t)c * MF * 64, J.fin.z + (size_t)c * MF,
                  J.fin.S_lo ? J.fin.S_lo + (size_t)c * MF * 64 : nullptr,
                  J.fin.z_lo ? J.fin.z_lo + (size_t)c * MF : nullptr};
    // G^(N): zero at the true end of a sequence, or handed in by the backward
    // of a later segment (eq. 18)
    if (J.gio.S_in) {
      s2 = StateRef{J.gio.S_in + (size_t)c * MF * 64, J.gio.z_in + (size_t)c * MF, nullptr, nullptr};
      s2_rowmajor = true;
    } else {
      s2 = StateRef{nullptr, nullptr, nullptr, nullptr};
    }
  }
  // the first tile of the sequence hands on G^(0), the gradient with respect
  // to the state the sequence started from
  const bool seq_first = n == 0 && t == 0 && J.gio.S_out != nullptr;
  const int* f1 = J.flag1 + ((size_t)c * J.nt + snext) * FLAG_STRIDE;
  const int* f2 = J.flag2 + ((size_t)c * J.nt + snext) * FLAG_STRIDE;
  float* own1 = J.slot1 + ((size_t)c * J.nt + t) * C::E;
  float* own2 = J.slot2 + ((size_t)c * J.nt + t) * C::E;
  int* of1 = J.flag1 + ((size_t)c * J.nt + t) * FLAG_STRIDE;
  int* of2 = J.flag2 + ((size_t)c * J.nt + t) * FLAG_STRIDE;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int row = 32 * (warp & 3) + (tid & 31);
  const int cg = warp >> 2;
  const int gl = tid - GRP;     // index inside the chain group (warps 8-15)
  const int cq = 2 * (cg - 2);  // chain group: column groups cq, cq + 1
  if (tid == 0) {
    abort_ = 0;
    for (int i = 0; i < NBAR; ++i) mbar_init(smem_u32(&mb[i]), 1);
    mbar_fence_init();
  }
  if (tid == POLL) {
    // while the tiles stream in: the hand-off buffers of ring slot n % R are
    // free once slice n+R's dk/dv part has read them (tril(A) is written in
    // the A row-sum loop, the rest after join1)
    const bool ok = flag_poll2(t < J.nRtiles ? J.kvread + tf * FLAG_STRIDE : nullptr,
                               n + J.ring + 1, nullptr, 0, J.err);
    gfail[1] = ok ? 0 : 1;
  } else if (tid == 0) {
    // the four row tiles by TMA (rows past the chain's end read as zero)
    const uint32_t bar = smem_u32(&mb[MB_TILES]);
    mbar_expect_tx(bar, 4 * ROWT);
    tma_load_3d(smem_u32(sQ), J.tq, row0, c, bar);
    tma_load_3d(smem_u32(sK), J.tk, row0, c, bar);
    tma_load_3d(smem_u32(sV), J.tv, row0, c, bar);
    tma_load_3d(smem_u32(sDo), J.tdo, row0, c, bar);
  }
  // The rollback chain's flag is usually set before this tile starts: read it
  // now, so that its round trip overlaps the loads (an acquire fence follows
  // when it is used); the chain polls only if it was not set yet.
  int early1 = 0, early2 = 0;
  if (tid == GRP && linked) early1 = ld_relaxed_gpu(f1);
  // this thread's 16 columns of its out row, fetched while the tiles stream in
  uint4 orow[2] = {make_uint4(0, 0, 0, 0), make_uint4(0, 0, 0, 0)};
  if (row < valid) {
    const uint4* src = reinterpret_cast<const uint4*>(J.Out + g0 + (size_t)row * D + 16 * cg);
    orow[0] = src[0];
    orow[1] = src[1];
  }
  if (tid == 0) gfail[0] = 0;
  grid_dependency_wait();  // Omega (bf16), slots and buffers belong to earlier kernels
  if (tid == 0) {
    const uint32_t bar = smem_u32(&mb[MB_OMEGA]);
    mbar_expect_tx(bar, 2 * C::OMB);
    tma_load_2d(smem_u32(sOm), J.tom, 0, bar);
    tma_load_2d(smem_u32(sOl), J.tom, MF, bar);
  }
  __syncthreads();  // the barriers' initialisation is seen by every thread
  if (!mbar_wait(smem_u32(&mb[MB_TILES]), 0, J.err)) abort_ = 1;
  if (!mbar_wait(smem_u32(&mb[MB_OMEGA]), 0, J.err)) abort_ = 1;
  __syncthreads();
  if (abort_) goto teardown;
  {
    const bool rv = row < valid;
    float* redN = reinterpret_cast<float*>(sPhiQ);  // 6 KB scratch below Omega lo
    {
      float part = 0.f;  // <dout_r, out_r> over this thread's 16 columns
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const uint4 g = ld_chunk(sDo, T, row, 16 * cg + 8 * h);
        const uint32_t ow[4] = {orow[h].x, orow[h].y, orow[h].z, orow[h].w};
        const uint32_t gw[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          float o0, o1, g0f, g1f;
          unpack_bf16(ow[i], o0, o1);
          unpack_bf16(gw[i], g0f, g1f);
          part = fmaf(o0, g0f, fmaf(o1, g1f, part));
        }
      }
      redN[cg * T + row] = row_norm2_part(sQ, row, cg);
      redN[(NG + cg) * T + row] = row_norm2_part(sK, row, cg);
      redN[(2 * NG + cg) * T + row] = part;
    }
    publish();
    const float q2 = group_total(redN, row), k2 = group_total(redN + NG * T, row);
    const float rowdot = group_total(redN + 2 * NG * T, row);
    const uint32_t tmem = tmem_base;
    const uint32_t trow = tmem + ((uint32_t)(32 * (warp & 3)) << 16);
    if (tid == 0) {
      // K first: the rollback chain needs only Delta_t
      const uint32_t aQ = smem_u32(sQ), aK = smem_u32(sK), aOm = smem_u32(sOm);
      const uint32_t aOl = smem_u32(sOl);
      for (int k0 = 0; k0 < D; k0 += 16) {
        mma(tmem + 256, kmaj(aK, T, k0), kmaj(aOm, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
        mma(tmem + 256, kmaj(aK, T, k0), kmaj(aOl, MF, k0), idesc_bf16(T, MF, 0, 0), 1);
      }
      mma_commit(smem_u32(&mb[0]));
      for (int k0 = 0; k0 < D; k0 += 16) {
        mma(tmem, kmaj(aQ, T, k0), kmaj(aOm, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
        mma(tmem, kmaj(aQ, T, k0), kmaj(aOl, MF, k0), idesc_bf16(T, MF, 0, 0), 1);
      }
      mma_commit(smem_u32(&mb[1]));
    }
    if (!mbar_wait(smem_u32(&mb[0]), 0, J.err)) abort_ = 1;
    tc_fence_after();
    __syncthreads();
    if (abort_) goto teardown;
    fill_ones(sOnes, tid);  // the K tile is no longer read
    feature_epilogue<MF, FEAT>(trow + 256, sPhiK, row, cg, k2, rv);
    publish();
    // the dk/dv part of this tile takes phiK and tril(A) from here (phiQ stays
    // in shared memory)
    uint8_t* img = J.img + tf * ((size_t)C::FEATB + 2 * ROWT);
    if (tid == 0 || (C::MH > 1 && tid == 32)) {
      // Delta_t = phiK^T [V | 1], one feature half per issuing thread
      const int h = tid == 0 ? 0 : 1;
      const uint32_t aPK = smem_u32(sPhiK), aV = smem_u32(sV), aOnes = smem_u32(sOnes);
      for (int k0 = 0; k0 < T; k0 += 16) {
        const uint64_t ad = mnmaj(aPK + h * 2 * ROWT, k0, ROWT);
        mma(tmem + 256 + 64 * h, ad, mnmaj(aV, k0, ROWT), idesc_bf16(T, 64, 1, 1), k0 > 0);
        mma(tmem + 384 + 16 * h, ad, kmaj(aOnes, 16, k0), idesc_bf16(T, 16, 1, 0), k0 > 0);
      }
      mma_commit(smem_u32(&mb[h == 0 ? 2 : 6]));
    }
    if (warp < 8) {
      // ---- compute group: g(Q), then A and dout V^T, and A's row sums
      if (!mbar_wait(smem_u32(&mb[1]), 0, J.err)) gfail[0] = 1;
      tc_fence_after();
      group_bar(1);
      if (gfail[0]) goto join1;
      feature_cols<MF, FEAT>(trow, sPhiQ, row, 32 * cg, MF, 64, q2, rv);
      group_publish(1);
      if (tid == 0) {
        const uint32_t aPQ = smem_u32(sPhiQ), aPK = smem_u32(sPhiK);
        const uint32_t aDo = smem_u32(sDo), aV = smem_u32(sV);
        for (int k0 = 0; k0 < MF; k0 += 16)  // A = phiQ phiK^T
          mma(tmem, kmaj(aPQ, T, k0), kmaj(aPK, T, k0), idesc_bf16(T, T, 0, 0), k0 > 0);
        for (int k0 = 0; k0 < D; k0 += 16)  // dout V^T (scaled by 1/den below)
          mma(tmem + 128, kmaj(aDo, T, k0), kmaj(aV, T, k0), idesc_bf16(T, T, 0, 0), k0 > 0);
        mma_commit(smem_u32(&mb[3]));
      }
      if (!mbar_wait(smem_u32(&mb[3]), 0, J.err)) gfail[0] = 1;
      tc_fence_after();
      group_bar(1);
      if (gfail[0]) goto join1;
      float rs = 0.f;  // the rounded masked A values of this thread's columns
      uint8_t* imgA = img + C::FEATB;
#pragma unroll 1
      for (int c0 = 32 * cg; c0 < T; c0 += 64) {
        float v[32];
        tmem_ld32(trow + c0, v);
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          const float x0 = (c0 + i <= row) ? v[i] : 0.f;
          const float x1 = (c0 + i + 1 <= row) ? v[i + 1] : 0.f;
          pk[i / 2] = pack_bf16(x0, x1);
          float r0, r1;
          unpack_bf16(pk[i / 2], r0, r1);
          rs += r0 + r1;
        }
#pragma unroll
        for (int q = 0; q < 4; ++q)  // tril(A) for the dk/dv side: a warp writes 512 bytes
          reinterpret_cast<uint4*>(imgA)[((c0 >> 3) + q) * T + row] =
              make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
      }
      redA[cg * T + row] = rs;  // V is no longer read: its tile holds the partials
    } else {
      // ---- chain group, rollback (eq. 17 per tile): the state before this
      // tile is the state after it minus Delta_t.  The prefix after this tile
      // is acquired and loaded while the Delta_t products run.
      if (linked && gl == 0 && !gfail[1]) {
        if (early1 == wnext)
          fence_acq_rel_gpu();
        else if (!flag_poll(f1, wnext, J.err))
          gfail[1] = 1;
      }
      group_bar(2);
      if (gfail[1]) goto join1;
      // every load of the prefix after this tile before any store: one L2 trip
      float sv[C::MH][2][16], sz[C::MH];
#pragma unroll
      for (int h = 0; h < C::MH; ++h) {
        const int m = 128 * h + row;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          if (linked)
            ld_lm16(s1.S, h, cq + j, row, sv[h][j]);
          else
            ld_row16f(s1.S + (size_t)m * 64 + 16 * (cq + j), sv[h][j]);
        }
        sz[h] = cq == 0 ? __ldcg(s1.z + m) : 0.f;
      }
      if (s1.S_lo) {
#pragma unroll
        for (int h = 0; h < C::MH; ++h)
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            float lo[16];
            ld_row16f(s1.S_lo + (size_t)(128 * h + row) * 64 + 16 * (cq + j), lo);
#pragma unroll
            for (int i = 0; i < 16; ++i) sv[h][j][i] += lo[i];
          }
      }
      if (cq == 0 && s1.z_lo) {
#pragma unroll
        for (int h = 0; h < C::MH; ++h) sz[h] += __ldcg(s1.z_lo + 128 * h + row);
      }
      if (!mbar_wait(smem_u32(&mb[2]), 0, J.err)) gfail[1] = 1;
      if (C::MH > 1 && !mbar_wait(smem_u32(&mb[6]), 0, J.err)) gfail[1] = 1;
      tc_fence_after();
      group_bar(2);
      if (gfail[1]) goto join1;
#pragma unroll
      for (int h = 0; h < C::MH; ++h) {
        const int m = 128 * h + row;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          float d[16];
          tmem_ld16(trow + 256 + 64 * h + 16 * (cq + j), d);
#pragma unroll
          for (int i = 0; i < 16; ++i) sv[h][j][i] -= d[i];
          st_lm16(own1, h, cq + j, row, sv[h][j]);
          st_tile16(sS, MF, m, 16 * (cq + j), sv[h][j]);
        }
      }
      if (cq == 0) {
#pragma unroll
        for (int h = 0; h < C::MH; ++h) {
          const int m = 128 * h + row;
          float dz;
          tmem_ld1(trow + 384 + 16 * h, dz);
          const float z = sz[h] - dz;
          __stcg(own1 + MF * 64 + m, z);
          sZ[m] = z;
        }
      }
      // the prefix after this tile is read only here: drop it from L2 (before
      // the release, so that it comes before the slot's next writer), unless it
      // sits in this tile's own slot (one-tile slices), just rewritten
      if (linked && snext != t) discard_l2(s1.S, (size_t)C::E * 4, gl, GRP);
      group_bar(2);  // every slot write of the group is issued
      if (gl == 0) st_release_gpu(of1, n + 1);
    }
  join1:
    __syncthreads();
    if (gfail[0] | gfail[1]) goto teardown;
    // the state-gradient chain's flag, read ahead of its use (see early1)
    if (tid == GRP && linked) early2 = ld_relaxed_gpu(f2);
    // phiK's tile image, while the MMAs of the next phases run (the tile is
    // overwritten by u once the copy has read it); Q, read again after them,
    // back into L2
    if (tid == GRP) bulk_store(img, smem_u32(sPhiK), C::FEATB);
    if (tid == GRP + 32) prefetch_l2(J.Q + g0, (uint32_t)valid * 128u);
    {
      // g(Q) . z_t over this thread's feature columns
      constexpr int W = MF / NG;
      float zd = 0.f;
#pragma unroll
      for (int f0 = cg * W; f0 < (cg + 1) * W; f0 += 16) {
        float f[16];
        ld_feat16(sPhiQ, row, f0, f);
#pragma unroll
        for (int i = 0; i < 16; ++i) zd = fmaf(f[i], sZ[f0 + i], zd);
      }
      redZ[cg * T + row] = zd;
    }
    __syncthreads();
    const float den = redA[row] + redA[T + row] + group_total(redZ, row);
    const bool live = rv && den != 0.f;
    const float inv = live ? 1.f / den : 0.f;
    const float dden = live ? -rowdot * inv : 0.f;
    // dnum = dout / den, in place of dout (this thread's 16 columns)
#pragma unroll
    for (int c8 = 16 * cg; c8 < 16 * cg + 16; c8 += 8) {
      const uint4 g = ld_chunk(sDo, T, row, c8);
      const uint32_t gw[4] = {g.x, g.y, g.z, g.w};
      uint32_t pw[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float g0f, g1f;
        unpack_bf16(gw[i], g0f, g1f);
        pw[i] = pack_bf16(g0f * inv, g1f * inv);
      }
      st_chunk(sDo, T, row, c8, make_uint4(pw[0], pw[1], pw[2], pw[3]));
    }
    {
      // dA = tril(dnum V^T + dden), this thread's 32 columns
      float v[32];
      const int c0 = 32 * cg;
      tmem_ld32(trow + 128 + c0, v);
      uint32_t pk[16];
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        const float x0 = (live && c0 + i <= row) ? fmaf(v[i], inv, dden) : 0.f;
        const float x1 = (live && c0 + i + 1 <= row) ? fmaf(v[i + 1], inv, dden) : 0.f;
        pk[i / 2] = pack_bf16(x0, x1);
      }
#pragma unroll
      for (int q = 0; q < 4; ++q)
        st_chunk(sdA, T, row, c0 + 8 * q, make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]));
    }
    // dden as the first row of a K-major [16][128] operand (other rows zero)
#pragma unroll
    for (int r16 = 4 * cg; r16 < 4 * cg + 4; ++r16)
      *reinterpret_cast<__nv_bfloat16*>(sDd + tile_off(16, r16, row)) =
          __float2bfloat16_rn(r16 == 0 ? dden : 0.f);
    if (rv && cg == 0) {
      float* rsw = J.rowstat + (tf * T + row) * 2;
      rsw[0] = den;
      rsw[1] = dden;
    }
    publish();
    if (tid == 0) {
      const uint32_t aDn = smem_u32(sDo), aS = smem_u32(sS), adA = smem_u32(sdA);
      const uint32_t aPK = smem_u32(sPhiK);
      for (int k0 = 0; k0 < D; k0 += 16)  // dnum S_t^T
        mma(tmem + 256, kmaj(aDn, T, k0), kmaj(aS, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
      for (int k0 = 0; k0 < T; k0 += 16)  // + dA phiK
        mma(tmem + 256, kmaj(adA, T, k0), mnmaj(aPK, k0, ROWT), idesc_bf16(T, MF, 0, 1), 1);
      mma_commit(smem_u32(&mb[4]));
    } else if (tid == 32) {
      // Gd = phiQ^T [dnum | dden], from a second issuing thread
      const uint32_t aDn = smem_u32(sDo), aPQ = smem_u32(sPhiQ), aDd = smem_u32(sDd);
      for (int h = 0; h < C::MH; ++h)
        for (int k0 = 0; k0 < T; k0 += 16) {
          const uint64_t ad = mnmaj(aPQ + h * 2 * ROWT, k0, ROWT);
          mma(tmem + 64 * h, ad, mnmaj(aDn, k0, ROWT), idesc_bf16(T, 64, 1, 1), k0 > 0);
          mma(tmem + 128 + 16 * h, ad, kmaj(aDd, 16, k0), idesc_bf16(T, 16, 1, 0), k0 > 0);
        }
      mma_commit(smem_u32(&mb[7]));
    }
    if (!mbar_wait(smem_u32(&mb[4]), 0, J.err)) abort_ = 1;
    if (!mbar_wait(smem_u32(&mb[7]), 0, J.err)) abort_ = 1;
    if (tid == GRP) bulk_wait_read();  // u goes to phiK's tile next
    tc_fence_after();
    __syncthreads();
    if (abort_) goto teardown;
    if (warp < 8) {
      // ---- compute group: Q and Omega again (dq = u Omega - q sum(u),
      // dOmega += u^T q), u = (dphiQ + dden z_t) (.) g'(Q), then the products
      if (tid == 0) {
        const uint32_t bar = smem_u32(&mb[MB_RELOAD]);
        mbar_expect_tx(bar, ROWT + C::OMB);
        tma_load_3d(smem_u32(sQ), J.tq, row0, c, bar);
        tma_load_2d(smem_u32(sOm), J.tom, 0, bar);
      }
      float usum = 0.f;
      const float rscale = rsqrtf((float)MF);
#pragma unroll 1
      for (int c0 = 32 * cg; c0 < MF; c0 += 64) {
        float v[32];
        tmem_ld32(trow + 256 + c0, v);
        uint32_t pk[16];
#pragma unroll
        for (int s16 = 0; s16 < 32; s16 += 16) {
          float f[16];
          ld_feat16(sPhiQ, row, c0 + s16, f);
#pragma unroll
          for (int i = 0; i < 16; i += 2) {
            float u0 = fmaf(dden, sZ[c0 + s16 + i], v[s16 + i]);
            float u1 = fmaf(dden, sZ[c0 + s16 + i + 1], v[s16 + i + 1]);
            if (FEAT == SLIM_FEAT_EXP) {
              u0 *= f[i];
              u1 *= f[i + 1];
            } else {
              u0 = f[i] > 0.f ? u0 * rscale : 0.f;
              u1 = f[i + 1] > 0.f ? u1 * rscale : 0.f;
            }
            if (!live) u0 = u1 = 0.f;
            pk[(s16 + i) / 2] = pack_bf16(u0, u1);
            float r0, r1;
            unpack_bf16(pk[(s16 + i) / 2], r0, r1);
            usum += r0 + r1;
          }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q)
          st_chunk(sU, T, row, c0 + 8 * q, make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]));
      }
      redU[cg * T + row] = usum;
      if (!mbar_wait(smem_u32(&mb[MB_RELOAD]), 0, J.err)) gfail[0] = 1;
      group_publish(1);
      // dq and the dOmega partial go to the columns dphiQ held, so Gd stays
      // readable for the chain group; one issuing thread each
      if (tid == 0) {
        const uint32_t aU = smem_u32(sU), aOm = smem_u32(sOm);
        for (int k0 = 0; k0 < MF; k0 += 16)
          mma(tmem + 256, kmaj(aU, T, k0), mnmaj(aOm, k0, C::OMB), idesc_bf16(T, 64, 0, 1), k0 > 0);
        mma_commit(smem_u32(&mb[5]));
      } else if (tid == 32) {
        const uint32_t aU = smem_u32(sU), aQ = smem_u32(sQ);
        for (int h = 0; h < C::MH; ++h)
          for (int k0 = 0; k0 < T; k0 += 16)
            mma(tmem + 320 + 64 * h, mnmaj(aU + h * 2 * ROWT, k0, ROWT), mnmaj(aQ, k0, ROWT),
                idesc_bf16(T, 64, 1, 1), k0 > 0);
        mma_commit(smem_u32(&mb[8]));
      }
    } else {
      // ---- chain group, state gradient (eq. 18): G_t = the prefix after this
      // tile (zero at the end of the sequence); G_t + Gd_t goes on to tile t-1
      if (linked && gl == 0) {
        if (early2 == wnext)
          fence_acq_rel_gpu();
        else if (!flag_poll(f2, wnext, J.err))
          gfail[1] = 1;
      }
      group_bar(2);
      if (gfail[1]) goto join2;
      float gs[C::MH][2][16], gzs[C::MH];
#pragma unroll
      for (int h = 0; h < C::MH; ++h) {
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          if (s2.S && s2_rowmajor) {
            ld_row16f(s2.S + (size_t)(128 * h + row) * 64 + 16 * (cq + j), gs[h][j]);
          } else if (s2.S) {
            ld_lm16(s2.S, h, cq + j, row, gs[h][j]);
          } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) gs[h][j][i] = 0.f;
          }
        }
        gzs[h] = (s2.z && cq == 0) ? __ldcg(s2.z + 128 * h + row) : 0.f;
      }
#pragma unroll
      for (int h = 0; h < C::MH; ++h) {
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          st_lm16_bf16(J.gS + tf * MF * 64, h, cq + j, row, gs[h][j]);  // G_t(S), dk/dv side
          float gd[16];
          tmem_ld16(trow + 64 * h + 16 * (cq + j), gd);
#pragma unroll
          for (int i = 0; i < 16; ++i) gs[h][j][i] += gd[i];
          st_lm16(own2, h, cq + j, row, gs[h][j]);
          if (seq_first)
            st_f32x16(J.gio.S_out + ((size_t)c * MF + 128 * h + row) * 64 + 16 * (cq + j), gs[h][j]);
        }
      }
      if (cq == 0) {
#pragma unroll
        for (int h = 0; h < C::MH; ++h) {
          const int m = 128 * h + row;
          float gdz;
          tmem_ld1(trow + 128 + 16 * h, gdz);
          J.gz[tf * MF + m] = gzs[h];
          __stcg(own2 + MF * 64 + m, gzs[h] + gdz);
          if (seq_first) J.gio.z_out[(size_t)c * MF + m] = gzs[h] + gdz;
        }
      }
      if (linked && snext != t) discard_l2(s2.S, (size_t)C::E * 4, gl, GRP);
      group_bar(2);  // every slot write of the group is issued
      if (gl == 0) st_release_gpu(of2, n + 1);
    }
  join2:
    __syncthreads();
    // K and V, which the dk/dv part reads next, back into L2
    if (tid == GRP) prefetch_l2(J.K + g0, (uint32_t)valid * 128u);
    if (tid == GRP + 32) prefetch_l2(J.V + g0, (uint32_t)valid * 128u);
    {
      float us = 0.f;
      if (FEAT == SLIM_FEAT_EXP) us = redU[row] + redU[T + row];
      // the dq products were issued in every case: let them land
      if (!mbar_wait(smem_u32(&mb[5]), 0, J.err)) abort_ = 1;
      if (!mbar_wait(smem_u32(&mb[8]), 0, J.err)) abort_ = 1;
      tc_fence_after();
      __syncthreads();
      if (abort_ | gfail[0] | gfail[1]) goto teardown;
      // the partial joins the key side's in the dk/dv part (through L2)
      float* dqp = J.domq + tf * (size_t)(MF * 64);
      float v[16];
#pragma unroll
      for (int h = 0; h < C::MH; ++h) {
        tmem_ld16(trow + 320 + 64 * h + 16 * cg, v);
        st_lm16(dqp, h, cg, row, v);
      }
      // the hand-off to the dk/dv part is complete once phiK's bulk copy is:
      // the part follows in this CTA, after a barrier
      if (tid == GRP) bulk_wait_done();
      float xq[16];
      ld_feat16(sQ, row, 16 * cg, xq);
      tmem_ld16(trow + 256 + 16 * cg, v);
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = fmaf(-us, xq[i], v[i]);
      if (rv) st_row16(J.dq + g0 + (size_t)row * D + 16 * cg, v);
    }
    if (tid == 0) done_ = 1;  // reached only when no wait gave up
  }
  TC_TEARDOWN_KEEP();
}

// ================================================================== backward, dk/dv side
struct BwdKVJob {
  const CUtensorMap *tk, *tv, *tom;  // tensor maps (in the launch's parameters)
  const __nv_bfloat16 *Q, *K, *V, *dOut, *om16;
  // from the dq part of the same tile, indexed by (chain, tile) of a full slice
  const __nv_bfloat16* gS;   // [chains][ntf][MF][64] G_t(S)
  const float *gz, *rowstat;
  const float* domq;         // [chains][ntf][MF][64] lane-major: the dq part's u^T q
  const uint8_t* img;        // [chains][ntf][...] phiK's tile image, tril(A) lane-major
  int* kvread;               // set to n + 1 once this part has read them
  int L, a, b, ntn, ntf, n;  // slice n = rows [a, a+b), ntn tiles; ntf: full slice
  __nv_bfloat16 *dk, *dv;
  // dOmega: per-position sums over slices N-1 .. n of the tiles' partials
  float* acc;                // [chains][ntf][MF][64] lane-major
  int* accflag;              // [chains][ntf]: n + 1 once slice n has added its partial
  int n1tiles;               // tiles of slice n+1 per chain (0: no such slice)
  int* sums_done;            // slice 0 only: counter of final sums written
  int* err;
};

// The dk/dv part of a tile, run by the CTA that ran its dq part: phiQ is still
// in shared memory, and the rest of the hand-off was written by this CTA and
// is read back from L2.  The TMEM columns are the caller's.
template <int MF, int FEAT>
__device__ __forceinline__ void role_bwd_kv(const BwdKVJob& J, int t, int c, uint8_t* smem_raw,
                                            uint64_t* mb, uint32_t& tmem_base, int& abort_) {
  using C = Cfg<MF>;
  uint8_t* base = align1024(smem_raw);
  uint8_t* sPhiQ = base;               // later: u
  uint8_t* sU = sPhiQ;
  uint8_t* sPhiK = sPhiQ + C::FEATB;
  uint8_t* sX = sPhiK + C::FEATB;      // [A | G_t] -> [dA | G_t] -> [K | red | Omega]
  uint8_t* sA = sX;
  uint8_t* sKr = sX;
  float* redU = reinterpret_cast<float*>(sX + ROWT);
  uint8_t* sOm = sX + 2 * ROWT;
  uint8_t* sG = sOm;
  uint8_t* sV = sOm + C::OMB;
  uint8_t* sDn = sV + ROWT;            // dnum, as the dq part left it (its sDo)
  float* sGz = reinterpret_cast<float*>(sDn + ROWT);
  const int row0 = J.a + t * T;
  const int valid = min(T, J.b - t * T);
  const size_t g0 = ((size_t)c * J.L + row0) * D;
  const size_t tf = (size_t)c * J.ntf + t;  // hand-off buffers, flags, dOmega sums
  const bool acc_first = t >= J.n1tiles;
  float den = 0.f, dden = 0.f;
  __shared__ __align__(8) uint64_t mb_img;  // phiK's tile, initialised by one thread
  const int tid = threadIdx.x, warp = tid >> 5;
  const int row = 32 * (warp & 3) + (tid & 31);
  const int cg = warp >> 2;
  if (tid == 0) {
    abort_ = 0;
    for (int i_ = 0; i_ < NBAR; ++i_) mbar_init(smem_u32(&mb[i_]), 1);
    mbar_fence_init();
  }
  uint8_t* const img = const_cast<uint8_t*>(J.img) + tf * ((size_t)C::FEATB + 2 * ROWT);
  if (tid == POLL) {
    // phiK, tril(A), G_t, g_t(z), the row statistics and the dOmega partial
    // come from the dq part of this tile, which this CTA ran before a barrier
    // (its bulk copy waited for and fenced); phiK's tile by a bulk copy
    // completing on mb_img
    const uint32_t bar = smem_u32(&mb_img);
    mbar_init(bar, 1);
    mbar_fence_init();
    fence_proxy_async_global();
    mbar_expect_tx(bar, C::FEATB + ROWT);
    bulk_load(smem_u32(sPhiK), img, C::FEATB, bar);
    tma_load_3d(smem_u32(sV), J.tv, row0, c, bar);  // and the V tile
  }
  // every other load at once: G_t (lane-major -> its tile), tril(A)
  // (lane-major -> its tile), the row statistics and g_t(z)
  if (row < valid) {
    const float* rsr = J.rowstat + (tf * T + row) * 2;
    den = __ldcg(rsr);
    dden = __ldcg(rsr + 1);
  }
  // (dnum = dout / den is still in its tile: the dq part left it there)
  load_lm_bf16(sG, MF, J.gS + tf * MF * 64, tid);
  {
    const uint8_t* imgA = img + C::FEATB;
    for (int k = tid; k < T * T / 8; k += NTHR)
      cp_async16(smem_u32(sA) + tile_off(T, k % T, 8 * (k / T)), imgA + (size_t)k * 16, 16u);
  }
  for (int m = tid; m < MF; m += NTHR) sGz[m] = __ldcg(J.gz + tf * MF + m);
  cp_async_wait_all();
  __syncthreads();  // rows were copied by other threads
  {
    const bool rv = row < valid;
    const uint32_t tmem = tmem_base;
    const uint32_t trow = tmem + ((uint32_t)(32 * (warp & 3)) << 16);
    Sync sy{mb, 0, J.err};
    const bool live = rv && den != 0.f;
    if (!live) dden = 0.f;
    if (!mbar_wait(smem_u32(&mb_img), 0, J.err)) abort_ = 1;  // phiK's and V's tiles
    publish();
    if (abort_) goto teardown;
    // every thread has what it needs of the hand-off but the dOmega partial
    // (read at the end): drop it from L2, it is not read again
    discard_l2(img, (size_t)C::FEATB + 2 * ROWT, tid, NTHR);
    discard_l2(J.gS + tf * MF * 64, (size_t)MF * 64 * 2, tid, NTHR);
    discard_l2(J.gz + tf * MF, (size_t)MF * 4, tid, NTHR);
    discard_l2(J.rowstat + tf * T * 2, (size_t)T * 2 * 4, tid, NTHR);
    if (tid == 0) {
      const uint32_t aDn = smem_u32(sDn), aV = smem_u32(sV);
      for (int k0 = 0; k0 < D; k0 += 16)  // dnum V^T
        mma(tmem + 128, kmaj(aDn, T, k0), kmaj(aV, T, k0), idesc_bf16(T, T, 0, 0), k0 > 0);
      mma_commit(sy.bar(0));
      const uint32_t aA = smem_u32(sA), aPK = smem_u32(sPhiK);
      const uint32_t aG = smem_u32(sG);
      for (int k0 = 0; k0 < T; k0 += 16)  // dV = A^T dnum
        mma(tmem, mnmaj(aA, k0, ROWT), mnmaj(aDn, k0, ROWT), idesc_bf16(T, 64, 1, 1), k0 > 0);
      for (int k0 = 0; k0 < MF; k0 += 16)  // + phiK G_t(S)
        mma(tmem, kmaj(aPK, T, k0), mnmaj(aG, k0, C::OMB), idesc_bf16(T, 64, 0, 1), 1);
      mma_commit(sy.bar(1));
    } else if (tid == 32) {
      // dphiK = V G_t(S)^T, from a second issuing thread
      const uint32_t aG = smem_u32(sG), aV = smem_u32(sV);
      for (int k0 = 0; k0 < D; k0 += 16)
        mma(tmem + 256, kmaj(aV, T, k0), kmaj(aG, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
      mma_commit(sy.bar(2));
    }
    TC_WAIT(sy);
    TC_WAIT(sy);
    TC_WAIT(sy);
    {
      float v[16];
      tmem_ld16(trow + 16 * cg, v);  // dv
      if (rv) st_row16(J.dv + g0 + (size_t)row * D + 16 * cg, v);
    }
    {  // dA = tril(dnum V^T + dden) -> smem, this thread's 32 columns
      float v[32];
      const int c0 = 32 * cg;
      tmem_ld32(trow + 128 + c0, v);
      uint32_t pk[16];
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        const float x0 = (live && c0 + i <= row) ? v[i] + dden : 0.f;
        const float x1 = (live && c0 + i + 1 <= row) ? v[i + 1] + dden : 0.f;
        pk[i / 2] = pack_bf16(x0, x1);
      }
#pragma unroll
      for (int q = 0; q < 4; ++q)
        st_chunk(sA, T, row, c0 + 8 * q, make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]));
    }
    publish();
    if (tid == 0) {
      const uint32_t adA = smem_u32(sA), aPQ = smem_u32(sPhiQ);
      for (int k0 = 0; k0 < T; k0 += 16)  // dphiK += dA^T phiQ
        mma(tmem + 256, mnmaj(adA, k0, ROWT), mnmaj(aPQ, k0, ROWT), idesc_bf16(T, MF, 1, 1), 1);
      mma_commit(sy.bar(3));
    }
    TC_WAIT(sy);
    // K and Omega again (dk = u Omega - k sum(u), dOmega += u^T k), overlapping the epilogue
    if (tid == 0) {
      const uint32_t bar = smem_u32(&mb[MB_RELOAD]);
      mbar_expect_tx(bar, ROWT + C::OMB);
      tma_load_3d(smem_u32(sKr), J.tk, row0, c, bar);
      tma_load_2d(smem_u32(sOm), J.tom, 0, bar);
    }
    {
      // dphiK (+ g_z) -> u (into the phiQ tile), this thread's columns
      constexpr int W = MF / NG;
      float usum = 0.f;
      const float rscale = rsqrtf((float)MF);
#pragma unroll 1
      for (int c0 = cg * W; c0 < (cg + 1) * W; c0 += 32) {
        float v[32];
        tmem_ld32(trow + 256 + c0, v);
        uint32_t pk[16];
#pragma unroll
        for (int s16 = 0; s16 < 32; s16 += 16) {
          float f[16];
          ld_feat16(sPhiK, row, c0 + s16, f);
#pragma unroll
          for (int i = 0; i < 16; i += 2) {
            float u0 = v[s16 + i] + sGz[c0 + s16 + i];
            float u1 = v[s16 + i + 1] + sGz[c0 + s16 + i + 1];
            if (FEAT == SLIM_FEAT_EXP) {
              u0 *= f[i];
              u1 *= f[i + 1];
            } else {
              u0 = f[i] > 0.f ? u0 * rscale : 0.f;
              u1 = f[i + 1] > 0.f ? u1 * rscale : 0.f;
            }
            if (!rv) u0 = u1 = 0.f;
            pk[(s16 + i) / 2] = pack_bf16(u0, u1);
            float r0, r1;
            unpack_bf16(pk[(s16 + i) / 2], r0, r1);
            usum += r0 + r1;
          }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q)
          st_chunk(sU, T, row, c0 + 8 * q, make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]));
      }
      redU[cg * T + row] = usum;
    }
    if (!mbar_wait(smem_u32(&mb[MB_RELOAD]), 0, J.err)) abort_ = 1;
    publish();
    if (abort_) goto teardown;
    if (tid == 0) {
      const uint32_t aU = smem_u32(sU), aOm = smem_u32(sOm);
      for (int k0 = 0; k0 < MF; k0 += 16)
        mma(tmem, kmaj(aU, T, k0), mnmaj(aOm, k0, C::OMB), idesc_bf16(T, 64, 0, 1), k0 > 0);
      mma_commit(sy.bar(4));
    } else if (tid == 32) {
      // the dOmega partial, from a second issuing thread
      const uint32_t aU = smem_u32(sU), aK = smem_u32(sKr);
      for (int h = 0; h < C::MH; ++h)
        for (int k0 = 0; k0 < T; k0 += 16)
          mma(tmem + 64 + 64 * h, mnmaj(aU + h * 2 * ROWT, k0, ROWT), mnmaj(aK, k0, ROWT),
              idesc_bf16(T, 64, 1, 1), k0 > 0);
      mma_commit(sy.bar(5));
    }
    float us = 0.f;
    if (FEAT == SLIM_FEAT_EXP) {
#pragma unroll
      for (int g = 0; g < NG; ++g) us += redU[g * T + row];
    }
    // the dq part's dOmega partial, fetched while the last products run
    const float* dqp = J.domq + tf * (size_t)(MF * 64);
    float wq[C::MH][16];
#pragma unroll
    for (int h = 0; h < C::MH; ++h) ld_lm16(dqp, h, cg, row, wq[h]);
    // slice n+1's dOmega sum at this position, added to after the next waits
    if (tid == POLL && !acc_first &&
        !flag_poll(J.accflag + tf * FLAG_STRIDE, J.n + 2, J.err))
      abort_ = 1;
    TC_WAIT(sy);
    TC_WAIT(sy);
    {
      // the tile's partial (key side + the dq part's query side) goes onto the
      // running dOmega sum at this position (or starts it): one add per
      // slice, in slice order
      float* accp = J.acc + tf * (size_t)(MF * 64);
      float v[16];
#pragma unroll
      for (int h = 0; h < C::MH; ++h) {
        tmem_ld16(trow + 64 + 64 * h + 16 * cg, v);
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] += wq[h][i];
        if (acc_first)
          st_lm16(accp, h, cg, row, v);
        else
          red_lm16(accp, h, cg, row, v);
      }
      __syncthreads();
      discard_l2(dqp, (size_t)MF * 64 * 4, tid, NTHR);
      __syncthreads();  // every discard of the hand-off comes before the release
      if (tid == 0) {  // warp 0 waits for the releases while the others store dk
        st_release_gpu(J.accflag + tf * FLAG_STRIDE, J.n + 1);
        if (J.sums_done) red_release_gpu(J.sums_done, 1);
        st_release_gpu(J.kvread + tf * FLAG_STRIDE, J.n + 1);  // hand-off buffers read
      }
      float xk[16];
      ld_feat16(sKr, row, 16 * cg, xk);
      tmem_ld16(trow + 16 * cg, v);
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = fmaf(-us, xk[i], v[i]);
      if (rv) st_row16(J.dk + g0 + (size_t)row * D + 16 * cg, v);
    }
  }
  TC_TEARDOWN_KEEP();
}

// ================================================================== launches
// Final dOmega reduction of the per-position sums (both sides, lane-major),
// in two stages with fixed ranges and orders, so dOmega is reproducible:
//   stage 1, CTA r < nsums: sums[r] = positions [r*per, (r+1)*per) summed in order
//   stage 2, CTA s: dOmega = sums[0] + ... + sums[nsums-1] over its share of
//            the elements
constexpr int RS1 = 128, RS2 = 32;  // most CTAs of stages 1 and 2
struct RedJob {
  const float* part;  // stage 1: [nparts][M*64] lane-major per-position sums
  int nparts;
  float* sums;        // [nsums][M*64]: stage 1 out, stage 2 in
  int nsums;          // stage-1 CTAs, a multiple of 4
  int nsplit;         // stage-2 CTAs
  float* domega;      // [M][64]
  int n;              // M * 64
};

// Stage 1 streaming its positions through shared memory: NSLOT slots of one
// position each, filled by bulk copies (one thread, mbarrier per slot), so
// NSLOT positions are in flight; the sum is taken in the same order.
constexpr int NSLOT = 3;
__device__ __forceinline__ void reduce_stage1_bulk(const RedJob& J, int r, uint8_t* smem,
                                                   uint64_t* mb, int* err) {
  const int per = (J.nparts + J.nsums - 1) / J.nsums;
  const int i0 = min(J.nparts, r * per), cnt = min(J.nparts, i0 + per) - i0;
  const int n4 = J.n / 4, tid = threadIdx.x;
  const uint32_t bytes = (uint32_t)J.n * 4;
  constexpr int QMAX = 256 * 64 / 4 / NTHR;
  float4 acc[QMAX];
#pragma unroll
  for (int k = 0; k < QMAX; ++k) acc[k] = make_float4(0.f, 0.f, 0.f, 0.f);
  if (tid == 0) {
    for (int sl = 0; sl < NSLOT; ++sl) mbar_init(smem_u32(&mb[sl]), 1);
    mbar_fence_init();
    fence_proxy_async_global();  // the sums were acquired by this thread
    for (int sl = 0; sl < NSLOT && sl < cnt; ++sl) {
      mbar_expect_tx(smem_u32(&mb[sl]), bytes);
      bulk_load(smem_u32(smem + (size_t)sl * bytes), J.part + (size_t)(i0 + sl) * J.n, bytes,
                smem_u32(&mb[sl]));
    }
  }
  __syncthreads();
  bool ok = true;
  for (int k = 0; k < cnt; ++k) {
    const int sl = k % NSLOT;
    if (!mbar_wait(smem_u32(&mb[sl]), (uint32_t)((k / NSLOT) & 1), err)) ok = false;
    const float4* src = reinterpret_cast<const float4*>(smem + (size_t)sl * bytes);
#pragma unroll
    for (int q = 0; q < QMAX; ++q) {
      const int e = tid + q * NTHR;
      if (e < n4) {
        const float4 x = src[e];
        acc[q].x += x.x;
        acc[q].y += x.y;
        acc[q].z += x.z;
        acc[q].w += x.w;
      }
    }
    __syncthreads();  // the slot is read by every thread
    if (tid == 0 && ok && k + NSLOT < cnt) {
      fence_async_smem();
      mbar_expect_tx(smem_u32(&mb[sl]), bytes);
      bulk_load(smem_u32(smem + (size_t)sl * bytes), J.part + (size_t)(i0 + k + NSLOT) * J.n, bytes,
                smem_u32(&mb[sl]));
    }
  }
  float4* dst = reinterpret_cast<float4*>(J.sums + (size_t)r * J.n);
#pragma unroll
  for (int q = 0; q < QMAX; ++q) {
    const int e = tid + q * NTHR;
    if (e < n4) __stcg(dst + e, acc[q]);
  }
}

// Stage 2: CTA s owns float4 indices [s*share, (s+1)*share); thread (q, part)
// sums the range sums [part*nsums/4, (part+1)*nsums/4) of float4 q in order,
// and the four parts are then added in order through shared scratch red4[NTHR].
__device__ __forceinline__ void reduce_stage2(const RedJob& J, int s, float4* red4) {
  const int n4 = J.n / 4, share = (n4 + J.nsplit - 1) / J.nsplit;
  static_assert(NTHR % 4 == 0, "stage 2 splits the ranges in four");
  constexpr int QPER = NTHR / 4;  // float4 per round
  constexpr int BATCH = 16;       // loads in flight per thread
  const int tid = threadIdx.x, ql = tid % QPER, part = tid / QPER;
  const int R4 = J.nsums / 4, end = min(n4, (s + 1) * share);
  for (int q0 = s * share; q0 < end; q0 += QPER) {
    const int q = q0 + ql;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (q < end) {
      for (int r0 = 0; r0 < R4; r0 += BATCH) {
        float4 x[BATCH];
#pragma unroll
        for (int r = 0; r < BATCH; ++r)
          if (r0 + r < R4)
            x[r] = __ldcg(reinterpret_cast<const float4*>(J.sums + (size_t)(part * R4 + r0 + r) * J.n) + q);
#pragma unroll
        for (int r = 0; r < BATCH; ++r)
          if (r0 + r < R4) {
            acc.x += x[r].x;
            acc.y += x[r].y;
            acc.z += x[r].z;
            acc.w += x[r].w;
          }
      }
    }
    red4[tid] = acc;
    __syncthreads();
    if (part == 0 && q < end) {
      float4 t = red4[ql];
#pragma unroll
      for (int k = 1; k < 4; ++k) {
        const float4 u = red4[k * QPER + ql];
        t.x += u.x;
        t.y += u.y;
        t.z += u.z;
        t.w += u.w;
      }
      // lane-major float4 q holds row 128h + row, columns 16cg + 4i .. +3
      const int row = q & 127, rest = q >> 7, i = rest & 3;
      const int cg = (rest >> 2) % NG, h = rest / (4 * NG);
      float* o = J.domega + (128 * h + row) * 64 + 16 * cg + 4 * i;
      o[0] = t.x;
      o[1] = t.y;
      o[2] = t.z;
      o[3] = t.w;
    }
    __syncthreads();
  }
}

// ------------------------------------------------------------------ forward launch
// Every tile of every slice in one launch.  A tile waits only on tiles earlier
// in its chain; the CTAs take their tile from a counter rather than from
// blockIdx, so the tiles handed out so far always belong to CTAs that are
// running and every awaited tile is in progress whatever order the CTAs are
// dispatched in.  (The counter is zeroed by the call's memset.)
template <int MF, int FEAT>
__global__ void __launch_bounds__(NTHR, 1) k_tc_fwd(const __grid_constant__ FwdJob J) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t mbar[NBAR];
  __shared__ uint32_t tmem_base;
  __shared__ int abort_;
  __shared__ int ticket;
  if (threadIdx.x == 0) ticket = atomicAdd(J.ticket, 1);
  __syncthreads();
  role_fwd<MF, FEAT>(J, ticket / J.chains, ticket % J.chains, smem_raw, mbar, tmem_base, abort_);
}

// ------------------------------------------------------------------ backward launch
// The backward is one launch too.  Its items (one per tile, running the
// tile's dq part and then its dk/dv part, and the final dOmega reduction
// CTAs) are handed out by the same kind of counter, in stage order: stage j =
// 0 .. N-1 holds the tiles of slice N-1-j, last tile first, chains inside a
// tile position, and the final dOmega reduction (stage 1, then stage 2) comes
// last.  Every wait of an item is on items of earlier stages or on earlier
// tiles of its own chain, which hold lower tickets:
//   tile of slice n       <- its chain (slice n's later tiles, slice n+1's first),
//                            slice n+R's tile at its position (hand-off buffers
//                            of ring slot n % R, R >= 2), slice n+1's tile at its
//                            position (dOmega sum)
//   reduction stage 1     <- every tile of slice 0 (the last to add to a sum)
//   reduction stage 2     <- stage 1
// so the lowest unfinished item never waits and the launch always progresses.
struct BwdSched {
  int N, chains, nt, ntl;  // slices, chains, tiles of a full slice and of the last
  int r1n, r2n;            // final dOmega stage-1 and stage-2 CTAs
};
enum { IT_TILE = 0, IT_R1 = 2, IT_R2 = 3 };
struct BwdItem {
  int kind, n, idx;  // role, slice, index among the role's items of the slice
};

__host__ __device__ inline int sched_tiles(const BwdSched& s, int n) {
  return s.chains * (n == s.N - 1 ? s.ntl : s.nt);
}
__host__ __device__ inline long long sched_items(const BwdSched& s) {
  long long n = s.r1n + s.r2n;
  for (int k = 0; k < s.N; ++k) n += sched_tiles(s, k);
  return n;
}
// Item of ticket x: stage 0 is the last slice (possibly shorter), stages 1 ..
// N-1 all have chains * nt items.
__host__ __device__ inline BwdItem sched_locate(const BwdSched& s, int x) {
  const int first = sched_tiles(s, s.N - 1);
  if (x < first) return BwdItem{IT_TILE, s.N - 1, x};
  x -= first;
  const int full = s.chains * s.nt;
  const int k = x / full;
  if (k < s.N - 1) return BwdItem{IT_TILE, s.N - 2 - k, x - k * full};
  x -= (s.N - 1) * full;
  if (x < s.r1n) return BwdItem{IT_R1, 0, x};
  return BwdItem{IT_R2, 0, x - s.r1n};
}

struct BwdJob {
  CUtensorMap tq, tk, tv, tdo, tom;  // see FwdJob; the parts point at these
  BwdSched s;
  BwdQJob q;   // slice fields set per item
  BwdKVJob kv;
  RedJob red;
  int L, Cs;
  int* ticket;
  // hand-off ring: slot k (slice n uses n % ring) holds, at hand + k hand_slot,
  // G_t(S) bf16 [chains][nt][M][64], then g_t(z), the row statistics, the dq
  // part's dOmega partials and the tile images at the given offsets; its flag
  // array (kvread) is hflag + k * chains * nt * FLAG_STRIDE
  uint8_t* hand;
  size_t hand_slot, off_gz, off_rs, off_dq, off_img;
  int ring;
  int* hflag;
  float* acc;       // [chains][nt][M*64] per-position dOmega sums
  int* accflag;     // [chains][nt]
  int *sums_done, *r1done;  // slice-0 tiles done, final stage-1 CTAs done
};

template <int MF, int FEAT>
__global__ void __launch_bounds__(NTHR, 1) k_tc_bwd(const __grid_constant__ BwdJob J) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t mbar[2 * NBAR];  // the dq part's, then the dk/dv part's
  __shared__ uint32_t tmem_base;
  __shared__ int abort_, done_;
  __shared__ int ticket;
  if (threadIdx.x == 0) ticket = atomicAdd(J.ticket, 1);
  __syncthreads();
  const BwdItem it = sched_locate(J.s, ticket);
  const int n = it.n, N = J.s.N;
  if (it.kind == IT_TILE) {
    const int a = n * J.Cs, b = min(J.Cs, J.L - a), ntn = (b + T - 1) / T;
    const int n1 = n + 1 < N ? (n + 1 == N - 1 ? J.s.ntl : J.s.nt) : 0;
    const size_t tiles = (size_t)J.s.chains * J.s.nt;
    const int slot = n % J.ring;
    uint8_t* hs = J.hand + slot * J.hand_slot;
    int* hf = J.hflag + (size_t)slot * tiles * FLAG_STRIDE;
    BwdQJob q = J.q;
    q.tq = &J.tq;
    q.tk = &J.tk;
    q.tv = &J.tv;
    q.tdo = &J.tdo;
    q.tom = &J.tom;
    q.a = a;
    q.b = b;
    q.ntn = ntn;
    q.n = n;
    q.gS = reinterpret_cast<__nv_bfloat16*>(hs);
    q.gz = reinterpret_cast<float*>(hs + J.off_gz);
    q.rowstat = reinterpret_cast<float*>(hs + J.off_rs);
    q.domq = reinterpret_cast<float*>(hs + J.off_dq);
    q.img = hs + J.off_img;
    q.kvread = hf;
    q.ring = J.ring;
    q.nRtiles = n + J.ring < N ? (n + J.ring == N - 1 ? J.s.ntl : J.s.nt) : 0;
    BwdKVJob kv = J.kv;
    kv.tk = &J.tk;
    kv.tv = &J.tv;
    kv.tom = &J.tom;
    kv.a = a;
    kv.b = b;
    kv.ntn = ntn;
    kv.n = n;
    kv.gS = q.gS;
    kv.gz = q.gz;
    kv.rowstat = q.rowstat;
    kv.domq = q.domq;
    kv.img = q.img;
    kv.kvread = hf;
    kv.acc = J.acc;
    kv.accflag = J.accflag;
    kv.n1tiles = n1;
    kv.sums_done = n == 0 ? J.sums_done : nullptr;
    // one TMEM allocation (all 512 columns) serves both parts of the tile
    if (threadIdx.x == 0) done_ = 0;
    if (threadIdx.x < 32) tmem_alloc(smem_u32(&tmem_base), 512);
    role_bwd_q<MF, FEAT>(q, it.idx, smem_raw, mbar, tmem_base, abort_, done_);
    __syncthreads();
    // the dk/dv part runs only after a complete dq part (a wait that gave up
    // has left the error word set; the part would wait on what never comes)
    if (done_) {
      tc_fence_after();
      // the dq part's order: last tile first, chains inside a position
      role_bwd_kv<MF, FEAT>(kv, ntn - 1 - it.idx / J.s.chains, it.idx % J.s.chains, smem_raw,
                            mbar + NBAR, tmem_base, abort_);
    }
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x < 32) tmem_dealloc(tmem_base, 512);
    return;
  }
  // final dOmega reduction over every position
  if (threadIdx.x == 0) {
    abort_ = 0;
    const int want = it.kind == IT_R1 ? J.red.nparts : J.s.r1n;
    if (!counter_poll(it.kind == IT_R1 ? J.sums_done : J.r1done, want, J.q.err)) abort_ = 1;
  }
  __syncthreads();
  if (abort_) return;
  if (it.kind == IT_R1) {
    reduce_stage1_bulk(J.red, it.idx, align1024(smem_raw), mbar, J.q.err);
    __syncthreads();
    if (threadIdx.x == 0) red_release_gpu(J.r1done, 1);
  } else {
    reduce_stage2(J.red, it.idx, reinterpret_cast<float4*>(align1024(smem_raw)));
  }
}

// ================================================================== small kernels
// Omega as a bf16 pair: hi = bf16(Omega), lo = bf16(Omega - hi), so the
// projections X Omega^T = X hi^T + X lo^T carry ~16 mantissa bits.
// Thread 0 also stores the call's report-counter address (see give_up).
__global__ void k_omega_bf16(const float* om, __nv_bfloat16* om16, int n, int* err,
                             unsigned* rep) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i == 0) set_report(err, rep);
  if (i < n) {
    const __nv_bfloat16 hi = __float2bfloat16_rn(om[i]);
    om16[i] = hi;
    om16[n + i] = __float2bfloat16_rn(om[i] - __bfloat162float(hi));
  }
}

// ================================================================== host
namespace {

struct Geo {
  int chains, MF, Cs, nt, N;
  int E;
};

Geo geometry(const Problem& p) {
  Geo g;
  g.chains = p.chains();
  g.MF = p.M;
  g.Cs = p.slice_len();
  g.nt = (g.Cs + T - 1) / T;
  g.N = p.num_slices();
  g.E = g.MF * 65;
  return g;
}

// The chain slots hold one prefix per (chain, tile of a slice): a slice's
// tiles overwrite the previous slice's only after reading them.  The buffers
// a tile's dq part hands to its dk/dv part form a ring of R slots (slice n
// uses n % R): slice n-R's tile reuses a slot once slice n's tile has read it.
// R is at least 2 and large enough that those two items are KV_LEAD tickets
// apart, so that the wait is almost never taken even when slices are short.
// dOmega is summed per (chain, tile position) over the slices and reduced
// once at the end.
constexpr int KV_LEAD = 320;  // about two waves of tile CTAs
constexpr int MAX_RING = 16;
int handoff_ring(const Geo& g) {
  const int stage = g.chains * g.nt;  // items of a full stage
  const int r = 1 + (KV_LEAD + stage - 1) / stage;
  return r < 2 ? 2 : (r > MAX_RING ? MAX_RING : r);
}
struct Ws {
  int* err;
  int* flags;  // every flag and counter of the call, zeroed together
  int nflags;
  int *flag1, *flag2;         // [chains][nt] chain flags, FLAG_STRIDE ints each
  int* hflag;                 // [ring][chains][nt] hand-off flags (backward)
  int* accflag;               // [chains][nt]: dOmega sums (backward)
  int *sums_done, *r1done;    // final reduction counters (backward)
  int* ticket;
  __nv_bfloat16* om16;
  float *slot1, *slot2;
  // hand-off ring (see BwdJob): per slot G_t(S), g_t(z), the row statistics,
  // the dq parts' dOmega partials and per tile phiK (T x M bf16) and tril(A)
  // (T x T bf16)
  uint8_t* hand;
  size_t hand_slot, off_gz, off_rs, off_dq, off_img;
  int ring;
  float* acc;    // [chains][nt][M*64]
  float* rsums;  // [RS1][M*64]
};

Ws carve(Carver& cv, const Geo& g, bool bwd) {
  Ws w{};
  const size_t C = g.chains, tiles = C * g.nt, FS = FLAG_STRIDE;
  w.err = cv.take<int>(64);
  w.ring = bwd ? handoff_ring(g) : 0;
  w.nflags = (int)((bwd ? (3 + (size_t)w.ring) * tiles + 2 : 2 * tiles) * FS + FS);
  w.flags = cv.take<int>(w.nflags);
  int* f = w.flags;
  w.flag1 = f;
  w.flag2 = f + tiles * FS;
  f += 2 * tiles * FS;
  if (bwd) {
    w.hflag = f;
    f += (size_t)w.ring * tiles * FS;
    w.accflag = f;
    f += tiles * FS;
    w.sums_done = f;
    w.r1done = f + FS;
    f += 2 * FS;
  }
  w.ticket = f;
  w.om16 = cv.take<__nv_bfloat16>((size_t)2 * g.MF * D);
  w.slot1 = cv.take<float>(tiles * g.E);
  if (bwd) {
    w.slot2 = cv.take<float>(tiles * g.E);
    // byte offsets inside a slot (all multiples of 16)
    w.off_gz = tiles * g.MF * D * 2;
    w.off_rs = w.off_gz + tiles * g.MF * 4;
    w.off_dq = w.off_rs + tiles * T * 2 * 4;
    w.off_img = w.off_dq + tiles * g.MF * D * 4;
    w.hand_slot = (w.off_img + tiles * ((size_t)2 * T * g.MF + 2 * T * T) + 255) & ~size_t(255);
    w.hand = cv.take<uint8_t>(w.ring * w.hand_slot);
    w.acc = cv.take<float>(tiles * (size_t)g.MF * D);
    w.rsums = cv.take<float>((size_t)RS1 * g.MF * D);
  }
  return w;
}

// dynamic shared memory of each role (plus 1 KB for 1024-byte alignment)
template <int MF>
constexpr size_t smem_fwd() {
  return 1024 + 2 * Cfg<MF>::FEATB + 3 * ROWT + Cfg<MF>::OMB + 8192 + 2 * T * 4 + 16;
}
template <int MF>
constexpr size_t smem_bwd() { return 1024 + 2 * Cfg<MF>::FEATB + 4 * ROWT + Cfg<MF>::OMB + MF * 4 + 16; }
static_assert(smem_fwd<256>() <= 232448 && smem_bwd<256>() <= 232448,
              "a tile CTA must fit in 227 KB of shared memory");
static_assert(NTHR * sizeof(float4) <= smem_bwd<128>() - 1024, "stage-2 scratch fits");
static_assert(NSLOT * 128 * 64 * 4 <= smem_bwd<128>() - 1024 &&
                  NSLOT * 256 * 64 * 4 <= smem_bwd<256>() - 1024,
              "stage-1 slots fit");

template <int MF, int FEAT>
cudaError_t configure() {
  static bool configured[kMaxDevices] = {};
  bool* done = device_flag(configured);
  if (done == nullptr) return cudaErrorInvalidDevice;
  if (*done) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(k_tc_fwd<MF, FEAT>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem_fwd<MF>());
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_tc_bwd<MF, FEAT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem_bwd<MF>());
  if (e != cudaSuccess) return e;
  *done = true;
  return cudaSuccess;
}

// cuTensorMapEncodeTiled from the driver (through the runtime's entry-point
// query, so the library needs no link against libcuda).
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_tiled() {
  static const EncodeTiledFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      p = nullptr;
    cudaGetLastError();
    return reinterpret_cast<EncodeTiledFn>(p);
  }();
  return fn;
}
// [chains][L][64] bf16 rows, 128 bytes each: box {64, 128, 1} (one row tile),
// 128-byte swizzle; rows at or past L read as zero.
bool rows_map(CUtensorMap* m, const void* base, int chains, int L) {
  const EncodeTiledFn fn = encode_tiled();
  if (!fn) return false;
  const cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)L, (cuuint64_t)chains};
  const cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)L * D * 2};
  const cuuint32_t box[3] = {(cuuint32_t)D, (cuuint32_t)T, 1};
  const cuuint32_t es[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
// Omega's bf16 hi rows then lo rows, [2 M][64]: box {64, M}.
bool omega_map(CUtensorMap* m, const void* om16, int MF) {
  const EncodeTiledFn fn = encode_tiled();
  if (!fn) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)2 * MF};
  const cuuint64_t strides[1] = {(cuuint64_t)D * 2};
  const cuuint32_t box[2] = {(cuuint32_t)D, (cuuint32_t)MF};
  const cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(om16), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

#define TC_TRY(x)                                  \
  do {                                             \
    cudaError_t e_ = (x);                          \
    if (e_ != cudaSuccess) return SLIM_ERR_CUDA;   \
  } while (0)

unsigned nblk(long long n) { return (unsigned)((n + 255) / 256); }

// Launch as a programmatic dependent of the previous kernel in the stream:
// the kernel may start while its predecessor drains and waits for it inside
// (grid_dependency_wait).
template <typename... KArgs, typename... Args>
cudaError_t launch_dep(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Slice n: rows [a, a+b) and its tile count.
struct Slice {
  int a, b, nt;
};
Slice slice_of(const Problem& p, const Geo& g, int n) {
  Slice r;
  r.a = n * g.Cs;
  r.b = (p.L - r.a < g.Cs) ? p.L - r.a : g.Cs;
  r.nt = (r.b + T - 1) / T;
  return r;
}

cudaError_t prepare(const Ws& w, const Geo& g, const float* omega, unsigned* rep,
                    cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(w.err, 0, sizeof(int), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(w.flags, 0, (size_t)w.nflags * sizeof(int), s);
  if (e != cudaSuccess) return e;
  prof::Scope ps(prof::K_TC_PREP, s);
  k_omega_bf16<<<nblk(g.MF * D), 256, 0, s>>>(omega, w.om16, g.MF * D, w.err, rep);  // hi and lo
  return cudaGetLastError();
}

template <int MF, int FEAT>
slim_status fwd_impl(const Problem& p, const __nv_bfloat16* q, const __nv_bfloat16* k,
                     const __nv_bfloat16* v, const float* omega, __nv_bfloat16* out,
                     const StateOut& st, const StateInit& init, unsigned* rep, void* workspace,
                     cudaStream_t s) {
  TC_TRY((configure<MF, FEAT>()));
  const Geo g = geometry(p);
  Carver cv(workspace);
  const Ws w = carve(cv, g, false);
  // every tile of every slice in one launch, in sequence order, chains inside
  // a tile position.  Algorithmic work per row: 8dM (phiQ, phiK, Delta, readout).
  const int P = (g.N - 1) * g.nt + slice_of(p, g, g.N - 1).nt;
  FwdJob J{{}, {}, {}, {}, q, k, v, w.om16, p.L, g.Cs, g.N, g.nt, P, g.chains, w.slot1, w.flag1,
           w.ticket, out, st, init, w.err};
  // the tensor maps first: a failure leaves nothing launched
  if (!rows_map(&J.tq, q, g.chains, p.L) || !rows_map(&J.tk, k, g.chains, p.L) ||
      !rows_map(&J.tv, v, g.chains, p.L) || !omega_map(&J.tom, w.om16, MF))
    return SLIM_ERR_CUDA;
  TC_TRY(prepare(w, g, omega, rep, s));
  const double rows = (double)g.chains * p.L, MD = (double)MF * D;
  prof::Scope ps(prof::K_TC_FWD, s, rows * 8.0 * MD, rows * D * 2.0 * 4);
  TC_TRY(launch_dep(k_tc_fwd<MF, FEAT>, dim3(P * g.chains), dim3(NTHR), smem_fwd<MF>(), s, J));
  return SLIM_OK;
}

// Final reduction: stage-1 CTAs each sum at least 8 positions, at most RS1
// CTAs, a multiple of 4; stage 2 takes a quarter as many (at least 4).
void reduction_split(const Geo& g, int& r1n, int& r2n) {
  const int nparts = g.chains * g.nt;
  r1n = nparts / 8;
  r1n = r1n < 4 ? 4 : (r1n > RS1 ? RS1 : r1n);
  r1n -= r1n % 4;
  r2n = r1n / 4 < 4 ? 4 : (r1n / 4 > RS2 ? RS2 : r1n / 4);
}

template <int MF, int FEAT>
slim_status bwd_impl(const Problem& p, const __nv_bfloat16* q, const __nv_bfloat16* k,
                     const __nv_bfloat16* v, const float* omega, const __nv_bfloat16* out,
                     const __nv_bfloat16* dout, const StateIn& st, const GradIO& gio,
                     __nv_bfloat16* dq, __nv_bfloat16* dk, __nv_bfloat16* dv, float* domega,
                     unsigned* rep, void* workspace, cudaStream_t s) {
  TC_TRY((configure<MF, FEAT>()));
  const Geo g = geometry(p);
  Carver cv(workspace);
  const Ws w = carve(cv, g, true);
  const int N = g.N;
  BwdJob J{};
  // the tensor maps first: a failure leaves nothing launched
  if (!rows_map(&J.tq, q, g.chains, p.L) || !rows_map(&J.tk, k, g.chains, p.L) ||
      !rows_map(&J.tv, v, g.chains, p.L) || !rows_map(&J.tdo, dout, g.chains, p.L) ||
      !omega_map(&J.tom, w.om16, MF))
    return SLIM_ERR_CUDA;
  TC_TRY(prepare(w, g, omega, rep, s));
  J.s.N = N;
  J.s.chains = g.chains;
  J.s.nt = g.nt;
  J.s.ntl = slice_of(p, g, N - 1).nt;
  reduction_split(g, J.s.r1n, J.s.r2n);
  // slice 0 (C rows, or all L rows) has a tile at every position, so its
  // tiles close every dOmega sum
  // slice fields (a, b, ntn, n and the per-slice buffers) are set per item
  J.q = BwdQJob{nullptr, nullptr, nullptr, nullptr, nullptr, q, k, v, out, dout, w.om16, st, p.L, 0, 0, 0, 0, N, g.nt, g.chains, w.slot1,
                w.slot2, w.flag1, w.flag2, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr,
                0, 0, dq, w.err, gio};
  J.kv = BwdKVJob{nullptr, nullptr, nullptr, q, k, v, dout, w.om16, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr,
                  p.L, 0, 0, 0, g.nt, 0, dk, dv, nullptr, nullptr, 0, nullptr, w.err};
  J.red = RedJob{w.acc, g.chains * g.nt, w.rsums, J.s.r1n, J.s.r2n, domega, MF * D};
  J.L = p.L;
  J.Cs = g.Cs;
  J.ticket = w.ticket;
  J.hand = w.hand;
  J.hand_slot = w.hand_slot;
  J.off_gz = w.off_gz;
  J.off_rs = w.off_rs;
  J.off_dq = w.off_dq;
  J.off_img = w.off_img;
  J.ring = w.ring;
  J.hflag = w.hflag;
  J.accflag = w.accflag;
  J.acc = w.acc;
  J.sums_done = w.sums_done;
  J.r1done = w.r1done;
  // Algorithmic work per row: dq part 14dM (phiQ, phiK, rollback Delta,
  // dphiQ, G, dq, dOmega), dk/dv part 8dM (dV, dphiK, dk, dOmega).
  const double rows = (double)g.chains * p.L, MD = (double)MF * D;
  const long long items = sched_items(J.s);
  prof::Scope ps(prof::K_TC_BWD, s, rows * 22.0 * MD, rows * D * 2.0 * 12);
  TC_TRY(launch_dep(k_tc_bwd<MF, FEAT>, dim3((unsigned)items), dim3(NTHR), smem_bwd<MF>(), s, J));
  return SLIM_OK;
}

}  // namespace

bool supports(const Problem& p) {
  return p.dtype == SLIM_BF16 && p.d == D && (p.M == 128 || p.M == 256) &&
         p.feature != SLIM_FEAT_SQUARE && p.slice_len() >= 64;
}

size_t workspace_bytes(const Problem& p, bool bwd) {
  Carver cv(nullptr);
  carve(cv, geometry(p), bwd);
  return cv.bytes();
}

int bwd_schedule(const Problem& p, int* items, int cap, int* ring) {
  const Geo g = geometry(p);
  if (ring) *ring = handoff_ring(g);
  BwdSched sc{};
  sc.N = g.N;
  sc.chains = g.chains;
  sc.nt = g.nt;
  sc.ntl = slice_of(p, g, g.N - 1).nt;
  reduction_split(g, sc.r1n, sc.r2n);
  const long long n = sched_items(sc);
  for (long long x = 0; x < n && x < cap; ++x) {
    const BwdItem it = sched_locate(sc, (int)x);
    items[3 * x] = it.kind;
    items[3 * x + 1] = it.n;
    items[3 * x + 2] = it.idx;
  }
  return (int)n;
}

#define TC_DISPATCH(FN, ...)                                                        \
  do {                                                                              \
    if (p.M == 256)                                                                 \
      return p.feature == SLIM_FEAT_EXP ? FN<256, SLIM_FEAT_EXP>(__VA_ARGS__)       \
                                        : FN<256, SLIM_FEAT_RELU>(__VA_ARGS__);     \
    return p.feature == SLIM_FEAT_EXP ? FN<128, SLIM_FEAT_EXP>(__VA_ARGS__)         \
                                      : FN<128, SLIM_FEAT_RELU>(__VA_ARGS__);       \
  } while (0)

slim_status fwd(const Problem& p, const void* q, const void* k, const void* v,
                const float* omega, void* out, const StateOut& st, const StateInit& init,
                unsigned* report, void* workspace, cudaStream_t s) {
  using B16 = __nv_bfloat16;
  TC_DISPATCH(fwd_impl, p, (const B16*)q, (const B16*)k, (const B16*)v, omega, (B16*)out, st,
              init, report, workspace, s);
}

slim_status bwd(const Problem& p, const void* q, const void* k, const void* v,
                const float* omega, const void* out, const void* dout, const StateIn& st,
                const GradIO& gio, void* dq, void* dk, void* dv, float* domega,
                unsigned* report, void* workspace, cudaStream_t s) {
  using B16 = __nv_bfloat16;
  TC_DISPATCH(bwd_impl, p, (const B16*)q, (const B16*)k, (const B16*)v, omega, (const B16*)out,
              (const B16*)dout, st, gio, (B16*)dq, (B16*)dk, (B16*)dv, domega, report, workspace,
              s);
}

}  // namespace tc
}  // namespace slim
