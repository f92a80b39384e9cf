// Tensor-core (tcgen05) path of libslim: bf16 inputs, d = 64, M in {128, 256}.
//
// Same slice algorithm as the fp32 path (Algorithm 1, App. B block form with
// masked tile products), with tiles of T = 128 rows, one CTA of 128 threads
// per (tile, chain).  Every tile product is a chain of tcgen05 MMAs on
// 128-byte-swizzled bf16 shared-memory operands with an fp32 accumulator in
// tensor memory; thread r of the CTA owns row r (TMEM lane r) in the
// epilogues.  Per slice:
//
//   forward   tc_delta : phiK = g(K_t), Delta_t = phiK^T [V_t | 1]
//             scan     : P_t = B + sum_{t'<t} Delta_t', B += sum Delta_t
//             tc_fwd   : phiQ, phiK, A = tril(phiQ phiK^T),
//                        num = phiQ S_t + A V_t, den = phiQ z_t + rowsum A
//   backward  tc_delta, scan(rollback, eq. 17)
//             tc_bwd_q : den, dnum = dout/den, dden = -<dout,out>/den,
//                        dA = tril(dnum V^T + dden), dphiQ = dnum S_t^T +
//                        dden z_t + dA phiK, Gd_t = phiQ^T [dnum | dden],
//                        dq = u Omega - q sum(u), dOmega partial u^T q
//             scan     : G_t = G + sum_{t'>t} Gd_t' (eq. 18)
//             tc_bwd_kv: dV = A^T dnum + phiK G_t(S), dphiK = dA^T phiQ +
//                        V G_t(S)^T + g_t(z), dk = u Omega - k sum(u),
//                        dOmega partial += u^T k
//             reduce   : dOmega += sum of partials (fixed order)
//
// The state rows of the workspace hold [S (M x 64) | z (M)] per tile (E =
// 65 M floats), exactly what the shared scan carries.
#include <math.h>

#include "common.cuh"
#include "profiler.h"
#include "scan.h"
#include "scan_dev.cuh"
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

// fp32 [R][64] global -> bf16 row tile (R rows), all NTHR threads.  Every
// thread issues all of its loads before converting, so they are in flight
// together.
template <int R>
__device__ __forceinline__ void load_f32_rows64(uint8_t* tile, const float* g, int tid) {
  constexpr int PER = R * 8 / NTHR;  // 16-byte bf16 chunks per thread
  static_assert(R * 8 % NTHR == 0, "rows must split evenly over the CTA");
  float4 a[PER], b[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) {
    const int e = tid + i * NTHR, r = e >> 3, c = (e & 7) * 8;
    a[i] = *reinterpret_cast<const float4*>(g + (size_t)r * 64 + c);
    b[i] = *reinterpret_cast<const float4*>(g + (size_t)r * 64 + c + 4);
  }
#pragma unroll
  for (int i = 0; i < PER; ++i) {
    const int e = tid + i * NTHR, r = e >> 3, c = (e & 7) * 8;
    st_chunk(tile, R, r, c, make_uint4(pack_bf16(a[i].x, a[i].y), pack_bf16(a[i].z, a[i].w),
                                       pack_bf16(b[i].x, b[i].y), pack_bf16(b[i].z, b[i].w)));
  }
}

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
template <int MF, int FEAT>
__device__ __forceinline__ float feature_epilogue(uint32_t trow, uint8_t* phi, int r, int cg,
                                                  float x2, bool valid,
                                                  const float* z = nullptr) {
  constexpr int W = MF / NG;
  float dz = 0.f;  // sum over this thread's columns of bf16(phi) * z
  // exp map: phi = 2^(p log2e - (|x|^2/2) log2e - log2 sqrt(M))
  const float bias = -0.5f * x2 * kLog2e - 0.5f * log2f((float)MF);
  const float relu_scale = rsqrtf((float)MF);
#pragma unroll 1
  for (int c0 = cg * W; c0 < (cg + 1) * W; c0 += 32) {
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
      if (z) {
        float ra, rb;
        unpack_bf16(pk[i / 2], ra, rb);
        dz = fmaf(ra, z[c0 + i], fmaf(rb, z[c0 + i + 1], dz));
      }
    }
#pragma unroll
    for (int q = 0; q < 4; ++q)
      st_chunk(phi, T, r, c0 + 8 * q, make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]));
  }
  return dz;
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
__device__ __forceinline__ void st_row16(__nv_bfloat16* dst, const float* v) {
  uint4* d = reinterpret_cast<uint4*>(dst);
  d[0] = make_uint4(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]), pack_bf16(v[4], v[5]),
                    pack_bf16(v[6], v[7]));
  d[1] = make_uint4(pack_bf16(v[8], v[9]), pack_bf16(v[10], v[11]), pack_bf16(v[12], v[13]),
                    pack_bf16(v[14], v[15]));
}
__device__ __forceinline__ void st_f32x16(float* dst, const float* v) {
  float4* o = reinterpret_cast<float4*>(dst);
#pragma unroll
  for (int i = 0; i < 4; ++i) o[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
}

struct Sync {
  uint32_t mbar;
  uint32_t phase;
  int* err;
  __device__ bool wait() {
    const bool ok = mbar_wait(mbar, phase, err);
    phase ^= 1u;
    tc_fence_after();
    return ok;
  }
};

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
    mbar_init(smem_u32(&mbar), 1);                      \
    mbar_fence_init();                                  \
  }                                                     \
  if (warp == 0) tmem_alloc(smem_u32(&tmem_base), 512)

#define TC_TEARDOWN()                                   \
  teardown:                                             \
  tc_fence_before();                                    \
  __syncthreads();                                      \
  if (warp == 0) tmem_dealloc(tmem_base, 512)

// ================================================================== tc_delta
template <int MF, int FEAT>
__device__ __forceinline__ void role_delta(const __nv_bfloat16* __restrict__ K, const __nv_bfloat16* __restrict__ V,
               const __nv_bfloat16* __restrict__ om16, int L, int a, int b, int nt,
               float* __restrict__ delta, int* err,
    int t, int c, uint8_t* smem_raw, uint64_t& mbar, uint32_t& tmem_base, int& abort_) {
  using C = Cfg<MF>;
  uint8_t* base = align1024(smem_raw);
  uint8_t* sK = base;
  uint8_t* sV = sK + ROWT;
  uint8_t* sOm = sV + ROWT;
  uint8_t* sPhi = sOm + C::OMB;
  uint8_t* sOnes = sPhi + C::FEATB;  // [16][128] K-major, all ones
  const int row0 = a + t * T;
  const int valid = min(T, b - t * T);
  const size_t g0 = ((size_t)c * L + row0) * D;
  TC_PROLOGUE();
  load_rows64(sK, T, K + g0, valid, tid, NTHR);
  load_rows64(sV, T, V + g0, valid, tid, NTHR);
  grid_dependency_wait();  // Omega (bf16) and the delta buffer belong to earlier kernels
  load_rows64(sOm, MF, om16, MF, tid, NTHR);
  load_rows64(sPhi, MF, om16 + MF * D, MF, tid, NTHR);  // Omega lo, until phi overwrites it
  cp_async_wait_all();
  __syncthreads();  // rows were copied by other threads
  {
    float* redN = reinterpret_cast<float*>(sOnes);  // scratch until the ones are written
    redN[cg * T + row] = row_norm2_part(sK, row, cg);
    publish();
    const float x2 = group_total(redN, row);
    const uint32_t tmem = tmem_base;
    const uint32_t trow = tmem + ((uint32_t)(32 * (warp & 3)) << 16);
    Sync sy{smem_u32(&mbar), 0u, err};
    if (tid == 0) {
      const uint32_t aK = smem_u32(sK), aOm = smem_u32(sOm), aOl = smem_u32(sPhi);
      for (int k0 = 0; k0 < D; k0 += 16) {
        mma(tmem, kmaj(aK, T, k0), kmaj(aOm, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
        mma(tmem, kmaj(aK, T, k0), kmaj(aOl, MF, k0), idesc_bf16(T, MF, 0, 0), 1);
      }
      mma_commit(sy.mbar);
    }
    TC_WAIT(sy);
    for (int e = tid; e < 4096 / 16; e += NTHR)
      reinterpret_cast<uint4*>(sOnes)[e] = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
    feature_epilogue<MF, FEAT>(trow, sPhi, row, cg, x2, row < valid);
    publish();
    if (tid == 0) {
      const uint32_t aPhi = smem_u32(sPhi), aV = smem_u32(sV), aOnes = smem_u32(sOnes);
      for (int h = 0; h < C::MH; ++h)
        for (int k0 = 0; k0 < T; k0 += 16) {
          const uint64_t ad = mnmaj(aPhi + h * 2 * ROWT, k0, ROWT);
          mma(tmem + 256 + 64 * h, ad, mnmaj(aV, k0, ROWT), idesc_bf16(T, 64, 1, 1), k0 > 0);
          mma(tmem + 384 + 16 * h, ad, kmaj(aOnes, 16, k0), idesc_bf16(T, 16, 1, 0), k0 > 0);
        }
      mma_commit(sy.mbar);
    }
    TC_WAIT(sy);
    float* dst = delta + ((size_t)c * nt + t) * C::E;
    for (int h = 0; h < C::MH; ++h) {
      const int m = 128 * h + row;
      float v[16];
      tmem_ld16(trow + 256 + 64 * h + 16 * cg, v);
      st_f32x16(dst + (size_t)m * 64 + 16 * cg, v);
      if (cg == 0) {
        float zz;
        tmem_ld1(trow + 384 + 16 * h, zz);
        dst[MF * 64 + m] = zz;
      }
    }
  }
  TC_TEARDOWN();
}

// ================================================================== tc_fwd
template <int MF, int FEAT>
__device__ __forceinline__ void role_fwd(const __nv_bfloat16* __restrict__ Q, const __nv_bfloat16* __restrict__ K,
             const __nv_bfloat16* __restrict__ V, const __nv_bfloat16* __restrict__ om16,
             const float* __restrict__ pfx, int L, int a, int b, int nt,
             __nv_bfloat16* __restrict__ out, int* err,
    int t, int c, uint8_t* smem_raw, uint64_t& mbar, uint32_t& tmem_base, int& abort_) {
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
  float* sZ = reinterpret_cast<float*>(sV + ROWT);
  float* red = sZ + MF;            // [NG][128] row-sum partials
  const int row0 = a + t * T;
  const int valid = min(T, b - t * T);
  const size_t g0 = ((size_t)c * L + row0) * D;
  const float* P = pfx + ((size_t)c * nt + t) * C::E;
  TC_PROLOGUE();
  load_rows64(sQ, T, Q + g0, valid, tid, NTHR);
  load_rows64(sK, T, K + g0, valid, tid, NTHR);
  load_rows64(sV, T, V + g0, valid, tid, NTHR);
  grid_dependency_wait();  // the state prefixes come from the scan just before
  load_rows64(sOm, MF, om16, MF, tid, NTHR);
  load_rows64(sPhiK, MF, om16 + MF * D, MF, tid, NTHR);  // Omega lo, until phiK overwrites it
  for (int m = tid; m < MF; m += NTHR) sZ[m] = P[MF * 64 + m];
  cp_async_wait_all();
  __syncthreads();  // rows were copied by other threads
  {
    const bool rv = row < valid;
    float* redN = reinterpret_cast<float*>(sPhiQ);  // phiQ is written only after phase 1
    redN[cg * T + row] = row_norm2_part(sQ, row, cg);
    redN[(NG + cg) * T + row] = row_norm2_part(sK, row, cg);
    publish();
    const float q2 = group_total(redN, row), k2 = group_total(redN + NG * T, row);
    const uint32_t tmem = tmem_base;
    const uint32_t trow = tmem + ((uint32_t)(32 * (warp & 3)) << 16);
    Sync sy{smem_u32(&mbar), 0u, err};
    if (tid == 0) {
      // two commits: the phiQ epilogue runs while the K projection is computed
      const uint32_t aQ = smem_u32(sQ), aK = smem_u32(sK), aOm = smem_u32(sOm);
      const uint32_t aOl = smem_u32(sPhiK);
      for (int k0 = 0; k0 < D; k0 += 16) {
        mma(tmem, kmaj(aQ, T, k0), kmaj(aOm, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
        mma(tmem, kmaj(aQ, T, k0), kmaj(aOl, MF, k0), idesc_bf16(T, MF, 0, 0), 1);
      }
      mma_commit(sy.mbar);
      for (int k0 = 0; k0 < D; k0 += 16) {
        mma(tmem + 256, kmaj(aK, T, k0), kmaj(aOm, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
        mma(tmem + 256, kmaj(aK, T, k0), kmaj(aOl, MF, k0), idesc_bf16(T, MF, 0, 0), 1);
      }
      mma_commit(sy.mbar);
    }
    TC_WAIT(sy);  // Q projection done
    float* redZ = reinterpret_cast<float*>(sQ);  // Q is dead; A is written after the next waits
    redZ[cg * T + row] = feature_epilogue<MF, FEAT>(trow, sPhiQ, row, cg, q2, rv, sZ);
    TC_WAIT(sy);  // K projection done: Omega is no longer needed, S_t takes its place
    load_f32_rows64<MF>(sS, P, tid);
    feature_epilogue<MF, FEAT>(trow + 256, sPhiK, row, cg, k2, rv);
    publish();
    if (tid == 0) {
      const uint32_t aPQ = smem_u32(sPhiQ), aPK = smem_u32(sPhiK), aS = smem_u32(sS);
      for (int k0 = 0; k0 < MF; k0 += 16) {
        mma(tmem, kmaj(aPQ, T, k0), kmaj(aPK, T, k0), idesc_bf16(T, T, 0, 0), k0 > 0);
        mma(tmem + 128, kmaj(aPQ, T, k0), mnmaj(aS, k0, C::OMB), idesc_bf16(T, 64, 0, 1), k0 > 0);
      }
      mma_commit(sy.mbar);
    }
    const float dz = group_total(redZ, row);  // phiQ z_t
    TC_WAIT(sy);
    {
      // A: inclusive causal mask, bf16; row sum of the rounded values
      float v[32];
      const int c0 = 32 * cg;
      tmem_ld32(trow + c0, v);
      uint32_t pk[16];
      float rs = 0.f;
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
      red[cg * T + row] = rs;
    }
    publish();
    if (tid == 0) {
      const uint32_t aA = smem_u32(sA), aV = smem_u32(sV);
      for (int k0 = 0; k0 < T; k0 += 16)
        mma(tmem + 128, kmaj(aA, T, k0), mnmaj(aV, k0, ROWT), idesc_bf16(T, 64, 0, 1), 1);
      mma_commit(sy.mbar);
    }
    float rs = 0.f;
#pragma unroll
    for (int g = 0; g < NG; ++g) rs += red[g * T + row];
    TC_WAIT(sy);
    {
      const float den = rs + dz;
      const float inv = den != 0.f ? 1.f / den : 0.f;
      float v[16];
      tmem_ld16(trow + 128 + 16 * cg, v);  // every lane loads (warp-aligned op)
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] *= inv;
      if (rv) st_row16(out + g0 + (size_t)row * D + 16 * cg, v);
    }
  }
  TC_TEARDOWN();
}

// ================================================================== tc_bwd_q
template <int MF, int FEAT>
__device__ __forceinline__ void role_bwd_q(const __nv_bfloat16* __restrict__ Q, const __nv_bfloat16* __restrict__ K,
               const __nv_bfloat16* __restrict__ V, const __nv_bfloat16* __restrict__ Out,
               const __nv_bfloat16* __restrict__ dOut, const __nv_bfloat16* __restrict__ om16,
               const float* __restrict__ pfx, int L, int a, int b, int nt,
               __nv_bfloat16* __restrict__ dq, float* __restrict__ gdelta,
               float* __restrict__ rowstat, float* __restrict__ part, int* err,
    int t, int c, uint8_t* smem_raw, uint64_t& mbar, uint32_t& tmem_base, int& abort_) {
  using C = Cfg<MF>;
  uint8_t* base = align1024(smem_raw);
  uint8_t* sPhiQ = base;
  uint8_t* sPhiK = sPhiQ + C::FEATB;  // later: u
  uint8_t* sU = sPhiK;
  uint8_t* sX = sPhiK + C::FEATB;     // [Q | K | Omega] -> [dA (2 tiles) | S_t] -> [Q | red | Omega]
  uint8_t* sQ = sX;
  uint8_t* sK = sX + ROWT;
  uint8_t* sdA = sX;
  uint8_t* sOm = sX + 2 * ROWT;
  uint8_t* sS = sOm;
  float* redU = reinterpret_cast<float*>(sX + ROWT);  // [NG][128], phase 4
  uint8_t* sV = sOm + C::OMB;         // later: dden as a K-major [16][128] operand + row sums
  uint8_t* sDd = sV;
  float* redA = reinterpret_cast<float*>(sV + 8192);  // [NG][128], phase 2
  uint8_t* sDo = sV + ROWT;           // dout, then dnum in place
  float* sZ = reinterpret_cast<float*>(sDo + ROWT);
  const int row0 = a + t * T;
  const int valid = min(T, b - t * T);
  const size_t g0 = ((size_t)c * L + row0) * D;
  const float* P = pfx + ((size_t)c * nt + t) * C::E;
  TC_PROLOGUE();
  load_rows64(sQ, T, Q + g0, valid, tid, NTHR);
  load_rows64(sK, T, K + g0, valid, tid, NTHR);
  load_rows64(sV, T, V + g0, valid, tid, NTHR);
  load_rows64(sDo, T, dOut + g0, valid, tid, NTHR);
  // this thread's 16 columns of its out row, fetched while the tiles stream in
  uint4 orow[2] = {make_uint4(0, 0, 0, 0), make_uint4(0, 0, 0, 0)};
  if (row < valid) {
    const uint4* src = reinterpret_cast<const uint4*>(Out + g0 + (size_t)row * D + 16 * cg);
    orow[0] = src[0];
    orow[1] = src[1];
  }
  grid_dependency_wait();  // the state prefixes come from the scan just before
  load_rows64(sOm, MF, om16, MF, tid, NTHR);
  load_rows64(sPhiK, MF, om16 + MF * D, MF, tid, NTHR);  // Omega lo, until phiK overwrites it
  for (int m = tid; m < MF; m += NTHR) sZ[m] = P[MF * 64 + m];
  cp_async_wait_all();
  __syncthreads();  // rows were copied by other threads
  {
    const bool rv = row < valid;
    float* redN = reinterpret_cast<float*>(sPhiQ);  // phiQ is written only after phase 1
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
    Sync sy{smem_u32(&mbar), 0u, err};
    if (tid == 0) {
      // two commits: the phiQ epilogue runs while the K projection is computed
      const uint32_t aQ = smem_u32(sQ), aK = smem_u32(sK), aOm = smem_u32(sOm);
      const uint32_t aOl = smem_u32(sPhiK);
      for (int k0 = 0; k0 < D; k0 += 16) {
        mma(tmem, kmaj(aQ, T, k0), kmaj(aOm, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
        mma(tmem, kmaj(aQ, T, k0), kmaj(aOl, MF, k0), idesc_bf16(T, MF, 0, 0), 1);
      }
      mma_commit(sy.mbar);
      for (int k0 = 0; k0 < D; k0 += 16) {
        mma(tmem + 256, kmaj(aK, T, k0), kmaj(aOm, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
        mma(tmem + 256, kmaj(aK, T, k0), kmaj(aOl, MF, k0), idesc_bf16(T, MF, 0, 0), 1);
      }
      mma_commit(sy.mbar);
    }
    TC_WAIT(sy);  // Q projection done
    float* redZ = reinterpret_cast<float*>(sQ);  // Q is dead; dA is written after the next waits
    redZ[cg * T + row] = feature_epilogue<MF, FEAT>(trow, sPhiQ, row, cg, q2, rv, sZ);
    TC_WAIT(sy);  // K projection done: S_t replaces Omega
    load_f32_rows64<MF>(sS, P, tid);
    feature_epilogue<MF, FEAT>(trow + 256, sPhiK, row, cg, k2, rv);
    publish();
    if (tid == 0) {
      const uint32_t aPQ = smem_u32(sPhiQ), aPK = smem_u32(sPhiK);
      const uint32_t aDo = smem_u32(sDo), aV = smem_u32(sV);
      for (int k0 = 0; k0 < MF; k0 += 16)
        mma(tmem, kmaj(aPQ, T, k0), kmaj(aPK, T, k0), idesc_bf16(T, T, 0, 0), k0 > 0);
      for (int k0 = 0; k0 < D; k0 += 16)  // dout V^T (scaled by 1/den below)
        mma(tmem + 128, kmaj(aDo, T, k0), kmaj(aV, T, k0), idesc_bf16(T, T, 0, 0), k0 > 0);
      mma_commit(sy.mbar);
    }
    const float dz = group_total(redZ, row);
    TC_WAIT(sy);
    {
      float v[32];
      tmem_ld32(trow + 32 * cg, v);
      float rs = 0.f;
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        const float x0 = (32 * cg + i <= row) ? v[i] : 0.f;
        const float x1 = (32 * cg + i + 1 <= row) ? v[i + 1] : 0.f;
        float r0, r1;
        unpack_bf16(pack_bf16(x0, x1), r0, r1);
        rs += r0 + r1;
      }
      redA[cg * T + row] = rs;  // V is no longer read: its tile holds the partials
    }
    __syncthreads();
    float rs = 0.f;
#pragma unroll
    for (int g = 0; g < NG; ++g) rs += redA[g * T + row];
    const float den = rs + dz;
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
    for (int n = 4 * cg; n < 4 * cg + 4; ++n)
      *reinterpret_cast<__nv_bfloat16*>(sDd + tile_off(16, n, row)) =
          __float2bfloat16_rn(n == 0 ? dden : 0.f);
    if (rv && cg == 0) {
      float* rsw = rowstat + (((size_t)c * nt + t) * T + row) * 2;
      rsw[0] = den;
      rsw[1] = dden;
    }
    publish();
    if (tid == 0) {
      const uint32_t aDn = smem_u32(sDo), aS = smem_u32(sS), adA = smem_u32(sdA);
      const uint32_t aPK = smem_u32(sPhiK), aPQ = smem_u32(sPhiQ), aDd = smem_u32(sDd);
      for (int k0 = 0; k0 < D; k0 += 16)  // dnum S_t^T
        mma(tmem + 256, kmaj(aDn, T, k0), kmaj(aS, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
      for (int k0 = 0; k0 < T; k0 += 16)  // + dA phiK
        mma(tmem + 256, kmaj(adA, T, k0), mnmaj(aPK, k0, ROWT), idesc_bf16(T, MF, 0, 1), 1);
      for (int h = 0; h < C::MH; ++h)
        for (int k0 = 0; k0 < T; k0 += 16) {  // Gd = phiQ^T [dnum | dden]
          const uint64_t ad = mnmaj(aPQ + h * 2 * ROWT, k0, ROWT);
          mma(tmem + 64 * h, ad, mnmaj(aDn, k0, ROWT), idesc_bf16(T, 64, 1, 1), k0 > 0);
          mma(tmem + 128 + 16 * h, ad, kmaj(aDd, 16, k0), idesc_bf16(T, 16, 1, 0), k0 > 0);
        }
      mma_commit(sy.mbar);
    }
    TC_WAIT(sy);
    // Q and Omega again (for dq = u Omega - q sum(u) and dOmega += u^T q); the
    // copies overlap the epilogue below
    load_rows64(sQ, T, Q + g0, valid, tid, NTHR);
    load_rows64(sOm, MF, om16, MF, tid, NTHR);
    {
      float* dst = gdelta + ((size_t)c * nt + t) * C::E;
      for (int h = 0; h < C::MH; ++h) {
        const int m = 128 * h + row;
        float v[16];
        tmem_ld16(trow + 64 * h + 16 * cg, v);
        st_f32x16(dst + (size_t)m * 64 + 16 * cg, v);
        if (cg == 0) {
          float zz;
          tmem_ld1(trow + 128 + 16 * h, zz);
          dst[MF * 64 + m] = zz;
        }
      }
    }
    {
      // dphiQ (+ dden z_t) -> u (into the phiK tile), this thread's columns
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
    }
    cp_async_wait_all();
    publish();
    if (tid == 0) {
      const uint32_t aU = smem_u32(sU), aOm = smem_u32(sOm), aQ = smem_u32(sQ);
      for (int k0 = 0; k0 < MF; k0 += 16)
        mma(tmem, kmaj(aU, T, k0), mnmaj(aOm, k0, C::OMB), idesc_bf16(T, 64, 0, 1), k0 > 0);
      for (int h = 0; h < C::MH; ++h)
        for (int k0 = 0; k0 < T; k0 += 16)
          mma(tmem + 64 + 64 * h, mnmaj(aU + h * 2 * ROWT, k0, ROWT), mnmaj(aQ, k0, ROWT),
              idesc_bf16(T, 64, 1, 1), k0 > 0);
      mma_commit(sy.mbar);
    }
    float us = 0.f;
    if (FEAT == SLIM_FEAT_EXP) {
#pragma unroll
      for (int g = 0; g < NG; ++g) us += redU[g * T + row];
    }
    TC_WAIT(sy);
    {
      float xq[16];
      ld_feat16(sQ, row, 16 * cg, xq);
      float v[16];
      tmem_ld16(trow + 16 * cg, v);
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = fmaf(-us, xq[i], v[i]);
      if (rv) st_row16(dq + g0 + (size_t)row * D + 16 * cg, v);
      float* dst = part + ((size_t)c * nt + t) * (size_t)(MF * 64);
      for (int h = 0; h < C::MH; ++h) {
        const int m = 128 * h + row;
        tmem_ld16(trow + 64 + 64 * h + 16 * cg, v);
        st_f32x16(dst + (size_t)m * 64 + 16 * cg, v);
      }
    }
  }
  TC_TEARDOWN();
}

// ================================================================== tc_bwd_kv
template <int MF, int FEAT>
__device__ __forceinline__ void role_bwd_kv(const __nv_bfloat16* __restrict__ Q, const __nv_bfloat16* __restrict__ K,
                const __nv_bfloat16* __restrict__ V, const __nv_bfloat16* __restrict__ dOut,
                const __nv_bfloat16* __restrict__ om16, const float* __restrict__ gsfx,
                const float* __restrict__ rowstat, int L, int a, int b, int nt,
                __nv_bfloat16* __restrict__ dk, __nv_bfloat16* __restrict__ dv,
                float* __restrict__ part, int* err,
    int t, int c, uint8_t* smem_raw, uint64_t& mbar, uint32_t& tmem_base, int& abort_) {
  using C = Cfg<MF>;
  uint8_t* base = align1024(smem_raw);
  uint8_t* sPhiQ = base;               // later: u
  uint8_t* sU = sPhiQ;
  uint8_t* sPhiK = sPhiQ + C::FEATB;
  uint8_t* sX = sPhiK + C::FEATB;      // [Q | K | Omega] -> [A | G_t] -> [dA | G_t] -> [K | red | Omega]
  uint8_t* sQ = sX;
  uint8_t* sK = sX + ROWT;
  uint8_t* sA = sX;
  uint8_t* sKr = sX;
  float* redU = reinterpret_cast<float*>(sX + ROWT);
  uint8_t* sOm = sX + 2 * ROWT;
  uint8_t* sG = sOm;
  uint8_t* sV = sOm + C::OMB;
  uint8_t* sDn = sV + ROWT;            // dout, then dnum in place
  float* sGz = reinterpret_cast<float*>(sDn + ROWT);
  const int row0 = a + t * T;
  const int valid = min(T, b - t * T);
  const size_t g0 = ((size_t)c * L + row0) * D;
  const float* G = gsfx + ((size_t)c * nt + t) * C::E;
  TC_PROLOGUE();
  load_rows64(sQ, T, Q + g0, valid, tid, NTHR);
  load_rows64(sK, T, K + g0, valid, tid, NTHR);
  load_rows64(sV, T, V + g0, valid, tid, NTHR);
  load_rows64(sDn, T, dOut + g0, valid, tid, NTHR);
  grid_dependency_wait();  // G suffixes (scan) and row statistics (tc_bwd_q) are earlier kernels'
  load_rows64(sOm, MF, om16, MF, tid, NTHR);
  load_rows64(sPhiK, MF, om16 + MF * D, MF, tid, NTHR);  // Omega lo, until phiK overwrites it
  for (int m = tid; m < MF; m += NTHR) sGz[m] = G[MF * 64 + m];
  float den = 0.f, dden = 0.f;
  if (row < valid) {
    const float* rsr = rowstat + (((size_t)c * nt + t) * T + row) * 2;
    den = rsr[0];
    dden = rsr[1];
  }
  cp_async_wait_all();
  __syncthreads();  // rows were copied by other threads
  {
    const bool rv = row < valid;
    const bool live = rv && den != 0.f;
    const float inv = live ? 1.f / den : 0.f;
    if (!live) dden = 0.f;
    float* redN = reinterpret_cast<float*>(sPhiQ);  // phiQ is written only after phase 1
    redN[cg * T + row] = row_norm2_part(sQ, row, cg);
    redN[(NG + cg) * T + row] = row_norm2_part(sK, row, cg);
#pragma unroll
    for (int c8 = 16 * cg; c8 < 16 * cg + 16; c8 += 8) {  // dnum = dout / den, in place
      const uint4 g = ld_chunk(sDn, T, row, c8);
      const uint32_t gw[4] = {g.x, g.y, g.z, g.w};
      uint32_t pw[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float g0f, g1f;
        unpack_bf16(gw[i], g0f, g1f);
        pw[i] = pack_bf16(g0f * inv, g1f * inv);
      }
      st_chunk(sDn, T, row, c8, make_uint4(pw[0], pw[1], pw[2], pw[3]));
    }
    publish();
    const float q2 = group_total(redN, row), k2 = group_total(redN + NG * T, row);
    const uint32_t tmem = tmem_base;
    const uint32_t trow = tmem + ((uint32_t)(32 * (warp & 3)) << 16);
    Sync sy{smem_u32(&mbar), 0u, err};
    if (tid == 0) {
      // two commits: the phiQ epilogue runs while the K projection is computed
      const uint32_t aQ = smem_u32(sQ), aK = smem_u32(sK), aOm = smem_u32(sOm);
      const uint32_t aOl = smem_u32(sPhiK);
      for (int k0 = 0; k0 < D; k0 += 16) {
        mma(tmem, kmaj(aQ, T, k0), kmaj(aOm, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
        mma(tmem, kmaj(aQ, T, k0), kmaj(aOl, MF, k0), idesc_bf16(T, MF, 0, 0), 1);
      }
      mma_commit(sy.mbar);
      for (int k0 = 0; k0 < D; k0 += 16) {
        mma(tmem + 256, kmaj(aK, T, k0), kmaj(aOm, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
        mma(tmem + 256, kmaj(aK, T, k0), kmaj(aOl, MF, k0), idesc_bf16(T, MF, 0, 0), 1);
      }
      mma_commit(sy.mbar);
    }
    TC_WAIT(sy);  // Q projection done
    feature_epilogue<MF, FEAT>(trow, sPhiQ, row, cg, q2, rv);
    TC_WAIT(sy);  // K projection done: G_t(S) replaces Omega
    load_f32_rows64<MF>(sG, G, tid);
    feature_epilogue<MF, FEAT>(trow + 256, sPhiK, row, cg, k2, rv);
    publish();
    if (tid == 0) {
      const uint32_t aPQ = smem_u32(sPhiQ), aPK = smem_u32(sPhiK);
      const uint32_t aDn = smem_u32(sDn), aV = smem_u32(sV);
      for (int k0 = 0; k0 < MF; k0 += 16)
        mma(tmem, kmaj(aPQ, T, k0), kmaj(aPK, T, k0), idesc_bf16(T, T, 0, 0), k0 > 0);
      for (int k0 = 0; k0 < D; k0 += 16)  // dnum V^T
        mma(tmem + 128, kmaj(aDn, T, k0), kmaj(aV, T, k0), idesc_bf16(T, T, 0, 0), k0 > 0);
      mma_commit(sy.mbar);
    }
    TC_WAIT(sy);
    {  // A -> smem (masked, bf16), this thread's 32 columns
      float v[32];
      const int c0 = 32 * cg;
      tmem_ld32(trow + c0, v);
      uint32_t pk[16];
#pragma unroll
      for (int i = 0; i < 32; i += 2)
        pk[i / 2] = pack_bf16((c0 + i <= row) ? v[i] : 0.f, (c0 + i + 1 <= row) ? v[i + 1] : 0.f);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        st_chunk(sA, T, row, c0 + 8 * q, make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]));
    }
    publish();
    if (tid == 0) {
      const uint32_t aA = smem_u32(sA), aDn = smem_u32(sDn), aPK = smem_u32(sPhiK);
      const uint32_t aG = smem_u32(sG), aV = smem_u32(sV);
      for (int k0 = 0; k0 < T; k0 += 16)  // dV = A^T dnum
        mma(tmem, mnmaj(aA, k0, ROWT), mnmaj(aDn, k0, ROWT), idesc_bf16(T, 64, 1, 1), k0 > 0);
      for (int k0 = 0; k0 < MF; k0 += 16)  // + phiK G_t(S)
        mma(tmem, kmaj(aPK, T, k0), mnmaj(aG, k0, C::OMB), idesc_bf16(T, 64, 0, 1), 1);
      for (int k0 = 0; k0 < D; k0 += 16)  // dphiK = V G_t(S)^T
        mma(tmem + 256, kmaj(aV, T, k0), kmaj(aG, MF, k0), idesc_bf16(T, MF, 0, 0), k0 > 0);
      mma_commit(sy.mbar);
    }
    TC_WAIT(sy);
    {
      float v[16];
      tmem_ld16(trow + 16 * cg, v);  // dv
      if (rv) st_row16(dv + g0 + (size_t)row * D + 16 * cg, v);
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
      mma_commit(sy.mbar);
    }
    TC_WAIT(sy);
    // K and Omega again (dk = u Omega - k sum(u), dOmega += u^T k), overlapping the epilogue
    load_rows64(sKr, T, K + g0, valid, tid, NTHR);
    load_rows64(sOm, MF, om16, MF, tid, NTHR);
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
    cp_async_wait_all();
    publish();
    if (tid == 0) {
      const uint32_t aU = smem_u32(sU), aOm = smem_u32(sOm), aK = smem_u32(sKr);
      for (int k0 = 0; k0 < MF; k0 += 16)
        mma(tmem, kmaj(aU, T, k0), mnmaj(aOm, k0, C::OMB), idesc_bf16(T, 64, 0, 1), k0 > 0);
      for (int h = 0; h < C::MH; ++h)
        for (int k0 = 0; k0 < T; k0 += 16)
          mma(tmem + 64 + 64 * h, mnmaj(aU + h * 2 * ROWT, k0, ROWT), mnmaj(aK, k0, ROWT),
              idesc_bf16(T, 64, 1, 1), k0 > 0);
      mma_commit(sy.mbar);
    }
    float us = 0.f;
    if (FEAT == SLIM_FEAT_EXP) {
#pragma unroll
      for (int g = 0; g < NG; ++g) us += redU[g * T + row];
    }
    TC_WAIT(sy);
    {
      float xk[16];
      ld_feat16(sKr, row, 16 * cg, xk);
      float v[16];
      tmem_ld16(trow + 16 * cg, v);
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = fmaf(-us, xk[i], v[i]);
      if (rv) st_row16(dk + g0 + (size_t)row * D + 16 * cg, v);
      float* dst = part + ((size_t)c * nt + t) * (size_t)(MF * 64);
      for (int h = 0; h < C::MH; ++h) {
        const int m = 128 * h + row;
        tmem_ld16(trow + 64 + 64 * h + 16 * cg, v);
        float4* o = reinterpret_cast<float4*>(dst + (size_t)m * 64 + 16 * cg);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          float4 x = o[i];
          x.x += v[4 * i];
          x.y += v[4 * i + 1];
          x.z += v[4 * i + 2];
          x.w += v[4 * i + 3];
          o[i] = x;
        }
      }
    }
  }
  TC_TEARDOWN();
}

// ================================================================== launches
// One launch runs tiles of up to four roles (independent work of different
// slices, longest role first so the short ones fill the last wave); CTA b of
// a role handles tile b % nt of chain b / nt.
struct DeltaJob {
  const __nv_bfloat16 *K, *V, *om16;
  int L, a, b, nt;
  float* delta;
  int* err;
};
struct FwdJob {
  const __nv_bfloat16 *Q, *K, *V, *om16;
  const float* pfx;
  int L, a, b, nt;
  __nv_bfloat16* out;
  int* err;
};
struct BwdQJob {
  const __nv_bfloat16 *Q, *K, *V, *Out, *dOut, *om16;
  const float* pfx;
  int L, a, b, nt;
  __nv_bfloat16* dq;
  float *gdelta, *rowstat, *part;
  int* err;
};
struct BwdKVJob {
  const __nv_bfloat16 *Q, *K, *V, *dOut, *om16;
  const float *gsfx, *rowstat;
  int L, a, b, nt;
  __nv_bfloat16 *dk, *dv;
  float* part;
  int* err;
};
struct TileJobs {
  int n_kv, n_q, n_fwd, n_delta;  // CTAs of each role, in dispatch order
  BwdKVJob kv;
  BwdQJob q;
  FwdJob f;
  DeltaJob d;
};

template <int MF, int FEAT>
__global__ void __launch_bounds__(NTHR, 1) k_tc_tiles(const __grid_constant__ TileJobs J) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t mbar;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_;
  int b = blockIdx.x;
  if (b < J.n_kv) {
    const BwdKVJob& p = J.kv;
    role_bwd_kv<MF, FEAT>(p.Q, p.K, p.V, p.dOut, p.om16, p.gsfx, p.rowstat, p.L, p.a, p.b, p.nt,
                          p.dk, p.dv, p.part, p.err, b % p.nt, b / p.nt, smem_raw, mbar,
                          tmem_base, abort_);
    return;
  }
  b -= J.n_kv;
  if (b < J.n_q) {
    const BwdQJob& p = J.q;
    role_bwd_q<MF, FEAT>(p.Q, p.K, p.V, p.Out, p.dOut, p.om16, p.pfx, p.L, p.a, p.b, p.nt, p.dq,
                         p.gdelta, p.rowstat, p.part, p.err, b % p.nt, b / p.nt, smem_raw, mbar,
                         tmem_base, abort_);
    return;
  }
  b -= J.n_q;
  if (b < J.n_fwd) {
    const FwdJob& p = J.f;
    role_fwd<MF, FEAT>(p.Q, p.K, p.V, p.om16, p.pfx, p.L, p.a, p.b, p.nt, p.out, p.err, b % p.nt,
                       b / p.nt, smem_raw, mbar, tmem_base, abort_);
    return;
  }
  b -= J.n_fwd;
  if (b < J.n_delta) {
    const DeltaJob& p = J.d;
    role_delta<MF, FEAT>(p.K, p.V, p.om16, p.L, p.a, p.b, p.nt, p.delta, p.err, b % p.nt,
                         b / p.nt, smem_raw, mbar, tmem_base, abort_);
  }
}

// The small steps between tile launches: up to two state scans (the
// forward/rollback carry of one slice and the state-gradient carry of
// another), and the two stages of the dOmega reduction of earlier slices.
constexpr int RSPLIT = 64;
struct ScanJob {
  float *buf, *hi, *lo;
  int chains, nt, E4, mode, blocks;
};
struct SmallJobs {
  ScanJob scan[2];
  int nscan;
  // stage 1: sums[split][e] = sum of partials of one range (blocks = r1_bx * RSPLIT)
  const float* r1_part;
  float* r1_sums;
  int r1_nparts, r1_bx;
  // stage 2: domega[e] += sum over the RSPLIT sums, in order
  const float* r2_sums;
  float* r2_domega;
  int r2_blocks;
  int n;  // M * 64
};

__global__ void __launch_bounds__(256) k_tc_small(const __grid_constant__ SmallJobs J) {
  grid_dependency_wait();
  int b = blockIdx.x;
  for (int i = 0; i < J.nscan; ++i) {
    const ScanJob& q = J.scan[i];
    if (b < q.blocks) {
      scan_thread(reinterpret_cast<float4*>(q.buf), reinterpret_cast<float4*>(q.hi),
                  reinterpret_cast<float4*>(q.lo), q.chains, q.nt, q.E4, q.mode,
                  (long long)b * 256 + threadIdx.x);
      return;
    }
    b -= q.blocks;
  }
  if (b < J.r1_bx * RSPLIT) {
    const int e = (b % J.r1_bx) * 256 + threadIdx.x, split = b / J.r1_bx;
    if (e >= J.n) return;
    const int per = (J.r1_nparts + RSPLIT - 1) / RSPLIT;
    const int i0 = split * per, i1 = min(J.r1_nparts, i0 + per);
    float s = 0.f;
#pragma unroll 4
    for (int i = i0; i < i1; ++i) s += J.r1_part[(size_t)i * J.n + e];
    J.r1_sums[(size_t)split * J.n + e] = s;
    return;
  }
  b -= J.r1_bx * RSPLIT;
  if (b < J.r2_blocks) {
    const int e = b * 256 + threadIdx.x;
    if (e >= J.n) return;
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < RSPLIT; ++i) s += J.r2_sums[(size_t)i * J.n + e];
    J.r2_domega[e] += s;
  }
}

// ================================================================== small kernels
// Omega as a bf16 pair: hi = bf16(Omega), lo = bf16(Omega - hi), so the
// projections X Omega^T = X hi^T + X lo^T carry ~16 mantissa bits.
__global__ void k_omega_bf16(const float* om, __nv_bfloat16* om16, int n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) {
    const __nv_bfloat16 hi = __float2bfloat16_rn(om[i]);
    om16[i] = hi;
    om16[n + i] = __float2bfloat16_rn(om[i] - __bfloat162float(hi));
  }
}

// state pair [chains][E] <-> S_state [chains][M][64], z_state [chains][M]
// (the pair is normalised: hi is the rounded state, lo its residual)
__global__ void k_tc_state_out(const float* hi, const float* lo, StateOut st, int chains, int MF) {
  grid_dependency_wait();
  const long long E = (long long)MF * 65;
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= chains * E) return;
  const long long c = i / E, e = i % E;
  if (e < (long long)MF * 64) {
    st.S[c * MF * 64 + e] = hi[i];
    if (st.S_lo) st.S_lo[c * MF * 64 + e] = lo[i];
  } else {
    st.z[c * MF + (e - (long long)MF * 64)] = hi[i];
    if (st.z_lo) st.z_lo[c * MF + (e - (long long)MF * 64)] = lo[i];
  }
}
__global__ void k_tc_state_in(StateIn st, float* hi, float* lo, int chains, int MF) {
  const long long E = (long long)MF * 65;
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= chains * E) return;
  const long long c = i / E, e = i % E;
  if (e < (long long)MF * 64) {
    hi[i] = st.S[c * MF * 64 + e];
    lo[i] = st.S_lo ? st.S_lo[c * MF * 64 + e] : 0.f;
  } else {
    hi[i] = st.z[c * MF + (e - (long long)MF * 64)];
    lo[i] = st.z_lo ? st.z_lo[c * MF + (e - (long long)MF * 64)] : 0.f;
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

// Every per-slice buffer has two slots (slice n uses slot n % 2), because
// consecutive slices overlap in the pipelined launches.
struct Ws {
  int* err;
  __nv_bfloat16* om16;
  float *st_hi, *st_lo;
  float* delta[2];
  float *g_hi, *g_lo;
  float *gdelta[2], *rowstat[2], *part[2], *rsums[2];
};

Ws carve(Carver& cv, const Geo& g, bool bwd) {
  Ws w{};
  const size_t C = g.chains;
  w.err = cv.take<int>(64);
  w.om16 = cv.take<__nv_bfloat16>((size_t)2 * g.MF * D);
  w.st_hi = cv.take<float>(C * g.E);
  w.st_lo = cv.take<float>(C * g.E);
  for (int k = 0; k < 2; ++k) w.delta[k] = cv.take<float>(C * g.nt * g.E);
  if (bwd) {
    w.g_hi = cv.take<float>(C * g.E);
    w.g_lo = cv.take<float>(C * g.E);
    for (int k = 0; k < 2; ++k) {
      w.gdelta[k] = cv.take<float>(C * g.nt * g.E);
      w.rowstat[k] = cv.take<float>(C * g.nt * T * 2);
      w.part[k] = cv.take<float>(C * g.nt * (size_t)g.MF * D);
      w.rsums[k] = cv.take<float>((size_t)RSPLIT * g.MF * D);
    }
  }
  return w;
}

// dynamic shared memory of each role (plus 1 KB for 1024-byte alignment)
template <int MF>
constexpr size_t smem_delta() { return 1024 + 2 * ROWT + Cfg<MF>::OMB + Cfg<MF>::FEATB + 4096; }
template <int MF>
constexpr size_t smem_fwd() {
  return 1024 + 2 * Cfg<MF>::FEATB + 3 * ROWT + Cfg<MF>::OMB + MF * 4 + NG * T * 4;
}
template <int MF>
constexpr size_t smem_bwd() { return 1024 + 2 * Cfg<MF>::FEATB + 4 * ROWT + Cfg<MF>::OMB + MF * 4; }
template <int MF>
constexpr size_t smem_max() {
  return smem_bwd<MF>() > smem_fwd<MF>() ? smem_bwd<MF>() : smem_fwd<MF>();
}

template <int MF, int FEAT>
cudaError_t configure() {
  static bool done = false;
  if (done) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(k_tc_tiles<MF, FEAT>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem_max<MF>());
  if (e != cudaSuccess) return e;
  done = true;
  return cudaSuccess;
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

template <int MF, int FEAT>
cudaError_t launch_tiles(cudaStream_t s, const TileJobs& J, double flops, double bytes,
                         prof::Kid kid) {
  const int n = J.n_kv + J.n_q + J.n_fwd + J.n_delta;
  if (n == 0) return cudaSuccess;
  size_t smem = 0;
  if (J.n_kv || J.n_q) smem = smem_bwd<MF>();
  if (J.n_fwd && smem_fwd<MF>() > smem) smem = smem_fwd<MF>();
  if (J.n_delta && smem_delta<MF>() > smem) smem = smem_delta<MF>();
  prof::Scope ps(kid, s, flops, bytes);
  return launch_dep(k_tc_tiles<MF, FEAT>, dim3(n), dim3(NTHR), smem, s, J);
}

cudaError_t launch_small(cudaStream_t s, SmallJobs& J, prof::Kid kid) {
  int blocks = J.r1_bx * RSPLIT + J.r2_blocks;
  for (int i = 0; i < J.nscan; ++i) blocks += J.scan[i].blocks;
  if (blocks == 0) return cudaSuccess;
  prof::Scope ps(kid, s);
  return launch_dep(k_tc_small, dim3(blocks), dim3(256), 0, s, J);
}

ScanJob scan_job(float* buf, float* hi, float* lo, int chains, int nt, int E, ScanMode mode) {
  ScanJob j;
  j.buf = buf;
  j.hi = hi;
  j.lo = lo;
  j.chains = chains;
  j.nt = nt;
  j.E4 = E / 4;
  j.mode = (int)mode;
  j.blocks = (int)nblk((long long)chains * (E / 4));
  return j;
}

template <int MF, int FEAT>
slim_status fwd_impl(const Problem& p, const __nv_bfloat16* q, const __nv_bfloat16* k,
                     const __nv_bfloat16* v, const float* omega, __nv_bfloat16* out,
                     const StateOut& st, void* workspace, cudaStream_t s) {
  TC_TRY((configure<MF, FEAT>()));
  const Geo g = geometry(p);
  Carver cv(workspace);
  const Ws w = carve(cv, g, false);
  const size_t SE = (size_t)g.chains * g.E;
  TC_TRY(cudaMemsetAsync(w.err, 0, sizeof(int), s));
  TC_TRY(cudaMemsetAsync(w.st_hi, 0, SE * sizeof(float), s));
  TC_TRY(cudaMemsetAsync(w.st_lo, 0, SE * sizeof(float), s));
  {
    prof::Scope ps(prof::K_TC_PREP, s);
    k_omega_bf16<<<nblk(MF * D), 256, 0, s>>>(omega, w.om16, MF * D);  // hi and lo
    TC_TRY(cudaGetLastError());
  }
  const double MD = (double)MF * D;
  auto delta_job = [&](int n) {
    const Slice sl = slice_of(p, g, n);
    return DeltaJob{k, v, w.om16, p.L, sl.a, sl.b, sl.nt, w.delta[n & 1], w.err};
  };
  // Pipeline: the deltas of slice n+1 are computed in the launch that reads
  // slice n's state prefixes.  Algorithmic work per row: delta 4dM (phiK,
  // Delta), forward 4dM (phiQ, readout); phiK recomputation and the 128 x 128
  // tile products are not counted.
  for (int n = -1; n < g.N; ++n) {
    TileJobs J{};
    double rows = 0.0;
    if (n >= 0) {
      const Slice sl = slice_of(p, g, n);
      J.f = FwdJob{q, k, v, w.om16, w.delta[n & 1], p.L, sl.a, sl.b, sl.nt, out, w.err};
      J.n_fwd = sl.nt * g.chains;
      rows += (double)g.chains * sl.b;
    }
    if (n + 1 < g.N) {
      const Slice sl = slice_of(p, g, n + 1);
      J.d = delta_job(n + 1);
      J.n_delta = sl.nt * g.chains;
      rows += (double)g.chains * sl.b;
    }
    TC_TRY((launch_tiles<MF, FEAT>(s, J, rows * 4.0 * MD, rows * D * 2.0 * 3, prof::K_TC_FWD)));
    if (n + 1 < g.N) {
      SmallJobs S{};
      S.scan[0] = scan_job(w.delta[(n + 1) & 1], w.st_hi, w.st_lo, g.chains,
                           slice_of(p, g, n + 1).nt, g.E, SCAN_FWD);
      S.nscan = 1;
      S.n = MF * D;
      TC_TRY(launch_small(s, S, prof::K_TC_SCAN));
    }
  }
  {
    prof::Scope ps(prof::K_STATE, s);
    TC_TRY(launch_dep(k_tc_state_out, dim3(nblk((long long)SE)), dim3(256), 0, s,
                      (const float*)w.st_hi, (const float*)w.st_lo, st, g.chains, MF));
  }
  return SLIM_OK;
}

template <int MF, int FEAT>
slim_status bwd_impl(const Problem& p, const __nv_bfloat16* q, const __nv_bfloat16* k,
                     const __nv_bfloat16* v, const float* omega, const __nv_bfloat16* out,
                     const __nv_bfloat16* dout, const StateIn& st,
                     __nv_bfloat16* dq, __nv_bfloat16* dk, __nv_bfloat16* dv, float* domega,
                     void* workspace, cudaStream_t s) {
  TC_TRY((configure<MF, FEAT>()));
  const Geo g = geometry(p);
  Carver cv(workspace);
  const Ws w = carve(cv, g, true);
  const size_t SE = (size_t)g.chains * g.E;
  const int N = g.N;
  TC_TRY(cudaMemsetAsync(w.err, 0, sizeof(int), s));
  TC_TRY(cudaMemsetAsync(domega, 0, (size_t)MF * D * sizeof(float), s));
  TC_TRY(cudaMemsetAsync(w.g_hi, 0, SE * sizeof(float), s));
  TC_TRY(cudaMemsetAsync(w.g_lo, 0, SE * sizeof(float), s));
  {
    prof::Scope ps(prof::K_TC_PREP, s);
    k_omega_bf16<<<nblk(MF * D), 256, 0, s>>>(omega, w.om16, MF * D);
    TC_TRY(cudaGetLastError());
    k_tc_state_in<<<nblk((long long)SE), 256, 0, s>>>(st, w.st_hi, w.st_lo, g.chains, MF);
    TC_TRY(cudaGetLastError());
  }
  const double MD = (double)MF * D;
  const unsigned r_bx = nblk(MF * D);
  auto valid = [&](int n) { return n >= 0 && n < N; };
  // Stage j of the reverse walk (slices n = N-1 .. 0):
  //   tiles j : dk/dv side of slice N-j, dq side of slice N-1-j, deltas of slice N-2-j
  //   small j : rollback scan of slice N-2-j, state-gradient scan of slice N-1-j,
  //             dOmega reduction stage 1 of slice N-j and stage 2 of slice N+1-j
  // Algorithmic work per row: delta 4dM (phiK, rollback Delta), dq side 10dM,
  // dk/dv side 8dM.
  for (int j = -1; j <= N + 1; ++j) {
    if (j >= 0) {
      TileJobs J{};
      double fl = 0.0, by = 0.0;
      const int nkv = N - j, nq = N - 1 - j, nd = N - 2 - j;
      if (j >= 1 && valid(nkv)) {
        const Slice sl = slice_of(p, g, nkv);
        J.kv = BwdKVJob{q, k, v, dout, w.om16, w.gdelta[nkv & 1], w.rowstat[nkv & 1], p.L, sl.a,
                        sl.b, sl.nt, dk, dv, w.part[nkv & 1], w.err};
        J.n_kv = sl.nt * g.chains;
        fl += (double)g.chains * sl.b * 8.0 * MD;
        by += (double)g.chains * sl.b * D * 2.0 * 6;
      }
      if (valid(nq)) {
        const Slice sl = slice_of(p, g, nq);
        J.q = BwdQJob{q, k, v, out, dout, w.om16, w.delta[nq & 1], p.L, sl.a, sl.b, sl.nt, dq,
                      w.gdelta[nq & 1], w.rowstat[nq & 1], w.part[nq & 1], w.err};
        J.n_q = sl.nt * g.chains;
        fl += (double)g.chains * sl.b * 10.0 * MD;
        by += (double)g.chains * sl.b * D * 2.0 * 6;
      }
      if (valid(nd)) {
        const Slice sl = slice_of(p, g, nd);
        J.d = DeltaJob{k, v, w.om16, p.L, sl.a, sl.b, sl.nt, w.delta[nd & 1], w.err};
        J.n_delta = sl.nt * g.chains;
        fl += (double)g.chains * sl.b * 4.0 * MD;
        by += (double)g.chains * sl.b * D * 2.0 * 2;
      }
      TC_TRY((launch_tiles<MF, FEAT>(s, J, fl, by, prof::K_TC_BWD)));
    } else {
      // prologue: deltas of the last slice
      const Slice sl = slice_of(p, g, N - 1);
      TileJobs J{};
      J.d = DeltaJob{k, v, w.om16, p.L, sl.a, sl.b, sl.nt, w.delta[(N - 1) & 1], w.err};
      J.n_delta = sl.nt * g.chains;
      TC_TRY((launch_tiles<MF, FEAT>(s, J, (double)g.chains * sl.b * 4.0 * MD,
                                     (double)g.chains * sl.b * D * 2.0 * 2, prof::K_TC_BWD)));
    }
    SmallJobs S{};
    S.n = MF * D;
    const int nr = N - 2 - j, ng = N - 1 - j, nx1 = N - j, nx2 = N + 1 - j;
    if (valid(nr))
      S.scan[S.nscan++] = scan_job(w.delta[nr & 1], w.st_hi, w.st_lo, g.chains,
                                   slice_of(p, g, nr).nt, g.E, SCAN_ROLLBACK);
    if (j >= 0 && valid(ng))
      S.scan[S.nscan++] = scan_job(w.gdelta[ng & 1], w.g_hi, w.g_lo, g.chains,
                                   slice_of(p, g, ng).nt, g.E, SCAN_GREV);
    if (j >= 1 && valid(nx1)) {
      S.r1_part = w.part[nx1 & 1];
      S.r1_sums = w.rsums[nx1 & 1];
      S.r1_nparts = g.chains * slice_of(p, g, nx1).nt;
      S.r1_bx = (int)r_bx;
    }
    if (j >= 2 && valid(nx2)) {
      S.r2_sums = w.rsums[nx2 & 1];
      S.r2_domega = domega;
      S.r2_blocks = (int)r_bx;
    }
    TC_TRY(launch_small(s, S, prof::K_TC_SCAN));
  }
  return SLIM_OK;
}

}  // namespace

bool supports(const Problem& p) {
  return p.dtype == SLIM_BF16 && p.d == D && (p.M == 128 || p.M == 256) && p.slice_len() >= 64;
}

size_t workspace_bytes(const Problem& p, bool bwd) {
  Carver cv(nullptr);
  carve(cv, geometry(p), bwd);
  return cv.bytes();
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
                const float* omega, void* out, const StateOut& st, void* workspace,
                cudaStream_t s) {
  using B16 = __nv_bfloat16;
  TC_DISPATCH(fwd_impl, p, (const B16*)q, (const B16*)k, (const B16*)v, omega, (B16*)out, st,
              workspace, s);
}

slim_status bwd(const Problem& p, const void* q, const void* k, const void* v,
                const float* omega, const void* out, const void* dout, const StateIn& st,
                void* dq, void* dk, void* dv, float* domega, void* workspace, cudaStream_t s) {
  using B16 = __nv_bfloat16;
  TC_DISPATCH(bwd_impl, p, (const B16*)q, (const B16*)k, (const B16*)v, omega, (const B16*)out,
              (const B16*)dout, st, (B16*)dq, (B16*)dk, (B16*)dv, domega, workspace, s);
}

}  // namespace tc
}  // namespace slim
