// fp32-compute path of libslim: every supported (d, M, dtype, feature) that the
// tcgen05 tile kernels do not take.  Operands and intermediates are fp32; the
// contractions run as warp MMAs on bf16 pieces of them (k_mma), the feature
// map and the scans on the FP32 pipe.
//
// One slice of Algorithm 1 at a time.  Inside a slice the rows are cut into
// tiles of T rows and every step is a small batched contraction over
// (chain, tile) -- App. B's "block" evaluation with the block's prefix sums
// written as masked matrix products:
//
//   forward, slice n (Sec. 3.2, eqs. 14-16):
//     phiQ, phiK = g(Q), g(K)                    (F, row-wise)
//     Delta_t    = phiK_t^T [V_t | 1]            (the tile's sum of T_l)
//     P_t        = B + sum_{t'<t} Delta_t'       (state before tile t)
//     A_t        = tril(phiQ_t phiK_t^T)         (inclusive causal mask)
//     [num|den]  = phiQ_t P_t + A_t [V_t | 1];  out = num / den   (eq. 4)
//     B         += sum_t Delta_t
//   backward, slice n (Sec. 3.3, eqs. 17-18), from B^(n), G^(n):
//     B -= sum_t Delta_t                          (eq. 17), then P_t as above
//     dnum = dout/den, dden = -<dout, out>/den,  W = [dnum | dden]
//     dA_t   = tril(W_t [V_t | 1]^T)
//     dphiQ  = W_t P_t^T + dA_t phiK_t
//     Gd_t   = phiQ_t^T W_t;   G_t = G + sum_{t'>t} Gd_t'   (reversed prefix sum)
//     dphiK  = dA_t^T phiQ_t + [V_t | 1] G_t^T
//     dV     = A_t^T dnum + phiK_t G_t(S part)
//     G     += sum_t Gd_t                           (eq. 18)
//     feature VJP: dq, dk; dOmega += u^T x
// The state B and its gradient G are carried as fp32 value/error pairs so the
// rollback returns the forward's state to within the pair's precision.
#include <math.h>

#include "common.cuh"
#include "profiler.h"
#include "scan.h"
#include "simt_path.h"

namespace slim {
namespace simt {

constexpr int GT = 64;  // output tile width of the contraction kernel
constexpr int GK = 16;  // reduction chunk (one k16 MMA step)

struct Mat {
  const float* p;
  long long b0, b1;  // batch strides (batch z = z0 * nb1 + z1)
  long long rs, cs;  // element (i, k) at p + i*rs + k*cs
};
struct OutMat {
  float* p;
  long long b0, b1, rs, cs;
};

struct GemmP {
  int m, n, k;
  Mat a, b;
  OutMat c;
  int nb1;
  int zoff;      // first batch index of this launch
  float beta;    // C = A B + beta * C
  int causal;    // C(i, j) = 0 for j > i
  // optional epilogue C(i, j) -= X(i, j) * s(i)
  const float* sx;
  long long sx_b0, sx_rs;
  const float* ss;
  long long ss_b0;
};

// ------------------------------------------------------------------ tensor-core contraction
// x = h + m + l with bf16 pieces: h = bf16(x), m = bf16(x - h), l = bf16(x - h - m)
// (each difference is exact in fp32), 24 bits of x in NS = 3 pieces, 16 in 2.
template <int NS>
__device__ __forceinline__ void split_bf16(float x, float (&pc)[NS]) {
#pragma unroll
  for (int i = 0; i < NS; ++i) {
    pc[i] = __bfloat162float(__float2bfloat16_rn(x));
    x = __fsub_rn(x, pc[i]);
  }
}
__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}
// D += A B for one m16n8k16 tile: A 16 x 16 bf16 (row-major fragment), B
// 16 x 8 bf16 (column fragment), D fp32; one warp.
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// C[m x n] = sum_k A[m x k] B[k x n], batched over blockIdx.z, on the tensor
// cores with warp MMAs: m16 tiles fit the 16-row tiles of short slices, where
// tcgen05's smallest M, 64, would leave three quarters of every MMA empty.  Each
// operand element is split once, when its chunk is staged, into NS bf16
// pieces; shared memory holds the pieces as bf16 pairs along k, so a
// fragment register is one 32-bit load.  The pieces' products with
// i + j < NS are summed into fp32 accumulators, smallest first: NS = 3 (6
// products, 24-bit operands) keeps fp32 problems' products to about 2^-24,
// NS = 2 (3 products, 16-bit operands) serves bf16 problems.  Warp (wm, wn)
// of a group owns rows 16 wm .. 16 wm + 15 and columns WN wn .. WN wn + WN - 1
// of the CTA tile.  A CTA's threads form KS groups; group g takes the reduction
// chunks g, g + KS, ... and the groups' partial tiles are summed in group order
// at the end (a fixed order: the result does not depend on scheduling), so
// that small tiles of long reductions still fill the SMs.  The 65th
// column of an n = 64q + 1 product is summed in fp32 FMA from the pieces by
// the group's first TM threads.
template <int TM, int TN, int KS, int NS>
__global__ void __launch_bounds__(((TM / 16) * (TN >= 32 ? TN / 32 : 1) * 32) * KS) k_mma(GemmP P) {
  constexpr int WN = TN >= 32 ? 32 : TN;          // columns per warp
  constexpr int NB = WN / 8;                      // n8 blocks per warp
  constexpr int NT = (TM / 16) * (TN / WN) * 32;  // threads per group
  constexpr int K2 = GK / 2;                      // k pairs per chunk
  constexpr int LA = TM + 8, LB = TN + 8;         // row strides (words): conflict-free fragments
  constexpr int ASZ = 2 * NS * K2 * LA, BSZ = 2 * NS * K2 * LB;  // words, two buffers
  constexpr int RED = 4 * NB + 1;  // floats a thread hands to group 0
  constexpr int SMW = KS * (ASZ + BSZ);
  static_assert(KS == 1 || (KS - 1) * NT * RED <= SMW, "reduction scratch");
  static_assert(TM * K2 % NT == 0 && TN * K2 % NT == 0, "staging split");
  __shared__ __align__(16) uint32_t sm[SMW];
  const int tid = threadIdx.x, grp = tid / NT, lt = tid % NT;
  // piece q of the k pair kk2 of row r (A) / column n (B) of buffer bf
  uint32_t* Ap = sm + grp * (ASZ + BSZ);
  uint32_t* Bp = Ap + ASZ;
  auto aw = [&](int bf, int q, int kk2, int r) -> uint32_t& { return Ap[((bf * NS + q) * K2 + kk2) * LA + r]; };
  auto bw = [&](int bf, int q, int kk2, int n) -> uint32_t& { return Bp[((bf * NS + q) * K2 + kk2) * LB + n]; };
  constexpr int PA = TM * K2 / NT, PB = TN * K2 / NT;  // k pairs a thread stages
  const int z = blockIdx.z + P.zoff;
  const int z0 = z / P.nb1, z1 = z % P.nb1;
  const float* A = P.a.p + z0 * P.a.b0 + z1 * P.a.b1;
  const float* Bm = P.b.p + z0 * P.b.b0 + z1 * P.b.b1;
  const int i0 = blockIdx.y * TM, j0 = blockIdx.x * TN;
  const int warp = lt / 32, lane = lt % 32, g = lane >> 2, t = lane & 3;
  const int wm = warp / (TN / WN), wn = warp % (TN / WN);
  const bool a_kc = P.a.cs == 1, b_nc = P.b.cs == 1;
  float acc[NB][4];
#pragma unroll
  for (int nb = 0; nb < NB; ++nb)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[nb][c] = 0.f;
  const bool ext = TN == GT && P.n - j0 == GT + 1;
  float acc_e = 0.f;

  // pair e of a chunk: (kk2, row) of A and (kk2, col) of B, laid out so that
  // consecutive threads read consecutive addresses of the contiguous dimension
  float ra[PA][2], rb[PB][2], rx[2] = {0.f, 0.f};
  // Each thread stages the same (pair, row) slots of every chunk: its element
  // addresses are fixed bases plus k0 times the operand's k stride.
  const float* pa[PA];
  int ka[PA];
  bool oka[PA];
#pragma unroll
  for (int i = 0; i < PA; ++i) {
    const int e = lt + i * NT;
    const int kk2 = a_kc ? e % K2 : e / TM, r = a_kc ? e / K2 : e % TM;
    oka[i] = i0 + r < P.m;
    ka[i] = 2 * kk2;
    pa[i] = A + (oka[i] ? (long long)(i0 + r) * P.a.rs + 2LL * kk2 * P.a.cs : 0);
  }
  const float* pb[PB];
  int kb[PB];
  bool okb[PB];
#pragma unroll
  for (int i = 0; i < PB; ++i) {
    const int e = lt + i * NT;
    const int kb2 = b_nc ? e / TN : e % K2, cb = b_nc ? e % TN : e / K2;
    okb[i] = j0 + cb < P.n;
    kb[i] = 2 * kb2;
    pb[i] = Bm + (okb[i] ? 2LL * kb2 * P.b.rs + (long long)(j0 + cb) * P.b.cs : 0);
  }
  const long long ak = P.a.cs, bk = P.b.rs;  // k strides
  auto fetch = [&](int k0) {
    if (ext && lt < K2) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int gk = k0 + 2 * lt + h;
        rx[h] = gk < P.k ? Bm[gk * P.b.rs + (j0 + GT) * P.b.cs] : 0.f;
      }
    }
#pragma unroll
    for (int i = 0; i < PA; ++i) {
      const float* src = pa[i] + k0 * ak;
      const int gk = k0 + ka[i];
      ra[i][0] = (oka[i] && gk < P.k) ? src[0] : 0.f;
      ra[i][1] = (oka[i] && gk + 1 < P.k) ? src[ak] : 0.f;
    }
#pragma unroll
    for (int i = 0; i < PB; ++i) {
      const float* src = pb[i] + k0 * bk;
      const int gk = k0 + kb[i];
      rb[i][0] = (okb[i] && gk < P.k) ? src[0] : 0.f;
      rb[i][1] = (okb[i] && gk + 1 < P.k) ? src[bk] : 0.f;
    }
  };
  auto put_pieces = [&](uint32_t* w0, int stride, const float (&x)[2]) {
    float p0[NS], p1[NS];
    split_bf16<NS>(x[0], p0);
    split_bf16<NS>(x[1], p1);
#pragma unroll
    for (int q = 0; q < NS; ++q) w0[q * stride] = pack2(p0[q], p1[q]);
  };
  auto stage = [&](int bf) {
    if (ext && lt < K2) put_pieces(&bw(bf, 0, lt, GT), K2 * LB, rx);
#pragma unroll
    for (int i = 0; i < PA; ++i) {
      const int e = lt + i * NT;
      const int kk2 = a_kc ? e % K2 : e / TM, r = a_kc ? e / K2 : e % TM;
      put_pieces(&aw(bf, 0, kk2, r), K2 * LA, ra[i]);
    }
#pragma unroll
    for (int i = 0; i < PB; ++i) {
      const int e = lt + i * NT;
      const int kb2 = b_nc ? e / TN : e % K2, cb = b_nc ? e % TN : e / K2;
      put_pieces(&bw(bf, 0, kb2, cb), K2 * LB, rb[i]);
    }
  };
  // the fp32 value (to the pieces' precision) of a staged element pair
  auto unpieces = [&](const uint32_t* w0, int stride, float& lo, float& hi) {
    lo = hi = 0.f;
#pragma unroll
    for (int q = NS - 1; q >= 0; --q) {
      __nv_bfloat162 v = *reinterpret_cast<const __nv_bfloat162*>(&w0[q * stride]);
      lo += __low2float(v);
      hi += __high2float(v);
    }
  };

  const int steps = (P.k + GK * KS - 1) / (GK * KS);
  fetch(grp * GK);
  stage(0);
  __syncthreads();
  int buf = 0;
  const int ar = 16 * wm + g;  // this thread's fragment rows ar and ar + 8
  for (int st = 0; st < steps; ++st) {
    const bool more = st + 1 < steps;
    if (more) fetch((grp + (st + 1) * KS) * GK);
    // register i of the A fragment: k pair t + 4 (i / 2) of row ar + 8 (i % 2)
    uint32_t af[NS][4];
#pragma unroll
    for (int q = 0; q < NS; ++q)
#pragma unroll
      for (int i = 0; i < 4; ++i) af[q][i] = aw(buf, q, t + 4 * (i >> 1), ar + 8 * (i & 1));
#pragma unroll
    for (int nb = 0; nb < NB; ++nb) {
      const int col = WN * wn + 8 * nb + g;
      uint32_t bfr[NS][2];
#pragma unroll
      for (int q = 0; q < NS; ++q)
#pragma unroll
        for (int i = 0; i < 2; ++i) bfr[q][i] = bw(buf, q, t + 4 * i, col);
      // products of pieces (i, j) with i + j < NS, smallest first
#pragma unroll
      for (int o = NS - 1; o >= 0; --o)
#pragma unroll
        for (int i = 0; i <= o; ++i) mma16816(acc[nb], af[i], bfr[o - i]);
    }
    if (ext && lt < TM) {
#pragma unroll
      for (int kk2 = 0; kk2 < K2; ++kk2) {
        float a0, a1, b0, b1;
        unpieces(&aw(buf, 0, kk2, lt), K2 * LA, a0, a1);
        unpieces(&bw(buf, 0, kk2, GT), K2 * LB, b0, b1);
        acc_e = fmaf(a1, b1, fmaf(a0, b0, acc_e));
      }
    }
    if (more) stage(buf ^ 1);
    __syncthreads();
    buf ^= 1;
  }

  if (KS > 1) {
    // groups 1..KS-1 hand their partial tiles to group 0 (element v of
    // thread lt of group g at red[((g - 1) RED + v) NT + lt]), summed in
    // group order
    float* smf = reinterpret_cast<float*>(sm);
    if (grp > 0) {
      float* red = smf + (grp - 1) * RED * NT + lt;
#pragma unroll
      for (int nb = 0; nb < NB; ++nb)
#pragma unroll
        for (int c = 0; c < 4; ++c) red[(4 * nb + c) * NT] = acc[nb][c];
      red[4 * NB * NT] = acc_e;
    }
    __syncthreads();
    if (grp > 0) return;
#pragma unroll 1
    for (int gg = 1; gg < KS; ++gg) {
      const float* red = smf + (gg - 1) * RED * NT + lt;
#pragma unroll
      for (int nb = 0; nb < NB; ++nb)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[nb][c] += red[(4 * nb + c) * NT];
      acc_e += red[4 * NB * NT];
    }
  }

  float* Cm = P.c.p + z0 * P.c.b0 + z1 * P.c.b1;
  auto put = [&](int i, int j, float v) {
    if (P.causal && j > i) v = 0.f;
    if (P.sx) v -= P.sx[z0 * P.sx_b0 + i * P.sx_rs + j] * P.ss[z0 * P.ss_b0 + i];
    float* dst = Cm + i * P.c.rs + j * P.c.cs;
    if (P.beta != 0.f) v += P.beta * *dst;
    *dst = v;
  };
#pragma unroll
  for (int nb = 0; nb < NB; ++nb)
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int i = i0 + ar + 8 * (c >> 1), j = j0 + WN * wn + 8 * nb + 2 * t + (c & 1);
      if (i < P.m && j < P.n) put(i, j, acc[nb][c]);
    }
  if (ext && lt < TM && i0 + lt < P.m) put(i0 + lt, j0 + GT, acc_e);
}

// ------------------------------------------------------------------ per-slice staging
// Loads rows [a, a+b) of every chain, converts to fp32, applies the feature
// map.  Rows b..Cp-1 of the padded tile are zero everywhere (including the
// ones column of [V | 1]), so they add nothing to any contraction.
constexpr int kPrepFeat = 128;  // features per projection chunk

// Omega in the layout the projections read, built once per call: chunk c of
// kPrepFeat features is a [d][kPrepFeat] block (feature index contiguous,
// zero past M), and omn[m] = |omega_m|.
__global__ void k_omega_prep(const float* __restrict__ omega, int M, int d, float* omT,
                             float* omn) {
  const int nch = (M + kPrepFeat - 1) / kPrepFeat;
  const long long n = (long long)nch * d * kPrepFeat;
  for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < n;
       e += (long long)gridDim.x * blockDim.x) {
    const int mm = (int)(e % kPrepFeat);
    const long long cj = e / kPrepFeat;
    const int j = (int)(cj % d), c = (int)(cj / d);
    const int m = c * kPrepFeat + mm;
    omT[e] = m < M ? omega[(size_t)m * d + j] : 0.f;
  }
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) / 32, lane = threadIdx.x % 32;
  const int nw = gridDim.x * blockDim.x / 32;
  for (int m = warp; m < M; m += nw) {
    float t = 0.f;
    for (int j = lane; j < d; j += 32) t = fmaf(omega[(size_t)m * d + j], omega[(size_t)m * d + j], t);
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (lane == 0) omn[m] = sqrtf(t);
  }
}

// R rows per CTA (2R vectors: R queries, then R keys).  One staged chunk of
// Omega serves all of them, in blocks of 32 vectors; R = 64 when the rows fit
// (d <= 64), so that the chunk is staged once per 128 vectors, not 32.
template <typename T, int R>
__global__ void __launch_bounds__(256) k_prep(
    const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v,
    const T* __restrict__ dout, const T* __restrict__ out,
    const float* __restrict__ omT_g, const float* __restrict__ omn_g,
    int L, int ld, int M, int a, int b, int Cp, int feature, int sides, float inv_sqrt_m,
    float* Xq, float* Xk, float* Vx, float* phiQ, float* phiK, float* dout32, float* rowdot) {
  extern __shared__ __align__(16) float sm[];
  static_assert(R % 16 == 0, "vector blocks");
  const int d = 1 << ld;           // d is a power of two (16 .. 128)
  float* omT = sm;                 // [d][kPrepFeat]: a chunk of Omega, transposed
  float* xs = omT + d * kPrepFeat; // [2R][d]
  float* xn2 = xs + 2 * R * d;     // [2R]
  const int c = blockIdx.y, r0 = blockIdx.x * R, tid = threadIdx.x;
  const int dp = d + 1;
  const size_t rowbase = (size_t)c * L + a;

  for (int e = tid; e < R * d; e += 256) {
    const int rr = e >> ld, j = e & (d - 1), r = r0 + rr;
    float xq = 0.f, xk = 0.f, xv = 0.f;
    if (r < b) {
      size_t g = (rowbase + r) * d + j;
      xq = Io<T>::load(q, g);
      xk = Io<T>::load(k, g);
      xv = Io<T>::load(v, g);
    }
    xs[rr * d + j] = xq;
    xs[(R + rr) * d + j] = xk;
    size_t o = ((size_t)c * Cp + r) * d + j;
    Xq[o] = xq;
    Xk[o] = xk;
    Vx[((size_t)c * Cp + r) * dp + j] = xv;
    if (dout32) dout32[o] = (r < b) ? Io<T>::load(dout, (rowbase + r) * d + j) : 0.f;
  }
  for (int rr = tid; rr < R; rr += 256)
    Vx[((size_t)c * Cp + r0 + rr) * dp + d] = (r0 + rr < b) ? 1.f : 0.f;
  __syncthreads();

  const int warp = tid / 32, lane = tid % 32;
  for (int vec = warp; vec < 2 * R; vec += 8) {
    float s = 0.f;
    for (int j = lane; j < d; j += 32) s = fmaf(xs[vec * d + j], xs[vec * d + j], s);
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) xn2[vec] = s;
  }
  if (rowdot) {
    for (int rr = warp; rr < R; rr += 8) {
      const int r = r0 + rr;
      float s = 0.f;
      if (r < b)
        for (int j = lane; j < d; j += 32) {
          size_t g = (rowbase + r) * d + j;
          s = fmaf(Io<T>::load(dout, g), Io<T>::load(out, g), s);
        }
      for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      if (lane == 0) rowdot[(size_t)c * Cp + r] = s;
    }
  }

  if (feature == SLIM_FEAT_SQUARE) {
    // elementwise quadratic map g(x)_i = x_i^2, M = d (Sec. 4): no Omega
    __syncthreads();
    for (int e = tid; e < 2 * R * d; e += 256) {
      const int vec = e >> ld, m = e & (d - 1), r = r0 + vec % R;
      const float x = xs[vec * d + m];
      float* dst = (vec < R) ? phiQ : phiK;
      dst[((size_t)c * Cp + r) * M + m] = (r < b) ? x * x : 0.f;
    }
    return;
  }
  // error bound of an fp32 dot product of length d, times a safety factor 2
  const float gamma = 2.f * (float)(d + 2) * 5.9604645e-08f;
  // The projections x . omega_m, 128 features at a time: thread (f, grp) owns
  // features m0 + 2f and m0 + 2f + 1 of vectors vbase .. vbase + 7, reading
  // four x values per vector as one float4 and two Omega values as one float2
  // (64 FMAs per 12 shared-memory loads).  Each dot product is summed in j
  // order, one fmaf per term.
  const int f = tid % 64, grp = tid / 64;
  for (int m0 = 0; m0 < M; m0 += kPrepFeat) {
    __syncthreads();
    {
      const float4* src = reinterpret_cast<const float4*>(omT_g + (size_t)(m0 / kPrepFeat) * d * kPrepFeat);
      float4* dst = reinterpret_cast<float4*>(omT);
      for (int e = tid; e < d * kPrepFeat / 4; e += 256) dst[e] = src[e];
    }
    __syncthreads();
    for (int vb = 0; vb < 2 * R / 32; ++vb) {
    const int vbase = vb * 32 + grp * 8;  // this thread's vectors vbase .. vbase + 7
    // sides: bit 0 the query features, bit 1 the key features (the
    // non-causal sweeps need one side each); vectors 0..R-1 are queries
    if (!(sides & (vbase < R ? 1 : 2))) continue;
    float acc[8][2];
#pragma unroll
    for (int vv = 0; vv < 8; ++vv) acc[vv][0] = acc[vv][1] = 0.f;
    for (int j = 0; j < d; j += 4) {
      float2 o[4];
#pragma unroll
      for (int t = 0; t < 4; ++t)
        o[t] = *reinterpret_cast<const float2*>(&omT[(j + t) * kPrepFeat + 2 * f]);
#pragma unroll
      for (int vv = 0; vv < 8; ++vv) {
        const float4 x = *reinterpret_cast<const float4*>(&xs[(vbase + vv) * d + j]);
        acc[vv][0] = fmaf(x.x, o[0].x, acc[vv][0]);
        acc[vv][1] = fmaf(x.x, o[0].y, acc[vv][1]);
        acc[vv][0] = fmaf(x.y, o[1].x, acc[vv][0]);
        acc[vv][1] = fmaf(x.y, o[1].y, acc[vv][1]);
        acc[vv][0] = fmaf(x.z, o[2].x, acc[vv][0]);
        acc[vv][1] = fmaf(x.z, o[2].y, acc[vv][1]);
        acc[vv][0] = fmaf(x.w, o[3].x, acc[vv][0]);
        acc[vv][1] = fmaf(x.w, o[3].y, acc[vv][1]);
      }
    }
    // features m0 + 2f and m0 + 2f + 1 (M is even: both exist or neither)
    const int m = m0 + 2 * f;
    if (m < M) {
#pragma unroll
      for (int vv = 0; vv < 8; ++vv) {
        const int vec = vbase + vv;
        const int rr = vec % R, r = r0 + rr;
        float phi[2] = {0.f, 0.f};
        if (r < b) {
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const float dot = acc[vv][h];
            if (feature == SLIM_FEAT_EXP) {
              phi[h] = expf(dot - 0.5f * xn2[vec]) * inv_sqrt_m;
            } else if (fabsf(dot) <= gamma * omn_g[m + h] * sqrtf(xn2[vec])) {
              // The sign of omega.x decides ReLU's branch; near zero it is
              // recomputed as a compensated dot product (FMA TwoProduct and
              // TwoSum, about 48 bits, Ogita-Rump-Oishi Dot2) so that the
              // decision is the exact one.
              float sh = 0.f, sl = 0.f;
              for (int j = 0; j < d; ++j) {
                const float xw = xs[vec * d + j], ow = omT[j * kPrepFeat + 2 * f + h];
                const float p = __fmul_rn(xw, ow), ep = __fmaf_rn(xw, ow, -p);
                float t, e;
                two_sum(sh, p, t, e);
                sh = t;
                sl = __fadd_rn(sl, __fadd_rn(e, ep));
              }
              const float a32 = __fadd_rn(sh, sl);
              phi[h] = a32 > 0.f ? a32 * inv_sqrt_m : 0.f;
            } else {
              phi[h] = dot > 0.f ? dot * inv_sqrt_m : 0.f;
            }
          }
        }
        float* dst = (vec < R) ? phiQ : phiK;
        *reinterpret_cast<float2*>(&dst[((size_t)c * Cp + r) * M + m]) = make_float2(phi[0], phi[1]);
      }
    }
    }
  }
}

template <typename T>
__global__ void k_finalize_out(const float* numden, T* out, int L, int d, int a, int b, int Cp,
                               int chains) {
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (long long)chains * b * d) return;
  const int j = (int)(idx % d);
  const long long rc = idx / d;
  const int r = (int)(rc % b), c = (int)(rc / b);
  const float* row = numden + ((size_t)c * Cp + r) * (d + 1);
  const float den = row[d];
  Io<T>::store(out, ((size_t)c * L + a + r) * d + j, den != 0.f ? row[j] / den : 0.f);
}

__global__ void k_dstat(const float* numden, const float* dout32, const float* rowdot, float* W,
                        int d, int b, int Cp, int chains) {
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const int dp = d + 1;
  if (idx >= (long long)chains * Cp * dp) return;
  const int j = (int)(idx % dp);
  const long long rc = idx / dp;
  const int r = (int)(rc % Cp);
  const float den = numden[rc * dp + d];
  float w = 0.f;
  if (r < b && den != 0.f) w = (j < d) ? dout32[rc * d + j] / den : -rowdot[rc] / den;
  W[idx] = w;
}

// u = dphi * phi (exp) or dphi * 1[phi > 0] / sqrt(M) (ReLU), in place; row sums.
__global__ void k_vjp_prep(float* dphi, const float* phi, float* usum, int M, int rows,
                           int feature, float inv_sqrt_m) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) / 32, lane = threadIdx.x % 32;
  if (warp >= rows) return;
  float* u = dphi + (size_t)warp * M;
  const float* p = phi + (size_t)warp * M;
  float s = 0.f;
  for (int m = lane; m < M; m += 32) {
    float x = (feature == SLIM_FEAT_EXP) ? u[m] * p[m] : (p[m] > 0.f ? u[m] * inv_sqrt_m : 0.f);
    u[m] = x;
    s += x;
  }
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) usum[warp] = s;
}

// Quadratic map: dX = 2 x (.) dphi (M = d, so both are [rows][d]).
__global__ void k_vjp_square(const float* dphi, const float* X, float* stage, long long n) {
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx < n) stage[idx] = 2.f * X[idx] * dphi[idx];
}

template <typename T>
__global__ void k_store(const float* stage, T* dst, int L, int d, int a, int b, int Cp,
                        int chains) {
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (long long)chains * b * d) return;
  const int j = (int)(idx % d);
  const long long rc = idx / d;
  const int r = (int)(rc % b), c = (int)(rc / b);
  Io<T>::store(dst, ((size_t)c * L + a + r) * d + j, stage[((size_t)c * Cp + r) * d + j]);
}

// dOmega += the sum of a launch's partials (per chain and row split), in a
// fixed order, compensated (TwoSum) so that the number of partials does not
// show in the fp32 result.
__global__ void k_reduce_domega(const float* part, float* domega, int parts, int MD) {
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= MD) return;
  float s = domega[e], c = 0.f;
  for (int i = 0; i < parts; ++i) {
    float t, err;
    two_sum(s, part[(size_t)i * MD + e], t, err);
    s = t;
    c += err;
  }
  domega[e] = s + c;
}

// The pair is kept normalised (|lo| <= ulp(hi)/2), so hi is the rounded state
// and lo its residual.
__global__ void k_state_out(const float* hi, const float* lo, StateOut st, int chains, int M,
                            int d) {
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const int dp = d + 1;
  if (idx >= (long long)chains * M * dp) return;
  const int j = (int)(idx % dp);
  const long long cm = idx / dp;
  if (j < d) {
    st.S[cm * d + j] = hi[idx];
    if (st.S_lo) st.S_lo[cm * d + j] = lo[idx];
  } else {
    st.z[cm] = hi[idx];
    if (st.z_lo) st.z_lo[cm] = lo[idx];
  }
}

__global__ void k_state_in(StateIn st, float* hi, float* lo, int chains, int M, int d) {
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const int dp = d + 1;
  if (idx >= (long long)chains * M * dp) return;
  const int j = (int)(idx % dp);
  const long long cm = idx / dp;
  if (j < d) {
    hi[idx] = st.S[cm * d + j];
    lo[idx] = st.S_lo ? st.S_lo[cm * d + j] : 0.f;
  } else {
    hi[idx] = st.z[cm];
    lo[idx] = st.z_lo ? st.z_lo[cm] : 0.f;
  }
}

// ------------------------------------------------------------------ host side
namespace {

constexpr int kGroupRows = 1024;  // rows per launch when short slices are grouped
constexpr int kSplitCtas = 304;   // dOmega contractions: about two waves of 152 SMs

struct Geo {
  int chains, d, dp, M, Cs, T, nt, Cp, N;  // Cs: rows per launch sequence (a slice or a group)
  int ks;        // row splits of the dOmega contractions (divides nt)
  int ns;        // bf16 pieces per operand element in the tensor-core contractions
};

Geo geometry(const Problem& p) {
  Geo g;
  g.chains = p.chains();
  g.d = p.d;
  g.dp = p.d + 1;
  g.M = p.M;
  g.Cs = p.slice_len();
  if (g.Cs < 64 && g.Cs % 16 == 0 && p.L > g.Cs) {
    // Short slices (16, 32 or 48 rows): one tile per slice (T = C) and
    // kGroupRows / C consecutive slices per launch.  The scan over a launch's
    // tiles forms the state at every slice boundary (eq. 16) and the backward's
    // reverse scan every rolled-back state (eq. 17), so each slice is evaluated
    // as on its own; grouping trades workspace (kGroupRows rows, not C) for a
    // launch sequence per group instead of per slice.
    g.T = g.Cs;
    const long long whole = ((long long)p.L + g.T - 1) / g.T * g.T;  // L in whole slices
    const long long rows = (long long)(kGroupRows / g.T) * g.T;
    g.Cs = (int)(rows < whole ? rows : whole);
  } else {
    g.T = g.Cs >= 64 ? 64 : ((g.Cs + 15) / 16) * 16;
    if (g.T < 16) g.T = 16;
  }
  g.nt = (g.Cs + g.T - 1) / g.T;
  g.Cp = g.nt * g.T;
  g.N = p.L == 0 ? 0 : (p.L + g.Cs - 1) / g.Cs;
  // dOmega = sum over rows of u^T x is M x d per chain: few CTAs with a long
  // reduction.  Split the rows into ks runs of whole tiles, one partial each.
  const int mn = ((g.M + GT - 1) / GT) * ((g.d + GT - 1) / GT);
  const int want = (kSplitCtas + g.chains * mn - 1) / (g.chains * mn);
  g.ks = 1;
  for (int k = 2; k <= g.nt && k <= want; ++k)
    if (g.nt % k == 0) g.ks = k;
  // fp32 problems: 3 pieces (24 bits); bf16 problems: 2 (16 bits)
  g.ns = p.dtype == SLIM_F32 ? 3 : 2;
  return g;
}

struct Ws {
  int* err;
  float *st_hi, *st_lo, *g_hi, *g_lo;
  float *Xq, *Xk, *Vx, *phiQ, *phiK, *delta, *A, *numden, *omT, *omn;
  float *dout32, *rowdot, *W, *dA, *dphiQ, *dphiK, *gdelta, *usum_q, *usum_k, *stage, *pOm;
};

Ws carve(Carver& cv, const Geo& g, bool bwd) {
  Ws w{};
  const size_t C = g.chains;
  w.err = cv.take<int>(64);
  w.st_hi = cv.take<float>(C * g.M * g.dp);
  w.st_lo = cv.take<float>(C * g.M * g.dp);
  w.Xq = cv.take<float>(C * g.Cp * g.d);
  w.Xk = cv.take<float>(C * g.Cp * g.d);
  w.Vx = cv.take<float>(C * g.Cp * g.dp);
  w.phiQ = cv.take<float>(C * g.Cp * g.M);
  w.phiK = cv.take<float>(C * g.Cp * g.M);
  w.delta = cv.take<float>(C * g.nt * g.M * g.dp);
  w.A = cv.take<float>(C * g.nt * g.T * g.T);
  w.numden = cv.take<float>(C * g.Cp * g.dp);
  w.omT = cv.take<float>((size_t)((g.M + kPrepFeat - 1) / kPrepFeat) * kPrepFeat * g.d);
  w.omn = cv.take<float>(g.M);
  if (bwd) {
    w.g_hi = cv.take<float>(C * g.M * g.dp);
    w.g_lo = cv.take<float>(C * g.M * g.dp);
    w.dout32 = cv.take<float>(C * g.Cp * g.d);
    w.rowdot = cv.take<float>(C * g.Cp);
    w.W = cv.take<float>(C * g.Cp * g.dp);
    w.dA = cv.take<float>(C * g.nt * g.T * g.T);
    w.dphiQ = cv.take<float>(C * g.Cp * g.M);
    w.dphiK = cv.take<float>(C * g.Cp * g.M);
    w.gdelta = cv.take<float>(C * g.nt * g.M * g.dp);
    w.usum_q = cv.take<float>(C * g.Cp);
    w.usum_k = cv.take<float>(C * g.Cp);
    w.stage = cv.take<float>(C * g.Cp * g.d);
    w.pOm = cv.take<float>(C * g.ks * g.M * g.d);
  }
  return w;
}

Mat mat(const float* p, long long b0, long long b1, long long rs, long long cs) {
  return Mat{p, b0, b1, rs, cs};
}
OutMat omat(float* p, long long b0, long long b1, long long rs, long long cs) {
  return OutMat{p, b0, b1, rs, cs};
}

cudaError_t gemm(cudaStream_t s, int ns, int m, int n, int k, Mat a, Mat b, OutMat c,
                 int nb0, int nb1,
                 float beta, int causal, const float* sx = nullptr, long long sx_b0 = 0,
                 long long sx_rs = 0, const float* ss = nullptr, long long ss_b0 = 0) {
  const int nz = nb0 * nb1;
  for (int z = 0; z < nz; z += 65535) {
    GemmP P{m, n, k, a, b, c, nb1, z, beta, causal, sx, sx_b0, sx_rs, ss, ss_b0};
    const int zc = (nz - z < 65535) ? nz - z : 65535;
    // rows per CTA tile: 16 or 32 for the short tiles of grouped slices;
    // columns: 16 for products only that wide
    const int tn = n <= 16 ? 16 : GT;
    const int tm = (m <= 16 || tn == 16) ? 16 : (m <= 32 ? 32 : 64);
    // reduction groups per CTA for the small tiles, when the reduction has
    // at least two chunks per group (fewer with 3 pieces: shared memory)
    const int want = tn == 16 ? (ns == 2 ? 8 : 4)
                              : (tm == 16 ? (ns == 2 ? 4 : 2) : (tm == 32 ? 2 : 1));
    const int ks = (k >= 2 * GK * want) ? want : 1;
    // n = 64 q + 1 (the [V | 1] operands): the last 64-column tile takes the
    // extra column
    const int nx = (tn == GT && n > GT && n % GT == 1) ? n / GT : (n + tn - 1) / tn;
    dim3 grid(nx, (m + tm - 1) / tm, zc);
    prof::Scope ps(prof::K_GEMM, s, 2.0 * m * n * k * zc);
    const int nthr = (tm / 16) * (tn >= 32 ? tn / 32 : 1) * 32 * ks;
#define SLIM_MMA_LAUNCH(NS, K16, K64)                                                 \
    if (tn == 16) {                                                                   \
      if (ks > 1) k_mma<16, 16, K16, NS><<<grid, nthr, 0, s>>>(P);                    \
      else k_mma<16, 16, 1, NS><<<grid, nthr, 0, s>>>(P);                             \
    } else if (tm == 16) {                                                            \
      if (ks > 1) k_mma<16, GT, K64, NS><<<grid, nthr, 0, s>>>(P);                    \
      else k_mma<16, GT, 1, NS><<<grid, nthr, 0, s>>>(P);                             \
    } else if (tm == 32) {                                                            \
      if (ks > 1) k_mma<32, GT, 2, NS><<<grid, nthr, 0, s>>>(P);                      \
      else k_mma<32, GT, 1, NS><<<grid, nthr, 0, s>>>(P);                             \
    } else {                                                                          \
      k_mma<64, GT, 1, NS><<<grid, nthr, 0, s>>>(P);                                  \
    }
    if (ns == 2) {
      SLIM_MMA_LAUNCH(2, 8, 4)
    } else {
      SLIM_MMA_LAUNCH(3, 4, 2)
    }
#undef SLIM_MMA_LAUNCH
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

unsigned blocks(long long n, int t = 256) { return (unsigned)((n + t - 1) / t); }

#define SLIM_TRY(x)                                   \
  do {                                                \
    cudaError_t e_ = (x);                             \
    if (e_ != cudaSuccess) return SLIM_ERR_CUDA;      \
  } while (0)

template <typename T>
cudaError_t launch_prep(cudaStream_t s, const Problem& p, const Geo& g, const Ws& w,
                        const void* q, const void* k, const void* v, const void* dout,
                        const void* out, const float* omega, int a, int b, bool bwd,
                        int sides = 3) {
  // 64 rows per CTA where they fit (d <= 64, whole blocks of the slice buffer)
  const bool wide = g.d <= 64 && g.Cp % 64 == 0;
  const int R = wide ? 64 : 16;
  const size_t smem = (g.d * kPrepFeat + 2 * R * g.d + 2 * R) * sizeof(float);
  static bool attr_set[kMaxDevices] = {};  // per dtype instantiation and device
  bool* set = device_flag(attr_set);
  if (set == nullptr) return cudaErrorInvalidDevice;
  if (!*set) {
    cudaError_t e = cudaFuncSetAttribute(k_prep<T, 16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         96 * 1024);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(k_prep<T, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize, 96 * 1024);
    if (e != cudaSuccess) return e;
    *set = true;
  }
  dim3 grid(g.Cp / R, g.chains);
  const float inv_sqrt_m = (float)(1.0 / sqrt((double)g.M));
  const double rows = (double)g.chains * b;
  int ld = 0;
  while ((1 << ld) < g.d) ++ld;
  prof::Scope ps(prof::K_PREP, s, (sides == 3 ? 4.0 : 2.0) * rows * g.d * g.M,
                 rows * g.d * sizeof(T) * (bwd ? 5.0 : 3.0));
  auto kern = wide ? k_prep<T, 64> : k_prep<T, 16>;
  kern<<<grid, 256, smem, s>>>(
      (const T*)q, (const T*)k, (const T*)v, bwd ? (const T*)dout : nullptr,
      bwd ? (const T*)out : nullptr, w.omT, w.omn, p.L, ld, g.M, a, b, g.Cp,
      (int)p.feature, sides, inv_sqrt_m, w.Xq, w.Xk, w.Vx, w.phiQ, w.phiK, bwd ? w.dout32 : nullptr,
      bwd ? w.rowdot : nullptr);
  return cudaGetLastError();
}

// Omega's projection layout and row norms, once per call (no Omega for the
// quadratic map).
cudaError_t omega_prep(cudaStream_t s, const Problem& p, const Geo& g, const Ws& w,
                       const float* omega) {
  if (p.feature == SLIM_FEAT_SQUARE || p.L == 0 || omega == nullptr) return cudaSuccess;
  prof::Scope ps(prof::K_PREP, s);
  k_omega_prep<<<64, 256, 0, s>>>(omega, g.M, g.d, w.omT, w.omn);
  return cudaGetLastError();
}

// Delta_t = phiK_t^T [V_t | 1]  (M x dp per tile)
cudaError_t tile_deltas(cudaStream_t s, const Geo& g, const Ws& w) {
  const long long T = g.T, M = g.M, dp = g.dp, Cp = g.Cp, nt = g.nt;
  return gemm(s, g.ns, g.M, g.dp, g.T, mat(w.phiK, Cp * M, T * M, 1, M), mat(w.Vx, Cp * dp, T * dp, dp, 1),
              omat(w.delta, nt * M * dp, M * dp, dp, 1), g.chains, g.nt, 0.f, 0);
}

// A_t = tril(phiQ_t phiK_t^T); [num | den] = phiQ_t P_t + A_t [V_t | 1].
// den_only: the backward, which has the forward's output, needs only the
// denominator column (phiQ_t z_t + rowsum A_t), not num.
cudaError_t scores_and_readout(cudaStream_t s, const Geo& g, const Ws& w, bool den_only) {
  const long long T = g.T, M = g.M, dp = g.dp, Cp = g.Cp, nt = g.nt;
  const long long c0 = den_only ? g.d : 0;  // first column computed
  const int nc = den_only ? 1 : g.dp;
  cudaError_t e = gemm(s, g.ns, g.T, g.T, g.M, mat(w.phiQ, Cp * M, T * M, M, 1),
                       mat(w.phiK, Cp * M, T * M, 1, M), omat(w.A, nt * T * T, T * T, T, 1),
                       g.chains, g.nt, 0.f, 1);
  if (e != cudaSuccess) return e;
  e = gemm(s, g.ns, g.T, nc, g.M, mat(w.phiQ, Cp * M, T * M, M, 1),
           mat(w.delta + c0, nt * M * dp, M * dp, dp, 1),
           omat(w.numden + c0, Cp * dp, T * dp, dp, 1), g.chains, g.nt, 0.f, 0);
  if (e != cudaSuccess) return e;
  return gemm(s, g.ns, g.T, nc, g.T, mat(w.A, nt * T * T, T * T, T, 1),
              mat(w.Vx + c0, Cp * dp, T * dp, dp, 1), omat(w.numden + c0, Cp * dp, T * dp, dp, 1),
              g.chains, g.nt, 1.f, 0);
}

cudaError_t scan(cudaStream_t s, const Geo& g, float* buf, float* hi, float* lo, ScanMode mode) {
  return launch_scan(s, buf, hi, lo, g.chains, g.nt, g.M * g.dp, mode, prof::K_SCAN);
}

template <typename T>
slim_status fwd_impl(const Problem& p, const void* q, const void* k, const void* v,
                     const float* omega, void* out, const StateOut& st, const StateInit& init,
                     void* workspace, cudaStream_t s) {
  const Geo g = geometry(p);
  Carver cv(workspace);
  const Ws w = carve(cv, g, false);
  const size_t E = (size_t)g.chains * g.M * g.dp;
  SLIM_TRY(cudaMemsetAsync(w.err, 0, sizeof(int), s));
  SLIM_TRY(omega_prep(s, p, g, w, omega));
  if (init.S) {
    // B^(0) from an earlier segment (eq. 16 with n - 1 = 0 carried in)
    prof::Scope ps(prof::K_STATE, s);
    k_state_in<<<blocks((long long)E), 256, 0, s>>>(StateIn{init.S, init.z, init.S_lo, init.z_lo},
                                                    w.st_hi, w.st_lo, g.chains, g.M, g.d);
    SLIM_TRY(cudaGetLastError());
  } else {
    SLIM_TRY(cudaMemsetAsync(w.st_hi, 0, E * sizeof(float), s));
    SLIM_TRY(cudaMemsetAsync(w.st_lo, 0, E * sizeof(float), s));
  }
  for (int n = 0; n < g.N; ++n) {
    const int a = n * g.Cs, b = (p.L - a < g.Cs) ? p.L - a : g.Cs;
    SLIM_TRY(launch_prep<T>(s, p, g, w, q, k, v, nullptr, nullptr, omega, a, b, false));
    SLIM_TRY(tile_deltas(s, g, w));
    SLIM_TRY(scan(s, g, w.delta, w.st_hi, w.st_lo, SCAN_FWD));
    SLIM_TRY(scores_and_readout(s, g, w, false));
    { prof::Scope ps(prof::K_FINALIZE, s, 0.0, (double)g.chains * b * g.d * sizeof(T));
    k_finalize_out<T><<<blocks((long long)g.chains * b * g.d), 256, 0, s>>>(
        w.numden, (T*)out, p.L, g.d, a, b, g.Cp, g.chains); }
    SLIM_TRY(cudaGetLastError());
  }
  {
    prof::Scope ps(prof::K_STATE, s);
    k_state_out<<<blocks((long long)E), 256, 0, s>>>(w.st_hi, w.st_lo, st,
                                                     g.chains, g.M, g.d);
  }
  SLIM_TRY(cudaGetLastError());
  return SLIM_OK;
}

template <typename IO>
slim_status bwd_impl(const Problem& p, const void* q, const void* k, const void* v,
                     const float* omega, const void* out, const void* dout,
                     const StateIn& st, const GradIO& gio, void* dq, void* dk, void* dv,
                     float* domega, void* workspace, cudaStream_t s) {
  const Geo g = geometry(p);
  Carver cv(workspace);
  const Ws w = carve(cv, g, true);
  const long long T = g.T, M = g.M, d = g.d, dp = g.dp, Cp = g.Cp, nt = g.nt;
  const size_t E = (size_t)g.chains * g.M * g.dp;
  SLIM_TRY(cudaMemsetAsync(w.err, 0, sizeof(int), s));
  SLIM_TRY(omega_prep(s, p, g, w, omega));
  if (domega) SLIM_TRY(cudaMemsetAsync(domega, 0, (size_t)g.M * g.d * sizeof(float), s));
  const bool square = p.feature == SLIM_FEAT_SQUARE;
  { prof::Scope ps(prof::K_STATE, s);
  k_state_in<<<blocks((long long)E), 256, 0, s>>>(st, w.st_hi, w.st_lo, g.chains,
                                                  g.M, g.d); }
  SLIM_TRY(cudaGetLastError());
  if (gio.S_in) {
    // G^(N) handed in by the backward of a later segment (eq. 18)
    prof::Scope ps(prof::K_STATE, s);
    k_state_in<<<blocks((long long)E), 256, 0, s>>>(StateIn{gio.S_in, gio.z_in, nullptr, nullptr},
                                                    w.g_hi, w.g_lo, g.chains, g.M, g.d);
    SLIM_TRY(cudaGetLastError());
  } else {
    SLIM_TRY(cudaMemsetAsync(w.g_hi, 0, E * sizeof(float), s));
    SLIM_TRY(cudaMemsetAsync(w.g_lo, 0, E * sizeof(float), s));
  }
  const float inv_sqrt_m = (float)(1.0 / sqrt((double)g.M));

  for (int n = g.N - 1; n >= 0; --n) {
    const int a = n * g.Cs, b = (p.L - a < g.Cs) ? p.L - a : g.Cs;
    SLIM_TRY(launch_prep<IO>(s, p, g, w, q, k, v, dout, out, omega, a, b, true));
    SLIM_TRY(tile_deltas(s, g, w));
    SLIM_TRY(scan(s, g, w.delta, w.st_hi, w.st_lo, SCAN_ROLLBACK));
    SLIM_TRY(scores_and_readout(s, g, w, true));
    { prof::Scope ps(prof::K_DSTAT, s);
    k_dstat<<<blocks((long long)g.chains * Cp * dp), 256, 0, s>>>(w.numden, w.dout32, w.rowdot, w.W,
                                                               g.d, b, g.Cp, g.chains); }
    SLIM_TRY(cudaGetLastError());
    // dA_t = tril(W_t [V_t | 1]^T)
    SLIM_TRY(gemm(s, g.ns, g.T, g.T, g.dp, mat(w.W, Cp * dp, T * dp, dp, 1),
                  mat(w.Vx, Cp * dp, T * dp, 1, dp), omat(w.dA, nt * T * T, T * T, T, 1),
                  g.chains, g.nt, 0.f, 1));
    // dphiQ = W_t P_t^T + dA_t phiK_t
    SLIM_TRY(gemm(s, g.ns, g.T, g.M, g.dp, mat(w.W, Cp * dp, T * dp, dp, 1),
                  mat(w.delta, nt * M * dp, M * dp, 1, dp), omat(w.dphiQ, Cp * M, T * M, M, 1),
                  g.chains, g.nt, 0.f, 0));
    SLIM_TRY(gemm(s, g.ns, g.T, g.M, g.T, mat(w.dA, nt * T * T, T * T, T, 1),
                  mat(w.phiK, Cp * M, T * M, M, 1), omat(w.dphiQ, Cp * M, T * M, M, 1), g.chains,
                  g.nt, 1.f, 0));
    // Gd_t = phiQ_t^T W_t, then G_t = G + sum_{t' > t} Gd_t'
    SLIM_TRY(gemm(s, g.ns, g.M, g.dp, g.T, mat(w.phiQ, Cp * M, T * M, 1, M),
                  mat(w.W, Cp * dp, T * dp, dp, 1), omat(w.gdelta, nt * M * dp, M * dp, dp, 1),
                  g.chains, g.nt, 0.f, 0));
    SLIM_TRY(scan(s, g, w.gdelta, w.g_hi, w.g_lo, SCAN_GREV));
    // dphiK = dA_t^T phiQ_t + [V_t | 1] G_t^T
    SLIM_TRY(gemm(s, g.ns, g.T, g.M, g.T, mat(w.dA, nt * T * T, T * T, 1, T),
                  mat(w.phiQ, Cp * M, T * M, M, 1), omat(w.dphiK, Cp * M, T * M, M, 1), g.chains,
                  g.nt, 0.f, 0));
    SLIM_TRY(gemm(s, g.ns, g.T, g.M, g.dp, mat(w.Vx, Cp * dp, T * dp, dp, 1),
                  mat(w.gdelta, nt * M * dp, M * dp, 1, dp), omat(w.dphiK, Cp * M, T * M, M, 1),
                  g.chains, g.nt, 1.f, 0));
    // dV = A_t^T dnum + phiK_t G_t(S)
    SLIM_TRY(gemm(s, g.ns, g.T, g.d, g.T, mat(w.A, nt * T * T, T * T, 1, T),
                  mat(w.W, Cp * dp, T * dp, dp, 1), omat(w.stage, Cp * d, T * d, d, 1), g.chains,
                  g.nt, 0.f, 0));
    SLIM_TRY(gemm(s, g.ns, g.T, g.d, g.M, mat(w.phiK, Cp * M, T * M, M, 1),
                  mat(w.gdelta, nt * M * dp, M * dp, dp, 1), omat(w.stage, Cp * d, T * d, d, 1),
                  g.chains, g.nt, 1.f, 0));
    { prof::Scope ps(prof::K_STORE, s, 0.0, (double)g.chains * b * g.d * sizeof(IO));
    k_store<IO><<<blocks((long long)g.chains * b * g.d), 256, 0, s>>>(w.stage, (IO*)dv, p.L, g.d,
                                                                      a, b, g.Cp, g.chains); }
    SLIM_TRY(cudaGetLastError());
    // feature VJPs
    const int rows = g.chains * g.Cp;
    if (square) {
      // dX = 2 x (.) dphi; no Omega, so no dOmega
      const long long n = (long long)rows * g.d;
      { prof::Scope ps(prof::K_VJP, s);
      k_vjp_square<<<blocks(n), 256, 0, s>>>(w.dphiQ, w.Xq, w.stage, n); }
      SLIM_TRY(cudaGetLastError());
      { prof::Scope ps(prof::K_STORE, s, 0.0, (double)g.chains * b * g.d * sizeof(IO));
      k_store<IO><<<blocks((long long)g.chains * b * g.d), 256, 0, s>>>(w.stage, (IO*)dq, p.L, g.d,
                                                                        a, b, g.Cp, g.chains); }
      SLIM_TRY(cudaGetLastError());
      { prof::Scope ps(prof::K_VJP, s);
      k_vjp_square<<<blocks(n), 256, 0, s>>>(w.dphiK, w.Xk, w.stage, n); }
      SLIM_TRY(cudaGetLastError());
      { prof::Scope ps(prof::K_STORE, s, 0.0, (double)g.chains * b * g.d * sizeof(IO));
      k_store<IO><<<blocks((long long)g.chains * b * g.d), 256, 0, s>>>(w.stage, (IO*)dk, p.L, g.d,
                                                                        a, b, g.Cp, g.chains); }
      SLIM_TRY(cudaGetLastError());
      continue;
    }
    { prof::Scope ps(prof::K_VJP, s);
    k_vjp_prep<<<blocks((long long)rows * 32), 256, 0, s>>>(w.dphiQ, w.phiQ, w.usum_q, g.M, rows,
                                                            (int)p.feature, inv_sqrt_m); }
    SLIM_TRY(cudaGetLastError());
    { prof::Scope ps(prof::K_VJP, s);
    k_vjp_prep<<<blocks((long long)rows * 32), 256, 0, s>>>(w.dphiK, w.phiK, w.usum_k, g.M, rows,
                                                            (int)p.feature, inv_sqrt_m); }
    SLIM_TRY(cudaGetLastError());
    const bool ex = p.feature == SLIM_FEAT_EXP;
    // dX = u Omega (- x sum u for the exp map)
    SLIM_TRY(gemm(s, g.ns, g.Cp, g.d, g.M, mat(w.dphiQ, Cp * M, 0, M, 1), mat(omega, 0, 0, d, 1),
                  omat(w.stage, Cp * d, 0, d, 1), g.chains, 1, 0.f, 0, ex ? w.Xq : nullptr,
                  Cp * d, d, w.usum_q, Cp));
    { prof::Scope ps(prof::K_STORE, s, 0.0, (double)g.chains * b * g.d * sizeof(IO));
    k_store<IO><<<blocks((long long)g.chains * b * g.d), 256, 0, s>>>(w.stage, (IO*)dq, p.L, g.d,
                                                                      a, b, g.Cp, g.chains); }
    SLIM_TRY(cudaGetLastError());
    SLIM_TRY(gemm(s, g.ns, g.Cp, g.d, g.M, mat(w.dphiK, Cp * M, 0, M, 1), mat(omega, 0, 0, d, 1),
                  omat(w.stage, Cp * d, 0, d, 1), g.chains, 1, 0.f, 0, ex ? w.Xk : nullptr,
                  Cp * d, d, w.usum_k, Cp));
    { prof::Scope ps(prof::K_STORE, s, 0.0, (double)g.chains * b * g.d * sizeof(IO));
    k_store<IO><<<blocks((long long)g.chains * b * g.d), 256, 0, s>>>(w.stage, (IO*)dk, p.L, g.d,
                                                                      a, b, g.Cp, g.chains); }
    SLIM_TRY(cudaGetLastError());
    // dOmega partials per chain and row split: u_q^T x_q + u_k^T x_k
    const long long kc = (long long)(g.nt / g.ks) * T, ks = g.ks;
    SLIM_TRY(gemm(s, g.ns, g.M, g.d, (int)kc, mat(w.dphiQ, Cp * M, kc * M, 1, M),
                  mat(w.Xq, Cp * d, kc * d, d, 1), omat(w.pOm, ks * M * d, M * d, d, 1), g.chains,
                  g.ks, 0.f, 0));
    SLIM_TRY(gemm(s, g.ns, g.M, g.d, (int)kc, mat(w.dphiK, Cp * M, kc * M, 1, M),
                  mat(w.Xk, Cp * d, kc * d, d, 1), omat(w.pOm, ks * M * d, M * d, d, 1), g.chains,
                  g.ks, 1.f, 0));
    { prof::Scope ps(prof::K_REDUCE, s);
    k_reduce_domega<<<blocks((long long)M * d), 256, 0, s>>>(w.pOm, domega, g.chains * g.ks,
                                                             (int)(M * d)); }
    SLIM_TRY(cudaGetLastError());
  }
  if (gio.S_out) {
    // G^(0): the gradient with respect to the state this segment started from
    prof::Scope ps(prof::K_STATE, s);
    k_state_out<<<blocks((long long)E), 256, 0, s>>>(w.g_hi, w.g_lo,
                                                     StateOut{gio.S_out, gio.z_out, nullptr, nullptr},
                                                     g.chains, g.M, g.d);
    SLIM_TRY(cudaGetLastError());
  }
  return SLIM_OK;
}

// ------------------------------------------------------------------ non-causal form
// Eq. 2 without the mask: one global state B = sum over all rows (eq. 3 at
// l = L) serves every row.  Memory stays O(C): the forward reads the slices
// twice (accumulate B, then read it out), the backward twice as well (query
// side, which also accumulates G = grad_B, then key/value side, which reads G).

// Feature-map VJP of one side of a slice: u = dphi * g'(x) in place, dX stored
// to rows [a, a+b) of dst, and the side's dOmega partial added to domega.
template <typename IO>
cudaError_t side_vjp(cudaStream_t s, const Problem& p, const Geo& g, const Ws& w, float* dphi,
                     const float* phi, const float* X, float* usum, const float* omega, void* dst,
                     float* domega, int a, int b) {
  const long long M = g.M, d = g.d, Cp = g.Cp;
  const int rows = g.chains * g.Cp;
  cudaError_t e;
  if (p.feature == SLIM_FEAT_SQUARE) {
    const long long n = (long long)rows * g.d;
    { prof::Scope ps(prof::K_VJP, s);
    k_vjp_square<<<blocks(n), 256, 0, s>>>(dphi, X, w.stage, n); }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  } else {
    { prof::Scope ps(prof::K_VJP, s);
    k_vjp_prep<<<blocks((long long)rows * 32), 256, 0, s>>>(dphi, phi, usum, g.M, rows,
                                                            (int)p.feature,
                                                            (float)(1.0 / sqrt((double)g.M))); }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const bool ex = p.feature == SLIM_FEAT_EXP;
    e = gemm(s, g.ns, g.Cp, g.d, g.M, mat(dphi, Cp * M, 0, M, 1), mat(omega, 0, 0, d, 1),
             omat(w.stage, Cp * d, 0, d, 1), g.chains, 1, 0.f, 0, ex ? X : nullptr, Cp * d, d,
             usum, Cp);
    if (e != cudaSuccess) return e;
    const long long kc = (long long)(g.nt / g.ks) * g.T, ks = g.ks;
    e = gemm(s, g.ns, g.M, g.d, (int)kc, mat(dphi, Cp * M, kc * M, 1, M),
             mat(X, Cp * d, kc * d, d, 1), omat(w.pOm, ks * M * d, M * d, d, 1), g.chains, g.ks,
             0.f, 0);
    if (e != cudaSuccess) return e;
    { prof::Scope ps(prof::K_REDUCE, s);
    k_reduce_domega<<<blocks((long long)M * d), 256, 0, s>>>(w.pOm, domega, g.chains * g.ks,
                                                             (int)(M * d)); }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  { prof::Scope ps(prof::K_STORE, s, 0.0, (double)g.chains * b * g.d * sizeof(IO));
  k_store<IO><<<blocks((long long)g.chains * b * g.d), 256, 0, s>>>(w.stage, (IO*)dst, p.L, g.d,
                                                                    a, b, g.Cp, g.chains); }
  return cudaGetLastError();
}

template <typename T>
slim_status fwd_bidir_impl(const Problem& p, const void* q, const void* k, const void* v,
                           const float* omega, void* out, const StateOut& st, void* workspace,
                           cudaStream_t s) {
  const Geo g = geometry(p);
  Carver cv(workspace);
  const Ws w = carve(cv, g, false);
  const long long TT = g.T, M = g.M, dp = g.dp, Cp = g.Cp;
  const size_t E = (size_t)g.chains * g.M * g.dp;
  SLIM_TRY(cudaMemsetAsync(w.err, 0, sizeof(int), s));
  SLIM_TRY(omega_prep(s, p, g, w, omega));
  SLIM_TRY(cudaMemsetAsync(w.st_hi, 0, E * sizeof(float), s));
  SLIM_TRY(cudaMemsetAsync(w.st_lo, 0, E * sizeof(float), s));
  // sweep 1: B = sum over every tile of every slice of g(K)^T [V | 1]
  for (int n = 0; n < g.N; ++n) {
    const int a = n * g.Cs, b = (p.L - a < g.Cs) ? p.L - a : g.Cs;
    SLIM_TRY(launch_prep<T>(s, p, g, w, q, k, v, nullptr, nullptr, omega, a, b, false, 2));
    SLIM_TRY(tile_deltas(s, g, w));
    SLIM_TRY(scan(s, g, w.delta, w.st_hi, w.st_lo, SCAN_FWD));
  }
  { prof::Scope ps(prof::K_STATE, s);
  k_state_out<<<blocks((long long)E), 256, 0, s>>>(w.st_hi, w.st_lo, st, g.chains, g.M, g.d); }
  SLIM_TRY(cudaGetLastError());
  // sweep 2: [num | den] = g(Q) B, out = num / den
  for (int n = 0; n < g.N; ++n) {
    const int a = n * g.Cs, b = (p.L - a < g.Cs) ? p.L - a : g.Cs;
    SLIM_TRY(launch_prep<T>(s, p, g, w, q, k, v, nullptr, nullptr, omega, a, b, false, 1));
    SLIM_TRY(gemm(s, g.ns, g.T, g.dp, g.M, mat(w.phiQ, Cp * M, TT * M, M, 1),
                  mat(w.st_hi, M * dp, 0, dp, 1), omat(w.numden, Cp * dp, TT * dp, dp, 1),
                  g.chains, g.nt, 0.f, 0));
    { prof::Scope ps(prof::K_FINALIZE, s, 0.0, (double)g.chains * b * g.d * sizeof(T));
    k_finalize_out<T><<<blocks((long long)g.chains * b * g.d), 256, 0, s>>>(
        w.numden, (T*)out, p.L, g.d, a, b, g.Cp, g.chains); }
    SLIM_TRY(cudaGetLastError());
  }
  return SLIM_OK;
}

template <typename IO>
slim_status bwd_bidir_impl(const Problem& p, const void* q, const void* k, const void* v,
                           const float* omega, const void* out, const void* dout,
                           const StateIn& st, void* dq, void* dk, void* dv, float* domega,
                           void* workspace, cudaStream_t s) {
  const Geo g = geometry(p);
  Carver cv(workspace);
  const Ws w = carve(cv, g, true);
  const long long T = g.T, M = g.M, d = g.d, dp = g.dp, Cp = g.Cp, nt = g.nt;
  const size_t E = (size_t)g.chains * g.M * g.dp;
  SLIM_TRY(cudaMemsetAsync(w.err, 0, sizeof(int), s));
  SLIM_TRY(omega_prep(s, p, g, w, omega));
  if (domega) SLIM_TRY(cudaMemsetAsync(domega, 0, (size_t)g.M * g.d * sizeof(float), s));
  { prof::Scope ps(prof::K_STATE, s);
  k_state_in<<<blocks((long long)E), 256, 0, s>>>(st, w.st_hi, w.st_lo, g.chains, g.M, g.d); }
  SLIM_TRY(cudaGetLastError());
  SLIM_TRY(cudaMemsetAsync(w.g_hi, 0, E * sizeof(float), s));
  SLIM_TRY(cudaMemsetAsync(w.g_lo, 0, E * sizeof(float), s));
  // sweep 1, query side: W = [dnum | dden], dphiQ = W B^T, G += g(Q)^T W
  for (int n = 0; n < g.N; ++n) {
    const int a = n * g.Cs, b = (p.L - a < g.Cs) ? p.L - a : g.Cs;
    SLIM_TRY(launch_prep<IO>(s, p, g, w, q, k, v, dout, out, omega, a, b, true, 1));
    // den = g(Q) z: the only column of [num | den] the gradients need
    SLIM_TRY(gemm(s, g.ns, g.T, 1, g.M, mat(w.phiQ, Cp * M, T * M, M, 1),
                  mat(w.st_hi + d, M * dp, 0, dp, 1), omat(w.numden + d, Cp * dp, T * dp, dp, 1),
                  g.chains, g.nt, 0.f, 0));
    { prof::Scope ps(prof::K_DSTAT, s);
    k_dstat<<<blocks((long long)g.chains * Cp * dp), 256, 0, s>>>(w.numden, w.dout32, w.rowdot,
                                                                  w.W, g.d, b, g.Cp, g.chains); }
    SLIM_TRY(cudaGetLastError());
    SLIM_TRY(gemm(s, g.ns, g.T, g.M, g.dp, mat(w.W, Cp * dp, T * dp, dp, 1),
                  mat(w.st_hi, M * dp, 0, 1, dp), omat(w.dphiQ, Cp * M, T * M, M, 1),
                  g.chains, g.nt, 0.f, 0));
    SLIM_TRY(gemm(s, g.ns, g.M, g.dp, g.T, mat(w.phiQ, Cp * M, T * M, 1, M),
                  mat(w.W, Cp * dp, T * dp, dp, 1), omat(w.gdelta, nt * M * dp, M * dp, dp, 1),
                  g.chains, g.nt, 0.f, 0));
    SLIM_TRY(scan(s, g, w.gdelta, w.g_hi, w.g_lo, SCAN_GREV));
    SLIM_TRY(side_vjp<IO>(s, p, g, w, w.dphiQ, w.phiQ, w.Xq, w.usum_q, omega, dq, domega, a, b));
  }
  // sweep 2, key/value side: dphiK = [V | 1] G^T, dV = g(K) G_S
  for (int n = 0; n < g.N; ++n) {
    const int a = n * g.Cs, b = (p.L - a < g.Cs) ? p.L - a : g.Cs;
    SLIM_TRY(launch_prep<IO>(s, p, g, w, q, k, v, nullptr, nullptr, omega, a, b, false, 2));
    SLIM_TRY(gemm(s, g.ns, g.T, g.M, g.dp, mat(w.Vx, Cp * dp, T * dp, dp, 1),
                  mat(w.g_hi, M * dp, 0, 1, dp), omat(w.dphiK, Cp * M, T * M, M, 1), g.chains,
                  g.nt, 0.f, 0));
    SLIM_TRY(gemm(s, g.ns, g.T, g.d, g.M, mat(w.phiK, Cp * M, T * M, M, 1),
                  mat(w.g_hi, M * dp, 0, dp, 1), omat(w.stage, Cp * d, T * d, d, 1), g.chains,
                  g.nt, 0.f, 0));
    { prof::Scope ps(prof::K_STORE, s, 0.0, (double)g.chains * b * g.d * sizeof(IO));
    k_store<IO><<<blocks((long long)g.chains * b * g.d), 256, 0, s>>>(w.stage, (IO*)dv, p.L, g.d,
                                                                      a, b, g.Cp, g.chains); }
    SLIM_TRY(cudaGetLastError());
    SLIM_TRY(side_vjp<IO>(s, p, g, w, w.dphiK, w.phiK, w.Xk, w.usum_k, omega, dk, domega, a, b));
  }
  return SLIM_OK;
}

}  // namespace

size_t workspace_bytes(const Problem& p, bool bwd) {
  const Geo g = geometry(p);
  Carver cv(nullptr);
  carve(cv, g, bwd);
  return cv.bytes();
}

slim_status fwd(const Problem& p, const void* q, const void* k, const void* v,
                const float* omega, void* out, const StateOut& st, const StateInit& init,
                void* workspace, cudaStream_t s) {
  if (p.dtype == SLIM_BF16)
    return fwd_impl<__nv_bfloat16>(p, q, k, v, omega, out, st, init, workspace, s);
  return fwd_impl<float>(p, q, k, v, omega, out, st, init, workspace, s);
}

slim_status bwd(const Problem& p, const void* q, const void* k, const void* v,
                const float* omega, const void* out, const void* dout, const StateIn& st,
                const GradIO& gio, void* dq, void* dk, void* dv, float* domega, void* workspace,
                cudaStream_t s) {
  if (p.dtype == SLIM_BF16)
    return bwd_impl<__nv_bfloat16>(p, q, k, v, omega, out, dout, st, gio, dq, dk, dv,
                                   domega, workspace, s);
  return bwd_impl<float>(p, q, k, v, omega, out, dout, st, gio, dq, dk, dv, domega,
                         workspace, s);
}

}  // namespace simt
}  // namespace slim

namespace slim {
namespace simt {

slim_status fwd_bidir(const Problem& p, const void* q, const void* k, const void* v,
                      const float* omega, void* out, const StateOut& st, void* workspace,
                      cudaStream_t s) {
  if (p.dtype == SLIM_BF16)
    return fwd_bidir_impl<__nv_bfloat16>(p, q, k, v, omega, out, st, workspace, s);
  return fwd_bidir_impl<float>(p, q, k, v, omega, out, st, workspace, s);
}

slim_status bwd_bidir(const Problem& p, const void* q, const void* k, const void* v,
                      const float* omega, const void* out, const void* dout, const StateIn& st,
                      void* dq, void* dk, void* dv, float* domega, void* workspace,
                      cudaStream_t s) {
  if (p.dtype == SLIM_BF16)
    return bwd_bidir_impl<__nv_bfloat16>(p, q, k, v, omega, out, dout, st, dq, dk, dv, domega,
                                         workspace, s);
  return bwd_bidir_impl<float>(p, q, k, v, omega, out, dout, st, dq, dk, dv, domega, workspace,
                               s);
}

}  // namespace simt
}  // namespace slim
