// A stack of s residual causal linear-attention layers run the memory-efficient
// way of Algorithm 1: slices in the outer loop, layers in the inner loop, one
// carried state per layer (the s rows of B in Sec. 3.2), and the reverse sweep
// of Algorithm 2 with a per-layer rollback (eq. 17) and state gradient (eq. 18).
//
// Layer r maps each row of its input X^(r-1) to q = k = v = u, the row scaled
// to a root-mean-square of d^(-1/4) (u = d^(-1/4) x / sqrt(mean(x^2) + eps), a
// parameter-free row normalisation in place of the layer norm of the paper's
// model, Sec. 2.2 eqs. 5-6), runs attention with its own Omega_r and adds the output
// back: X^(r) = X^(r-1) + Att_r(u, u, u).
// Each (slice, layer) step is one call of the segment entry points
// (slim_fwd_from / slim_bwd_from) on the slice's rows, gathered into a
// contiguous buffer, so the work runs in the same kernels as a single layer.
// Memory beyond inputs and outputs: one slice's activations per layer, the
// per-layer states and state gradients, and one call's workspace -- O(C), not
// O(L) (Sec. 3.4).
#include <stdint.h>
#include <string.h>

#include "common.cuh"
#include "profiler.h"
#include "stack.h"

namespace slim {
namespace stack {
namespace {

// (hi, lo) -= (dhi, dlo): the rollback of eq. 17 on an fp32 value/error pair
__global__ void k_pair_sub(float* hi, float* lo, const float* dhi, const float* dlo, long long n) {
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  float h = hi[i], l = lo[i];
  pair_add(h, l, -dhi[i]);
  pair_add(h, l, -dlo[i]);
  hi[i] = h;
  lo[i] = l;
}
constexpr float kNormEps = 1e-6f;
constexpr int kRowThreads = 256;  // threads per block of the row kernels

// Row kernels: thread `sub` of a row's d/8 lanes owns elements 8 sub .. 8 sub + 7
// and moves them as one 16-byte (bf16) or two 16-byte (fp32) accesses; the
// slice buffers are workspace rows of d contiguous elements, 16-byte aligned.
// A block serves kRowThreads / (d/8) rows.
__device__ __forceinline__ void ld8(const float* p, float* v) {
  const float4 a = reinterpret_cast<const float4*>(p)[0], b = reinterpret_cast<const float4*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void st8(float* p, const float* v) {
  reinterpret_cast<float4*>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
  reinterpret_cast<float4*>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
}
__device__ __forceinline__ void ld8(const __nv_bfloat16* p, float* v) {
  const uint4 r = *reinterpret_cast<const uint4*>(p);
  const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const __nv_bfloat162 h = *reinterpret_cast<const __nv_bfloat162*>(&w[i]);
    v[2 * i] = __low2float(h);
    v[2 * i + 1] = __high2float(h);
  }
}
__device__ __forceinline__ void st8(__nv_bfloat16* p, const float* v) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
    w[i] = *reinterpret_cast<const uint32_t*>(&h);
  }
  *reinterpret_cast<uint4*>(p) = make_uint4(w[0], w[1], w[2], w[3]);
}
// the value a store of x in the dtype reads back as
__device__ __forceinline__ float as_dtype(float x, const float*) { return x; }
__device__ __forceinline__ float as_dtype(float x, const __nv_bfloat16*) {
  return __bfloat162float(__float2bfloat16_rn(x));
}
// sum over the lpr lanes of a row (aligned groups of a power of two)
__device__ __forceinline__ float row_sum(float v, int lpr) {
  for (int o = lpr >> 1; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// This thread's row and first element.  Threads past the last row stay to the
// end (their lanes take part in the row sums' shuffles) and touch no memory.
struct RowPos {
  bool ok;  // the row exists
  size_t o; // element offset of this thread's 8 (0 when !ok)
};
__device__ __forceinline__ RowPos row_pos(int d, long long rows) {
  const int lpr = d >> 3;
  const long long row = (long long)blockIdx.x * (kRowThreads / lpr) + threadIdx.x / lpr;
  const bool ok = row < rows;
  return RowPos{ok, ok ? (size_t)row * d + (threadIdx.x % lpr) * 8 : 0};
}

// u = scale * x / sqrt(mean(x^2) + eps) for one row, from this thread's 8
// values v; the lanes of a row meet in row_sum, so every lane takes part
template <typename T>
__device__ __forceinline__ void norm8(const float* v, T* ur, int d, float scale, bool ok) {
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) ss = fmaf(v[i], v[i], ss);
  const float inv = scale / sqrtf(row_sum(ss, d >> 3) / d + kNormEps);
  float u[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) u[i] = v[i] * inv;
  if (ok) st8(ur, u);
}

// the first layer's u from the slice's rows
template <typename T>
__global__ void __launch_bounds__(kRowThreads) k_rownorm(const T* x, T* u, int d, float scale,
                                                         long long rows) {
  const RowPos rp = row_pos(d, rows);
  float v[8] = {};
  if (rp.ok) ld8(x + rp.o, v);
  norm8(v, u + rp.o, d, scale, rp.ok);
}

// the residual connection out = x + y (fp32 sum rounded to the dtype), then,
// when u is given, the next layer's u from the rounded out (the value the next
// layer's recompute reads back)
template <typename T>
__global__ void __launch_bounds__(kRowThreads) k_residual_norm(const T* x, const T* y, T* out,
                                                               T* u, int d, float scale,
                                                               long long rows) {
  const RowPos rp = row_pos(d, rows);
  float a[8] = {}, b[8] = {};
  if (rp.ok) {
    ld8(x + rp.o, a);
    ld8(y + rp.o, b);
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) a[i] = as_dtype(a[i] + b[i], x);
  if (rp.ok) st8(out + rp.o, a);
  if (u) norm8(a, u + rp.o, d, scale, rp.ok);
}

// dX (fp32) += u'(x)^T g with g = dq + dk + dv (q = k = v = u(x)):
//   dx += (scale / r) (g - x mean(g x) / r^2),  r = sqrt(mean(x^2) + eps),
// and the next layer down's upstream gradient (the new dX) as the dtype into
// dout.  For the top layer (first) the old dX is dout itself: the slice's dy.
template <typename T>
__global__ void __launch_bounds__(kRowThreads) k_dx_accum(float* dx, const T* x, const T* dq,
                                                          const T* dk, const T* dv, T* dout,
                                                          int d, float scale, long long rows,
                                                          int first) {
  const RowPos rp = row_pos(d, rows);
  const size_t o = rp.o;
  float xv[8] = {}, g[8] = {}, t[8] = {};
  if (rp.ok) {
    ld8(x + o, xv);
    ld8(dq + o, g);
    ld8(dk + o, t);
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) g[i] += t[i];
  if (rp.ok) ld8(dv + o, t);
  float ss = 0.f, gx = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    g[i] += t[i];
    ss = fmaf(xv[i], xv[i], ss);
    gx = fmaf(g[i], xv[i], gx);
  }
  const int lpr = d >> 3;
  const float r2 = row_sum(ss, lpr) / d + kNormEps;
  const float m = row_sum(gx, lpr) / d / r2;
  const float f = scale / sqrtf(r2);
  if (!rp.ok) return;  // after the last shuffle
  if (first)
    ld8(dout + o, t);
  else
    ld8(dx + o, t);
#pragma unroll
  for (int i = 0; i < 8; ++i) t[i] += f * (g[i] - xv[i] * m);
  st8(dx + o, t);
  st8(dout + o, t);
}
__global__ void k_add(float* acc, const float* x, long long n) {
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) acc[i] += x[i];
}

struct Geo {
  int chains, Cs, N, s;
  size_t rows;   // chains * Cs: elements of a slice buffer / d
  size_t st;     // chains * M * d, state elements
  size_t zt;     // chains * M
  size_t esz;    // dtype bytes
  size_t inner;  // workspace of one segment call
};

unsigned nb(long long n) { return (unsigned)((n + 255) / 256); }
// blocks of the row kernels for `rows` rows of d elements
unsigned nrb(long long rows, int d) {
  const long long per = kRowThreads / (d / 8);
  return (unsigned)((rows + per - 1) / per);
}
// every launch of this file is counted (and timed when the profiler is on),
// with the bytes it must move
#define STACK_LAUNCH(bytes, ...)                          \
  do {                                                    \
    prof::Scope ps_(prof::K_STACK, s, 0.0, (double)(bytes)); \
    __VA_ARGS__;                                          \
  } while (0)

// rows [a, a+b) of every chain: [chains][L][d] <-> [chains][b][d], one
// strided copy
cudaError_t gather(const void* src, void* dst, const Geo& g, int L, int d, int a, int b,
                   cudaStream_t s) {
  const size_t row = (size_t)d * g.esz;
  return cudaMemcpy2DAsync(dst, b * row, static_cast<const char*>(src) + a * row, L * row,
                           b * row, g.chains, cudaMemcpyDeviceToDevice, s);
}
cudaError_t scatter(const void* src, void* dst, const Geo& g, int L, int d, int a, int b,
                    cudaStream_t s) {
  const size_t row = (size_t)d * g.esz;
  return cudaMemcpy2DAsync(static_cast<char*>(dst) + a * row, L * row, src, b * row, b * row,
                           g.chains, cudaMemcpyDeviceToDevice, s);
}

struct Ws {
  uint8_t** xin;  // backward: [s] each layer's slice input; forward: two, ping-pong
  uint8_t** yout; // [s] layer outputs on the slice
  float *Sb, *zb, *Slb, *zlb;   // [s] running states (backward), value/error pairs
  float *Se, *ze, *Sle, *zle;   // [s] states at the slice's end (backward)
  float *dS, *dz, *dSl, *dzl;   // one slice's own contribution (rollback)
  float *G, *gz, *G2, *gz2;     // [s] state gradients, double-buffered
  float *dx;                    // fp32 dX of the slice
  uint8_t *dout, *dq, *dk, *dv, *scratch_y;
  uint8_t* u;                   // the normalised rows of one layer's slice input
  float* dom;                   // one call's dOmega
  float *Ssc, *zsc;             // a recompute's end state, not needed
  void* inner;
};

size_t inner_bytes(const Problem& p, int Cs) {
  size_t f = 0, b = 0;
  slim_fwd_workspace_size(p.B, p.H, Cs, p.d, p.M, Cs, p.dtype, p.feature, &f);
  slim_bwd_workspace_size(p.B, p.H, Cs, p.d, p.M, Cs, p.dtype, p.feature, &b);
  return f > b ? f : b;
}

Ws carve(Carver& cv, const Problem& p, const Geo& g, bool bwd, uint8_t** xin_ptrs,
         uint8_t** y_ptrs) {
  Ws w{};
  const size_t sb = g.rows * p.d * g.esz;
  // the segment calls' workspace first: its error word is then the stack
  // workspace's first word, where slim_check_device_error reads it
  w.inner = cv.take<uint8_t>(g.inner);
  w.xin = xin_ptrs;
  w.yout = y_ptrs;
  for (int r = 0; r < (bwd ? g.s : 2); ++r) xin_ptrs[r] = cv.take<uint8_t>(sb);
  if (bwd) {
    for (int r = 0; r < g.s; ++r) y_ptrs[r] = cv.take<uint8_t>(sb);
    const size_t S = g.s * g.st, Z = g.s * g.zt;
    w.Sb = cv.take<float>(S); w.zb = cv.take<float>(Z);
    w.Slb = cv.take<float>(S); w.zlb = cv.take<float>(Z);
    w.Se = cv.take<float>(S); w.ze = cv.take<float>(Z);
    w.Sle = cv.take<float>(S); w.zle = cv.take<float>(Z);
    w.dS = cv.take<float>(g.st); w.dz = cv.take<float>(g.zt);
    w.dSl = cv.take<float>(g.st); w.dzl = cv.take<float>(g.zt);
    w.G = cv.take<float>(S); w.gz = cv.take<float>(Z);
    w.G2 = cv.take<float>(S); w.gz2 = cv.take<float>(Z);
    w.dx = cv.take<float>(g.rows * p.d);
    w.dout = cv.take<uint8_t>(sb);
    w.dq = cv.take<uint8_t>(sb);
    w.dk = cv.take<uint8_t>(sb);
    w.dv = cv.take<uint8_t>(sb);
    w.scratch_y = cv.take<uint8_t>(sb);
    w.dom = cv.take<float>((size_t)p.M * p.d);
    w.Ssc = cv.take<float>(g.st);
    w.zsc = cv.take<float>(g.zt);
  } else {
    y_ptrs[0] = cv.take<uint8_t>(sb);
  }
  w.u = cv.take<uint8_t>(sb);
  return w;
}

Geo geometry(const Problem& p, int layers) {
  Geo g;
  g.chains = p.chains();
  g.Cs = p.slice_len();
  g.N = p.num_slices();
  g.s = layers;
  g.rows = (size_t)g.chains * g.Cs;
  g.st = (size_t)g.chains * p.M * p.d;
  g.zt = (size_t)g.chains * p.M;
  g.esz = p.dtype == SLIM_BF16 ? 2 : 4;
  g.inner = inner_bytes(p, g.Cs);
  return g;
}

#define ST_TRY(x)                                \
  do {                                           \
    cudaError_t e_ = (x);                        \
    if (e_ != cudaSuccess) return SLIM_ERR_CUDA; \
  } while (0)
#define ST_CALL(x)                               \
  do {                                           \
    slim_status s_ = (x);                        \
    if (s_ != SLIM_OK) return s_;                \
  } while (0)

template <typename T>
slim_status fwd_impl(const Problem& p, int layers, const T* x, const float* omegas, T* y,
                     float* S_state, float* z_state, float* S_lo, float* z_lo, void* workspace,
                     cudaStream_t s) {
  const Geo g = geometry(p, layers);
  Carver cv(workspace);
  uint8_t* xin[65];
  uint8_t* yo[64];
  const Ws w = carve(cv, p, g, false, xin, yo);
  const int d = p.d, M = p.M;
  const float scale = powf((float)d, -0.25f);
  T* U = reinterpret_cast<T*>(w.u);
  for (int n = 0; n < g.N; ++n) {
    const int a = n * g.Cs, b = (p.L - a < g.Cs) ? p.L - a : g.Cs;
    const long long rows = (long long)g.chains * b;
    const double sb = (double)rows * d * g.esz;  // bytes of one slice tensor
    T* X = reinterpret_cast<T*>(w.xin[0]);
    T* X2 = reinterpret_cast<T*>(w.xin[1]);
    T* Y = reinterpret_cast<T*>(w.yout[0]);
    ST_TRY(gather(x, X, g, p.L, d, a, b, s));
    STACK_LAUNCH(2 * sb, k_rownorm<T><<<nrb(rows, d), kRowThreads, 0, s>>>(X, U, d, scale, rows));
    ST_TRY(cudaGetLastError());
    for (int r = 0; r < layers; ++r) {
      float* Sr = S_state + (size_t)r * g.st;
      float* zr = z_state + (size_t)r * g.zt;
      float* Slr = S_lo ? S_lo + (size_t)r * g.st : nullptr;
      float* zlr = z_lo ? z_lo + (size_t)r * g.zt : nullptr;
      const float* om = omegas ? omegas + (size_t)r * M * d : nullptr;
      // layer r on the slice, from its state after the previous slice (in place)
      ST_CALL(slim_fwd_from(U, U, U, om, p.B, p.H, b, d, M, b, p.dtype, p.feature,
                            n ? Sr : nullptr, n ? zr : nullptr, n ? Slr : nullptr,
                            n ? zlr : nullptr, Y, Sr, zr, Slr, zlr, w.inner, g.inner, s));
      const bool next = r + 1 < layers;
      STACK_LAUNCH((next ? 4 : 3) * sb, k_residual_norm<T><<<nrb(rows, d), kRowThreads, 0, s>>>(
                                            X, Y, X2, next ? U : nullptr, d, scale, rows));
      ST_TRY(cudaGetLastError());
      T* t = X;
      X = X2;
      X2 = t;
    }
    ST_TRY(scatter(X, y, g, p.L, d, a, b, s));
  }
  return SLIM_OK;
}

template <typename T>
slim_status bwd_impl(const Problem& p, int layers, const T* x, const float* omegas, const T* dy,
                     const float* S_state, const float* z_state, const float* S_lo,
                     const float* z_lo, T* dx, float* domegas, void* workspace, cudaStream_t s) {
  const Geo g = geometry(p, layers);
  Carver cv(workspace);
  uint8_t* xin[65];
  uint8_t* yo[64];
  const Ws w = carve(cv, p, g, true, xin, yo);
  const int d = p.d, M = p.M;
  const size_t S = (size_t)layers * g.st, Z = (size_t)layers * g.zt;
  // running states start at the final states B^(N) (value/error pairs)
  ST_TRY(cudaMemcpyAsync(w.Sb, S_state, S * 4, cudaMemcpyDeviceToDevice, s));
  ST_TRY(cudaMemcpyAsync(w.zb, z_state, Z * 4, cudaMemcpyDeviceToDevice, s));
  if (S_lo) ST_TRY(cudaMemcpyAsync(w.Slb, S_lo, S * 4, cudaMemcpyDeviceToDevice, s));
  else ST_TRY(cudaMemsetAsync(w.Slb, 0, S * 4, s));
  if (z_lo) ST_TRY(cudaMemcpyAsync(w.zlb, z_lo, Z * 4, cudaMemcpyDeviceToDevice, s));
  else ST_TRY(cudaMemsetAsync(w.zlb, 0, Z * 4, s));
  if (domegas) ST_TRY(cudaMemsetAsync(domegas, 0, (size_t)layers * M * d * 4, s));
  float *G = w.G, *gz = w.gz, *G2 = w.G2, *gz2 = w.gz2;
  const float scale = powf((float)d, -0.25f);
  T* U = reinterpret_cast<T*>(w.u);
  for (int n = g.N - 1; n >= 0; --n) {
    const int a = n * g.Cs, b = (p.L - a < g.Cs) ? p.L - a : g.Cs;
    const long long rows = (long long)g.chains * b;
    const double sb = (double)rows * d * g.esz;
    ST_TRY(gather(x, w.xin[0], g, p.L, d, a, b, s));
    STACK_LAUNCH(2 * sb, k_rownorm<T><<<nrb(rows, d), kRowThreads, 0, s>>>(
                             reinterpret_cast<const T*>(w.xin[0]), U, d, scale, rows));
    ST_TRY(cudaGetLastError());
    // recompute the slice layer by layer, rolling each layer's state back
    for (int r = 0; r < layers; ++r) {
      const T* X = reinterpret_cast<const T*>(w.xin[r]);
      const float* om = omegas ? omegas + (size_t)r * M * d : nullptr;
      float* Sb = w.Sb + r * g.st;
      float* zb = w.zb + r * g.zt;
      float* Slb = w.Slb + r * g.st;
      float* zlb = w.zlb + r * g.zt;
      // the state at the slice's end, for the layer's backward
      ST_TRY(cudaMemcpyAsync(w.Se + r * g.st, Sb, g.st * 4, cudaMemcpyDeviceToDevice, s));
      ST_TRY(cudaMemcpyAsync(w.ze + r * g.zt, zb, g.zt * 4, cudaMemcpyDeviceToDevice, s));
      ST_TRY(cudaMemcpyAsync(w.Sle + r * g.st, Slb, g.st * 4, cudaMemcpyDeviceToDevice, s));
      ST_TRY(cudaMemcpyAsync(w.zle + r * g.zt, zlb, g.zt * 4, cudaMemcpyDeviceToDevice, s));
      // eq. 17: B_r -= the slice's sum of T_l (its own contribution, from zero)
      ST_CALL(slim_fwd_from(U, U, U, om, p.B, p.H, b, d, M, b, p.dtype, p.feature, nullptr,
                            nullptr, nullptr, nullptr, w.scratch_y, w.dS, w.dz, w.dSl, w.dzl,
                            w.inner, g.inner, s));
      STACK_LAUNCH(24.0 * g.st, k_pair_sub<<<nb(g.st), 256, 0, s>>>(Sb, Slb, w.dS, w.dSl, (long long)g.st));
      STACK_LAUNCH(24.0 * g.zt, k_pair_sub<<<nb(g.zt), 256, 0, s>>>(zb, zlb, w.dz, w.dzl, (long long)g.zt));
      ST_TRY(cudaGetLastError());
      // the layer's output on the slice from the rolled-back state
      T* Y = reinterpret_cast<T*>(w.yout[r]);
      ST_CALL(slim_fwd_from(U, U, U, om, p.B, p.H, b, d, M, b, p.dtype, p.feature, Sb, zb, Slb,
                            zlb, Y, w.Ssc, w.zsc, nullptr, nullptr, w.inner, g.inner, s));
      // the next layer's input and its u; the top layer's output is not needed
      if (r + 1 < layers) {
        STACK_LAUNCH(4 * sb, k_residual_norm<T><<<nrb(rows, d), kRowThreads, 0, s>>>(
                                 X, Y, reinterpret_cast<T*>(w.xin[r + 1]), U, d, scale, rows));
        ST_TRY(cudaGetLastError());
      }
    }
    // back through the layers: dX^(r-1) = dX^(r) + u'(X^(r-1))^T (dq + dk + dv);
    // the top layer's upstream gradient is the slice's dy
    ST_TRY(gather(dy, w.dout, g, p.L, d, a, b, s));
    for (int r = layers - 1; r >= 0; --r) {
      const T* X = reinterpret_cast<const T*>(w.xin[r]);
      const float* om = omegas ? omegas + (size_t)r * M * d : nullptr;
      if (r + 1 < layers) {  // the top layer's u is still in place from the recompute
        STACK_LAUNCH(2 * sb, k_rownorm<T><<<nrb(rows, d), kRowThreads, 0, s>>>(X, U, d, scale, rows));
        ST_TRY(cudaGetLastError());
      }
      ST_CALL(slim_bwd_from(U, U, U, om, w.yout[r], w.dout, w.Se + r * g.st, w.ze + r * g.zt,
                            w.Sle + r * g.st, w.zle + r * g.zt, n + 1 < g.N ? G + r * g.st : nullptr,
                            n + 1 < g.N ? gz + r * g.zt : nullptr, p.B, p.H, b, d, M, b, p.dtype,
                            p.feature, w.dq, w.dk, w.dv, domegas ? w.dom : nullptr,
                            G2 + r * g.st, gz2 + r * g.zt, w.inner, g.inner, s));
      if (domegas) {
        STACK_LAUNCH(12.0 * M * d, k_add<<<nb((long long)M * d), 256, 0, s>>>(
                                       domegas + (size_t)r * M * d, w.dom, (long long)M * d));
        ST_TRY(cudaGetLastError());
      }
      const bool first = r == layers - 1;
      STACK_LAUNCH((double)rows * d * (6.0 * g.esz + (first ? 4 : 8)),
                   k_dx_accum<T><<<nrb(rows, d), kRowThreads, 0, s>>>(
                       w.dx, X, reinterpret_cast<const T*>(w.dq), reinterpret_cast<const T*>(w.dk),
                       reinterpret_cast<const T*>(w.dv), reinterpret_cast<T*>(w.dout), d, scale,
                       rows, first ? 1 : 0));
      ST_TRY(cudaGetLastError());
    }
    // dout now holds dX^(0) of the slice, rounded to the dtype
    ST_TRY(scatter(w.dout, dx, g, p.L, d, a, b, s));
    float* t = G; G = G2; G2 = t;
    t = gz; gz = gz2; gz2 = t;
  }
  return SLIM_OK;
}

}  // namespace

size_t workspace_bytes(const Problem& p, int layers, bool bwd) {
  const Geo g = geometry(p, layers);
  Carver cv(nullptr);
  uint8_t* xin[65];
  uint8_t* yo[64];
  carve(cv, p, g, bwd, xin, yo);
  return cv.bytes();
}

slim_status fwd(const Problem& p, int layers, const void* x, const float* omegas, void* y,
                float* S_state, float* z_state, float* S_lo, float* z_lo, void* workspace,
                cudaStream_t s) {
  if (p.dtype == SLIM_BF16)
    return fwd_impl<__nv_bfloat16>(p, layers, (const __nv_bfloat16*)x, omegas, (__nv_bfloat16*)y,
                                   S_state, z_state, S_lo, z_lo, workspace, s);
  return fwd_impl<float>(p, layers, (const float*)x, omegas, (float*)y, S_state, z_state, S_lo,
                         z_lo, workspace, s);
}

slim_status bwd(const Problem& p, int layers, const void* x, const float* omegas, const void* dy,
                const float* S_state, const float* z_state, const float* S_lo,
                const float* z_lo, void* dx, float* domegas, void* workspace, cudaStream_t s) {
  if (p.dtype == SLIM_BF16)
    return bwd_impl<__nv_bfloat16>(p, layers, (const __nv_bfloat16*)x, omegas,
                                   (const __nv_bfloat16*)dy, S_state, z_state, S_lo, z_lo,
                                   (__nv_bfloat16*)dx, domegas, workspace, s);
  return bwd_impl<float>(p, layers, (const float*)x, omegas, (const float*)dy, S_state, z_state,
                         S_lo, z_lo, (float*)dx, domegas, workspace, s);
}

}  // namespace stack
}  // namespace slim
