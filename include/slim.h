/*
 * libslim -- sliced causal linear (Performer) attention, forward and backward,
 * on one NVIDIA GB300 (sm_103a).
 *
 * The operation is the causal linear self-attention of eq. 2 of "Sub-Linear
 * Memory: How to Make Performers SLiM" (arXiv 2012.11346), for B*H
 * independent chains (batch x head):
 *
 *     out_i = sum_{j<=i} (g(q_i).g(k_j)) v_j  /  sum_{j<=i} g(q_i).g(k_j)
 *
 * evaluated the way Algorithm 1 prescribes: the sequence is cut into
 * N = ceil(L/C) slices of C rows (Sec. 3.2, the last slice may be shorter),
 * and only the prefix state B^(n) = (S, z) is carried from slice to slice:
 *
 *     S = sum_j g(k_j) v_j^T   ([M, d], the transpose of the paper's R, eq. 3)
 *     z = sum_j g(k_j)         ([M],    the paper's S, eq. 3)
 *
 * The backward pass walks the slices in reverse (Sec. 3.3): it recomputes
 * each slice, rolls the state back by subtraction (eq. 17) and carries the
 * state gradient G^(n) (eq. 18).  Memory beyond inputs and outputs is the
 * caller-provided workspace, whose size grows with C, not with L.
 *
 * Feature maps g: R^d -> R_+^M (Omega is [M, d], shared by all chains):
 *     SLIM_FEAT_EXP    : g(x)_m = exp(omega_m.x - |x|^2/2) / sqrt(M)   (FAVOR+)
 *     SLIM_FEAT_RELU   : g(x)_m = max(omega_m.x, 0) / sqrt(M), ReLU'(0) = 0
 *     SLIM_FEAT_SQUARE : g(x)_i = x_i^2, M = d -- the elementwise map of the
 *                        paper's experiments (Sec. 4).  Omega is not used (it
 *                        may be NULL) and dOmega is zero (domega may be NULL).
 * A row whose denominator is exactly 0 (possible with the ReLU map, and with
 * the quadratic map for all-zero inputs) gets output 0 and passes no
 * gradient.
 *
 * Conventions for every entry point
 *   - All tensor pointers are DEVICE pointers, contiguous, row-major, 16-byte
 *     aligned, and non-null -- except that when L = 0 the (empty) [B, H, L, d]
 *     tensors may be null.  q, k, v, out, dout, dq, dk, dv are [B, H, L, d] in `dtype`;
 *     omega and domega are [M, d] fp32; S_state is [B, H, M, d] fp32 and
 *     z_state is [B, H, M] fp32.
 *   - The caller owns every buffer, and the library allocates no device
 *     memory.  It never synchronises the device; all work is enqueued on
 *     `stream` (a cudaStream_t passed as void*; NULL is the legacy default
 *     stream).  Inputs must not be modified until that work completes, and a
 *     workspace serves one call at a time.
 *   - Arguments are validated before anything is enqueued.  On any error
 *     nothing has been launched, except SLIM_ERR_CUDA (a launch failed part
 *     way; outputs are then undefined).
 *   - Device-side waits (only the tensor-core kernels have any) are bounded
 *     (about a second).  A wait that gives up makes its call leave early
 *     (outputs undefined) and is reported as SLIM_ERR_TIMEOUT by the next
 *     slim_fwd / slim_bwd / *_from call on the same workspace once the failed
 *     work has finished, without blocking: that call then launches nothing.
 *     For this the library pins and maps, on the first tensor-core call in a
 *     process, one 4 KB page of its own static host memory
 *     (cudaHostRegister), where the kernels count such failures; the call's
 *     first kernel stores the counter's address in the workspace, so the
 *     report adds no copy and no launch.  slim_check_device_error reads the
 *     same failure by blocking instead.
 *   - A workspace's first 4 bytes are its device error word.  Every call
 *     clears it when it starts; a bounded wait that gives up sets it.
 *   - 1 <= C; C > L behaves as C = L.  L % C != 0 gives a shorter last slice.
 *   - Outputs are written in `dtype` rounded to nearest even.  The state
 *     carried between slices depends on the kernels serving the problem (see
 *     slim_path_for).  The fp32-compute kernels carry it as an fp32
 *     value/error pair (TwoSum) and accumulate the contractions in fp32
 *     FMA; their residual outputs (S_state_lo, z_state_lo) hold the pair's
 *     low part.
 *     The tensor-core kernels (bf16) chain plain fp32 prefixes from tile to
 *     tile, accumulate in fp32, and write zero residuals.
 *   - Supported: d in {16, 32, 64, 128}; M a multiple of 16 in [16, 256];
 *     dtype SLIM_F32 or SLIM_BF16; every feature map.  Other combinations
 *     return SLIM_ERR_UNSUPPORTED.
 */
#ifndef SLIM_H_
#define SLIM_H_

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SLIM_OK = 0,
  SLIM_ERR_INVALID_ARG = 1,   /* null/misaligned pointer, bad size, C < 1 ... */
  SLIM_ERR_UNSUPPORTED = 2,   /* valid but unsupported (d, M, dtype, feature) */
  SLIM_ERR_WORKSPACE = 3,     /* workspace pointer null or too small          */
  SLIM_ERR_CUDA = 4,          /* a CUDA launch or runtime call failed          */
  SLIM_ERR_TIMEOUT = 5        /* a bounded device-side wait gave up            */
} slim_status;

typedef enum { SLIM_F32 = 0, SLIM_BF16 = 1 } slim_dtype;
typedef enum { SLIM_FEAT_EXP = 0, SLIM_FEAT_RELU = 1, SLIM_FEAT_SQUARE = 2 } slim_feature;

/* Human-readable name of a status code (static storage, never NULL). */
const char* slim_status_string(slim_status status);

/* Library version as MAJOR*10000 + MINOR*100 + PATCH. */
int slim_version(void);

/*
 * Workspace bytes needed by slim_fwd / slim_bwd for this problem.  Pure host
 * computation (no CUDA call).  The size grows linearly with min(C, L) and with
 * B*H, and does not depend on L otherwise (Sec. 3.4: O(C) memory).
 * Returns SLIM_ERR_INVALID_ARG / SLIM_ERR_UNSUPPORTED as the entry points
 * would; *bytes is written only on SLIM_OK.
 */
slim_status slim_fwd_workspace_size(int B, int H, int L, int d, int M, int C,
                                    slim_dtype dtype, slim_feature feature,
                                    size_t* bytes);
slim_status slim_bwd_workspace_size(int B, int H, int L, int d, int M, int C,
                                    slim_dtype dtype, slim_feature feature,
                                    size_t* bytes);

/*
 * Forward sweep of Algorithm 1 (Sec. 3.2, eqs. 14-16) for one causal
 * linear-attention layer.
 *   q, k, v   [B,H,L,d] dtype, read-only.
 *   omega     [M,d] fp32, read-only; the random-feature matrix of g.
 *   out       [B,H,L,d] dtype, written: eq. 2 for every row.
 *   S_state   [B,H,M,d] fp32, written: final state S^(N) = sum_j g(k_j) v_j^T.
 *   z_state   [B,H,M]   fp32, written: final state z^(N) = sum_j g(k_j).
 *   S_state_lo, z_state_lo  same shapes, written if non-NULL: the low-order
 *             residual of the carried fp32 value/error pair (state = S_state +
 *             S_state_lo to about 48 bits; zero from the tensor-core kernels).
 *             Passing them back to slim_bwd lets the rollback of eq. 17 start
 *             from the unrounded state.  For fp32 problems they are part of
 *             the 1e-5 accuracy: an fp32-rounded z^(N) alone perturbs the
 *             early rows' denominators, which are small next to z^(N), by
 *             ~6e-8 * z^(N), and on long sequences that moves dq by about
 *             2e-5 (rel-L2; B4 H12 L8192 d64 M128, ReLU map).
 *   workspace device scratch of at least slim_fwd_workspace_size() bytes,
 *             256-byte aligned; contents on entry are ignored.
 * L = 0 is valid and only zeroes S_state / z_state.
 */
slim_status slim_fwd(const void* q, const void* k, const void* v, const float* omega,
                     int B, int H, int L, int d, int M, int C,
                     slim_dtype dtype, slim_feature feature,
                     void* out, float* S_state, float* z_state,
                     float* S_state_lo, float* z_state_lo,
                     void* workspace, size_t workspace_bytes, void* stream);

/*
 * Backward sweep of Algorithm 1 (Sec. 3.3, eqs. 17-18): the vector-Jacobian
 * product of eq. 2 for the upstream gradient dout, i.e. the gradients of
 * <dout, out> with respect to q, k, v and omega.
 *   q, k, v, omega  as for slim_fwd, read-only.
 *   out        [B,H,L,d] dtype, read-only: the output slim_fwd returned.
 *   dout       [B,H,L,d] dtype, read-only: upstream gradient.
 *   S_state, z_state  read-only: the final state B^(N) slim_fwd returned; the
 *              reverse walk starts from it and rolls it back slice by slice.
 *              Not modified, so a second call gives the same result.
 *   S_state_lo, z_state_lo  read-only, may be NULL (then taken as zero): the
 *              residuals slim_fwd wrote.
 *   dq, dk, dv [B,H,L,d] dtype, written.
 *   domega     [M,d] fp32, written (sum over all chains, queries and keys).
 *   workspace  at least slim_bwd_workspace_size() bytes, 256-byte aligned.
 * The same C as the forward is expected; any C gives the same result in exact
 * arithmetic (Sec. 4.2), differing only by rounding.
 */
slim_status slim_bwd(const void* q, const void* k, const void* v, const float* omega,
                     const void* out, const void* dout,
                     const float* S_state, const float* z_state,
                     const float* S_state_lo, const float* z_state_lo,
                     int B, int H, int L, int d, int M, int C,
                     slim_dtype dtype, slim_feature feature,
                     void* dq, void* dk, void* dv, float* domega,
                     void* workspace, size_t workspace_bytes, void* stream);

/*
 * A sequence cut into segments, one call per segment (streaming).  The slice
 * recurrence of Sec. 3.2 carries B^(n-1) into slice n (eq. 16), and the
 * reverse sweep of Sec. 3.3 carries the state gradient G^(n) back into slice
 * n (eq. 18, G^(N) = 0 only at the true end of the sequence).  These two
 * entry points expose both carries at the ends of a call, so that calls on
 * consecutive segments give the result of one call on the whole sequence:
 *
 *   slim_fwd_from: slim_fwd starting from the state B^(0) = (S_init, z_init)
 *     instead of zero -- typically the S_state / z_state (and residuals) an
 *     earlier segment's forward returned.  S_init [B,H,M,d] and z_init
 *     [B,H,M] fp32, read-only, both NULL (zero state) or both given;
 *     S_init_lo / z_init_lo optional residuals (NULL: zero), only with
 *     S_init.  The outputs may alias the inputs (S_state == S_init updates a
 *     running state in place).  The S_state it returns is the state after
 *     the segment, including B^(0).
 *
 *   slim_bwd_from: slim_bwd with the incoming state gradient G^(N) =
 *     (G_S_in [B,H,M,d], g_z_in [B,H,M] fp32, read-only; both NULL for zero)
 *     -- the gradient of the later segments' loss with respect to this
 *     segment's final state, i.e. the G_S_out / g_z_out of the later
 *     segment's slim_bwd_from -- and returning G^(0) in G_S_out / g_z_out
 *     (written if non-NULL, both or neither): the gradient with respect to
 *     the state this segment started from, to hand to the previous segment.
 *     S_state / z_state are this segment's final state as its slim_fwd_from
 *     returned it; the rollback ends at this segment's B^(0).  The dOmega of
 *     the segments add up to the whole sequence's.
 *
 * With all the extra pointers NULL they are slim_fwd and slim_bwd.
 */
slim_status slim_fwd_from(const void* q, const void* k, const void* v, const float* omega,
                          int B, int H, int L, int d, int M, int C,
                          slim_dtype dtype, slim_feature feature,
                          const float* S_init, const float* z_init,
                          const float* S_init_lo, const float* z_init_lo,
                          void* out, float* S_state, float* z_state,
                          float* S_state_lo, float* z_state_lo,
                          void* workspace, size_t workspace_bytes, void* stream);
slim_status slim_bwd_from(const void* q, const void* k, const void* v, const float* omega,
                          const void* out, const void* dout,
                          const float* S_state, const float* z_state,
                          const float* S_state_lo, const float* z_state_lo,
                          const float* G_S_in, const float* g_z_in,
                          int B, int H, int L, int d, int M, int C,
                          slim_dtype dtype, slim_feature feature,
                          void* dq, void* dk, void* dv, float* domega,
                          float* G_S_out, float* g_z_out,
                          void* workspace, size_t workspace_bytes, void* stream);

/*
 * The non-causal (bidirectional) form: eq. 2 without the causal mask, every
 * row reading every key,
 *     out_i = sum_j (g(q_i).g(k_j)) v_j / sum_j g(q_i).g(k_j),   j = 1..L,
 * so that one global state B = (S, z) (eq. 3 at the last row) serves every
 * row.  The paper treats the causal form; this is the same computation with
 * the prefix sums replaced by the full sum, with memory kept O(C) the same
 * way: the forward reads the slices twice (accumulate B, then read it out)
 * and the backward reads them twice (query side, accumulating the state
 * gradient G, then key/value side, reading G).  It runs on the fp32-compute
 * kernels for every supported problem.
 *   slim_bidir_workspace_size: workspace bytes (backward != 0: the backward's).
 *   slim_fwd_bidir: out and the global state S_state / z_state (written).
 *   slim_bwd_bidir: gradients of <dout, out>; S_state / z_state as
 *     slim_fwd_bidir returned them (read-only).
 * Arguments, layouts and errors as for slim_fwd / slim_bwd (the quadratic map
 * again needs no omega and writes no domega).  No device-side waits.
 */
slim_status slim_bidir_workspace_size(int B, int H, int L, int d, int M, int C,
                                      slim_dtype dtype, slim_feature feature, int backward,
                                      size_t* bytes);
slim_status slim_fwd_bidir(const void* q, const void* k, const void* v, const float* omega,
                           int B, int H, int L, int d, int M, int C,
                           slim_dtype dtype, slim_feature feature,
                           void* out, float* S_state, float* z_state,
                           void* workspace, size_t workspace_bytes, void* stream);
slim_status slim_bwd_bidir(const void* q, const void* k, const void* v, const float* omega,
                           const void* out, const void* dout,
                           const float* S_state, const float* z_state,
                           int B, int H, int L, int d, int M, int C,
                           slim_dtype dtype, slim_feature feature,
                           void* dq, void* dk, void* dv, float* domega,
                           void* workspace, size_t workspace_bytes, void* stream);

/*
 * A stack of `layers` (s) causal linear-attention layers with residual
 * connections, run the memory-efficient way of Algorithm 1 (Sec. 3.2-3.3):
 * the slices in the outer loop, the layers in the inner loop, one carried
 * state per layer (B is s x D1), and the reverse sweep of Algorithm 2 with a
 * rollback (eq. 17) and a state gradient (eq. 18) per layer.  Layer r maps
 * each row x of its input to q = k = v = u(x) = d^(-1/4) x / sqrt(mean(x^2)
 * + 1e-6) -- a parameter-free row normalisation standing in for the layer
 * norm of the paper's model (Sec. 2.2, eqs. 5-6), keeping every layer's features at the scale of
 * one layer's inputs -- runs attention with its own random-feature matrix
 * Omega_r (the F of Sec. 3.1) and adds its output back (the G):
 *     X^(r) = X^(r-1) + Att_r(u, u, u),   r = 1..s,   out: X^(s).
 * Each (slice, layer) step runs as one slim_fwd_from / slim_bwd_from call on
 * the slice's rows, gathered into the workspace.  Memory beyond inputs and
 * outputs: one slice's activations per layer, the per-layer states and state
 * gradients, and one segment call's workspace (O(C * s), not O(L)).
 *   x          [B,H,L,d] dtype: X^(0).  y: [B,H,L,d] dtype, written: X^(s).
 *   omegas     [layers][M][d] fp32 (may be NULL for the quadratic map).
 *   S_state, z_state  [layers][B,H,M,d], [layers][B,H,M] fp32: written by
 *              slim_stack_fwd (each layer's final state), read by
 *              slim_stack_bwd; S_state_lo / z_state_lo the residuals (both or
 *              neither), as for slim_fwd.
 *   dy         [B,H,L,d] dtype: the upstream gradient of X^(s).
 *   dx         [B,H,L,d] dtype, written: the gradient of <dy, X^(s)> w.r.t. x.
 *   domegas    [layers][M][d] fp32, written (NULL allowed for the quadratic map).
 *   layers     1 .. 64.  Workspace: slim_stack_workspace_size (backward != 0
 *              for slim_stack_bwd), 256-byte aligned; its first word is the
 *              device error word, as for slim_fwd.
 * Errors as for slim_fwd / slim_bwd.
 */
slim_status slim_stack_workspace_size(int B, int H, int L, int d, int M, int C, int layers,
                                      slim_dtype dtype, slim_feature feature, int backward,
                                      size_t* bytes);
slim_status slim_stack_fwd(const void* x, const float* omegas,
                           int B, int H, int L, int d, int M, int C, int layers,
                           slim_dtype dtype, slim_feature feature,
                           void* y, float* S_state, float* z_state,
                           float* S_state_lo, float* z_state_lo,
                           void* workspace, size_t workspace_bytes, void* stream);
slim_status slim_stack_bwd(const void* x, const float* omegas, const void* dy,
                           const float* S_state, const float* z_state,
                           const float* S_state_lo, const float* z_state_lo,
                           int B, int H, int L, int d, int M, int C, int layers,
                           slim_dtype dtype, slim_feature feature,
                           void* dx, float* domegas,
                           void* workspace, size_t workspace_bytes, void* stream);

/*
 * Which kernels serve this problem: *path = 1 for the tensor-core path
 * (tcgen05 MMAs, bf16 operands, fp32 accumulation; bf16 inputs with d = 64,
 * M in {128, 256} and slices of at least 64 rows), 0 for the fp32-compute
 * path (every other supported problem).  Setting the environment variable
 * SLIM_PATH=simt (read on every call) selects the fp32-compute path for every
 * problem.  Pure host computation.
 */
slim_status slim_path_for(int B, int H, int L, int d, int M, int C, slim_dtype dtype,
                          slim_feature feature, int* path);

/*
 * The order in which the tensor-core backward (one launch, Algorithm 1's
 * reverse sweep) hands out its work items; a pure host computation, for
 * inspecting and testing that order (no counterpart in the paper).  Ticket x
 * names item (role, slice, index), written to items[3x], items[3x+1],
 * items[3x+2] for x < min(*count, cap):
 *   role 0: tile index of the slice, dq part then dk/dv part in one CTA
 *           (tiles last first, chains inside a position: tile
 *           ntn-1-index/(B*H) of chain index%(B*H)),
 *   role 2: final dOmega reduction, stage 1 CTA index (slice 0),
 *   role 3: final dOmega reduction, stage 2 CTA index (slice 0).
 * *count receives the number of items.  items may be null when cap is 0.
 * *ring (when ring is not null) receives R, the slots of the ring through
 * which a tile's dq part hands its results to its dk/dv part (slot n % R;
 * slice n-R's tile at the same position waits until slice n's has read it).
 * Returns SLIM_ERR_UNSUPPORTED for problems the tensor-core path does not
 * take (see slim_path_for) and for L = 0.
 */
slim_status slim_bwd_schedule(int B, int H, int L, int d, int M, int C, slim_dtype dtype,
                              slim_feature feature, int* items, int cap, int* count,
                              int* ring);

/*
 * Reads the device error word that bounded waits in the kernels set when they
 * give up, and clears it.  Copies 4 bytes from the workspace on `stream` and
 * synchronises that stream (this call, unlike the others, blocks).  A failure
 * it reports is not reported again by the next call on the workspace.
 * Returns SLIM_OK, SLIM_ERR_TIMEOUT, or SLIM_ERR_CUDA.
 */
slim_status slim_check_device_error(void* workspace, void* stream);

/*
 * Launch accounting and per-kernel timing (a host-side runtime feature for
 * benchmarking; no counterpart in the paper).  Process-global, not
 * thread-safe.
 *
 * slim_launch_count: number of libslim kernel launches since load.
 * slim_profiler_enable(1): from now on every libslim kernel launch is
 *   bracketed by two CUDA events recorded on its stream; each launch site also
 *   tallies the algorithmic FLOPs and HBM bytes of the launch.
 * slim_profiler_read: waits for the recorded events, folds them into
 *   per-kernel totals and writes up to `cap` entries (one per kernel that ran);
 *   returns the number of entries, or -1 on a CUDA error.
 * slim_profiler_reset: drops all records and totals.
 */
typedef struct {
  char name[48];
  unsigned long long launches;
  double total_ms;  /* summed CUDA-event durations of the recorded launches */
  double flops;     /* algorithmic floating-point operations of those launches */
  double bytes;     /* algorithmic HBM bytes (reads + writes) of those launches */
} slim_kernel_stats;

unsigned long long slim_launch_count(void);
void slim_profiler_enable(int on);
void slim_profiler_reset(void);
int slim_profiler_read(slim_kernel_stats* stats, int cap);

/*
 * Diagnostic of the tensor-core building blocks (no counterpart in the
 * paper): one CTA computes D = A x B with a single chain of tcgen05 MMAs,
 * the operands staged in 128-byte-swizzled shared memory in K-major (0) or
 * MN-major (1) layout, so a caller can compare D against a reference.
 *   A  [128, K] bf16 row-major device; B [K, N] bf16 row-major device;
 *   D  [128, N] fp32 row-major device (written); err: device int, set to 1 if
 *   the MMA completion wait gave up.  K, N in {64, 128, 256}.
 */
slim_status slim_tc_selftest(int a_mn, int b_mn, int K, int N, const void* A, const void* B,
                             float* D, int* err, void* stream);

/*
 * Diagnostic of the failure path (no counterpart in the paper): one warp
 * waits on an mbarrier that nothing arrives at.  The wait gives up after its
 * time limit (about a second), sets the error word at the start of
 * `workspace` (a workspace as passed to slim_fwd/slim_bwd, at least 256
 * bytes) and the kernel returns.  Like slim_fwd/slim_bwd it takes part in the
 * non-blocking report: once the kernel has finished, the next slim_fwd /
 * slim_bwd on the same workspace returns SLIM_ERR_TIMEOUT (and launches
 * nothing), or slim_check_device_error reports it by blocking.  Nothing
 * faults and the context stays usable.
 */
slim_status slim_diag_wait_timeout(void* workspace, void* stream);

/*
 * Allocation-free forward (the paper has no counterpart; this is for callers
 * that cannot allocate device memory).  Some callers cannot call cudaMalloc or
 * any allocating routine where they run the forward -- code inside an
 * allocator or memory-pool callback, hosts that fix their device memory at
 * start-up, plug-ins whose host owns every allocation.  slim_fwd_noalloc is
 * slim_fwd with the workspace replaced by a scratch array that the library
 * itself reserves in device memory: SLIM_NOALLOC_SCRATCH_BYTES (16 MiB) on
 * every GPU that loads the library, held until the process exits.  The caller
 * still passes every input and output (same arguments and rules as slim_fwd,
 * minus the workspace).
 *   - Allocates nothing: no cudaMalloc, cudaFree or other allocating call
 *     (keep the launch profiler off, it creates CUDA events when on), and it
 *     does not take part in the non-blocking timeout report (which pins a
 *     host page on first use).
 *   - CUDA loads a library's device code on a device lazily, and that load
 *     reserves the array: the first libslim call that reaches a device does
 *     it.  Make a first call on each device at start-up, outside any context
 *     that must not allocate (and before any stream capture on the device).
 *   - Returns SLIM_ERR_WORKSPACE when the problem needs more scratch than
 *     SLIM_NOALLOC_SCRATCH_BYTES (compare slim_fwd_workspace_size); use
 *     slim_fwd with a caller workspace, or a smaller C or B*H, then.
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current.
 *   - All calls share the one array and it keeps the last call's contents;
 *     the call clears, on its stream, what must start at zero.  Calls that
 *     overlap on the GPU (different streams, or several host threads) race
 *     on the array and give wrong results: order them on one stream.
 */
#define SLIM_NOALLOC_SCRATCH_BYTES (16u * 1024u * 1024u)
slim_status slim_fwd_noalloc(const void* q, const void* k, const void* v, const float* omega,
                             int B, int H, int L, int d, int M, int C,
                             slim_dtype dtype, slim_feature feature,
                             void* out, float* S_state, float* z_state,
                             float* S_state_lo, float* z_state_lo, void* stream);

#ifdef __cplusplus
}
#endif

#endif  /* SLIM_H_ */
