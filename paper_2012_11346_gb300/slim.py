"""Python binding of libslim (ctypes): argument marshalling only.

Every computation runs in the CUDA kernels behind the C ABI declared in
include/slim.h.  PyTorch supplies device memory (outputs and workspace, so
torch.cuda.max_memory_allocated sees all of it) and the current stream.  There
is no CPU fallback: if libslim.so is missing or no GPU is present, the calls
raise.
"""
import ctypes
import os

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libslim.so")
_lib = None

DTYPES = {torch.float32: 0, torch.bfloat16: 1}
FEATURES = {"exp": 0, "relu": 1, "square": 2}
STATUS = {0: "SLIM_OK", 1: "SLIM_ERR_INVALID_ARG", 2: "SLIM_ERR_UNSUPPORTED",
          3: "SLIM_ERR_WORKSPACE", 4: "SLIM_ERR_CUDA", 5: "SLIM_ERR_TIMEOUT"}

_i, _p, _sz = ctypes.c_int, ctypes.c_void_p, ctypes.c_size_t

# (name, argtypes) for every symbol of include/slim.h
SIGNATURES = {
    "slim_status_string": ([_i], ctypes.c_char_p),
    "slim_version": ([], _i),
    "slim_fwd_workspace_size": ([_i] * 6 + [_i, _i, ctypes.POINTER(_sz)], _i),
    "slim_bwd_workspace_size": ([_i] * 6 + [_i, _i, ctypes.POINTER(_sz)], _i),
    "slim_fwd": ([_p] * 4 + [_i] * 6 + [_i, _i] + [_p] * 5 + [_p, _sz, _p], _i),
    "slim_bwd": ([_p] * 10 + [_i] * 6 + [_i, _i] + [_p] * 4 + [_p, _sz, _p], _i),
    "slim_fwd_from": ([_p] * 4 + [_i] * 6 + [_i, _i] + [_p] * 4 + [_p] * 5 + [_p, _sz, _p], _i),
    "slim_bwd_from": ([_p] * 12 + [_i] * 6 + [_i, _i] + [_p] * 4 + [_p] * 2 + [_p, _sz, _p], _i),
    "slim_bidir_workspace_size": ([_i] * 6 + [_i, _i, _i, ctypes.POINTER(_sz)], _i),
    "slim_fwd_bidir": ([_p] * 4 + [_i] * 6 + [_i, _i] + [_p] * 3 + [_p, _sz, _p], _i),
    "slim_bwd_bidir": ([_p] * 8 + [_i] * 6 + [_i, _i] + [_p] * 4 + [_p, _sz, _p], _i),
    "slim_stack_workspace_size": ([_i] * 7 + [_i, _i, _i, ctypes.POINTER(_sz)], _i),
    "slim_stack_fwd": ([_p] * 2 + [_i] * 7 + [_i, _i] + [_p] * 5 + [_p, _sz, _p], _i),
    "slim_stack_bwd": ([_p] * 7 + [_i] * 7 + [_i, _i] + [_p] * 2 + [_p, _sz, _p], _i),
    "slim_check_device_error": ([_p, _p], _i),
    "slim_launch_count": ([], ctypes.c_ulonglong),
    "slim_profiler_enable": ([_i], None),
    "slim_profiler_reset": ([], None),
    "slim_profiler_read": ([_p, _i], _i),
    "slim_tc_selftest": ([_i, _i, _i, _i, _p, _p, _p, _p, _p], _i),
    "slim_path_for": ([_i] * 6 + [_i, _i, ctypes.POINTER(_i)], _i),
    "slim_bwd_schedule": ([_i] * 6 + [_i, _i, _p, _i, ctypes.POINTER(_i), ctypes.POINTER(_i)],
                          _i),
    "slim_fwd_noalloc": ([_p] * 4 + [_i] * 6 + [_i, _i] + [_p] * 5 + [_p], _i),
    "slim_diag_wait_timeout": ([_p, _p], _i),
}


class KernelStats(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 48), ("launches", ctypes.c_ulonglong),
                ("total_ms", ctypes.c_double), ("flops", ctypes.c_double),
                ("bytes", ctypes.c_double)]


class SlimError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__(f"{where}: {status_string(status)}")


def library():
    """Loads libslim.so (built by paper_2012_11346_gb300.build); raises if absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"libslim.so not built ({_LIB_PATH}); run "
                               "python -m paper_2012_11346_gb300.build")
        lib = ctypes.CDLL(_LIB_PATH)
        for name, (args, res) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = res
        _lib = lib
    return _lib


def status_string(status):
    return library().slim_status_string(int(status)).decode()


def _check(status, where):
    if status != 0:
        raise SlimError(status, where)


def _dims(q, omega):
    B, H, L, d = q.shape
    M = omega.shape[0] if omega is not None else d
    return B, H, L, d, M


def workspace_size(B, H, L, d, M, C, dtype, feature, backward):
    n = _sz(0)
    fn = library().slim_bwd_workspace_size if backward else library().slim_fwd_workspace_size
    _check(fn(B, H, L, d, M, C, DTYPES[dtype], FEATURES[feature], ctypes.byref(n)),
           "workspace_size")
    return n.value


def path_for(B, H, L, d, M, C, dtype, feature):
    """1 if the tensor-core kernels serve this problem, 0 for the fp32 path."""
    r = _i(0)
    _check(library().slim_path_for(B, H, L, d, M, C, DTYPES[dtype], FEATURES[feature],
                                   ctypes.byref(r)), "slim_path_for")
    return r.value


def bwd_schedule(B, H, L, d, M, C, dtype, feature):
    """The tensor-core backward's item order and hand-off ring depth R: a list
    of (role, slice, index) per ticket (roles 0 dq side, 1 dk/dv side, 2 and 3
    the final dOmega reduction stages), and R."""
    lib, n, ring = library(), _i(0), _i(0)
    _check(lib.slim_bwd_schedule(B, H, L, d, M, C, DTYPES[dtype], FEATURES[feature], None, 0,
                                 ctypes.byref(n), None), "slim_bwd_schedule")
    buf = (_i * (3 * n.value))()
    _check(lib.slim_bwd_schedule(B, H, L, d, M, C, DTYPES[dtype], FEATURES[feature], buf, n.value,
                                 ctypes.byref(n), ctypes.byref(ring)), "slim_bwd_schedule")
    return [tuple(buf[3 * x:3 * x + 3]) for x in range(n.value)], ring.value


def _stream_handle(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _workspace(nbytes, device):
    return torch.empty(max(nbytes, 256), dtype=torch.uint8, device=device)


def _require_cuda(*ts):
    for t in ts:
        if not t.is_cuda:
            raise RuntimeError("libslim runs on CUDA tensors only (no CPU fallback)")
        if not t.is_contiguous():
            raise RuntimeError("libslim needs contiguous tensors")


def _ptr(t):
    return None if t is None else t.data_ptr()


def _opt_ptr(t):
    if t is None:
        return None
    _require_cuda(t)
    return t.data_ptr()


def forward(q, k, v, omega, C, feature="exp", workspace=None, stream=None, residuals=False,
            S_init=None, z_init=None, S_init_lo=None, z_init_lo=None):
    """slim_fwd (slim_fwd_from when an initial state is given): returns
    (out, S_state, z_state), or with residuals=True (out, S_state, z_state,
    S_state_lo, z_state_lo) -- the low-order parts of the carried state, which
    slim_bwd uses to start its rollback exactly.  S_init / z_init (and their
    residuals): the state B^(0) the sequence starts from, e.g. the state an
    earlier segment returned.  omega may be None for the quadratic map."""
    _require_cuda(q, k, v)
    B, H, L, d = q.shape
    M = omega.shape[0] if omega is not None else d
    out = torch.empty_like(q)
    S_state = torch.empty(B, H, M, d, dtype=torch.float32, device=q.device)
    z_state = torch.empty(B, H, M, dtype=torch.float32, device=q.device)
    S_lo = torch.empty_like(S_state) if residuals else None
    z_lo = torch.empty_like(z_state) if residuals else None
    need = workspace_size(B, H, L, d, M, C, q.dtype, feature, False)
    ws = workspace if workspace is not None else _workspace(need, q.device)
    args = (q.data_ptr(), k.data_ptr(), v.data_ptr(), _opt_ptr(omega), B, H, L, d, M, C,
            DTYPES[q.dtype], FEATURES[feature])
    tail = (out.data_ptr(), S_state.data_ptr(), z_state.data_ptr(), _ptr(S_lo), _ptr(z_lo),
            ws.data_ptr(), ws.numel(), _stream_handle(stream))
    if S_init is None and z_init is None:
        _check(library().slim_fwd(*args, *tail), "slim_fwd")
    else:
        _check(library().slim_fwd_from(*args, _opt_ptr(S_init), _opt_ptr(z_init),
                                       _opt_ptr(S_init_lo), _opt_ptr(z_init_lo), *tail),
               "slim_fwd_from")
    if residuals:
        return out, S_state, z_state, S_lo, z_lo
    return out, S_state, z_state


def backward(q, k, v, omega, out, dout, S_state, z_state, C, feature="exp", workspace=None,
             stream=None, S_lo=None, z_lo=None, G_S_in=None, g_z_in=None, return_state_grad=False):
    """slim_bwd (slim_bwd_from when a state gradient is handed in or asked
    for): returns (dq, dk, dv, domega), and with return_state_grad=True also
    (G_S, g_z) = G^(0), the gradient with respect to the state the sequence
    started from.  S_lo / z_lo: the residuals from forward(..., residuals=True),
    or None.  G_S_in / g_z_in: G^(N) from the backward of a later segment.
    For the quadratic map omega may be None; domega is then None."""
    _require_cuda(q, k, v, out, dout, S_state, z_state)
    B, H, L, d = q.shape
    M = omega.shape[0] if omega is not None else d
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    domega = (torch.empty(M, d, dtype=torch.float32, device=q.device)
              if omega is not None else None)
    need = workspace_size(B, H, L, d, M, C, q.dtype, feature, True)
    ws = workspace if workspace is not None else _workspace(need, q.device)
    G_S = g_z = None
    head = (q.data_ptr(), k.data_ptr(), v.data_ptr(), _opt_ptr(omega), out.data_ptr(),
            dout.data_ptr(), S_state.data_ptr(), z_state.data_ptr(), _ptr(S_lo), _ptr(z_lo))
    dims = (B, H, L, d, M, C, DTYPES[q.dtype], FEATURES[feature])
    grads = (dq.data_ptr(), dk.data_ptr(), dv.data_ptr(), _ptr(domega))
    tail = (ws.data_ptr(), ws.numel(), _stream_handle(stream))
    if G_S_in is None and g_z_in is None and not return_state_grad:
        _check(library().slim_bwd(*head, *dims, *grads, *tail), "slim_bwd")
    else:
        if return_state_grad:
            G_S = torch.empty(B, H, M, d, dtype=torch.float32, device=q.device)
            g_z = torch.empty(B, H, M, dtype=torch.float32, device=q.device)
        _check(library().slim_bwd_from(*head, _opt_ptr(G_S_in), _opt_ptr(g_z_in), *dims, *grads,
                                       _ptr(G_S), _ptr(g_z), *tail), "slim_bwd_from")
    if return_state_grad:
        return dq, dk, dv, domega, G_S, g_z
    return dq, dk, dv, domega


def bidir_workspace_size(B, H, L, d, M, C, dtype, feature, backward):
    n = _sz(0)
    _check(library().slim_bidir_workspace_size(B, H, L, d, M, C, DTYPES[dtype],
                                               FEATURES[feature], 1 if backward else 0,
                                               ctypes.byref(n)), "slim_bidir_workspace_size")
    return n.value


def forward_bidir(q, k, v, omega, C, feature="exp", workspace=None, stream=None):
    """slim_fwd_bidir (non-causal): returns (out, S_state, z_state), the state
    being the global sum over all rows."""
    _require_cuda(q, k, v)
    B, H, L, d, M = _dims(q, omega)
    out = torch.empty_like(q)
    S_state = torch.empty(B, H, M, d, dtype=torch.float32, device=q.device)
    z_state = torch.empty(B, H, M, dtype=torch.float32, device=q.device)
    ws = workspace if workspace is not None else _workspace(
        bidir_workspace_size(B, H, L, d, M, C, q.dtype, feature, False), q.device)
    _check(library().slim_fwd_bidir(q.data_ptr(), k.data_ptr(), v.data_ptr(), _opt_ptr(omega),
                                    B, H, L, d, M, C, DTYPES[q.dtype], FEATURES[feature],
                                    out.data_ptr(), S_state.data_ptr(), z_state.data_ptr(),
                                    ws.data_ptr(), ws.numel(), _stream_handle(stream)),
           "slim_fwd_bidir")
    return out, S_state, z_state


def backward_bidir(q, k, v, omega, out, dout, S_state, z_state, C, feature="exp", workspace=None,
                   stream=None):
    """slim_bwd_bidir (non-causal): returns (dq, dk, dv, domega)."""
    _require_cuda(q, k, v, out, dout, S_state, z_state)
    B, H, L, d, M = _dims(q, omega)
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    domega = (torch.empty(M, d, dtype=torch.float32, device=q.device)
              if omega is not None else None)
    ws = workspace if workspace is not None else _workspace(
        bidir_workspace_size(B, H, L, d, M, C, q.dtype, feature, True), q.device)
    _check(library().slim_bwd_bidir(q.data_ptr(), k.data_ptr(), v.data_ptr(), _opt_ptr(omega),
                                    out.data_ptr(), dout.data_ptr(), S_state.data_ptr(),
                                    z_state.data_ptr(), B, H, L, d, M, C, DTYPES[q.dtype],
                                    FEATURES[feature], dq.data_ptr(), dk.data_ptr(),
                                    dv.data_ptr(), _ptr(domega), ws.data_ptr(), ws.numel(),
                                    _stream_handle(stream)), "slim_bwd_bidir")
    return dq, dk, dv, domega


def stack_workspace_size(B, H, L, d, M, C, layers, dtype, feature, backward):
    n = _sz(0)
    _check(library().slim_stack_workspace_size(B, H, L, d, M, C, layers, DTYPES[dtype],
                                               FEATURES[feature], 1 if backward else 0,
                                               ctypes.byref(n)), "slim_stack_workspace_size")
    return n.value


def stack_forward(x, omegas, C, feature="exp", layers=None, workspace=None, stream=None,
                  residuals=True):
    """slim_stack_fwd: x [B,H,L,d]; omegas [layers, M, d] fp32 (None for the
    quadratic map, then give `layers`).  Returns (y, S_state, z_state[, S_lo,
    z_lo]) with per-layer states [layers, B, H, M, d] and [layers, B, H, M]."""
    _require_cuda(x)
    B, H, L, d = x.shape
    layers = omegas.shape[0] if omegas is not None else layers
    M = omegas.shape[1] if omegas is not None else d
    y = torch.empty_like(x)
    S = torch.empty(layers, B, H, M, d, dtype=torch.float32, device=x.device)
    z = torch.empty(layers, B, H, M, dtype=torch.float32, device=x.device)
    S_lo = torch.empty_like(S) if residuals else None
    z_lo = torch.empty_like(z) if residuals else None
    ws = workspace if workspace is not None else _workspace(
        stack_workspace_size(B, H, L, d, M, C, layers, x.dtype, feature, False), x.device)
    _check(library().slim_stack_fwd(x.data_ptr(), _opt_ptr(omegas), B, H, L, d, M, C, layers,
                                    DTYPES[x.dtype], FEATURES[feature], y.data_ptr(),
                                    S.data_ptr(), z.data_ptr(), _ptr(S_lo), _ptr(z_lo),
                                    ws.data_ptr(), ws.numel(), _stream_handle(stream)),
           "slim_stack_fwd")
    return (y, S, z, S_lo, z_lo) if residuals else (y, S, z)


def stack_backward(x, omegas, dy, S_state, z_state, C, feature="exp", S_lo=None, z_lo=None,
                   workspace=None, stream=None):
    """slim_stack_bwd: returns (dx, domegas) (domegas None without omegas)."""
    _require_cuda(x, dy, S_state, z_state)
    B, H, L, d = x.shape
    layers = S_state.shape[0]
    M = S_state.shape[3]
    dx = torch.empty_like(x)
    dom = (torch.empty(layers, M, d, dtype=torch.float32, device=x.device)
           if omegas is not None else None)
    ws = workspace if workspace is not None else _workspace(
        stack_workspace_size(B, H, L, d, M, C, layers, x.dtype, feature, True), x.device)
    _check(library().slim_stack_bwd(x.data_ptr(), _opt_ptr(omegas), dy.data_ptr(),
                                    S_state.data_ptr(), z_state.data_ptr(), _ptr(S_lo),
                                    _ptr(z_lo), B, H, L, d, M, C, layers, DTYPES[x.dtype],
                                    FEATURES[feature], dx.data_ptr(), _ptr(dom), ws.data_ptr(),
                                    ws.numel(), _stream_handle(stream)), "slim_stack_bwd")
    return dx, dom


def forward_into(q, k, v, omega, C, feature, out, S_state, z_state, workspace, stream=None,
                 S_lo=None, z_lo=None, S_init=None, z_init=None, S_init_lo=None, z_init_lo=None):
    """slim_fwd (slim_fwd_from with an initial state) into caller-allocated
    outputs and workspace (no allocation)."""
    B, H, L, d, M = _dims(q, omega)
    args = (q.data_ptr(), k.data_ptr(), v.data_ptr(), _ptr(omega), B, H, L, d, M, C,
            DTYPES[q.dtype], FEATURES[feature])
    tail = (out.data_ptr(), S_state.data_ptr(), z_state.data_ptr(), _ptr(S_lo), _ptr(z_lo),
            workspace.data_ptr(), workspace.numel(), _stream_handle(stream))
    if S_init is None:
        _check(library().slim_fwd(*args, *tail), "slim_fwd")
    else:
        _check(library().slim_fwd_from(*args, _ptr(S_init), _ptr(z_init), _ptr(S_init_lo),
                                       _ptr(z_init_lo), *tail), "slim_fwd_from")


def backward_into(q, k, v, omega, out, dout, S_state, z_state, C, feature, dq, dk, dv, domega,
                  workspace, stream=None, S_lo=None, z_lo=None, G_S_in=None, g_z_in=None,
                  G_S_out=None, g_z_out=None):
    """slim_bwd (slim_bwd_from with state gradients in or out) into
    caller-allocated gradients and workspace (no allocation)."""
    B, H, L, d, M = _dims(q, omega)
    head = (q.data_ptr(), k.data_ptr(), v.data_ptr(), _ptr(omega), out.data_ptr(),
            dout.data_ptr(), S_state.data_ptr(), z_state.data_ptr(), _ptr(S_lo), _ptr(z_lo))
    dims = (B, H, L, d, M, C, DTYPES[q.dtype], FEATURES[feature])
    grads = (dq.data_ptr(), dk.data_ptr(), dv.data_ptr(), _ptr(domega))
    tail = (workspace.data_ptr(), workspace.numel(), _stream_handle(stream))
    if G_S_in is None and G_S_out is None:
        _check(library().slim_bwd(*head, *dims, *grads, *tail), "slim_bwd")
    else:
        _check(library().slim_bwd_from(*head, _ptr(G_S_in), _ptr(g_z_in), *dims, *grads,
                                       _ptr(G_S_out), _ptr(g_z_out), *tail), "slim_bwd_from")


def forward_bidir_into(q, k, v, omega, C, feature, out, S_state, z_state, workspace, stream=None):
    """slim_fwd_bidir into caller-allocated outputs and workspace."""
    B, H, L, d, M = _dims(q, omega)
    _check(library().slim_fwd_bidir(q.data_ptr(), k.data_ptr(), v.data_ptr(), _ptr(omega),
                                    B, H, L, d, M, C, DTYPES[q.dtype], FEATURES[feature],
                                    out.data_ptr(), S_state.data_ptr(), z_state.data_ptr(),
                                    workspace.data_ptr(), workspace.numel(),
                                    _stream_handle(stream)), "slim_fwd_bidir")


def backward_bidir_into(q, k, v, omega, out, dout, S_state, z_state, C, feature, dq, dk, dv,
                        domega, workspace, stream=None):
    """slim_bwd_bidir into caller-allocated gradients and workspace."""
    B, H, L, d, M = _dims(q, omega)
    _check(library().slim_bwd_bidir(q.data_ptr(), k.data_ptr(), v.data_ptr(), _ptr(omega),
                                    out.data_ptr(), dout.data_ptr(), S_state.data_ptr(),
                                    z_state.data_ptr(), B, H, L, d, M, C, DTYPES[q.dtype],
                                    FEATURES[feature], dq.data_ptr(), dk.data_ptr(),
                                    dv.data_ptr(), _ptr(domega), workspace.data_ptr(),
                                    workspace.numel(), _stream_handle(stream)), "slim_bwd_bidir")


def check_device_error(workspace, stream=None):
    """Raises SlimError(SLIM_ERR_TIMEOUT) if a bounded device wait gave up."""
    _check(library().slim_check_device_error(workspace.data_ptr(), _stream_handle(stream)),
           "slim_check_device_error")


def launch_count():
    """Number of libslim kernel launches since the library was loaded."""
    return int(library().slim_launch_count())


def profiler_enable(on=True):
    library().slim_profiler_enable(1 if on else 0)


def profiler_reset():
    library().slim_profiler_reset()


def profiler_read():
    """Per-kernel totals since the last reset: list of dicts with name,
    launches, total_ms (CUDA events), flops and bytes (algorithmic)."""
    arr = (KernelStats * 64)()
    n = library().slim_profiler_read(ctypes.cast(arr, ctypes.c_void_p), 64)
    if n < 0:
        raise SlimError(4, "slim_profiler_read")
    return [{"name": arr[i].name.decode(), "launches": int(arr[i].launches),
             "total_ms": arr[i].total_ms, "flops": arr[i].flops, "bytes": arr[i].bytes}
            for i in range(min(n, 64))]


def tc_selftest(A, B, a_mn, b_mn):
    """D = A @ B through one chain of tcgen05 MMAs (diagnostic of the
    tensor-core operand layouts); A [128, K], B [K, N] bf16 CUDA tensors."""
    _require_cuda(A, B)
    K, N = B.shape
    D = torch.empty(A.shape[0], N, dtype=torch.float32, device=A.device)
    err = torch.zeros(1, dtype=torch.int32, device=A.device)
    _check(library().slim_tc_selftest(a_mn, b_mn, K, N, A.data_ptr(), B.data_ptr(), D.data_ptr(),
                                      err.data_ptr(), _stream_handle(None)), "slim_tc_selftest")
    return D, err


class SlimAttention(torch.autograd.Function):
    """Causal linear attention with the SLiM forward/backward (state carried
    across slices of C rows; backward by rollback, no stored activations)."""

    @staticmethod
    def forward(ctx, q, k, v, omega, C, feature):
        out, S, z, S_lo, z_lo = forward(q.contiguous(), k.contiguous(), v.contiguous(),
                                        omega.contiguous(), C, feature, residuals=True)
        ctx.save_for_backward(q, k, v, omega, out, S, z, S_lo, z_lo)
        ctx.C, ctx.feature = C, feature
        return out

    @staticmethod
    def backward(ctx, dout):
        q, k, v, omega, out, S, z, S_lo, z_lo = ctx.saved_tensors
        dq, dk, dv, domega = backward(q.contiguous(), k.contiguous(), v.contiguous(),
                                      omega.contiguous(), out, dout.contiguous(), S, z, ctx.C,
                                      ctx.feature, S_lo=S_lo, z_lo=z_lo)
        return dq, dk, dv, domega, None, None


def slim_attention(q, k, v, omega, C, feature="exp"):
    return SlimAttention.apply(q, k, v, omega, C, feature)
