"""ctypes binding of libgc.so (argument marshalling only).

Tensors passed to device entry points must be contiguous CUDA tensors of the
dtype the C header states; outputs not supplied by the caller are allocated
with torch.  Calls are asynchronous on torch's current stream, like the C
functions; gc_status() synchronises and reports device-detected data errors.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch  # loads the CUDA runtime libgc.so links against

_HERE = os.path.dirname(os.path.abspath(__file__))
library_path = os.path.join(_HERE, "libgc.so")
if not os.path.exists(library_path):
    raise ImportError(
        f"{library_path} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`"
        " (the gradient-coding path has no fallback without the CUDA library)")
lib = ctypes.CDLL(library_path)

GC_CYCLIC, GC_EXPLICIT = 0, 1
GC_F32, GC_BF16 = 0, 1
GC_LSQ, GC_LOGISTIC = 0, 1

_i, _sz, _p, _d, _f, _i64 = (ctypes.c_int, ctypes.c_size_t, ctypes.c_void_p, ctypes.c_double,
                             ctypes.c_float, ctypes.c_int64)


def _sig(name, res, *args):
    fn = getattr(lib, name)
    fn.restype = res
    fn.argtypes = list(args)
    return fn


_sig("gc_last_error", ctypes.c_char_p)
_sig("gc_version", _i)
_sig("gc_kernel_launches", ctypes.c_uint64)
_sig("gc_set_wait_limit", _i, _i64)
_sig("gc_inject_stall", _i, _i)
_sig("gc_set_decode_policy", _i, _i)
_sig("gc_workspace_init", _i, _p, _sz, _p)
_sig("gc_status", _i, _p, _p)
_sig("gc_make_assignment", _i, _i, _i, _i, _i, _p, _p, _p, _p)
_sig("gc_chunk_ordering", _i, _p, _i, _i, _i, _p, _p)
_sig("gc_trigger_workspace", _sz, _i)
_sig("gc_chunk_grads_batched_workspace", _sz, _i, _i, _i, _i)
_sig("gc_chunk_grads_batched", _i, _p, _p, _p, _i, _i, _i, _i, _i, _p, _p, _sz, _p)
_sig("gc_trigger_times", _i, _p, _i, _i, _i, _p, _i64, _i, _i, _p, _p, _p, _p, _sz, _p)
_sig("gc_chunk_grads_workspace", _sz, _i, _i, _i, _i)
_sig("gc_chunk_grads", _i, _p, _i, _p, _p, _i, _i, _i, _i, _p, _p, _p, _sz, _p)
_sig("gc_coeff_workspace", _sz, _i, _i, _i, _i, _i)
_sig("gc_find_encoding_coeff", _i, _p, _i, _p, _i, _i, _i, _p, _i, _p, _p, _p, _p, _p, _p, _p,
     _sz, _p)
_sig("gc_find_encoding_coeff_noalloc", _i, _p, _i, _p, _i, _i, _i, _p, _i, _p, _p, _p, _p, _p, _p,
     _p)
_sig("gc_encode_workspace", _sz, _i, _i, _i, _i, _i, _i)
_sig("gc_encode", _i, _p, _i, _p, _i, _i, _i, _p, _i, _p, _i, _p, _p, _sz, _p)
_sig("gc_encode_with_coeffs", _i, _p, _i, _p, _i, _i, _i, _p, _i, _p, _i, _p, _p)
_sig("gc_decode_tx", _i, _p, _i, _i, _p, _i, _i, _p, _p)
_sig("gc_decode_batch_workspace", _sz, _i, _i, _i, _i, _i, _i)
_sig("gc_decode_batch", _i, _p, _i, _p, _i, _i, _i, _p, _i, _p, _i, _p, _p, _p, _p, _p, _sz, _p)
_sig("gc_decode_plan_bytes", _sz, _i, _i, _i)
_sig("gc_decode_plan_workspace", _sz, _i, _i, _i, _i, _i)
_sig("gc_decode_plan", _i, _p, _i, _p, _i, _i, _i, _p, _i, _p, _sz, _p, _p, _p, _sz, _p)
_sig("gc_decode_prepare_bytes", _sz, _i, _i, _i, _i)
_sig("gc_decode_prepare", _i, _p, _i, _p, _i, _i, _i, _p, _sz, _p)
_sig("gc_decode_plan_prepared_workspace", _sz)
_sig("gc_decode_plan_prepared", _i, _p, _p, _i, _i, _i, _i, _p, _i, _p, _sz, _p, _p, _p, _sz, _p)
_sig("gc_decode_apply_workspace", _sz, _i, _i, _i, _i)
_sig("gc_decode_apply", _i, _p, _i, _i, _i, _p, _i, _p, _p, _p, _sz, _p)
_sig("gc_decode_combine_workspace", _sz, _i, _i, _i, _i)
_sig("gc_decode_combine", _i, _p, _i, _i, _i, _p, _i, _p, _p, _p, _sz, _p)
_sig("gc_mse_workspace", _sz, _i, _i, _i, _i, _i, _i)
_sig("gc_mse", _i, _p, _i, _p, _i, _i, _i, _p, _i, _p, _i, _p, _p, _p, _p, _sz, _p)
_sig("gc_sgd_step", _i, _p, _p, _i, _f, _i64, _p)
_sig("gc_live_step", _i, _p, _p, _i, _p, _i, _i, _i, _p, _p, _i, _f, _i64, _p, _p, _p, _p)


class GCError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"gc error {code}: {msg}")
        self.code = code


def gc_last_error() -> str:
    return lib.gc_last_error().decode()


def gc_version() -> int:
    return lib.gc_version()


def _check(rc: int) -> None:
    if rc != 0:
        raise GCError(rc, gc_last_error())


def block_length(d: int, ell: int) -> int:
    return -(-d // ell)


def _stream() -> int:
    return torch.cuda.current_stream().cuda_stream


def _dev(t, dtype, name, shape=None):
    """Device pointer of a contiguous CUDA tensor of the given dtype (None -> NULL)."""
    if t is None:
        return None
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    return t.data_ptr()


class Workspace:
    """Reusable device scratch buffer; grows on demand.  Its 256-byte status
    header is zeroed whenever a new buffer is allocated."""

    def __init__(self, device=None):
        self.device = torch.device(device) if device is not None else torch.device("cuda")
        self.buf = None

    def get(self, nbytes: int):
        nbytes = max(int(nbytes), 256)
        if self.buf is None or self.buf.numel() < nbytes:
            self.buf = None
            self.buf = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
            _check(lib.gc_workspace_init(self.buf.data_ptr(), nbytes, _stream()))
        return self.buf.data_ptr(), self.buf.numel()

    def status(self) -> None:
        if self.buf is not None:
            _check(lib.gc_status(self.buf.data_ptr(), _stream()))


def _ws(ws, nbytes, device):
    if ws is None:
        ws = Workspace(device)
    return ws, ws.get(nbytes)


def gc_status(ws: Workspace) -> None:
    """Synchronise and raise GCError if a kernel flagged bad data or a timeout."""
    ws.status()


# ---------------------------------------------------------------- assignment
def gc_make_assignment(N: int, m: int, delta: int, kind: int = GC_CYCLIC, explicit_order=None):
    """Host-only: (A N x m uint8, order m x delta int32, O N x m uint8) numpy arrays."""
    A = np.zeros((N, m), dtype=np.uint8)
    O = np.zeros((N, m), dtype=np.uint8)
    order = np.zeros((m, delta), dtype=np.int32)
    ex = None
    if explicit_order is not None:
        ex = np.ascontiguousarray(explicit_order, dtype=np.int32)
        if ex.shape != (m, delta):
            raise ValueError("explicit_order must be m x delta")
    _check(lib.gc_make_assignment(N, m, delta, kind, None if ex is None else ex.ctypes.data,
                                  A.ctypes.data, order.ctypes.data, O.ctypes.data))
    return A, order, O


def gc_chunk_ordering(A):
    """Host-only Algorithm 2: A (N x N, every row and column sum delta) ->
    (order m x delta int32, O N x m uint8) with every row sum of O equal to
    delta (delta + 1) / 2."""
    A = np.ascontiguousarray(np.asarray(A) != 0, dtype=np.uint8)
    N, m = A.shape
    delta = int(A[0].sum()) if N else 0
    order = np.zeros((m, max(delta, 1)), dtype=np.int32)
    O = np.zeros((N, m), dtype=np.uint8)
    _check(lib.gc_chunk_ordering(A.ctypes.data, N, m, delta, order.ctypes.data, O.ctypes.data))
    return order, O


def gc_trigger_times(order, N: int, m: int, delta: int, tau, ell: int, theta: int = 0, T=True,
                     psi=True, T_full=True, ws: Workspace | None = None):
    """Completion times and the encode-and-transmit trigger for nsim simulated
    realizations (tau: nsim x m float64 on the device, +inf = failed worker).
    Returns dict T (nsim float64), psi (nsim x m int32), T_full (nsim float64);
    pass a tensor to write into it or False to skip an output."""
    nsim = tau.shape[0]
    dev = tau.device

    def out(x, shape, dt):
        if x is True:
            return torch.empty(shape, dtype=dt, device=dev)
        return x if isinstance(x, torch.Tensor) else None
    T = out(T, (nsim,), torch.float64)
    psi = out(psi, (nsim, m), torch.int32)
    T_full = out(T_full, (nsim,), torch.float64)
    ws, (wp, wn) = _ws(ws, lib.gc_trigger_workspace(N), dev)
    _check(lib.gc_trigger_times(
        _dev(order, torch.int32, "order", (m, delta)), N, m, delta,
        _dev(tau, torch.float64, "tau", (nsim, m)), nsim, ell, theta,
        _dev(T, torch.float64, "T", (nsim,)), _dev(psi, torch.int32, "psi", (nsim, m)),
        _dev(T_full, torch.float64, "T_full", (nsim,)), wp, wn, _stream()))
    return {"T": T, "psi": psi, "T_full": T_full}


def gc_chunk_grads_batched(X, y, W, N: int, n_c: int, loss: int, G=None,
                           ws: Workspace | None = None):
    """Chunk gradients for n_w parameter vectors (rows of W) on the tensor
    cores: G (n_w x N x d float32).  X must be bfloat16."""
    n_w, d = W.shape
    if X.dtype != torch.bfloat16:
        raise TypeError("X must be bfloat16")
    if G is None:
        G = torch.empty(n_w, N, d, dtype=torch.float32, device=X.device)
    ws, (wp, wn) = _ws(ws, lib.gc_chunk_grads_batched_workspace(N, n_c, d, n_w), X.device)
    _check(lib.gc_chunk_grads_batched(
        _dev(X, torch.bfloat16, "X", (N * n_c, d)), _dev(y, torch.float32, "y", (N * n_c,)),
        _dev(W, torch.float32, "W", (n_w, d)), N, n_c, d, n_w, loss,
        _dev(G, torch.float32, "G", (n_w, N, d)), wp, wn, _stream()))
    return G


# ---------------------------------------------------------------- chunk gradients
def gc_chunk_grads_workspace(N, n_c, d, x_dtype):
    return lib.gc_chunk_grads_workspace(N, n_c, d, x_dtype)


def gc_chunk_grads(X, y, w, N: int, n_c: int, loss: int, G=None, loss_out=None,
                   ws: Workspace | None = None):
    """G (N x d float32) = per-chunk gradients; loss_out (1 float64) optional."""
    d = X.shape[1]
    x_dtype = GC_BF16 if X.dtype == torch.bfloat16 else GC_F32
    if X.dtype not in (torch.float32, torch.bfloat16):
        raise TypeError("X must be float32 or bfloat16")
    if X.shape[0] != N * n_c:
        raise ValueError("X must have N * n_c rows")
    if G is None:
        G = torch.empty(N, d, dtype=torch.float32, device=X.device)
    ws, (wp, wn) = _ws(ws, gc_chunk_grads_workspace(N, n_c, d, x_dtype), X.device)
    _check(lib.gc_chunk_grads(_dev(X, X.dtype, "X"), x_dtype, _dev(y, torch.float32, "y", (N * n_c,)),
                              _dev(w, torch.float32, "w", (d,)), N, n_c, d, loss,
                              _dev(G, torch.float32, "G", (N, d)),
                              _dev(loss_out, torch.float64, "loss_out"), wp, wn, _stream()))
    return G


# ---------------------------------------------------------------- Algorithm 1
def gc_coeff_workspace(N, m, delta, ell, npat):
    return lib.gc_coeff_workspace(N, m, delta, ell, npat)


def gc_find_encoding_coeff(R, ell, order, N, m, delta, psi, E=True, C=True, delta_out=True,
                           support=False, coef_err=True, est=True, ws: Workspace | None = None):
    """Batched Algorithm 1.  Boolean arguments request an output (allocated
    here); tensors are used as given.  Returns a dict of the outputs."""
    npat = psi.shape[0]
    dev = psi.device

    def out(flag, shape, dtype):
        if isinstance(flag, torch.Tensor):
            return flag
        return torch.empty(shape, dtype=dtype, device=dev) if flag else None

    res = {
        "E": out(E, (npat, m, delta, ell), torch.float64),
        "C": out(C, (npat, ell, N * ell), torch.float32),
        "delta": out(delta_out, (npat, N), torch.uint8),
        "support": out(support, (npat, N, m), torch.uint8),
        "coef_err": out(coef_err, (npat,), torch.float64),
        "est": out(est, (npat,), torch.float64),
    }
    ws, (wp, wn) = _ws(ws, gc_coeff_workspace(N, m, delta, ell, npat), dev)
    _check(lib.gc_find_encoding_coeff(
        _dev(R, torch.float64, "R", (ell, m)), ell, _dev(order, torch.int32, "order", (m, delta)),
        N, m, delta, _dev(psi, torch.int32, "psi", (npat, m)), npat,
        _dev(res["E"], torch.float64, "E"), _dev(res["C"], torch.float32, "C"),
        _dev(res["delta"], torch.uint8, "delta_out"), _dev(res["support"], torch.uint8, "support"),
        _dev(res["coef_err"], torch.float64, "coef_err"), _dev(res["est"], torch.float64, "est"),
        wp, wn, _stream()))
    return res


# ---------------------------------------------------------------- encode / decode
def gc_encode_workspace(N, m, delta, ell, npat, d):
    return lib.gc_encode_workspace(N, m, delta, ell, npat, d)


def gc_encode(R, ell, order, N, m, delta, psi, G, T=None, ws: Workspace | None = None):
    """Worker transmissions T (npat x m x L float32), eq. (2)."""
    npat = psi.shape[0]
    d = G.shape[1]
    L = block_length(d, ell)
    if T is None:
        T = torch.empty(npat, m, L, dtype=torch.float32, device=G.device)
    ws, (wp, wn) = _ws(ws, gc_encode_workspace(N, m, delta, ell, npat, d), G.device)
    _check(lib.gc_encode(_dev(R, torch.float64, "R", (ell, m)), ell,
                         _dev(order, torch.int32, "order", (m, delta)), N, m, delta,
                         _dev(psi, torch.int32, "psi", (npat, m)), npat,
                         _dev(G, torch.float32, "G", (N, d)), d,
                         _dev(T, torch.float32, "T", (npat, m, L)), wp, wn, _stream()))
    return T


def gc_encode_with_coeffs(E, ell, order, N, m, delta, psi, G, T=None):
    """Eq. (2) alone: transmissions from Algorithm 1's coefficients E
    (npat x m x delta x ell float64, as gc_find_encoding_coeff returns)."""
    npat = psi.shape[0]
    d = G.shape[1]
    L = block_length(d, ell)
    if T is None:
        T = torch.empty(npat, m, L, dtype=torch.float32, device=G.device)
    _check(lib.gc_encode_with_coeffs(_dev(E, torch.float64, "E", (npat, m, delta, ell)), ell,
                                     _dev(order, torch.int32, "order", (m, delta)), N, m, delta,
                                     _dev(psi, torch.int32, "psi", (npat, m)), npat,
                                     _dev(G, torch.float32, "G", (N, d)), d,
                                     _dev(T, torch.float32, "T", (npat, m, L)), _stream()))
    return T


def gc_decode_tx(R, ell, m, T, d, ghat=None):
    """PS decode of transmissions: ghat (npat x d float32)."""
    npat = T.shape[0]
    L = block_length(d, ell)
    if ghat is None:
        ghat = torch.empty(npat, d, dtype=torch.float32, device=T.device)
    _check(lib.gc_decode_tx(_dev(R, torch.float64, "R", (ell, m)), ell, m,
                            _dev(T, torch.float32, "T", (npat, m, L)), npat, d,
                            _dev(ghat, torch.float32, "ghat", (npat, d)), _stream()))
    return ghat


def gc_decode_batch_workspace(N, m, delta, ell, npat, d):
    return lib.gc_decode_batch_workspace(N, m, delta, ell, npat, d)


def gc_decode_batch(R, ell, order, N, m, delta, psi, G, Ghat=True, coef_err=True, est=True,
                    grad_mse=True, ws: Workspace | None = None):
    """Batched decode-combine.  Returns dict with Ghat (npat x d float32 or
    None), coef_err, est, grad_mse (npat float64 or None)."""
    npat = psi.shape[0]
    d = G.shape[1]
    dev = G.device

    def out(flag, shape, dtype):
        if isinstance(flag, torch.Tensor):
            return flag
        return torch.empty(shape, dtype=dtype, device=dev) if flag else None

    res = {
        "Ghat": out(Ghat, (npat, d), torch.float32),
        "coef_err": out(coef_err, (npat,), torch.float64),
        "est": out(est, (npat,), torch.float64),
        "grad_mse": out(grad_mse, (npat,), torch.float64),
    }
    ws, (wp, wn) = _ws(ws, gc_decode_batch_workspace(N, m, delta, ell, npat, d), dev)
    _check(lib.gc_decode_batch(
        _dev(R, torch.float64, "R", (ell, m)), ell, _dev(order, torch.int32, "order", (m, delta)),
        N, m, delta, _dev(psi, torch.int32, "psi", (npat, m)), npat,
        _dev(G, torch.float32, "G", (N, d)), d, _dev(res["Ghat"], torch.float32, "Ghat", (npat, d)),
        _dev(res["coef_err"], torch.float64, "coef_err"), _dev(res["est"], torch.float64, "est"),
        _dev(res["grad_mse"], torch.float64, "grad_mse"), wp, wn, _stream()))
    return res


def gc_decode_plan(R, ell, order, N, m, delta, psi, plan=None, coef_err=True, est=True,
                   ws: Workspace | None = None):
    """Algorithm 1 for every pattern into an opaque plan (uint8 device tensor)
    for gc_decode_apply.  Returns dict with plan, coef_err, est."""
    npat = psi.shape[0]
    dev = psi.device
    nb = lib.gc_decode_plan_bytes(N, ell, npat)
    if plan is None:
        plan = torch.empty(max(int(nb), 256), dtype=torch.uint8, device=dev)
    ce = coef_err if isinstance(coef_err, torch.Tensor) else (
        torch.empty(npat, dtype=torch.float64, device=dev) if coef_err else None)
    es = est if isinstance(est, torch.Tensor) else (
        torch.empty(npat, dtype=torch.float64, device=dev) if est else None)
    ws, (wp, wn) = _ws(ws, lib.gc_decode_plan_workspace(N, m, delta, ell, npat), dev)
    _check(lib.gc_decode_plan(_dev(R, torch.float64, "R", (ell, m)), ell,
                              _dev(order, torch.int32, "order", (m, delta)), N, m, delta,
                              _dev(psi, torch.int32, "psi", (npat, m)), npat,
                              _dev(plan, torch.uint8, "plan"), plan.numel(),
                              _dev(ce, torch.float64, "coef_err"), _dev(es, torch.float64, "est"),
                              wp, wn, _stream()))
    return {"plan": plan, "coef_err": ce, "est": es}


def gc_decode_prepare(R, ell, order, N, m, delta, prep=None):
    """Holders and the Algorithm 1 memo table for (R, assignment), once:
    a uint8 device buffer for gc_decode_plan_prepared."""
    nb = int(lib.gc_decode_prepare_bytes(N, m, delta, ell))
    if nb == 0:
        raise ValueError("unsupported shape for gc_decode_prepare")
    if prep is None:
        prep = torch.empty(nb, dtype=torch.uint8, device=R.device)
    _check(lib.gc_decode_prepare(_dev(R, torch.float64, "R", (ell, m)), ell,
                                 _dev(order, torch.int32, "order", (m, delta)), N, m, delta,
                                 _dev(prep, torch.uint8, "prep"), prep.numel(), _stream()))
    return prep


def gc_decode_plan_prepared(prep, R, ell, N, m, delta, psi, plan=None, coef_err=True, est=True,
                            ws: Workspace | None = None):
    """gc_decode_plan from a gc_decode_prepare buffer.  Returns dict with
    plan, coef_err, est."""
    npat = psi.shape[0]
    dev = psi.device
    nb = lib.gc_decode_plan_bytes(N, ell, npat)
    if plan is None:
        plan = torch.empty(max(int(nb), 256), dtype=torch.uint8, device=dev)
    ce = coef_err if isinstance(coef_err, torch.Tensor) else (
        torch.empty(npat, dtype=torch.float64, device=dev) if coef_err else None)
    es = est if isinstance(est, torch.Tensor) else (
        torch.empty(npat, dtype=torch.float64, device=dev) if est else None)
    ws, (wp, wn) = _ws(ws, lib.gc_decode_plan_prepared_workspace(), dev)
    _check(lib.gc_decode_plan_prepared(_dev(prep, torch.uint8, "prep"),
                                       _dev(R, torch.float64, "R", (ell, m)), ell, N, m, delta,
                                       _dev(psi, torch.int32, "psi", (npat, m)), npat,
                                       _dev(plan, torch.uint8, "plan"), plan.numel(),
                                       _dev(ce, torch.float64, "coef_err"),
                                       _dev(es, torch.float64, "est"), wp, wn, _stream()))
    return {"plan": plan, "coef_err": ce, "est": es}


def gc_decode_apply(plan, ell, N, npat, G, Ghat=True, grad_mse=True, ws: Workspace | None = None):
    """Ghat (npat x d) and/or grad_mse (npat) from a gc_decode_plan plan and G."""
    d = G.shape[1]
    dev = G.device
    if not isinstance(Ghat, torch.Tensor):
        Ghat = torch.empty(npat, d, dtype=torch.float32, device=dev) if Ghat else None
    if not isinstance(grad_mse, torch.Tensor):
        grad_mse = torch.empty(npat, dtype=torch.float64, device=dev) if grad_mse else None
    ws, (wp, wn) = _ws(ws, lib.gc_decode_apply_workspace(N, ell, npat, d), dev)
    _check(lib.gc_decode_apply(_dev(plan, torch.uint8, "plan"), ell, N, npat,
                               _dev(G, torch.float32, "G", (N, d)), d,
                               _dev(Ghat, torch.float32, "Ghat", (npat, d)),
                               _dev(grad_mse, torch.float64, "grad_mse"), wp, wn, _stream()))
    return {"Ghat": Ghat, "grad_mse": grad_mse}


def gc_set_wait_limit(cycles: int) -> None:
    """Testing aid: device waits give up after `cycles` clock cycles (0 = default)."""
    _check(lib.gc_set_wait_limit(int(cycles)))


GC_STALL_CHUNK_GRADS = 1
GC_STALL_COMBINE = 2
GC_STALL_BATCHED = 4


def gc_inject_stall(kernels: int) -> None:
    """Testing aid: the next launch of each selected kernel withholds its copies."""
    _check(lib.gc_inject_stall(int(kernels)))


GC_DECODE_AUTO = 0
GC_DECODE_DENSE = 1
GC_DECODE_RESIDUAL = 2


def gc_set_decode_policy(policy: int) -> None:
    """Path of the batched decode per 128-row tile: GC_DECODE_AUTO (default),
    GC_DECODE_DENSE (tensor-core GEMM) or GC_DECODE_RESIDUAL (sum of the
    chunk gradients plus the non-identity blocks).  Process-wide."""
    _check(lib.gc_set_decode_policy(int(policy)))


def gc_kernel_launches() -> int:
    return int(lib.gc_kernel_launches())


def gc_decode_combine_workspace(N, ell, npat, d):
    return lib.gc_decode_combine_workspace(N, ell, npat, d)


def gc_decode_combine(C, ell, N, G, Ghat=True, grad_mse=True, ws: Workspace | None = None):
    """Ghat (npat x d) = C . G for a decode matrix C (npat x ell x N*ell) from
    gc_find_encoding_coeff; grad_mse optional."""
    npat = C.shape[0]
    d = G.shape[1]
    dev = G.device
    if not isinstance(Ghat, torch.Tensor):
        Ghat = torch.empty(npat, d, dtype=torch.float32, device=dev) if Ghat else None
    if not isinstance(grad_mse, torch.Tensor):
        grad_mse = torch.empty(npat, dtype=torch.float64, device=dev) if grad_mse else None
    ws, (wp, wn) = _ws(ws, gc_decode_combine_workspace(N, ell, npat, d), dev)
    _check(lib.gc_decode_combine(_dev(C, torch.float32, "C", (npat, ell, N * ell)), ell, N, npat,
                                 _dev(G, torch.float32, "G", (N, d)), d,
                                 _dev(Ghat, torch.float32, "Ghat", (npat, d)),
                                 _dev(grad_mse, torch.float64, "grad_mse"), wp, wn, _stream()))
    return {"Ghat": Ghat, "grad_mse": grad_mse}


def gc_mse_workspace(N, m, delta, ell, npat, d):
    return lib.gc_mse_workspace(N, m, delta, ell, npat, d)


def gc_mse(R, ell, order, N, m, delta, psi, G, coef_err=True, est=True, grad_mse=True,
           ws: Workspace | None = None):
    """Error measures only; decoded gradients are never written."""
    npat = psi.shape[0]
    d = G.shape[1]
    dev = G.device

    def out(flag, shape, dtype):
        if isinstance(flag, torch.Tensor):
            return flag
        return torch.empty(shape, dtype=dtype, device=dev) if flag else None

    res = {
        "coef_err": out(coef_err, (npat,), torch.float64),
        "est": out(est, (npat,), torch.float64),
        "grad_mse": out(grad_mse, (npat,), torch.float64),
    }
    ws, (wp, wn) = _ws(ws, gc_mse_workspace(N, m, delta, ell, npat, d), dev)
    _check(lib.gc_mse(
        _dev(R, torch.float64, "R", (ell, m)), ell, _dev(order, torch.int32, "order", (m, delta)),
        N, m, delta, _dev(psi, torch.int32, "psi", (npat, m)), npat,
        _dev(G, torch.float32, "G", (N, d)), d, _dev(res["coef_err"], torch.float64, "coef_err"),
        _dev(res["est"], torch.float64, "est"), _dev(res["grad_mse"], torch.float64, "grad_mse"),
        wp, wn, _stream()))
    return res


def gc_sgd_step(w, ghat, lr: float, Ntil: int):
    """w -= lr * ghat / N~ in place."""
    d = w.shape[0]
    _check(lib.gc_sgd_step(_dev(w, torch.float32, "w", (d,)), _dev(ghat, torch.float32, "ghat", (d,)),
                           d, float(lr), int(Ntil), _stream()))
    return w


def gc_live_step(E, R, ell, order, N, m, delta, psi, G, w, lr: float, Ntil: int, T=None, ghat=None):
    """One live realization in one launch: eq. (2) transmissions, their PS
    decode and the update of w (in place).  E is the pattern's m x delta x ell
    float64 coefficients (a 1 x m x delta x ell batch is accepted), psi its m
    processed counts; T (m x L) and ghat (d) are written when given."""
    d = G.shape[1]
    L = block_length(d, ell)
    _check(lib.gc_live_step(_dev(E.reshape(m, delta, ell), torch.float64, "E", (m, delta, ell)),
                            _dev(R, torch.float64, "R", (ell, m)), ell,
                            _dev(order, torch.int32, "order", (m, delta)), N, m, delta,
                            _dev(psi.reshape(m), torch.int32, "psi", (m,)),
                            _dev(G, torch.float32, "G", (N, d)), d, float(lr), int(Ntil),
                            _dev(w, torch.float32, "w", (d,)),
                            None if T is None else _dev(T.reshape(m, L), torch.float32, "T", (m, L)),
                            None if ghat is None else _dev(ghat.reshape(d), torch.float32, "ghat", (d,)),
                            _stream()))
    return w
