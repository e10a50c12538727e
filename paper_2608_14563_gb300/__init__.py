"""Python binding of libfpo (include/fpo.h): the GB300 pseudogradient update of
Forward-Pass-Only MLP training.

Argument marshalling only: every function here passes device pointers, sizes
and the current CUDA stream to the C entry point of the same name; every step
of the computation runs in libfpo's CUDA kernels.  PyTorch supplies device
memory and streams.  There is no CPU fallback: importing this package fails
loudly when ``libfpo.so`` has not been built (``python -m
paper_2608_14563_gb300.build`` or ``__graft_entry__.build()``).
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libfpo.so")

F32, BF16 = 0, 1
OK = 0
MAX_GROUPED_LAYERS = 64
STAGE_EVENTS = 7
ES_AUTO, ES_RECOMPUTE, ES_STORED_LOGITS, ES_DIRECT = 0, 1, 2, 3
AUTO_T_CHUNK = 8192  # FPO_AUTO_T_CHUNK: tokens per error-matrix chunk when t_chunk is 0

if not os.path.exists(LIB_PATH):
    raise ImportError(f"libfpo.so is not built ({LIB_PATH} missing); run "
                      "`python -m paper_2608_14563_gb300.build` first")
_lib = ctypes.CDLL(LIB_PATH)
ABI_VERSION = 2  # FPO_ABI_VERSION of include/fpo.h that the structures below mirror
_lib.fpo_abi_version.restype = ctypes.c_int32
if _lib.fpo_abi_version() != ABI_VERSION:
    raise ImportError(f"libfpo.so reports ABI version {_lib.fpo_abi_version()}, this binding "
                      f"needs {ABI_VERSION}; rebuild it (`python -m paper_2608_14563_gb300.build`)")

_vp, _i64, _i32, _f32, _sz = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_float,
                              ctypes.c_size_t)


class ErrorSignalDesc(ctypes.Structure):
    """Mirror of fpo_error_signal_desc."""
    _fields_ = [("T", _i64), ("d", _i64), ("V", _i64), ("dtype", _i32), ("eps", _f32),
                ("min_rms", _f32), ("loss_scale", _f32), ("algo", _i32), ("t_chunk", _i64),
                ("stage_events", ctypes.POINTER(_vp)), ("stage_events_per_chunk", _i32)]


_lib.fpo_abi_version.restype = _i32
_lib.fpo_status_string.argtypes = [_i32]
_lib.fpo_status_string.restype = ctypes.c_char_p
_lib.fpo_set_wait_limit_ns.argtypes = [ctypes.c_uint64]
_lib.fpo_set_wait_limit_ns.restype = None
_lib.fpo_error_signal_stage_events.argtypes = [ctypes.POINTER(ErrorSignalDesc)]
_lib.fpo_error_signal_stage_events.restype = _i32
_lib.fpo_error_signal_workspace.argtypes = [ctypes.POINTER(ErrorSignalDesc)]
_lib.fpo_error_signal_workspace.restype = _sz
_lib.fpo_error_signal.argtypes = [ctypes.POINTER(ErrorSignalDesc), _vp, _vp, _vp, _vp, _vp, _vp,
                                  _vp, _vp, _sz, _vp]
_lib.fpo_error_signal.restype = _i32
_lib.fpo_layer_update_workspace.argtypes = []
_lib.fpo_layer_update_workspace.restype = _sz
_lib.fpo_layer_update.argtypes = [_i64, _i64, _i64, _i32, _vp, _vp, _f32, _vp, _vp, _vp, _vp,
                                  _sz, _vp]
_lib.fpo_layer_update.restype = _i32
_lib.fpo_layer_update_grouped.argtypes = [_i32, _i64, _i64, _i64, _i32, _vp,
                                          ctypes.POINTER(_vp), _f32, ctypes.POINTER(_vp),
                                          ctypes.POINTER(_vp), ctypes.POINTER(_vp), _vp, _sz, _vp]
_lib.fpo_layer_update_grouped.restype = _i32
_lib.fpo_layer_update_grouped_signals.argtypes = [_i32, _i64, _i64, _i64, _i32,
                                                  ctypes.POINTER(_vp), ctypes.POINTER(_vp), _f32,
                                                  ctypes.POINTER(_vp), ctypes.POINTER(_vp),
                                                  ctypes.POINTER(_vp), _vp, _sz, _vp]
_lib.fpo_layer_update_grouped_signals.restype = _i32
_lib.fpo_rmsnorm_vjp.argtypes = [_i64, _i64, _i32, _vp, _vp, _vp, _f32, _f32, _vp, _vp]
_lib.fpo_rmsnorm_vjp.restype = _i32
_lib.fpo_layer_signals.argtypes = [_i32, _i64, _i64, _i32, _vp, _vp, _vp, _vp, _vp, _f32, _f32,
                                   _vp, _vp]
_lib.fpo_layer_signals.restype = _i32


class OptimizerDesc(ctypes.Structure):
    """Mirror of fpo_optimizer_desc."""
    _fields_ = [("kind", _i32), ("clip", _i32), ("lr", _f32), ("momentum", _f32),
                ("beta1", _f32), ("beta2", _f32), ("adam_eps", _f32), ("weight_decay", _f32),
                ("clip_frac", _f32), ("step", _i64)]


OPT_SGD, OPT_SGD_MOMENTUM, OPT_ADAMW = 0, 1, 2
CLIP_NONE, CLIP_STEP, CLIP_GRADIENT = 0, 1, 2
_lib.fpo_layer_optimize_workspace.argtypes = [_i32, _i64, _i64]
_lib.fpo_layer_optimize_workspace.restype = _sz
_lib.fpo_layer_optimize_grouped.argtypes = [_i32, _i64, _i64, _i64, _i32, ctypes.POINTER(_vp),
                                            ctypes.POINTER(_vp), ctypes.POINTER(OptimizerDesc),
                                            ctypes.POINTER(_vp), ctypes.POINTER(_vp),
                                            ctypes.POINTER(_vp), ctypes.POINTER(_vp), _vp, _sz, _vp]
_lib.fpo_layer_optimize_grouped.restype = _i32
_lib.fpo_gate_up_signals.argtypes = [_i64, _i64, _i64, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                     _sz, _vp]
_lib.fpo_gate_up_signals.restype = _i32
_lib.fpo_cosine_workspace.argtypes = [_i64]
_lib.fpo_cosine_workspace.restype = _sz
_lib.fpo_cosine.argtypes = [_i64, _i32, _vp, _vp, _vp, _vp, _sz, _vp]
_lib.fpo_cosine.restype = _i32
_lib.fpo_get_device_status.argtypes = [_vp, _vp]
_lib.fpo_get_device_status.restype = _i32
_lib.fpo_cosine_grouped_workspace.argtypes = [_i32, _i64]
_lib.fpo_cosine_grouped_workspace.restype = _sz
_lib.fpo_cosine_grouped.argtypes = [_i32, _i64, _i32, ctypes.POINTER(_vp), ctypes.POINTER(_vp),
                                    _vp, _vp, _sz, _vp]
_lib.fpo_cosine_grouped.restype = _i32
_lib.fpo_layer_grad_cosine_workspace.argtypes = [_i32, _i64, _i64]
_lib.fpo_layer_grad_cosine_workspace.restype = _sz
_lib.fpo_layer_grad_cosine_grouped.argtypes = [_i32, _i64, _i64, _i64, _i32, _vp,
                                               ctypes.POINTER(_vp), ctypes.POINTER(_vp),
                                               ctypes.POINTER(_vp), _vp, _vp, _sz, _vp]
_lib.fpo_layer_grad_cosine_grouped.restype = _i32
_lib.fpo_norm_ratio_workspace.argtypes = [_i32, _i64]
_lib.fpo_norm_ratio_workspace.restype = _sz
_lib.fpo_norm_ratio.argtypes = [_i32, _i64, _i32, ctypes.POINTER(_vp), _i32, ctypes.POINTER(_vp),
                                ctypes.c_double, _vp, _vp, _sz, _vp]
_lib.fpo_norm_ratio.restype = _i32
_lib.fpo_h2d_copy.argtypes = [_i32, ctypes.POINTER(_vp), ctypes.POINTER(_vp),
                              ctypes.POINTER(_sz), _vp]
_lib.fpo_h2d_copy.restype = _i32
_lib.fpo_testing_direct_fixup_rows.argtypes = [ctypes.POINTER(ErrorSignalDesc), _vp, _vp]
_lib.fpo_testing_direct_fixup_rows.restype = _i64
_lib.fpo_testing_kernel_launches.argtypes = []
_lib.fpo_testing_kernel_launches.restype = ctypes.c_uint64
_lib.fpo_testing_set_gemm_variant.argtypes = [_i32]
_lib.fpo_testing_set_gemm_variant.restype = _i32


class FpoError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {status_string(code)}")
        self.code = code


def status_string(code: int) -> str:
    return _lib.fpo_status_string(int(code)).decode()


def abi_version() -> int:
    return _lib.fpo_abi_version()


def set_wait_limit_ns(ns: int) -> None:
    _lib.fpo_set_wait_limit_ns(int(ns))


def kernel_launches() -> int:
    """fpo_testing_kernel_launches: kernels this library has launched in this process."""
    return int(_lib.fpo_testing_kernel_launches())


def set_gemm_variant(variant: int) -> int:
    """fpo_testing_set_gemm_variant: 0 single-CTA, 1 CTA-pair tiles, 2 CTA-pair tiles with a
    256 x 512 projection (the default); a negative value only reads the current setting.  Returns the setting in
    force before the call."""
    if variant < 0:
        cur = _lib.fpo_testing_set_gemm_variant(0)
        _lib.fpo_testing_set_gemm_variant(cur)
        return cur
    return _lib.fpo_testing_set_gemm_variant(int(variant))


def _check(code: int, where: str) -> None:
    if code != OK:
        raise FpoError(code, where)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return F32
    raise TypeError(f"unsupported dtype {t.dtype}; libfpo takes bfloat16 or float32")


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libfpo takes CUDA tensors")
    if not t.is_contiguous():
        raise ValueError("libfpo takes contiguous tensors")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _nbytes(t: torch.Tensor) -> int:
    return t.numel() * t.element_size()


def _workspace(nbytes: int, device) -> torch.Tensor:
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


# --------------------------------------------------------------------------- error signal
def error_signal_desc(T, d, V, dtype=BF16, *, eps=1e-6, min_rms=0.5, loss_scale=None, t_chunk=0,
                      stage_events=None, algo=ES_AUTO, per_chunk_events=False):
    """fpo_error_signal_desc; ``stage_events`` is None or torch.cuda.Event objects that have
    been recorded once (so their CUDA handles exist): STAGE_EVENTS of them, or with
    ``per_chunk_events`` stage_event_count() of them (every token chunk's stages)."""
    s = (1.0 / T if T > 0 else 1.0) if loss_scale is None else loss_scale
    d = ErrorSignalDesc(int(T), int(d), int(V), int(dtype), float(eps), float(min_rms), float(s),
                        int(algo), int(t_chunk), None, 1 if per_chunk_events else 0)
    if stage_events is not None:
        need = stage_event_count(d)
        if len(stage_events) != need:
            raise ValueError(f"stage_events needs {need} events")
        ev = (_vp * need)(*[e.cuda_event for e in stage_events])
        d.stage_events = ctypes.cast(ev, ctypes.POINTER(_vp))
        d._keep = ev
    return d


def stage_event_count(desc: ErrorSignalDesc) -> int:
    """fpo_error_signal_stage_events: events the descriptor's stage-event layout needs."""
    return int(_lib.fpo_error_signal_stage_events(ctypes.byref(desc)))


def error_signal_workspace(desc: ErrorSignalDesc) -> int:
    return int(_lib.fpo_error_signal_workspace(ctypes.byref(desc)))


def error_signal(h, norm_w, W_U, targets, g_out, *, eps=1e-6, min_rms=0.5, loss_scale=None,
                 t_chunk=0, lse_out=None, loss_out=None, workspace=None, stream=None,
                 stage_events=None, algo=ES_AUTO, per_chunk_events=False):
    """fpo_error_signal: g~ = final-RMSNorm VJP of (softmax(z) - 1_y) W_U into ``g_out``.

    Returns the workspace tensor (its first word holds the device status).
    """
    T, d = h.shape
    V = W_U.shape[0]
    desc = error_signal_desc(T, d, V, _dtype_code(h), eps=eps, min_rms=min_rms,
                             loss_scale=loss_scale, t_chunk=t_chunk, stage_events=stage_events,
                             algo=algo, per_chunk_events=per_chunk_events)
    need = error_signal_workspace(desc)
    if workspace is None:
        workspace = _workspace(need, h.device)
    rc = _lib.fpo_error_signal(ctypes.byref(desc), _ptr(h), _ptr(norm_w), _ptr(W_U), _ptr(targets),
                               _ptr(g_out), _ptr(lse_out), _ptr(loss_out), _ptr(workspace),
                               _nbytes(workspace), _stream(stream))
    _check(rc, "fpo_error_signal")
    return workspace


def direct_fixup_rows(h, W_U, workspace, *, t_chunk=0, algo=ES_AUTO, stream=None) -> int:
    """fpo_testing_direct_fixup_rows: rows of the last token chunk of the latest error_signal
    call on ``workspace`` that the direct algorithm recomputed (-1: not the direct algorithm)."""
    T, d = h.shape
    desc = error_signal_desc(T, d, W_U.shape[0], _dtype_code(h), t_chunk=t_chunk, algo=algo)
    return int(_lib.fpo_testing_direct_fixup_rows(ctypes.byref(desc), _ptr(workspace),
                                                  _stream(stream)))


# --------------------------------------------------------------------------- layer update
def layer_update_workspace() -> int:
    return int(_lib.fpo_layer_update_workspace())


def layer_update(g, A, lr, *, W_master=None, W_out=None, G_out=None, workspace=None, stream=None):
    """fpo_layer_update: G = g~^T A ; W_master -= lr G ; W_out = cast(W_master)."""
    T, d = g.shape
    d_ff = A.shape[1]
    if workspace is None:
        workspace = _workspace(layer_update_workspace(), g.device)
    rc = _lib.fpo_layer_update(T, d, d_ff, _dtype_code(g), _ptr(g), _ptr(A), float(lr),
                               _ptr(W_master), _ptr(W_out), _ptr(G_out), _ptr(workspace),
                               _nbytes(workspace), _stream(stream))
    _check(rc, "fpo_layer_update")
    return workspace


def _ptr_array(ts, n):
    if ts is None:
        return None
    arr = (_vp * n)()
    for i, t in enumerate(ts):
        arr[i] = None if t is None else _ptr(t).value
    return arr


def layer_update_grouped(g, As, lr, *, W_masters=None, W_outs=None, G_outs=None, workspace=None,
                         stream=None):
    """fpo_layer_update_grouped over len(As) target layers in one launch."""
    n = len(As)
    T, d = g.shape
    d_ff = As[0].shape[1]
    if workspace is None:
        workspace = _workspace(layer_update_workspace(), g.device)
    rc = _lib.fpo_layer_update_grouped(n, T, d, d_ff, _dtype_code(g), _ptr(g), _ptr_array(As, n),
                                       float(lr), _ptr_array(W_masters, n), _ptr_array(W_outs, n),
                                       _ptr_array(G_outs, n), _ptr(workspace), _nbytes(workspace),
                                       _stream(stream))
    _check(rc, "fpo_layer_update_grouped")
    return workspace


def layer_update_grouped_signals(gs, As, lr, *, W_masters=None, W_outs=None, G_outs=None,
                                 workspace=None, stream=None):
    """fpo_layer_update_grouped_signals: layer l uses its own signal gs[l]."""
    n = len(As)
    T, d = gs[0].shape
    d_ff = As[0].shape[1]
    if workspace is None:
        workspace = _workspace(layer_update_workspace(), gs[0].device)
    rc = _lib.fpo_layer_update_grouped_signals(
        n, T, d, d_ff, _dtype_code(gs[0]), _ptr_array(gs, n), _ptr_array(As, n), float(lr),
        _ptr_array(W_masters, n), _ptr_array(W_outs, n), _ptr_array(G_outs, n), _ptr(workspace),
        _nbytes(workspace), _stream(stream))
    _check(rc, "fpo_layer_update_grouped_signals")
    return workspace


def optimizer_desc(kind=OPT_ADAMW, *, lr=1e-4, momentum=0.9, beta1=0.9, beta2=0.999, eps=1e-8,
                   weight_decay=0.01, clip=CLIP_STEP, clip_frac=0.01, step=1):
    return OptimizerDesc(int(kind), int(clip), float(lr), float(momentum), float(beta1),
                         float(beta2), float(eps), float(weight_decay), float(clip_frac), int(step))


def layer_optimize_workspace(n_layers, d, d_ff) -> int:
    return int(_lib.fpo_layer_optimize_workspace(int(n_layers), int(d), int(d_ff)))


def layer_optimize_grouped(gs, As, opt, W_masters, *, W_outs=None, states1=None, states2=None,
                           workspace=None, stream=None):
    """fpo_layer_optimize_grouped: G_l = g_l^T A_l, relative clip, optimizer step."""
    n = len(As)
    T, d = gs[0].shape
    d_ff = As[0].shape[1]
    if workspace is None:
        workspace = _workspace(layer_optimize_workspace(n, d, d_ff), gs[0].device)
    rc = _lib.fpo_layer_optimize_grouped(
        n, T, d, d_ff, _dtype_code(gs[0]), _ptr_array(gs, n), _ptr_array(As, n), ctypes.byref(opt),
        _ptr_array(W_masters, n), _ptr_array(W_outs, n), _ptr_array(states1, n),
        _ptr_array(states2, n), _ptr(workspace), _nbytes(workspace), _stream(stream))
    _check(rc, "fpo_layer_optimize_grouped")
    return workspace


def gate_up_signals(g, W3_init, a, b, dA, dB, *, workspace=None, stream=None):
    """fpo_gate_up_signals: SwiGLU W1/W2 signals through the cached W3_init feedback."""
    T, d = g.shape
    d_ff = W3_init.shape[1]
    if workspace is None:
        workspace = _workspace(layer_update_workspace(), g.device)
    rc = _lib.fpo_gate_up_signals(T, d, d_ff, _dtype_code(g), _ptr(g), _ptr(W3_init), _ptr(a),
                                  _ptr(b), _ptr(dA), _ptr(dB), _ptr(workspace), _nbytes(workspace),
                                  _stream(stream))
    _check(rc, "fpo_gate_up_signals")
    return workspace


def layer_signals(g, g_outs, *, m=None, gamma_post=None, x=None, gamma_pre=None, eps=1e-6,
                  min_rms=0.5, stream=None):
    """fpo_layer_signals: g_outs[l] = pre-MLP VJP at x[l] of (post-FFN VJP at m[l] of g);
    m / gamma_post and x / gamma_pre are lists with one entry per layer, or None."""
    n = len(g_outs)
    T, d = g.shape

    def arr(ts):
        if ts is None:
            return None
        if len(ts) != n:
            raise ValueError("one entry per layer expected")
        return _ptr_array(ts, n)

    rc = _lib.fpo_layer_signals(n, T, d, _dtype_code(g), _ptr(g), arr(m), arr(gamma_post), arr(x),
                                arr(gamma_pre), float(eps), float(min_rms), _ptr_array(g_outs, n),
                                _stream(stream))
    _check(rc, "fpo_layer_signals")
    return g_outs


def rmsnorm_vjp(g, x, gamma, g_out, *, eps=1e-6, min_rms=0.5, stream=None):
    """fpo_rmsnorm_vjp: the RMSNorm Jacobian (with the min-RMS clamp) applied to g at x."""
    T, d = x.shape
    rc = _lib.fpo_rmsnorm_vjp(T, d, _dtype_code(x), _ptr(g), _ptr(x), _ptr(gamma), float(eps),
                              float(min_rms), _ptr(g_out), _stream(stream))
    _check(rc, "fpo_rmsnorm_vjp")
    return g_out


# --------------------------------------------------------------------------- cosine
def cosine_workspace(n: int) -> int:
    return int(_lib.fpo_cosine_workspace(int(n)))


def cosine(X, Y, out=None, *, workspace=None, stream=None):
    """fpo_cosine: returns a device fp64 tensor [<X,Y>, |X|^2, |Y|^2, cos]."""
    n = X.numel()
    if out is None:
        out = torch.empty(4, dtype=torch.float64, device=X.device)
    if workspace is None:
        workspace = _workspace(cosine_workspace(n), X.device)
    rc = _lib.fpo_cosine(n, _dtype_code(X), _ptr(X), _ptr(Y), _ptr(out), _ptr(workspace),
                         _nbytes(workspace), _stream(stream))
    _check(rc, "fpo_cosine")
    return out


def cosine_grouped_workspace(n_layers: int, n: int) -> int:
    return int(_lib.fpo_cosine_grouped_workspace(int(n_layers), int(n)))


def cosine_grouped(X, Y, out=None, *, workspace=None, stream=None):
    """fpo_cosine_grouped: per layer [<X_l,Y_l>, |X_l|^2, |Y_l|^2, cos_l] as a device fp64
    tensor [len(X), 4]; X and Y are lists of same-size tensors of one dtype."""
    n_layers = len(X)
    if n_layers != len(Y) or n_layers == 0:
        raise ValueError("X and Y need one tensor per layer")
    n = X[0].numel()
    if any(t.numel() != n for t in list(X) + list(Y)):
        raise ValueError("every X_l and Y_l must have the same number of elements")
    if any(t.dtype != X[0].dtype for t in list(X) + list(Y)):
        raise TypeError("X and Y share one dtype")
    if out is None:
        out = torch.empty(n_layers, 4, dtype=torch.float64, device=X[0].device)
    if workspace is None:
        workspace = _workspace(cosine_grouped_workspace(n_layers, n), X[0].device)
    xarr = (_vp * n_layers)(*[_ptr(t) for t in X])
    yarr = (_vp * n_layers)(*[_ptr(t) for t in Y])
    rc = _lib.fpo_cosine_grouped(n_layers, n, _dtype_code(X[0]), xarr, yarr, _ptr(out),
                                 _ptr(workspace), _nbytes(workspace), _stream(stream))
    _check(rc, "fpo_cosine_grouped")
    return out


def layer_grad_cosine_workspace(n_layers: int, d: int, d_ff: int) -> int:
    return int(_lib.fpo_layer_grad_cosine_workspace(int(n_layers), int(d), int(d_ff)))


def layer_grad_cosine_grouped(g, As, Ys, G_outs, out=None, *, workspace=None, stream=None):
    """fpo_layer_grad_cosine_grouped: G_outs[l] = g^T As[l] and, per layer,
    [<G_l,Y_l>, |G_l|^2, |Y_l|^2, cos_l] as a device fp64 tensor [len(As), 4]."""
    n = len(As)
    if n == 0 or n != len(Ys) or n != len(G_outs):
        raise ValueError("As, Ys and G_outs need one tensor per layer")
    T, d = g.shape
    d_ff = As[0].shape[1]
    if out is None:
        out = torch.empty(n, 4, dtype=torch.float64, device=g.device)
    if workspace is None:
        workspace = _workspace(layer_grad_cosine_workspace(n, d, d_ff), g.device)
    arr = lambda ts: (_vp * n)(*[_ptr(t) for t in ts])  # noqa: E731
    rc = _lib.fpo_layer_grad_cosine_grouped(n, T, d, d_ff, _dtype_code(g), _ptr(g), arr(As),
                                            arr(Ys), arr(G_outs), _ptr(out), _ptr(workspace),
                                            _nbytes(workspace), _stream(stream))
    _check(rc, "fpo_layer_grad_cosine_grouped")
    return out


def norm_ratio_workspace(n_layers: int, n: int) -> int:
    return int(_lib.fpo_norm_ratio_workspace(int(n_layers), int(n)))


def norm_ratio(G, W, rel_step=0.01, out=None, *, workspace=None, stream=None):
    """fpo_norm_ratio: per layer [||G_l||^2, ||W_l||^2, ||G_l||/||W_l||, rel_step/ratio] as a
    device fp64 tensor [len(G), 4]; G and W are lists of same-size tensors."""
    n_layers = len(G)
    if n_layers != len(W) or n_layers == 0:
        raise ValueError("G and W need one tensor per layer")
    n = G[0].numel()
    if any(t.numel() != n for t in list(G) + list(W)):
        raise ValueError("every G_l and W_l must have the same number of elements")
    if any(t.dtype != G[0].dtype for t in G) or any(t.dtype != W[0].dtype for t in W):
        raise TypeError("the G_l share one dtype and the W_l share one dtype")
    if out is None:
        out = torch.empty(n_layers, 4, dtype=torch.float64, device=G[0].device)
    if workspace is None:
        workspace = _workspace(norm_ratio_workspace(n_layers, n), G[0].device)
    garr = (_vp * n_layers)(*[_ptr(t) for t in G])
    warr = (_vp * n_layers)(*[_ptr(t) for t in W])
    rc = _lib.fpo_norm_ratio(n_layers, n, _dtype_code(G[0]), garr, _dtype_code(W[0]), warr,
                             float(rel_step), _ptr(out), _ptr(workspace), _nbytes(workspace),
                             _stream(stream))
    _check(rc, "fpo_norm_ratio")
    return out


MAX_COPY_BUFFERS = 64


def h2d_copy(dsts, srcs, *, stream=None):
    """fpo_h2d_copy: copy page-locked host tensors srcs[i] into device tensors dsts[i]
    (contiguous, equal byte sizes) by SM loads, one kernel launch per MAX_COPY_BUFFERS
    pairs."""
    if len(dsts) != len(srcs):
        raise ValueError("h2d_copy takes as many destinations as sources")
    for d_t, s_t in zip(dsts, srcs):
        if s_t.is_cuda or not s_t.is_contiguous():
            raise ValueError("h2d_copy sources are contiguous host tensors")
        if d_t.numel() * d_t.element_size() != s_t.numel() * s_t.element_size():
            raise ValueError("h2d_copy source and destination sizes differ")
    for c in range(0, len(srcs), MAX_COPY_BUFFERS):
        ds, ss = dsts[c:c + MAX_COPY_BUFFERS], srcs[c:c + MAX_COPY_BUFFERS]
        n = len(ss)
        darr = (_vp * n)(*[_ptr(t).value for t in ds])
        sarr = (_vp * n)(*[t.data_ptr() for t in ss])
        barr = (_sz * n)(*[t.numel() * t.element_size() for t in ss])
        _check(_lib.fpo_h2d_copy(n, darr, sarr, barr, _stream(stream)), "fpo_h2d_copy")


def get_device_status(workspace, stream=None) -> int:
    """fpo_get_device_status: synchronise, read and clear the workspace's status word."""
    return int(_lib.fpo_get_device_status(_ptr(workspace), _stream(stream)))
