"""fp64 CPU oracle for the FPO pseudogradient update (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
and reference legs import this package.  It wraps ``oracle.c`` (plain C, fp64,
OpenMP over independent tokens) through ctypes and numpy; it shares no code
with the CUDA library and never imports it.

Each function follows one passage of the paper:

* :func:`error_signal`  Sec. 3.1 steps 2-4, Eq. (gproj), App. E Eq. (rmsnorm-vjp)
  with the min-RMS clamp.
* :func:`rmsnorm_vjp`   App. E Eq. (rmsnorm-vjp) at any norm (the per-layer post-FFN
  norm of OLMo-2 / Gemma 3, Sec. 3.2).
* :func:`layer_signal`  Sec. 3.1 step 4, Sec. 3.2: the layer-specific signal composed with
  the post-feedforward and / or pre-MLP RMSNorm Jacobians.
* :func:`gate_up_signals`  Sec. 3.1 step 5, Eq. (errh): W1/W2 signals of a SwiGLU MLP.
* :func:`pseudograd`    Sec. 3.1 step 5, Eq. (w3update).
* :func:`sgd_update`    App. A, fp32 master weights cast to bf16.
* :func:`optimizer_step`  Sec. 3.1 AdamW / SGD with momentum, App. A relative clip.
* :func:`cosine`        Sec. 2.2, Eq. (cosine).
* :func:`norm_ratio`    App. C update-magnitude ratios, Sec. C.2 implied SGD rate.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")

F32, BF16, F64 = 0, 1, 2

_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so with gcc (-O2, OpenMP)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", _SRC,
           "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = ctypes.CDLL(_LIB_PATH)
    vp, i64, dbl, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_double, ctypes.c_int
    lib.oracle_error_signal.argtypes = [i64, i64, i64, i32, vp, vp, vp, vp, dbl, dbl, dbl,
                                        vp, i64, vp, vp, vp, vp, vp, vp]
    lib.oracle_error_signal.restype = i32
    lib.oracle_rmsnorm_vjp.argtypes = [i64, i64, i32, vp, i32, vp, vp, dbl, dbl, vp]
    lib.oracle_rmsnorm_vjp.restype = i32
    lib.oracle_layer_signal.argtypes = [i64, i64, i32, vp, i32, vp, vp, vp, vp, dbl, dbl, vp]
    lib.oracle_layer_signal.restype = i32
    lib.oracle_gate_up_signals.argtypes = [i64, i64, i64, i32, vp, vp, vp, vp, vp, vp]
    lib.oracle_gate_up_signals.restype = i32
    lib.oracle_pseudograd.argtypes = [i64, i64, i64, i32, vp, i32, vp, vp, vp, i64, vp]
    lib.oracle_pseudograd.restype = i32
    lib.oracle_sgd_update.argtypes = [i64, vp, vp, dbl, vp, vp]
    lib.oracle_sgd_update.restype = None
    lib.oracle_optimizer_step.argtypes = [i64, i32, dbl, dbl, dbl, dbl, dbl, dbl, i64, i32, dbl,
                                          vp, vp, vp, vp, vp, vp, vp, vp]
    lib.oracle_optimizer_step.restype = dbl
    lib.oracle_f32_to_bf16.argtypes = [i64, vp, vp]
    lib.oracle_f32_to_bf16.restype = None
    lib.oracle_cosine.argtypes = [i64, i32, vp, vp, vp]
    lib.oracle_cosine.restype = None
    lib.oracle_mean_ce.argtypes = [i64, vp, vp]
    lib.oracle_norm_ratio.argtypes = [i64, i64, i32, vp, i32, vp, dbl, vp]
    lib.oracle_norm_ratio.restype = None
    lib.oracle_mean_ce.restype = dbl
    _lib = lib
    return lib


def _typed(a: np.ndarray):
    """Return (dtype code, contiguous array) for fp32 / fp64 / bf16-as-uint16."""
    a = np.ascontiguousarray(a)
    if a.dtype == np.float64:
        return F64, a
    if a.dtype == np.float32:
        return F32, a
    if a.dtype == np.uint16:  # raw bf16 bit patterns
        return BF16, a
    raise TypeError(f"oracle inputs must be float64, float32 or uint16 (bf16 bits), got {a.dtype}")


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def error_signal(h, w, W_U, y, *, eps=1e-6, min_rms=0.5, s=1.0, rows=None, want_e=False):
    """Steps 1-5 of the FPO error signal for every token (or the listed rows).

    ``h`` [T,d], ``w`` [d], ``W_U`` [V,d] share one dtype (float32/float64, or
    uint16 holding bf16 bits); ``y`` int32 [T].  Returns a dict of fp64 arrays:
    rho, lse, zy (target logit), g (= e W_U, Eq. gproj), g_tilde (after the
    final-norm VJP) and optionally e.
    """
    dt, h = _typed(h)
    dtw, w = _typed(w)
    dtu, W_U = _typed(W_U)
    if not (dt == dtw == dtu):
        raise TypeError("h, w and W_U must share one dtype")
    T, d = h.shape
    V = W_U.shape[0]
    y = np.ascontiguousarray(y, dtype=np.int32)
    if rows is None:
        n = T
        rows_arr = None
    else:
        rows_arr = np.ascontiguousarray(rows, dtype=np.int64)
        n = rows_arr.shape[0]
    out = {k: np.zeros(n) for k in ("rho", "lse", "zy")}
    out["g"] = np.zeros((n, d))
    out["g_tilde"] = np.zeros((n, d))
    e = np.zeros((n, V)) if want_e else None
    rc = _load().oracle_error_signal(T, d, V, dt, _ptr(h), _ptr(w), _ptr(W_U), _ptr(y),
                                     eps, min_rms, s, _ptr(rows_arr), n,
                                     _ptr(out["rho"]), _ptr(out["lse"]), _ptr(out["zy"]),
                                     _ptr(out["g"]), _ptr(out["g_tilde"]), _ptr(e))
    if rc == -2:
        raise ValueError("target or row index out of range")
    if rc != 0:
        raise ValueError(f"oracle_error_signal failed ({rc})")
    if want_e:
        out["e"] = e
    return out


def rmsnorm_vjp(g, x, gamma, *, eps=1e-6, min_rms=0.5):
    """App. E Eq. (rmsnorm-vjp) with the min-RMS clamp at norm input x, weight gamma.

    g, x: [T, d]; gamma: [d] (same dtype as x).  Returns fp64 [T, d].
    """
    dtg, g = _typed(g)
    dtx, x = _typed(x)
    dtw, gamma = _typed(gamma)
    if dtw != dtx:
        raise TypeError("x and gamma must share one dtype")
    T, d = x.shape
    if g.shape != x.shape or gamma.shape != (d,):
        raise ValueError("g and x must be [T, d] and gamma [d]")
    out = np.zeros((T, d))
    rc = _load().oracle_rmsnorm_vjp(T, d, dtg, _ptr(g), dtx, _ptr(x), _ptr(gamma), eps, min_rms,
                                    _ptr(out))
    if rc != 0:
        raise ValueError(f"oracle_rmsnorm_vjp failed ({rc})")
    return out


def layer_signal(g, m=None, gamma_post=None, x=None, gamma_pre=None, *, eps=1e-6, min_rms=0.5):
    """Sec. 3.1 step 4 / Sec. 3.2: compose g with the post-feedforward RMSNorm Jacobian at
    the MLP output m (weight gamma_post), then with the pre-MLP RMSNorm Jacobian at its
    input x (weight gamma_pre); a norm given as None is not composed.

    g, m, x: [T, d]; gammas: [d] (m, x and the gammas share one dtype).  Returns fp64 [T, d].
    """
    dtg, g = _typed(g)
    T, d = g.shape
    norms = [a for a in (m, gamma_post, x, gamma_pre) if a is not None]
    if (m is None) != (gamma_post is None) or (x is None) != (gamma_pre is None):
        raise ValueError("each norm needs both its input and its weight")
    typed = [_typed(a) for a in norms]
    if len({t for t, _ in typed}) > 1:
        raise TypeError("norm inputs and weights must share one dtype")
    dtn = typed[0][0] if typed else dtg
    arrs = iter(a for _, a in typed)
    mm = next(arrs) if m is not None else None
    gp = next(arrs) if m is not None else None
    xx = next(arrs) if x is not None else None
    gq = next(arrs) if x is not None else None
    for a in (mm, xx):
        if a is not None and a.shape != (T, d):
            raise ValueError("norm inputs must be [T, d] like g")
    for a in (gp, gq):
        if a is not None and a.shape != (d,):
            raise ValueError("norm weights must be [d]")
    out = np.zeros((T, d))
    rc = _load().oracle_layer_signal(T, d, dtg, _ptr(g), dtn, _ptr(mm), _ptr(gp), _ptr(xx),
                                     _ptr(gq), eps, min_rms, _ptr(out))
    if rc != 0:
        raise ValueError(f"oracle_layer_signal failed ({rc})")
    return out


def gate_up_signals(g, W3_init, a, b):
    """Sec. 3.1 step 5, Eq. (errh), SwiGLU: returns (dA, dB) fp64 [T, d_ff] with
    error_h = g W3_init, dA = error_h * b * silu'(a), dB = error_h * silu(a)."""
    dt, g = _typed(g)
    d2, W3_init = _typed(W3_init)
    d3, a = _typed(a)
    d4, b = _typed(b)
    if not (dt == d2 == d3 == d4):
        raise TypeError("g, W3_init, a and b must share one dtype")
    T, d = g.shape
    d_ff = W3_init.shape[1]
    if W3_init.shape[0] != d or a.shape != (T, d_ff) or b.shape != (T, d_ff):
        raise ValueError("shapes: g [T,d], W3_init [d,d_ff], a and b [T,d_ff]")
    dA = np.zeros((T, d_ff))
    dB = np.zeros((T, d_ff))
    rc = _load().oracle_gate_up_signals(T, d, d_ff, dt, _ptr(g), _ptr(W3_init), _ptr(a), _ptr(b),
                                        _ptr(dA), _ptr(dB))
    if rc != 0:
        raise ValueError(f"oracle_gate_up_signals failed ({rc})")
    return dA, dB


def pseudograd(g_tilde, A, pairs=None):
    """Eq. (w3update): G = g~^T A, [d, d_ff] fp64 (or the listed (i, j) entries)."""
    dtg, g_tilde = _typed(g_tilde)
    dta, A = _typed(A)
    T, d = g_tilde.shape
    d_ff = A.shape[1]
    if A.shape[0] != T:
        raise ValueError("g_tilde and A must have the same number of tokens")
    if pairs is None:
        G = np.zeros((d, d_ff))
        rc = _load().oracle_pseudograd(T, d, d_ff, dtg, _ptr(g_tilde), dta, _ptr(A),
                                       None, None, 0, _ptr(G))
    else:
        ii = np.ascontiguousarray(pairs[0], dtype=np.int64)
        jj = np.ascontiguousarray(pairs[1], dtype=np.int64)
        G = np.zeros(ii.shape[0])
        rc = _load().oracle_pseudograd(T, d, d_ff, dtg, _ptr(g_tilde), dta, _ptr(A),
                                       _ptr(ii), _ptr(jj), ii.shape[0], _ptr(G))
    if rc != 0:
        raise ValueError(f"oracle_pseudograd failed ({rc})")
    return G


def sgd_update(W_master, G, lr):
    """App. A: returns (W_new fp32, W_bf16 bits uint16) for W_master -= lr * G."""
    W = np.ascontiguousarray(W_master, dtype=np.float32)
    G = np.ascontiguousarray(G, dtype=np.float64)
    if W.shape != G.shape:
        raise ValueError("W_master and G must have the same shape")
    W_new = np.empty_like(W)
    W_b = np.empty(W.shape, dtype=np.uint16)
    _load().oracle_sgd_update(W.size, _ptr(W), _ptr(G), float(lr), _ptr(W_new), _ptr(W_b))
    return W_new, W_b


SGD, SGD_MOMENTUM, ADAMW = 0, 1, 2
CLIP_NONE, CLIP_UPDATE, CLIP_GRADIENT = 0, 1, 2


def optimizer_step(W_master, G, *, kind, lr, momentum=0.9, beta1=0.9, beta2=0.999, eps=1e-8,
                   weight_decay=0.01, t=1, clip=CLIP_NONE, frac=0.01, s1=None, s2=None):
    """Sec. 3.1 optimizers on the fp32 master with the App. A relative clip.

    Returns dict(W fp32, W_bf16 uint16, s1 fp32 or None, s2 fp32 or None, scale)."""
    W = np.ascontiguousarray(W_master, dtype=np.float32)
    G = np.ascontiguousarray(G, dtype=np.float64)
    if W.shape != G.shape:
        raise ValueError("W_master and G must have the same shape")
    z = np.zeros(W.shape, dtype=np.float32)
    s1 = z if s1 is None else np.ascontiguousarray(s1, dtype=np.float32)
    s2 = z if s2 is None else np.ascontiguousarray(s2, dtype=np.float32)
    W_new = np.empty_like(W)
    W_b = np.empty(W.shape, dtype=np.uint16)
    s1n = np.empty_like(W) if kind in (SGD_MOMENTUM, ADAMW) else None
    s2n = np.empty_like(W) if kind == ADAMW else None
    scale = _load().oracle_optimizer_step(W.size, kind, lr, momentum, beta1, beta2, eps,
                                          weight_decay, t, clip, frac, _ptr(W), _ptr(G), _ptr(s1),
                                          _ptr(s2), _ptr(W_new), _ptr(W_b), _ptr(s1n), _ptr(s2n))
    return {"W": W_new, "W_bf16": W_b, "s1": s1n, "s2": s2n, "scale": scale}


def f32_to_bf16_bits(x):
    """Round-to-nearest-even fp32 -> bf16, returned as uint16 bit patterns."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    _load().oracle_f32_to_bf16(x.size, _ptr(x), _ptr(out))
    return out


def bf16_bits_to_f64(b):
    """Exact value of bf16 bit patterns as fp64 (plain bit placement)."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def cosine(X, Y):
    """Eq. (cosine): returns (<X,Y>, |X|^2, |Y|^2, cos) in fp64."""
    dtx, X = _typed(X)
    dty, Y = _typed(Y)
    if dtx != dty or X.size != Y.size:
        raise TypeError("X and Y must have the same dtype and size")
    out = np.zeros(4)
    _load().oracle_cosine(X.size, dtx, _ptr(X.reshape(-1)), _ptr(Y.reshape(-1)), _ptr(out))
    return tuple(out)


def norm_ratio(G, W, rel=0.01):
    """App. C: per layer (||G_l||^2, ||W_l||^2, ||G_l||/||W_l||, rel/(||G_l||/||W_l||)) in fp64,
    for lists of same-size arrays G (one dtype) and W (one dtype); returns [L, 4]."""
    if len(G) != len(W):
        raise ValueError("G and W need one array per layer")
    typed_g = [_typed(x) for x in G]
    typed_w = [_typed(x) for x in W]
    n = typed_g[0][1].size if G else 0
    if any(a.size != n for _, a in typed_g + typed_w):
        raise ValueError("every G_l and W_l must have the same size")
    if len({t for t, _ in typed_g}) > 1 or len({t for t, _ in typed_w}) > 1:
        raise TypeError("the G_l share one dtype and the W_l share one dtype")
    g_arr = (ctypes.c_void_p * max(1, len(G)))(*[_ptr(a.reshape(-1)).value for _, a in typed_g])
    w_arr = (ctypes.c_void_p * max(1, len(W)))(*[_ptr(a.reshape(-1)).value for _, a in typed_w])
    out = np.zeros((len(G), 4))
    _load().oracle_norm_ratio(len(G), n, typed_g[0][0] if G else 0, g_arr,
                              typed_w[0][0] if W else 0, w_arr, float(rel), _ptr(out))
    return out


def mean_ce(lse, zy):
    """(1/T) sum_t (lse_t - z_{t,y_t}): the mean cross-entropy."""
    lse = np.ascontiguousarray(lse, dtype=np.float64)
    zy = np.ascontiguousarray(zy, dtype=np.float64)
    return _load().oracle_mean_ce(lse.size, _ptr(lse), _ptr(zy))
