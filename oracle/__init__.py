"""fp64 CPU oracle for Hidden Decoding's expansion and Stream-Factorized Attention.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this package.  The
product library (``paper_2607_08186_gb300``) never imports it and shares no
code with it.

The arithmetic lives in ``hdsfa_oracle.c`` (plain C, fp64, OpenMP over rows);
this module compiles it with gcc on first use and marshals torch/numpy arrays
to it.  Every function takes float tensors of any dtype and upcasts them to
fp64 exactly (bf16 -> fp64 is exact).

Citations (Hidden Decoding paper): Eq. 1 (expansion, and its adjoint into the n
tables), Eq. 2 (the final-stream positions the loss reads), Eq. 3 (token / stream
index), Eq. 4 (intra-stream mask), Fig. 2 (full and local cross-stream masks),
Sec. 2 "Setup" (standard causal softmax attention, grouped K/V heads per
Table 6), Sec. 3.1 (final-stream-only layers: the final-stream queries against all
keys), Sec. 3.2 (decoding with the expanded KV cache).  The backward is the
derivative of that forward (the paper does not write it out).

Pinned by ``tests/test_oracle_pins.py``; see the header of ``hdsfa_oracle.c``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np
import torch

WITHIN, CROSS, LOCAL = 0, 1, 2

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "hdsfa_oracle.c")
_LIB = os.path.join(_HERE, "libhdsfa_oracle.so")
_lock = threading.Lock()
_lib = None


class _Dims(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int64), ("L", ctypes.c_int64), ("n", ctypes.c_int64),
                ("Hq", ctypes.c_int64), ("Hkv", ctypes.c_int64), ("Dh", ctypes.c_int64),
                ("mode", ctypes.c_int), ("window", ctypes.c_int64), ("scale", ctypes.c_double)]


def build(force: bool = False) -> str:
    """Compile the oracle shared library with gcc (fp64, -O2, OpenMP)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            I64 = ctypes.c_int64
            lib.hdo_visible.restype = ctypes.c_int
            lib.hdo_visible.argtypes = [I64, I64, I64, ctypes.c_int, I64]
            lib.hdo_token_index.restype = I64
            lib.hdo_token_index.argtypes = [I64, I64]
            lib.hdo_stream_index.restype = I64
            lib.hdo_stream_index.argtypes = [I64, I64]
            lib.hdo_expand.restype = I64
            lib.hdo_expand.argtypes = [P, P, P, I64, I64, I64, I64, I64]
            lib.hdo_expand_bwd.restype = None
            lib.hdo_expand_bwd.argtypes = [P, P, P, I64, I64, I64, I64, I64]
            lib.hdo_select_final.restype = None
            lib.hdo_select_final.argtypes = [P, P, I64, I64, I64, I64]
            lib.hdo_select_final_bwd.restype = None
            lib.hdo_select_final_bwd.argtypes = [P, P, I64, I64, I64, I64]
            D = ctypes.POINTER(_Dims)
            lib.hdo_sfa_fwd.argtypes = [P, P, P, P, P, D]
            lib.hdo_sfa_fwd_rows.argtypes = [P, P, P, D, I64, P, P, P]
            lib.hdo_sfa_bwd_q_rows.argtypes = [P, P, P, P, D, I64, P, P, P, P]
            lib.hdo_sfa_bwd_kv_rows.argtypes = [P, P, P, P, P, P, D, I64, P, P, P]
            lib.hdo_sfa_bwd.argtypes = [P, P, P, P, P, P, P, P, P, D]
            lib.hdo_sfa_bwd_jacobian.argtypes = [P, P, P, P, P, P, P, D]
            lib.hdo_decode.restype = I64
            lib.hdo_decode.argtypes = [P, P, P, P, P, P, I64, I64, I64, I64, I64, I64, ctypes.c_double,
                                       ctypes.c_int, I64]
            lib.hdo_kv_append.restype = I64
            lib.hdo_kv_append.argtypes = [P, P, P, I64, I64, I64, I64]
            lib.hdo_num_threads.restype = ctypes.c_int
            _lib = lib
    return _lib


def num_threads() -> int:
    return int(_load().hdo_num_threads())


def _f64(t) -> np.ndarray:
    if isinstance(t, torch.Tensor):
        t = t.detach().to("cpu", torch.float64).numpy()
    return np.ascontiguousarray(t, dtype=np.float64)


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _dims(q, k, n, mode, scale, window):
    B, nL, Hq, Dh = q.shape
    Hkv = k.shape[2]
    if nL % n or Hq % Hkv:
        raise ValueError("bad shapes")
    if scale is None or scale <= 0:
        scale = 1.0 / float(Dh) ** 0.5
    return _Dims(B, nL // n, n, Hq, Hkv, Dh, int(mode), int(window), float(scale))


def visible(t: int, tk: int, n: int, mode: int, window: int = 0) -> bool:
    """Eq. 4 / Fig. 2 mask for 1-indexed expanded positions t (query) and tk (key)."""
    return bool(_load().hdo_visible(t, tk, n, mode, window))


def token_index(t: int, n: int) -> int:
    """Eq. 3: i(t) = ceil(t / n), 1-indexed."""
    return int(_load().hdo_token_index(t, n))


def stream_index(t: int, n: int) -> int:
    """Eq. 3: s(t) = ((t - 1) mod n) + 1, 1-indexed."""
    return int(_load().hdo_stream_index(t, n))


def expand(tables: torch.Tensor, ids: torch.Tensor):
    """Eq. 1 gather on bf16 bit patterns.  tables [n][V][D] bf16, ids [B][L] int32.

    Returns (out bf16 [B][n*L][D], count of out-of-range ids); an out-of-range id
    gives zero rows."""
    n, V, D = tables.shape
    B, L = ids.shape
    tb = np.ascontiguousarray(tables.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))
    ib = np.ascontiguousarray(ids.detach().cpu().to(torch.int32).numpy())
    out = np.empty((B, n * L, D), dtype=np.uint16)
    bad = _load().hdo_expand(_ptr(tb), _ptr(ib), _ptr(out), B, L, n, V, D)
    return torch.from_numpy(out.view(np.int16)).view(torch.bfloat16), int(bad)


def expand_bwd(dX: torch.Tensor, ids: torch.Tensor, n: int, V: int, dE: torch.Tensor | None = None):
    """Adjoint of the Eq. 1 gather: dE[k][x] += sum over tokens with id x of dX at
    stream k.  dX [B][n*L][D] (any float dtype, upcast to fp64), ids [B][L] int32.
    Returns dE fp64 [n][V][D] (a copy of `dE` plus the sums, or the sums alone)."""
    B, nL, D = dX.shape
    L = nL // n
    xd = _f64(dX)
    ib = np.ascontiguousarray(ids.detach().cpu().to(torch.int32).numpy())
    out = np.zeros((n, V, D), dtype=np.float64) if dE is None else _f64(dE).copy()
    _load().hdo_expand_bwd(_ptr(xd), _ptr(ib), _ptr(out), B, L, n, V, D)
    return torch.from_numpy(out)


def select_final(X: torch.Tensor, n: int):
    """Eq. 2 final-stream rows: Y[b][i] = X[b][i*n + n-1] (bf16 bit copy)."""
    B, nL, D = X.shape
    L = nL // n
    xb = np.ascontiguousarray(X.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))
    out = np.empty((B, L, D), dtype=np.uint16)
    _load().hdo_select_final(_ptr(xb), _ptr(out), B, L, n, D)
    return torch.from_numpy(out.view(np.int16)).view(torch.bfloat16)


def select_final_bwd(dY: torch.Tensor, n: int):
    """Adjoint of select_final: dY [B][L][D] bf16 back to the final-stream rows of a
    zero [B][n*L][D] tensor."""
    B, L, D = dY.shape
    yb = np.ascontiguousarray(dY.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))
    out = np.empty((B, n * L, D), dtype=np.uint16)
    _load().hdo_select_final_bwd(_ptr(yb), _ptr(out), B, L, n, D)
    return torch.from_numpy(out.view(np.int16)).view(torch.bfloat16)


def decode(q, k_cache, v_cache, lens, n: int, mode: int, scale: float | None = None, window: int = 0):
    """Decoding step over the expanded KV cache (Sec. 3.2 "Inference Cost"): the new
    token's n positions attend under the layer's mask to the lens[b] * n cached positions.
    q [B][n][Hq][Dh]; k_cache / v_cache [B][Lcap*n][Hkv][Dh]; lens [B] tokens in the cache
    (new token included).  Returns (O fp64 [B][n][Hq][Dh], LSE fp64 [B][Hq][n], number of
    sequences with lens outside [1, Lcap], which get zero rows and LSE = -inf)."""
    qa, ka, va = _f64(q), _f64(k_cache), _f64(v_cache)
    B, nq, Hq, Dh = qa.shape
    if nq != n or ka.shape[1] % n:
        raise ValueError("bad shapes")
    Lcap, Hkv = ka.shape[1] // n, ka.shape[2]
    if scale is None or scale <= 0:
        scale = 1.0 / float(Dh) ** 0.5
    la = np.ascontiguousarray(torch.as_tensor(lens).to(torch.int32).cpu().numpy())
    o = np.empty_like(qa)
    lse = np.empty((B, Hq, n))
    bad = _load().hdo_decode(_ptr(qa), _ptr(ka), _ptr(va), _ptr(la), _ptr(o), _ptr(lse), B, Lcap, n, Hq,
                             Hkv, Dh, float(scale), int(mode), int(window))
    return torch.from_numpy(o), torch.from_numpy(lse), int(bad)


def kv_append(new_rows, cache, lens, n: int):
    """The new token's n K (or V) rows into the cache at positions (lens[b]-1)*n + s,
    on bf16 bit patterns.  new_rows [B][n][Hkv][Dh], cache [B][Lcap*n][Hkv][Dh] (a copy is
    returned).  Returns (cache', number of sequences with lens outside [1, Lcap])."""
    B, nn, Hkv, Dh = new_rows.shape
    Lcap = cache.shape[1] // n
    nb = np.ascontiguousarray(new_rows.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))
    cb = np.ascontiguousarray(cache.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)).copy()
    la = np.ascontiguousarray(torch.as_tensor(lens).to(torch.int32).cpu().numpy())
    bad = _load().hdo_kv_append(_ptr(nb), _ptr(cb), _ptr(la), B, Lcap, n, Hkv * Dh)
    return torch.from_numpy(cb.view(np.int16)).view(torch.bfloat16), int(bad)


def sfa_fwd(q, k, v, n: int, mode: int, scale: float | None = None, window: int = 0):
    """Masked softmax attention forward over the expanded sequence.

    q [B][nL][Hq][Dh], k/v [B][nL][Hkv][Dh].  Returns (O fp64 same shape as q,
    LSE fp64 [B][Hq][nL])."""
    qa, ka, va = _f64(q), _f64(k), _f64(v)
    d = _dims(qa, ka, n, mode, scale, window)
    o = np.empty_like(qa)
    lse = np.empty((d.B, d.Hq, d.n * d.L), dtype=np.float64)
    _load().hdo_sfa_fwd(_ptr(qa), _ptr(ka), _ptr(va), _ptr(o), _ptr(lse), ctypes.byref(d))
    return torch.from_numpy(o), torch.from_numpy(lse)


def sfa_fwd_rows(q, k, v, n, mode, rows, scale=None, window=0):
    """Forward for selected rows; rows is an int64 [R][3] array of (b, h, p).
    Returns (O rows fp64 [R][Dh], LSE fp64 [R])."""
    qa, ka, va = _f64(q), _f64(k), _f64(v)
    d = _dims(qa, ka, n, mode, scale, window)
    r = np.ascontiguousarray(np.asarray(rows, dtype=np.int64).reshape(-1, 3))
    o = np.empty((r.shape[0], d.Dh))
    lse = np.empty((r.shape[0],))
    _load().hdo_sfa_fwd_rows(_ptr(qa), _ptr(ka), _ptr(va), ctypes.byref(d), r.shape[0], _ptr(r),
                             _ptr(o), _ptr(lse))
    return torch.from_numpy(o), torch.from_numpy(lse)


def _final_full(x, n):
    """[B][L][H][Dh] -> [B][nL][H][Dh] fp64 with x at the final-stream rows t*n + n-1, zero elsewhere."""
    xa = _f64(x)
    B, L, H, Dh = xa.shape
    full = np.zeros((B, n * L, H, Dh))
    full[:, n - 1::n] = xa
    return full


def sfa_fwd_final(q, k, v, n: int, mode: int, scale: float | None = None, window: int = 0):
    """Final-stream queries (the rows the loss reads, Eq. 2; the final-stream-only layers of
    Sec. 3.1): q [B][L][Hq][Dh] are the queries of positions t*n + n-1, attending to k / v
    [B][nL][Hkv][Dh] under the layer's mask.  By definition these are the forward's rows
    t*n + n-1.  Returns (O fp64 [B][L][Hq][Dh], LSE fp64 [B][Hq][L])."""
    qf = _final_full(q, n)
    B, nL, Hq, Dh = qf.shape
    L = nL // n
    rows = np.array([(b, h, t * n + n - 1) for b in range(B) for h in range(Hq) for t in range(L)], dtype=np.int64)
    o_rows, lse_rows = sfa_fwd_rows(qf, k, v, n, mode, rows, scale, window)
    o = o_rows.numpy().reshape(B, Hq, L, Dh).transpose(0, 2, 1, 3)
    return torch.from_numpy(np.ascontiguousarray(o)), lse_rows.reshape(B, Hq, L)


def sfa_bwd_final(q, k, v, dout, n: int, mode: int, scale: float | None = None, window: int = 0):
    """Gradients of the final-stream problem: the full backward with the queries and output
    gradients of every other position set to zero (a row with zero dO adds nothing to any
    gradient, and rows are independent).  Returns (dQ fp64 [B][L][Hq][Dh], dK, dV fp64
    [B][nL][Hkv][Dh])."""
    dq, dk, dv = sfa_bwd(_final_full(q, n), k, v, _final_full(dout, n), n, mode, scale, window)
    return dq[:, n - 1::n].contiguous(), dk, dv


def sfa_bwd(q, k, v, dout, n, mode, scale=None, window=0):
    """Full backward (reduced Jacobian form).  Returns (dQ, dK, dV) fp64."""
    qa, ka, va, da = _f64(q), _f64(k), _f64(v), _f64(dout)
    d = _dims(qa, ka, n, mode, scale, window)
    dq, dk, dv = np.empty_like(qa), np.empty_like(ka), np.empty_like(va)
    lse = np.empty((d.B, d.Hq, d.n * d.L))
    D = np.empty_like(lse)
    _load().hdo_sfa_bwd(_ptr(qa), _ptr(ka), _ptr(va), _ptr(da), _ptr(dq), _ptr(dk), _ptr(dv),
                        _ptr(lse), _ptr(D), ctypes.byref(d))
    return torch.from_numpy(dq), torch.from_numpy(dk), torch.from_numpy(dv)


def sfa_bwd_jacobian(q, k, v, dout, n, mode, scale=None, window=0):
    """Backward with the softmax Jacobian formed explicitly (small inputs only)."""
    qa, ka, va, da = _f64(q), _f64(k), _f64(v), _f64(dout)
    d = _dims(qa, ka, n, mode, scale, window)
    dq, dk, dv = np.empty_like(qa), np.empty_like(ka), np.empty_like(va)
    _load().hdo_sfa_bwd_jacobian(_ptr(qa), _ptr(ka), _ptr(va), _ptr(da), _ptr(dq), _ptr(dk),
                                 _ptr(dv), ctypes.byref(d))
    return torch.from_numpy(dq), torch.from_numpy(dk), torch.from_numpy(dv)


def sfa_bwd_q_rows(q, k, v, dout, n, mode, rows, scale=None, window=0):
    """dQ and the row statistics (LSE, D = sum P*dP) for rows (b, h, p)."""
    qa, ka, va, da = _f64(q), _f64(k), _f64(v), _f64(dout)
    d = _dims(qa, ka, n, mode, scale, window)
    r = np.ascontiguousarray(np.asarray(rows, dtype=np.int64).reshape(-1, 3))
    dq = np.empty((r.shape[0], d.Dh))
    lse = np.empty((r.shape[0],))
    D = np.empty((r.shape[0],))
    _load().hdo_sfa_bwd_q_rows(_ptr(qa), _ptr(ka), _ptr(va), _ptr(da), ctypes.byref(d),
                               r.shape[0], _ptr(r), _ptr(dq), _ptr(lse), _ptr(D))
    return torch.from_numpy(dq), torch.from_numpy(lse), torch.from_numpy(D)


def sfa_bwd_kv_rows(q, k, v, dout, n, mode, kv_rows, scale=None, window=0):
    """dK and dV for key rows (b, g, p').  Computes the statistics of every query
    row that can see one of the requested keys first (query rows at or after the
    earliest requested key, in the heads of the requested groups)."""
    qa, ka, va, da = _f64(q), _f64(k), _f64(v), _f64(dout)
    d = _dims(qa, ka, n, mode, scale, window)
    r = np.ascontiguousarray(np.asarray(kv_rows, dtype=np.int64).reshape(-1, 3))
    nL, grp = d.n * d.L, d.Hq // d.Hkv
    lse = np.zeros((d.B, d.Hq, nL))
    D = np.zeros_like(lse)
    need = []
    for b, g in sorted({(int(x[0]), int(x[1])) for x in r}):
        p0 = int(r[(r[:, 0] == b) & (r[:, 1] == g), 2].min())
        for h in range(g * grp, (g + 1) * grp):
            need.extend((b, h, p) for p in range(p0, nL))
    need = np.asarray(need, dtype=np.int64).reshape(-1, 3)
    if need.shape[0]:
        _, l_rows, D_rows = sfa_bwd_q_rows(qa, ka, va, da, n, mode, need, d.scale, window)
        lse[need[:, 0], need[:, 1], need[:, 2]] = l_rows.numpy()
        D[need[:, 0], need[:, 1], need[:, 2]] = D_rows.numpy()
    dk = np.empty((r.shape[0], d.Dh))
    dv = np.empty((r.shape[0], d.Dh))
    _load().hdo_sfa_bwd_kv_rows(_ptr(qa), _ptr(ka), _ptr(va), _ptr(da), _ptr(lse), _ptr(D),
                                ctypes.byref(d), r.shape[0], _ptr(r), _ptr(dk), _ptr(dv))
    return torch.from_numpy(dk), torch.from_numpy(dv)
