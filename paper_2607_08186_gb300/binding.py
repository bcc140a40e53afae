"""Thin ctypes binding over libhdsfa.so (C ABI in include/hdsfa.h).

Argument marshalling only: every step of the computation runs in the CUDA
kernels of libhdsfa.so.  Functions keep the C names and take torch CUDA tensors
(plain device memory); sizes are read from the tensor shapes.  There is no
CPU fallback: if the library is missing or a call fails, an exception is raised.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from .inputs import WITHIN, CROSS, LOCAL  # noqa: F401

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libhdsfa.so")
_lock = threading.Lock()
_lib = None

HD_OK = 0
HD_DEVBIT_INDEX = 1
HD_DEVBIT_TIMEOUT = 2


class HdError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {hd_status_string(code)} (code {code})")
        self.code = code


def lib():
    """Load libhdsfa.so (built by ``build.build()``); raise if it is missing."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(f"libhdsfa.so is not built ({LIB_PATH}); run "
                                   "paper_2607_08186_gb300.build.build() first")
            L = ctypes.CDLL(LIB_PATH)
            P, I, F, Z = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
            L.hd_selftest_bounded_wait.restype = I
            L.hd_selftest_bounded_wait.argtypes = [P, P, P]
            L.hd_expand_embed.restype = I
            L.hd_expand_embed.argtypes = [P, P, P, I, I, I, I, I, P, P]
            L.hd_expand_embed_bwd_workspace_bytes.restype = Z
            L.hd_expand_embed_bwd_workspace_bytes.argtypes = [I, I]
            L.hd_expand_embed_bwd.restype = I
            L.hd_expand_embed_bwd.argtypes = [P, P, P, I, I, I, I, I, P, Z, P, P]
            L.hd_expand_embed_bwd_plan.restype = I
            L.hd_expand_embed_bwd_plan.argtypes = [P, I, I, I, P, Z, P, P]
            L.hd_expand_embed_bwd_apply.restype = I
            L.hd_expand_embed_bwd_apply.argtypes = [P, P, I, I, I, I, I, P, Z, P]
            L.hd_select_final_stream.restype = I
            L.hd_select_final_stream.argtypes = [P, P, I, I, I, I, P]
            L.hd_select_final_stream_bwd.restype = I
            L.hd_select_final_stream_bwd.argtypes = [P, P, I, I, I, I, P]
            L.sfa_fwd_final.restype = I
            L.sfa_fwd_final.argtypes = [P, P, P, P, P, I, I, I, I, I, I, F, I, I, P, P]
            L.sfa_bwd_final_workspace_bytes.restype = Z
            L.sfa_bwd_final_workspace_bytes.argtypes = [I, I, I, I, I, I, I]
            L.sfa_bwd_final.restype = I
            L.sfa_bwd_final.argtypes = [P, P, P, P, P, P, P, P, P, I, I, I, I, I, I, F, I, I, P, Z, P, P]
            L.sfa_decode_workspace_bytes.restype = Z
            L.sfa_decode_workspace_bytes.argtypes = [I, I, I, I, I, I, I, I]
            L.sfa_decode.restype = I
            L.sfa_decode.argtypes = [P, P, P, P, P, P, I, I, I, I, I, I, I, F, I, I, P, Z, P, P]
            L.sfa_kv_append.restype = I
            L.sfa_kv_append.argtypes = [P, P, P, P, P, I, I, I, I, I, P, P]
            L.sfa_fwd.restype = I
            L.sfa_fwd.argtypes = [P, P, P, P, P, I, I, I, I, I, I, F, I, I, P, P]
            L.sfa_bwd_workspace_bytes.restype = Z
            L.sfa_bwd_workspace_bytes.argtypes = [I, I, I, I, I, I, I]
            L.sfa_bwd.restype = I
            L.sfa_bwd.argtypes = [P, P, P, P, P, P, P, P, P, I, I, I, I, I, I, F, I, I, P, Z, P, P]
            L.sfa_bwd_prep.restype = I
            L.sfa_bwd_prep.argtypes = [P, P, P, I, I, I, I, I, I, I, P, Z, P]
            L.sfa_bwd_row_terms.restype = I
            L.sfa_bwd_row_terms.argtypes = [P, P, P, I, I, I, I, I, I, I, P, Z, P]
            L.sfa_bwd_clear.restype = I
            L.sfa_bwd_clear.argtypes = [I, I, I, I, I, I, I, P, Z, P]
            L.sfa_bwd_main.restype = I
            L.sfa_bwd_main.argtypes = [P, P, P, P, P, P, I, I, I, I, I, I, F, I, I, P, Z, P, P]
            L.sfa_bwd_finalize.restype = I
            L.sfa_bwd_finalize.argtypes = [P, I, I, I, I, I, I, F, I, P, Z, P]
            L.sfa_bwd_noalloc.restype = I
            L.sfa_bwd_noalloc.argtypes = [P, P, P, P, P, P, P, P, P, I, I, I, I, I, I, F, I, I, P, P]
            L.hd_status_string.restype = ctypes.c_char_p
            L.hd_status_string.argtypes = [I]
            _lib = L
    return _lib


def hd_status_string(code: int) -> str:
    return lib().hd_status_string(int(code)).decode()


def hd_selftest_bounded_wait(dev_status, dev_result, stream=None):
    """Diagnostic: one warp's bounded wait on a barrier nothing arrives on runs out
    (about a second); HD_DEVBIT_TIMEOUT lands in dev_status, 0 in dev_result."""
    _check(lib().hd_selftest_bounded_wait(_p(dev_status), _p(dev_result), _stream(stream)),
           "hd_selftest_bounded_wait")


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(code: int, where: str):
    if code != HD_OK:
        raise HdError(code, where)


def hd_expand_embed(tables, ids, out, dev_status=None, stream=None):
    """out[b][t*n+s] = tables[s][ids[b][t]]  (Eq. 1).  tables [n][V][D] bf16,
    ids [B][L] int32, out [B][n*L][D] bf16."""
    n, V, D = tables.shape
    B, L = ids.shape
    _check(lib().hd_expand_embed(_p(tables), _p(ids), _p(out), B, L, n, V, D, _p(dev_status),
                                 _stream(stream)), "hd_expand_embed")
    return out


def hd_expand_embed_bwd_workspace_bytes(B, L) -> int:
    return int(lib().hd_expand_embed_bwd_workspace_bytes(B, L))


def hd_expand_embed_bwd(dout, ids, dtables, workspace, dev_status=None, stream=None):
    """dtables[s][v] += sum of dout[b][t*n+s] over tokens with ids[b][t] = v (adjoint of Eq. 1).
    dout [B][n*L][D] bf16, ids [B][L] int32, dtables [n][V][D] float32 (accumulated in place),
    workspace: uint8 CUDA tensor of >= hd_expand_embed_bwd_workspace_bytes(B, L) bytes."""
    n, V, D = dtables.shape
    B, L = ids.shape
    if dout.shape[1] != n * L:
        raise ValueError("dout.shape[1] must be n * L")
    _check(lib().hd_expand_embed_bwd(_p(dout), _p(ids), _p(dtables), B, L, n, V, D, _p(workspace),
                                     _wsb(workspace), _p(dev_status), _stream(stream)),
           "hd_expand_embed_bwd")
    return dtables


def hd_expand_embed_bwd_plan(ids, V, workspace, dev_status=None, stream=None):
    """The id-only part of hd_expand_embed_bwd: tokens sorted by id and each id's run,
    written into workspace for later hd_expand_embed_bwd_apply calls."""
    B, L = ids.shape
    _check(lib().hd_expand_embed_bwd_plan(_p(ids), B, L, int(V), _p(workspace), _wsb(workspace),
                                          _p(dev_status), _stream(stream)), "hd_expand_embed_bwd_plan")


def hd_expand_embed_bwd_apply(dout, dtables, workspace, L, stream=None):
    """dtables += the expansion backward of dout following the plan held in workspace
    (built by hd_expand_embed_bwd_plan for the same ids, B = dout.shape[0], L and V)."""
    n, V, D = dtables.shape
    B = dout.shape[0]
    if dout.shape[1] != n * L:
        raise ValueError("dout.shape[1] must be n * L")
    _check(lib().hd_expand_embed_bwd_apply(_p(dout), _p(dtables), B, L, n, V, D, _p(workspace),
                                           _wsb(workspace), _stream(stream)), "hd_expand_embed_bwd_apply")
    return dtables


def hd_select_final_stream(x, y, n, stream=None):
    """y[b][t] = x[b][t*n + n-1], the rows the loss reads (Eq. 2).  x [B][n*L][D], y [B][L][D] bf16."""
    B, L, D = y.shape
    if x.shape[1] != n * L:
        raise ValueError("x.shape[1] must be n * L")
    _check(lib().hd_select_final_stream(_p(x), _p(y), B, L, n, D, _stream(stream)),
           "hd_select_final_stream")
    return y


def hd_select_final_stream_bwd(dy, dx, n, stream=None):
    """dx[b][t*n + n-1] = dy[b][t], zero elsewhere.  dy [B][L][D], dx [B][n*L][D] bf16."""
    B, L, D = dy.shape
    if dx.shape[1] != n * L:
        raise ValueError("dx.shape[1] must be n * L")
    _check(lib().hd_select_final_stream_bwd(_p(dy), _p(dx), B, L, n, D, _stream(stream)),
           "hd_select_final_stream_bwd")
    return dx


def _attn_dims(q, k, n):
    B, nL, Hq, Dh = q.shape
    if nL % n:
        raise ValueError("q.shape[1] must be n * L")
    return B, nL // n, Hq, k.shape[2], Dh


def sfa_fwd(q, k, v, o, lse, n, mode, softmax_scale=0.0, window=0, dev_status=None, stream=None):
    """SFA forward (Eq. 4 / Fig. 2 masks).  q,o [B][nL][Hq][Dh], k,v [B][nL][Hkv][Dh] bf16;
    lse [B][Hq][nL] float32."""
    B, L, Hq, Hkv, Dh = _attn_dims(q, k, n)
    _check(lib().sfa_fwd(_p(q), _p(k), _p(v), _p(o), _p(lse), B, L, n, Hq, Hkv, Dh,
                         float(softmax_scale), int(mode), int(window), _p(dev_status),
                         _stream(stream)), "sfa_fwd")
    return o, lse


def sfa_bwd_workspace_bytes(B, L, n, Hq, Hkv, Dh, mode) -> int:
    return int(lib().sfa_bwd_workspace_bytes(B, L, n, Hq, Hkv, Dh, int(mode)))


def sfa_bwd(q, k, v, o, lse, dout, dq, dk, dv, n, mode, workspace, softmax_scale=0.0, window=0,
            dev_status=None, stream=None):
    """SFA backward.  workspace: uint8 CUDA tensor of >= sfa_bwd_workspace_bytes bytes."""
    B, L, Hq, Hkv, Dh = _attn_dims(q, k, n)
    _check(lib().sfa_bwd(_p(q), _p(k), _p(v), _p(o), _p(lse), _p(dout), _p(dq), _p(dk), _p(dv),
                         B, L, n, Hq, Hkv, Dh, float(softmax_scale), int(mode), int(window),
                         _p(workspace), _wsb(workspace),
                         _p(dev_status), _stream(stream)), "sfa_bwd")
    return dq, dk, dv


def _final_dims(q, k):
    B, L, Hq, Dh = q.shape
    if k.shape[1] % L:
        raise ValueError("k.shape[1] must be n * L")
    return B, L, k.shape[1] // L, Hq, k.shape[2], Dh


def sfa_fwd_final(q, k, v, o, lse, mode, softmax_scale=0.0, window=0, dev_status=None, stream=None):
    """Final-stream queries only (Eq. 2 rows; Sec. 3.1 final-stream-only layers): q, o [B][L][Hq][Dh],
    k, v [B][n*L][Hkv][Dh] bf16, lse [B][Hq][L] float32."""
    B, L, n, Hq, Hkv, Dh = _final_dims(q, k)
    _check(lib().sfa_fwd_final(_p(q), _p(k), _p(v), _p(o), _p(lse), B, L, n, Hq, Hkv, Dh, float(softmax_scale),
                               int(mode), int(window), _p(dev_status), _stream(stream)), "sfa_fwd_final")
    return o, lse


def sfa_bwd_final_workspace_bytes(B, L, n, Hq, Hkv, Dh, mode) -> int:
    return int(lib().sfa_bwd_final_workspace_bytes(B, L, n, Hq, Hkv, Dh, int(mode)))


def sfa_bwd_final(q, k, v, o, lse, dout, dq, dk, dv, mode, workspace, softmax_scale=0.0, window=0,
                  dev_status=None, stream=None):
    """Backward of sfa_fwd_final: dq [B][L][Hq][Dh], dk, dv [B][n*L][Hkv][Dh] (overwritten)."""
    B, L, n, Hq, Hkv, Dh = _final_dims(q, k)
    _check(lib().sfa_bwd_final(_p(q), _p(k), _p(v), _p(o), _p(lse), _p(dout), _p(dq), _p(dk), _p(dv), B, L, n, Hq,
                               Hkv, Dh, float(softmax_scale), int(mode), int(window), _p(workspace),
                               _wsb(workspace), _p(dev_status), _stream(stream)), "sfa_bwd_final")
    return dq, dk, dv


def sfa_decode_workspace_bytes(B, max_tokens, n, Hq, Hkv, Dh, mode, window=0) -> int:
    return int(lib().sfa_decode_workspace_bytes(B, max_tokens, n, Hq, Hkv, Dh, int(mode), int(window)))


def sfa_decode(q, k_cache, v_cache, lens, o, n, mode, workspace, max_tokens=None, lse=None, softmax_scale=0.0,
               window=0, dev_status=None, stream=None):
    """One decoding step (Sec. 3.2): the new token's n positions q [B][n][Hq][Dh] against
    the cache k_cache / v_cache [B][Lcap*n][Hkv][Dh] holding lens[b] tokens (int32 CUDA
    tensor [B]); o [B][n][Hq][Dh] bf16, lse [B][Hq][n] float32 or None.  max_tokens bounds
    every lens[b] (default: the cache capacity Lcap)."""
    B, nq, Hq, Dh = q.shape
    if nq != n or k_cache.shape[1] % n:
        raise ValueError("q.shape[1] must be n and k_cache.shape[1] a multiple of n")
    Lcap, Hkv = k_cache.shape[1] // n, k_cache.shape[2]
    T = Lcap if max_tokens is None else int(max_tokens)
    _check(lib().sfa_decode(_p(q), _p(k_cache), _p(v_cache), _p(lens), _p(o), _p(lse), B, T, Lcap, n, Hq, Hkv,
                            Dh, float(softmax_scale), int(mode), int(window), _p(workspace), _wsb(workspace),
                            _p(dev_status), _stream(stream)), "sfa_decode")
    return o


def sfa_kv_append(k_new, v_new, k_cache, v_cache, lens, n, dev_status=None, stream=None):
    """k_cache[b][(lens[b]-1)*n + s] = k_new[b][s] (and v): the new token's n K/V rows."""
    B, nn, Hkv, Dh = k_new.shape
    if nn != n:
        raise ValueError("k_new.shape[1] must be n")
    Lcap = k_cache.shape[1] // n
    _check(lib().sfa_kv_append(_p(k_new), _p(v_new), _p(k_cache), _p(v_cache), _p(lens), B, Lcap, n, Hkv, Dh,
                               _p(dev_status), _stream(stream)), "sfa_kv_append")


SFA_BWD_NOALLOC_MAX_BYTES = 64 << 20


def sfa_bwd_noalloc(q, k, v, o, lse, dout, dq, dk, dv, n, mode, softmax_scale=0.0, window=0,
                    dev_status=None, stream=None):
    """SFA backward with the library's fixed device workspace (no allocation anywhere,
    at most SFA_BWD_NOALLOC_MAX_BYTES of workspace).  Calls on one device share that
    workspace: order them (one stream, or events) so that none overlap."""
    B, L, Hq, Hkv, Dh = _attn_dims(q, k, n)
    _check(lib().sfa_bwd_noalloc(_p(q), _p(k), _p(v), _p(o), _p(lse), _p(dout), _p(dq), _p(dk),
                                 _p(dv), B, L, n, Hq, Hkv, Dh, float(softmax_scale), int(mode),
                                 int(window), _p(dev_status), _stream(stream)), "sfa_bwd_noalloc")
    return dq, dk, dv


def _wsb(ws):
    return ws.numel() * ws.element_size()


def sfa_bwd_prep(o, dout, lse, n, mode, workspace, Hkv, stream=None):
    """Phase 1 of sfa_bwd: delta = rowsum(dO * O), lse * log2(e), zeroed dQ accumulator."""
    B, nL, Hq, Dh = o.shape
    _check(lib().sfa_bwd_prep(_p(o), _p(dout), _p(lse), B, nL // n, n, Hq, Hkv, Dh, int(mode),
                              _p(workspace), _wsb(workspace), _stream(stream)), "sfa_bwd_prep")


def sfa_bwd_row_terms(o, dout, lse, n, mode, workspace, Hkv, stream=None):
    """The delta / lse half of sfa_bwd_prep (no zeroing of the dQ accumulator)."""
    B, nL, Hq, Dh = o.shape
    _check(lib().sfa_bwd_row_terms(_p(o), _p(dout), _p(lse), B, nL // n, n, Hq, Hkv, Dh, int(mode),
                                   _p(workspace), _wsb(workspace), _stream(stream)), "sfa_bwd_row_terms")


def sfa_bwd_clear(B, L, n, Hq, Hkv, Dh, mode, workspace, stream=None):
    """The other half: zero the workspace's fp32 dQ accumulator (independent of the forward)."""
    _check(lib().sfa_bwd_clear(B, L, n, Hq, Hkv, Dh, int(mode), _p(workspace), _wsb(workspace),
                               _stream(stream)), "sfa_bwd_clear")


def sfa_bwd_main(q, k, v, dout, dk, dv, n, mode, workspace, softmax_scale=0.0, window=0,
                 dev_status=None, stream=None):
    """Phase 2 of sfa_bwd: dK, dV and the fp32 dQ accumulator."""
    B, L, Hq, Hkv, Dh = _attn_dims(q, k, n)
    _check(lib().sfa_bwd_main(_p(q), _p(k), _p(v), _p(dout), _p(dk), _p(dv), B, L, n, Hq, Hkv, Dh,
                              float(softmax_scale), int(mode), int(window), _p(workspace),
                              _wsb(workspace), _p(dev_status), _stream(stream)), "sfa_bwd_main")


def sfa_bwd_finalize(dq, n, mode, workspace, Hkv, softmax_scale=0.0, stream=None):
    """Phase 3 of sfa_bwd: dq = bf16(scale * accumulator)."""
    B, nL, Hq, Dh = dq.shape
    _check(lib().sfa_bwd_finalize(_p(dq), B, nL // n, n, Hq, Hkv, Dh, float(softmax_scale), int(mode),
                                  _p(workspace), _wsb(workspace), _stream(stream)), "sfa_bwd_finalize")
