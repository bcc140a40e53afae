"""Host-only checks of the C ABI: the library builds, loads and exports every
symbol include/hdsfa.h declares; argument validation answers before anything is
launched (no GPU needed, no compute call reaches a kernel)."""
import ctypes
import os
import re

import pytest

from paper_2607_08186_gb300 import binding, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "hdsfa.h")


@pytest.fixture(scope="module")
def lib():
    build.build()
    return binding.lib()


def _declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s*([a-z_][a-z0-9_]*)\s*\(",
                                 src, flags=re.M)))


def test_header_declares_the_entry_points():
    names = _declared_functions()
    for want in ("hd_expand_embed", "sfa_fwd", "sfa_bwd", "sfa_bwd_workspace_bytes", "hd_status_string"):
        assert want in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared_functions():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    for code in range(7):
        assert binding.hd_status_string(code).startswith("HD_")
    assert "unknown" in binding.hd_status_string(99)


FAKE = 1 << 20  # 16-byte aligned non-null address; never dereferenced (validation fails first)


def _fwd(lib, B=1, L=8, n=2, Hq=4, Hkv=2, Dh=64, mode=0, window=0, ptr=FAKE):
    P = ctypes.c_void_p
    return lib.sfa_fwd(P(ptr), P(ptr), P(ptr), P(ptr), P(ptr), B, L, n, Hq, Hkv, Dh, 0.0, mode,
                       window, None, None)


def test_fwd_validation(lib):
    assert _fwd(lib, B=0) == 1
    assert _fwd(lib, L=-1) == 1
    assert _fwd(lib, n=0) == 1
    assert _fwd(lib, Hq=6, Hkv=4) == 1          # Hq % Hkv != 0
    assert _fwd(lib, mode=7) == 1
    assert _fwd(lib, mode=2, window=0) == 1     # LOCAL needs a window
    assert _fwd(lib, ptr=FAKE + 8) == 1         # misaligned
    assert _fwd(lib, ptr=0) == 1                # null
    assert _fwd(lib, Dh=96) == 2                # unsupported head dim
    assert _fwd(lib, Dh=32) == 2


def test_naive_within_mode_validation(lib):
    # the naive intra-stream schedule runs on the head-dim-128 tcgen05 kernels only, and
    # takes the CROSS problem's workspace; final-stream and decode calls reject it
    P, Z, F = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_float
    assert _fwd(lib, mode=3, Dh=64) == 2
    assert _fwd(lib, mode=3, Dh=256) == 2
    assert _fwd(lib, mode=3, Dh=128, ptr=FAKE + 8) == 1  # misaligned: rejected before any launch
    assert binding.sfa_bwd_workspace_bytes(1, 100, 4, 8, 2, 128, 3) == binding.sfa_bwd_workspace_bytes(
        1, 100, 4, 8, 2, 128, 1)
    assert binding.sfa_bwd_workspace_bytes(1, 100, 4, 8, 2, 64, 3) == 0
    assert lib.sfa_bwd_final_workspace_bytes(1, 64, 4, 8, 2, 128, 3) == 0
    assert lib.sfa_fwd_final(P(FAKE), P(FAKE), P(FAKE), P(FAKE), P(FAKE), 1, 64, 4, 8, 2, 128, F(0.0), 3, 0,
                             None, None) == 2
    assert binding.sfa_decode_workspace_bytes(1, 64, 4, 8, 2, 128, 3) == 0


def test_bwd_workspace_size(lib):
    B, L, n, Hq, Hkv, Dh = 1, 100, 4, 8, 2, 128
    ws = binding.sfa_bwd_workspace_bytes(B, L, n, Hq, Hkv, Dh, 0)
    rows = B * n * L * Hq
    assert ws >= rows * Dh * 4 + rows * 4
    assert binding.sfa_bwd_workspace_bytes(0, L, n, Hq, Hkv, Dh, 0) == 0
    assert binding.sfa_bwd_workspace_bytes(B, L, n, Hq, Hkv, 80, 0) == 0


def test_bwd_validation(lib):
    P = ctypes.c_void_p
    a = [P(FAKE)] * 9
    need = binding.sfa_bwd_workspace_bytes(1, 8, 2, 4, 2, 64, 0)
    assert lib.sfa_bwd(*a, 1, 8, 2, 4, 2, 64, 0.0, 0, 0, None, 0, None, None) == 4           # no workspace
    assert lib.sfa_bwd(*a, 1, 8, 2, 4, 2, 64, 0.0, 0, 0, P(FAKE), need - 1, None, None) == 4  # too small
    assert lib.sfa_bwd(*a, 1, 8, 2, 4, 2, 64, 0.0, 0, 0, P(FAKE + 16), need, None, None) == 4  # not 256-aligned
    assert lib.sfa_bwd(*a, 1, 8, 2, 5, 2, 64, 0.0, 0, 0, P(FAKE), need, None, None) == 1
    assert lib.sfa_bwd(*a, 1, 8, 2, 4, 2, 32, 0.0, 0, 0, P(FAKE), need, None, None) == 2


def test_expand_validation(lib):
    P = ctypes.c_void_p
    assert lib.hd_expand_embed(P(FAKE), P(FAKE), P(FAKE), 1, 4, 2, 16, 12, None, None) == 1  # D % 8
    assert lib.hd_expand_embed(P(FAKE), P(FAKE), P(FAKE + 2), 1, 4, 2, 16, 16, None, None) == 1
    assert lib.hd_expand_embed(P(FAKE), None, P(FAKE), 1, 4, 2, 16, 16, None, None) == 1
    assert lib.hd_expand_embed(P(FAKE), P(FAKE), P(FAKE), 1, 4, 0, 16, 16, None, None) == 1


def test_expand_bwd_workspace_size(lib):
    # sorted keys (u64, padded to a power of two, at least one 4096-key block), two
    # run lists of 16-byte records, one per token, two counters (16 bytes), and up to
    # 16384 tokens the rank counts, one u64 per token and 256-key tile
    assert lib.hd_expand_embed_bwd_workspace_bytes(1, 1) == 4096 * 8 + 2 * 16 + 16 + 8
    assert lib.hd_expand_embed_bwd_workspace_bytes(1, 4096) == 4096 * 8 + 2 * 4096 * 16 + 16 + 16 * 4096 * 8
    assert lib.hd_expand_embed_bwd_workspace_bytes(3, 1500) == 8192 * 8 + 2 * 4500 * 16 + 16 + 18 * 4500 * 8
    assert lib.hd_expand_embed_bwd_workspace_bytes(4, 4500) == 32768 * 8 + 2 * 18000 * 16 + 16  # bitonic
    assert lib.hd_expand_embed_bwd_workspace_bytes(0, 4) == 0
    assert lib.hd_expand_embed_bwd_workspace_bytes(1 << 16, 1 << 15) == 0  # B*L must stay below 2^31


def test_expand_bwd_validation(lib):
    P, Z = ctypes.c_void_p, ctypes.c_size_t
    ws = lib.hd_expand_embed_bwd_workspace_bytes(1, 4)

    def call(dout=FAKE, ids=FAKE, de=FAKE, B=1, L=4, n=2, V=16, D=16, w=FAKE, wb=ws):
        return lib.hd_expand_embed_bwd(P(dout), P(ids), P(de), B, L, n, V, D, P(w), Z(wb), None, None)

    assert call(D=12) == 1                     # D % 8
    assert call(dout=FAKE + 2) == 1            # misaligned
    assert call(ids=0) == 1                    # null ids
    assert call(ids=FAKE + 2) == 1             # ids not 4-byte aligned
    assert call(n=0) == 1 and call(V=0) == 1 and call(B=0) == 1
    assert call(wb=ws - 8) == 4                # workspace too small
    assert call(w=0) == 4
    assert call(n=1 << 20, D=1 << 12) == 2     # n*D beyond 2^31


def test_expand_bwd_plan_apply_validation(lib):
    P, Z = ctypes.c_void_p, ctypes.c_size_t
    ws = lib.hd_expand_embed_bwd_workspace_bytes(1, 4)
    assert lib.hd_expand_embed_bwd_plan(None, 1, 4, 16, P(FAKE), Z(ws), None, None) == 1
    assert lib.hd_expand_embed_bwd_plan(P(FAKE), 1, 4, 0, P(FAKE), Z(ws), None, None) == 1
    assert lib.hd_expand_embed_bwd_plan(P(FAKE), 1, 4, 16, P(FAKE), Z(ws - 1), None, None) == 4
    assert lib.hd_expand_embed_bwd_plan(P(FAKE), 1, 4, 16, P(FAKE + 8), Z(ws), None, None) == 4
    assert lib.hd_expand_embed_bwd_apply(P(FAKE), P(FAKE), 1, 4, 2, 16, 12, P(FAKE), Z(ws), None) == 1
    assert lib.hd_expand_embed_bwd_apply(P(FAKE), P(FAKE), 1, 4, 2, 16, 16, P(FAKE), Z(ws - 1), None) == 4
    assert lib.hd_expand_embed_bwd_apply(P(FAKE), P(FAKE + 4), 1, 4, 2, 16, 16, P(FAKE), Z(ws), None) == 1


def test_select_final_validation(lib):
    P = ctypes.c_void_p
    for f in (lib.hd_select_final_stream, lib.hd_select_final_stream_bwd):
        assert f(P(FAKE), P(FAKE), 1, 4, 2, 12, None) == 1
        assert f(P(FAKE + 4), P(FAKE), 1, 4, 2, 16, None) == 1
        assert f(P(FAKE), None, 1, 4, 2, 16, None) == 1
        assert f(P(FAKE), P(FAKE), 1, 0, 2, 16, None) == 1


def test_decode_workspace_and_validation(lib):
    P, Z, F = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_float
    need = lib.sfa_decode_workspace_bytes(1, 100, 4, 32, 8, 128, 1, 0)
    assert need > 0
    assert lib.sfa_decode_workspace_bytes(1, 100, 4, 32, 8, 96, 1, 0) == 0     # Dh 96
    assert lib.sfa_decode_workspace_bytes(1, 100, 4, 32, 6, 128, 1, 0) == 0    # Hq % Hkv
    assert lib.sfa_decode_workspace_bytes(1, 100, 4, 32, 8, 128, 2, 0) == 0    # LOCAL needs a window

    def call(q=FAKE, lens=FAKE, lse=None, B=1, T=100, Lcap=100, n=4, Hq=32, Hkv=8, Dh=128, mode=1, w=0,
             ws=FAKE, wsb=need):
        return lib.sfa_decode(P(q), P(FAKE), P(FAKE), P(lens), P(FAKE), P(lse), B, T, Lcap, n, Hq, Hkv, Dh, F(0.0),
                              mode, w, P(ws), Z(wsb), None, None)

    assert call(q=FAKE + 2) == 1
    assert call(lens=0) == 1 and call(lens=FAKE + 2) == 1
    assert call(lse=FAKE + 2) == 1
    assert call(T=101) == 1                    # max_tokens beyond the capacity
    assert call(Hkv=6) == 1 and call(B=0) == 1 and call(mode=3) == 1
    assert call(Dh=96) == 2
    assert call(wsb=need - 1) == 4
    assert call(ws=0) == 4


def test_kv_append_validation(lib):
    P = ctypes.c_void_p
    assert lib.sfa_kv_append(P(FAKE), P(FAKE), P(FAKE), P(FAKE), None, 1, 10, 4, 8, 128, None, None) == 1
    assert lib.sfa_kv_append(P(FAKE), P(FAKE + 8), P(FAKE), P(FAKE), P(FAKE), 1, 10, 4, 8, 128, None, None) == 1
    assert lib.sfa_kv_append(P(FAKE), P(FAKE), P(FAKE), P(FAKE), P(FAKE), 1, 0, 4, 8, 128, None, None) == 1
    assert lib.sfa_kv_append(P(FAKE), P(FAKE), P(FAKE), P(FAKE), P(FAKE), 1, 10, 4, 8, 12, None, None) == 1


def test_final_stream_validation(lib):
    P, Z, F = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_float
    assert lib.sfa_bwd_final_workspace_bytes(1, 64, 4, 8, 2, 128, 1) > 0
    assert lib.sfa_bwd_final_workspace_bytes(1, 64, 4, 8, 2, 256, 1) > 0
    assert lib.sfa_bwd_final_workspace_bytes(1, 64, 4, 8, 2, 80, 1) == 0     # unsupported head dim
    assert lib.sfa_fwd_final(P(FAKE), P(FAKE), P(FAKE), P(FAKE), P(FAKE + 4), 1, 64, 4, 8, 2, 128, F(0.0), 1, 0,
                             None, None) == 1
    assert lib.sfa_fwd_final(P(FAKE), P(FAKE), P(FAKE), P(FAKE), P(FAKE), 1, 64, 4, 8, 3, 128, F(0.0), 1, 0,
                             None, None) == 1
    assert lib.sfa_fwd_final(P(FAKE), P(FAKE), P(FAKE), P(FAKE), P(FAKE), 1, 64, 4, 8, 2, 96, F(0.0), 1, 0,
                             None, None) == 2
    a = [P(FAKE)] * 9
    assert lib.sfa_bwd_final(*a, 1, 64, 4, 8, 2, 96, F(0.0), 1, 0, P(FAKE), Z(1 << 30), None, None) == 2
    assert lib.sfa_bwd_final(*a, 1, 64, 4, 8, 2, 128, F(0.0), 1, 0, P(FAKE), Z(16), None, None) == 4
    assert lib.sfa_bwd_final(*a, 1, 64, 4, 8, 2, 256, F(0.0), 1, 0, P(FAKE), Z(16), None, None) == 4
