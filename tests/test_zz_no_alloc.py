"""sfa_bwd_noalloc: the SFA backward with the library's fixed device workspace.

The file is collected last, so the GPU test also runs after every other test of
the session (and passes alone in a fresh process too).  The entry point must give
what sfa_bwd gives with a workspace the caller allocates, call after call, while
the fixed array keeps whatever the previous call left in it.
"""
import ctypes

import pytest
import torch

from paper_2607_08186_gb300 import binding, build, inputs
from paper_2607_08186_gb300.inputs import AttnShape, CROSS, LOCAL, WITHIN

import guards
from parity import assert_grads_close, check_status, gpu_fwd

FAKE = 1 << 20  # 16-byte aligned non-null address; never dereferenced (validation fails first)


@pytest.fixture(scope="module")
def lib():
    build.build()
    return binding.lib()


def _noalloc(lib, B, L, n, Hq, Hkv, Dh, mode=0, window=0, ptr=FAKE):
    P = ctypes.c_void_p
    return lib.sfa_bwd_noalloc(*([P(ptr)] * 9), B, L, n, Hq, Hkv, Dh, 0.0, mode, window, None, None)


def test_rejects_sizes_beyond_the_fixed_workspace(lib):
    # B=1, L=4096, n=4, Hq=32, Dh=128: the fp32 dQ accumulator alone is 256 MiB
    assert binding.sfa_bwd_workspace_bytes(1, 4096, 4, 32, 8, 128, WITHIN) > binding.SFA_BWD_NOALLOC_MAX_BYTES
    assert _noalloc(lib, 1, 4096, 4, 32, 8, 128) == 7
    assert binding.hd_status_string(7).startswith("HD_ERR_SCRATCH_LIMIT")
    # argument errors answer like sfa_bwd's, before the array is looked at
    assert _noalloc(lib, 0, 8, 2, 4, 2, 64) == 1
    assert _noalloc(lib, 1, 8, 2, 5, 2, 64) == 1
    assert _noalloc(lib, 1, 8, 2, 4, 2, 64, mode=LOCAL, window=0) == 1
    assert _noalloc(lib, 1, 8, 2, 4, 2, 64, ptr=FAKE + 8) == 1
    assert _noalloc(lib, 1, 8, 2, 4, 2, 32) == 2


# (shape, mode, window); the later calls need less workspace than the first, so the
# array still holds the first call's data past their own.
# The first needs 63.5 MiB of the 64 MiB array (the split workspace's row terms sit at
# its top end; 16 K/V heads give a grid of 512 CTAs, so no head-chunk partial sums).
CALLS = [
    (AttnShape(1, 1000, 4, 32, 16, 128), WITHIN, 0),
    (AttnShape(1, 200, 4, 8, 2, 128), WITHIN, 0),
    (AttnShape(1, 96, 2, 4, 4, 64), CROSS, 0),
    (AttnShape(2, 70, 2, 4, 2, 128), LOCAL, 50),
]


@pytest.mark.gpu
def test_calls_in_a_row_match_sfa_bwd(lib):
    assert max(binding.sfa_bwd_workspace_bytes(s.B, s.L, s.n, s.Hq, s.Hkv, s.Dh, m) for s, m, _ in CALLS) \
        <= binding.SFA_BWD_NOALLOC_MAX_BYTES
    cases = []
    for i, (s, mode, window) in enumerate(CALLS):
        q, k, v, do = inputs.attn_inputs(s, seed=71 + i)
        st = torch.zeros(1, dtype=torch.int32, device="cuda")
        qd, kd, vd, o, lse = gpu_fwd(q, k, v, s.n, mode, 0.0, window, status=st)
        dod = do.cuda()
        ref = [guards.like(qd), guards.like(kd), guards.like(vd)]
        ws = guards.empty((binding.sfa_bwd_workspace_bytes(s.B, s.L, s.n, s.Hq, s.Hkv, s.Dh, mode),), torch.uint8)
        binding.sfa_bwd(qd, kd, vd, o, lse, dod, *ref, s.n, mode, ws, 0.0, window, dev_status=st)
        got = [guards.like(qd, float("nan")), guards.like(kd, float("nan")), guards.like(vd, float("nan"))]
        cases.append((s, mode, window, (qd, kd, vd, o, lse, dod), ref, got, st))
    # Two rounds of back-to-back calls on one stream.  The first noalloc call in this
    # context loads the module that holds the array (the one-time set-up), so the
    # device's free memory is read after the first round: across the second round it
    # must not drop (torch's cache emptied first; any device allocation takes at least a
    # 2 MiB page).
    for rnd in range(2):
        if rnd == 1:
            torch.cuda.synchronize()
            torch.cuda.empty_cache()
            before = torch.cuda.memory_allocated()
            free_before = torch.cuda.mem_get_info()[0]
        for s, mode, window, (qd, kd, vd, o, lse, dod), ref, got, st in cases:
            for t in got:
                t.fill_(float("nan"))
            binding.sfa_bwd_noalloc(qd, kd, vd, o, lse, dod, *got, s.n, mode, 0.0, window, dev_status=st)
        torch.cuda.synchronize()
        if rnd == 1:
            assert torch.cuda.memory_allocated() == before
            assert free_before - torch.cuda.mem_get_info()[0] < (1 << 20)
        for s, mode, window, _, ref, got, st in cases:
            check_status(st)
            assert_grads_close([(f"{name} {s} mode {mode} call {rnd}", g.cpu(), r.cpu())
                                for name, g, r in zip(("dq", "dk", "dv"), got, ref)])
