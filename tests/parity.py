"""Helpers for the GPU-vs-oracle parity tests (test infrastructure).

Tolerances (bf16 inputs, fp32 accumulation on the GPU, exact fp64 oracle):
  max |dO|   <= 2e-2      on the attention output
  max |dLSE| <= 1e-3      on the natural-log log-sum-exp
  rel-L2     <= 1e-2      on dQ, dK, dV  (||g - g_ref||_2 <= 1e-2 ||g_ref||_2 + abs floor)
  bit-exact               on the expansion gather
"""
from __future__ import annotations

import numpy as np
import torch

import guards
import oracle
from paper_2607_08186_gb300 import binding

TOL_O = 2e-2
TOL_LSE = 1e-3
TOL_GRAD = 1e-2


def check_status(st):
    """The device status word must stay clear (no bounded wait expired, no bad index)."""
    torch.cuda.synchronize()
    v = int(st.item())
    assert v == 0, f"device status bits set: {v:#x}"


def gpu_fwd(q, k, v, n, mode, scale=0.0, window=0, status=None):
    qd, kd, vd = q.cuda(), k.cuda(), v.cuda()
    B, nL, Hq, Dh = q.shape
    o = guards.like(qd)
    lse = guards.empty((B, Hq, nL), torch.float32)
    st = torch.zeros(1, dtype=torch.int32, device="cuda") if status is None else status
    binding.sfa_fwd(qd, kd, vd, o, lse, n, mode, scale or 0.0, window, dev_status=st)
    if status is None:
        check_status(st)
    return qd, kd, vd, o, lse


def gpu_fwd_bwd(q, k, v, do, n, mode, scale=0.0, window=0):
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    qd, kd, vd, o, lse = gpu_fwd(q, k, v, n, mode, scale, window, status=st)
    dod = do.cuda()
    B, nL, Hq, Dh = q.shape
    Hkv = k.shape[2]
    dq, dk, dv = guards.like(qd), guards.like(kd), guards.like(vd)
    wsb = binding.sfa_bwd_workspace_bytes(B, nL // n, n, Hq, Hkv, Dh, mode)
    ws = guards.empty((wsb,), torch.uint8, what="sfa_bwd workspace")
    binding.sfa_bwd(qd, kd, vd, o, lse, dod, dq, dk, dv, n, mode, ws, scale or 0.0, window, dev_status=st)
    check_status(st)
    return o.cpu(), lse.cpu(), dq.cpu(), dk.cpu(), dv.cpu()


def max_abs(a, b) -> float:
    return float((a.double() - b.double()).abs().max()) if a.numel() else 0.0


def rel_l2_ok(g, ref, tol=TOL_GRAD):
    g, ref = g.double(), ref.double()
    err = float(torch.linalg.vector_norm(g - ref))
    nrm = float(torch.linalg.vector_norm(ref))
    floor = 1e-6 * (ref.numel() ** 0.5)
    return err <= tol * nrm + floor, err / max(nrm, 1e-300)


def assert_fwd_close(o, lse, o_ref, lse_ref):
    eo, el = max_abs(o, o_ref), max_abs(lse, lse_ref)
    assert eo <= TOL_O, f"max|dO| {eo:.3e} > {TOL_O}"
    assert el <= TOL_LSE, f"max|dLSE| {el:.3e} > {TOL_LSE}"
    return eo, el


def assert_grads_close(pairs):
    out = {}
    for name, g, ref in pairs:
        ok, rel = rel_l2_ok(g, ref)
        assert ok, f"{name}: rel-L2 {rel:.3e} > {TOL_GRAD}"
        out[name] = rel
    return out


def group_slices(q, k, v, do, g, grp):
    """Tensors of K/V head g and its query heads (the oracle works per group)."""
    hs = slice(g * grp, (g + 1) * grp)
    return (q[:, :, hs].contiguous(), k[:, :, g:g + 1].contiguous(), v[:, :, g:g + 1].contiguous(),
            None if do is None else do[:, :, hs].contiguous())


def sample_rows(B, Hq, nL, count, seed, extra_p=()):
    """(b, h, p) rows: random ones plus fixed positions (tile edges, ends)."""
    g = torch.Generator().manual_seed(seed)
    rows = set()
    for _ in range(count):
        rows.add((int(torch.randint(0, B, (1,), generator=g)), int(torch.randint(0, Hq, (1,), generator=g)),
                  int(torch.randint(0, nL, (1,), generator=g))))
    for p in extra_p:
        if 0 <= p < nL:
            rows.add((0, 0, p))
            rows.add((B - 1, Hq - 1, p))
    return np.array(sorted(rows), dtype=np.int64)


def kv_sample_positions(nL, count, seed):
    """Key positions for full-size dK / dV checks, spread over the whole sequence: the
    first 128 positions (in a causal layer the keys that every later query sees, so
    their gradients sum over the most query tiles and heads), a 128-position band in
    the middle, and the last 384 positions (the shortest sums), plus both ends."""
    g = torch.Generator().manual_seed(seed)
    per = max(1, count // 3)
    bands = [(0, min(128, nL)), (max(0, nL // 2 - 64), min(nL, nL // 2 + 64)), (max(0, nL - 384), nL)]
    ps = {0, nL - 1}
    for lo, hi in bands:
        ps |= {int(x) for x in torch.randint(lo, hi, (per,), generator=g)}
    return sorted(ps)

