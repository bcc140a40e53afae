"""GPU parity of the final-stream problems (the L final-stream queries of Eq. 2 against
the layer's keys; the final-stream-only layers of Sec. 3.1) on the tcgen05 kernels,
against the oracle, through the C ABI.

Tolerances as for the full layers: max|dO| <= 2e-2, max|dLSE| <= 1e-3, gradients
rel-L2 <= 1e-2 (max|value| <= 1e-5 where the exact gradient is zero);
every call checks that the device status word stayed 0."""
import pytest
import torch

import oracle
from paper_2607_08186_gb300 import binding, build, inputs

import guards
from parity import kv_sample_positions

pytestmark = pytest.mark.gpu

WITHIN, CROSS, LOCAL = inputs.WITHIN, inputs.CROSS, inputs.LOCAL


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def _inputs(B, L, n, Hq, Hkv, Dh, seed):
    q = inputs.normal_bf16((B, L, Hq, Dh), seed)
    k = inputs.normal_bf16((B, n * L, Hkv, Dh), seed + 1)
    v = inputs.normal_bf16((B, n * L, Hkv, Dh), seed + 2)
    do = inputs.normal_bf16((B, L, Hq, Dh), seed + 3)
    return q, k, v, do


def _gpu(q, k, v, do, mode, window=0, bwd=True):
    B, L, Hq, Dh = q.shape
    n, Hkv = k.shape[1] // L, k.shape[2]
    qd, kd, vd = q.cuda(), k.cuda(), v.cuda()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    o = guards.empty((B, L, Hq, Dh), torch.bfloat16, 7.0)
    lse = guards.empty((B, Hq, L), torch.float32, 7.0)
    binding.sfa_fwd_final(qd, kd, vd, o, lse, mode, window=window, dev_status=st)
    out = {"o": o, "lse": lse}
    if bwd:
        dq = guards.like(qd, 7.0)
        dk, dv = guards.like(kd, 7.0), guards.like(vd, 7.0)
        ws = guards.empty((binding.sfa_bwd_final_workspace_bytes(B, L, n, Hq, Hkv, Dh, mode),), torch.uint8)
        binding.sfa_bwd_final(qd, kd, vd, o, lse, do.cuda(), dq, dk, dv, mode, ws, window=window, dev_status=st)
        out.update(dq=dq, dk=dk, dv=dv)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return {kk: t.cpu() for kk, t in out.items()}


def _rel(a, r):
    """rel-L2 error; for an all-zero reference (a single visible key: softmax 1, dS = 0)
    the largest magnitude in units of 1e-3 * 1e-2, i.e. passing at max|a| <= 1e-5, far
    above the ~1e-7 rounding residue of dP - delta and far below a real gradient."""
    den = float(r.norm())
    if den == 0:
        return float(a.double().abs().max()) / 1e-3
    return float((a.double() - r).norm()) / den


@pytest.mark.parametrize("mode,w", [(WITHIN, 0), (CROSS, 0), (LOCAL, 5), (LOCAL, 300)])
@pytest.mark.parametrize("B,L,n,Hq,Hkv", [(1, 64, 2, 4, 4), (2, 77, 4, 8, 2), (1, 200, 8, 4, 1), (1, 1, 4, 2, 1),
                                          (2, 129, 1, 4, 2), (1, 300, 3, 2, 2)])
def test_fwd_bwd_shapes(mode, w, B, L, n, Hq, Hkv):
    q, k, v, do = _inputs(B, L, n, Hq, Hkv, 128, L + n)
    got = _gpu(q, k, v, do, mode, w)
    o_r, lse_r = oracle.sfa_fwd_final(q, k, v, n, mode, window=w)
    assert float((got["o"].double() - o_r).abs().max()) <= 2e-2
    assert float((got["lse"].double() - lse_r).abs().max()) <= 1e-3
    g_r = oracle.sfa_bwd_final(q, k, v, do, n, mode, window=w)
    for name, r in zip(("dq", "dk", "dv"), g_r):
        assert _rel(got[name], r) <= 1e-2, (name, _rel(got[name], r))
    if mode == WITHIN:  # keys of streams 0..n-2 get exactly zero gradient
        for s in range(n - 1):
            assert torch.count_nonzero(got["dk"][:, s::n]) == 0 and torch.count_nonzero(got["dv"][:, s::n]) == 0


@pytest.mark.parametrize("mode,w", [(WITHIN, 0), (CROSS, 0), (LOCAL, 9)])
@pytest.mark.parametrize("B,L,n,Hq,Hkv,Dh", [(1, 70, 4, 24, 2, 256), (2, 40, 3, 4, 4, 256), (1, 90, 2, 4, 2, 64)])
def test_head_dims_256_and_64_fwd_bwd(mode, w, B, L, n, Hq, Hkv, Dh):
    # head dim 256 (the 80B final-stream-only layers: 24 over 2 heads, Table 6) and head
    # dim 64 run the final-stream geometry on their own kernel instantiations (head dim
    # 256: its own tcgen05 forward and the backward with two CTAs per key tile over the
    # head-dim halves; 64: the head-dim-64 instantiation of the tcgen05 backward)
    q, k, v, do = _inputs(B, L, n, Hq, Hkv, Dh, L + Dh)
    got = _gpu(q, k, v, do, mode, w)
    o_r, lse_r = oracle.sfa_fwd_final(q, k, v, n, mode, window=w)
    assert float((got["o"].double() - o_r).abs().max()) <= 2e-2
    assert float((got["lse"].double() - lse_r).abs().max()) <= 1e-3
    for name, r in zip(("dq", "dk", "dv"), oracle.sfa_bwd_final(q, k, v, do, n, mode, window=w)):
        assert _rel(got[name], r) <= 1e-2, (name, _rel(got[name], r))


@pytest.mark.parametrize("mode", [WITHIN, CROSS])
def test_fwd_head_dim_64(mode):
    q, k, v, do = _inputs(2, 150, 4, 4, 2, 64, 3)
    got = _gpu(q, k, v, do, mode, bwd=False)
    o_r, lse_r = oracle.sfa_fwd_final(q, k, v, 4, mode)
    assert float((got["o"].double() - o_r).abs().max()) <= 2e-2
    assert float((got["lse"].double() - lse_r).abs().max()) <= 1e-3


@pytest.mark.parametrize("mode", [WITHIN, CROSS])
def test_full_size_sampled(mode):
    # Qwen3-8B-class heads, 4096 tokens, n = 4 (16384 key positions): every output row's
    # forward statistics on sampled rows, dQ on sampled rows, dK / dV of keys from the
    # first 128 positions (the longest sums), a middle band and the last 384 positions
    B, L, n, Hq, Hkv, Dh = 1, 4096, 4, 32, 8, 128
    q, k, v, do = _inputs(B, L, n, Hq, Hkv, Dh, 11)
    got = _gpu(q, k, v, do, mode)
    gen = torch.Generator().manual_seed(1)
    ts = sorted({int(x) for x in torch.randint(0, L, (24,), generator=gen)} | {0, 127, 128, L - 1})
    hs = [0, 5, 13, 31]
    rows = [(0, h, t * n + n - 1) for h in hs for t in ts]
    qf, dof = oracle._final_full(q, n), oracle._final_full(do, n)
    o_r, lse_r = oracle.sfa_fwd_rows(qf, k, v, n, mode, rows)
    o_g = torch.stack([got["o"][0, p // n, h] for (_, h, p) in rows]).double()
    l_g = torch.tensor([float(got["lse"][0, h, p // n]) for (_, h, p) in rows], dtype=torch.float64)
    assert float((o_g - o_r).abs().max()) <= 2e-2
    assert float((l_g - lse_r).abs().max()) <= 1e-3
    dq_r, _, _ = oracle.sfa_bwd_q_rows(qf, k, v, dof, n, mode, rows)
    dq_g = torch.stack([got["dq"][0, p // n, h] for (_, h, p) in rows])
    assert _rel(dq_g, dq_r) <= 1e-2
    kv_rows = [(0, g, p) for g in (0, 7) for p in kv_sample_positions(n * L, 48, 2)]
    dk_r, dv_r = oracle.sfa_bwd_kv_rows(qf, k, v, dof, n, mode, kv_rows)
    dk_g = torch.stack([got["dk"][0, p, g] for (_, g, p) in kv_rows])
    dv_g = torch.stack([got["dv"][0, p, g] for (_, g, p) in kv_rows])
    assert _rel(dk_g, dk_r) <= 1e-2 and _rel(dv_g, dv_r) <= 1e-2
