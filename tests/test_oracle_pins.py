"""Pins for the fp64 CPU oracle: each test ties it to something other than itself.

- Golden worked examples the paper prints (Eq. 1, Eq. 3, Eq. 5) under tests/golden/.
- An independent (token, stream) characterisation of every mask, enumerated by brute force.
- Closed-form visible-pair counts.
- Library routines: torch's fp64 scaled_dot_product_attention (forward) and its
  autograd (backward) for the special cases that reduce to textbook causal attention.
- Exact special rows, probability-row invariants, and central finite differences.
- Adjoint identities <A x, y> = <x, A^T y> for the Eq. 1 gather and the Eq. 2 final-stream
  selection against their backward functions, plus torch index_add_ / indexing.
"""
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from paper_2607_08186_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_lines(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [ln.strip() for ln in f if ln.strip() and not ln.startswith("#")]


def _rand(shape, seed, dtype=torch.float64):
    g = torch.Generator().manual_seed(seed)
    return torch.randn(shape, generator=g, dtype=torch.float64).to(dtype)


# ------------------------------------------------------------------ Eq. 1 / 3 / 5
def _symbolic_tables(n, V, D=8):
    """Row x of table k holds (k+1, x) exactly in bf16 (small integers)."""
    t = torch.zeros(n, V, D)
    for k in range(n):
        t[k, :, 0] = k + 1
        t[k, :, 1] = torch.arange(V)
    return t.to(torch.bfloat16)


def _decode(row, ids_of_token):
    k = int(row[0].item())
    x = int(row[1].item())
    i = ids_of_token.index(x) + 1
    return f"E{k}(x{i})"


def test_eq1_worked_example_n2():
    golden = _golden_lines("eq1_expansion_n2.txt")
    ids = torch.tensor([[17, 42, 5]], dtype=torch.int32)  # x1, x2, x3 (distinct)
    out, bad = oracle.expand(_symbolic_tables(2, 64), ids)
    assert bad == 0
    seq = [_decode(out[0, t], ids[0].tolist()) for t in range(out.shape[1])]
    assert seq[: len(golden)] == golden
    assert seq[4:] == ["E1(x3)", "E2(x3)"]


def test_eq3_indices_golden():
    for line in _golden_lines("eq3_indices_n2.txt"):
        t, i, s = map(int, line.split())
        assert oracle.token_index(t, 2) == i
        assert oracle.stream_index(t, 2) == s


@pytest.mark.parametrize("n", [1, 2, 3, 4, 8])
def test_eq3_indices_invert_eq1(n):
    # Eq. 1 places stream k of token i at t = (i-1)n + k; Eq. 3 must recover (i, k).
    for i in range(1, 9):
        for k in range(1, n + 1):
            t = (i - 1) * n + k
            assert (oracle.token_index(t, n), oracle.stream_index(t, n)) == (i, k)


def test_expand_matches_torch_indexing_bit_exact():
    B, L, n, V, D = 2, 37, 4, 300, 24
    tables, ids = inputs.embed_inputs(B, L, n, V, D, seed=3)
    out, bad = oracle.expand(tables, ids)
    assert bad == 0
    ref = tables[:, ids.long()]                    # [n][B][L][D]
    ref = ref.permute(1, 2, 0, 3).reshape(B, n * L, D)  # token-major interleave
    assert torch.equal(out.view(torch.int16), ref.contiguous().view(torch.int16))


def test_expand_n1_is_embedding():
    tables, ids = inputs.embed_inputs(1, 50, 1, 128, 16, seed=4)
    out, _ = oracle.expand(tables, ids)
    ref = F.embedding(ids.long(), tables[0])
    assert torch.equal(out.view(torch.int16), ref.view(torch.int16))


def test_eq5_cyclic_replication_golden():
    # With tables replicated per Eq. 5, the 2n expansion repeats the n expansion's
    # rows stream-wise: stream k+n of the 2n sequence equals stream k.
    for line in _golden_lines("eq5_cyclic_replication.txt"):
        old, rest = line.split("->")
        new, names = rest.split(":")
        old, new = int(old), int(new)
        base = _symbolic_tables(old, 32)
        idx = [int(nm[1:]) - 1 for nm in names.split()]
        assert len(idx) == new
        grown = base[idx]
        ids = torch.tensor([[3, 9, 1, 30]], dtype=torch.int32)
        o_new, _ = oracle.expand(grown, ids)
        o_old, _ = oracle.expand(base, ids)
        L = ids.shape[1]
        for t in range(L):
            for k in range(new):
                assert torch.equal(o_new[0, t * new + k], o_old[0, t * old + (k % old)])


def test_expand_out_of_range_zero_rows():
    tables, ids = inputs.embed_inputs(1, 10, 2, 16, 8, seed=1)
    ids[0, 3] = 16
    ids[0, 7] = -1
    out, bad = oracle.expand(tables, ids)
    assert bad == 2
    assert torch.all(out[0, 6:8].float() == 0) and torch.all(out[0, 14:16].float() == 0)


# ------------------------------------------------------------------ Eq. 1 backward, Eq. 2
def _bf16_rand(shape, seed, scale=1.0):
    return (_rand(shape, seed) * scale).to(torch.bfloat16)


@pytest.mark.parametrize("n", [1, 2, 4])
def test_expand_bwd_is_adjoint_of_gather(n):
    # <gather(E), dX> = <E, gather^T(dX)>: a wrong stream, token or row index breaks it
    B, L, V, D = 2, 9, 13, 6
    E = _bf16_rand((n, V, D), 300 + n)
    g = torch.Generator().manual_seed(310 + n)
    ids = torch.randint(0, V, (B, L), generator=g, dtype=torch.int32)
    dX = _bf16_rand((B, n * L, D), 320 + n)
    X, bad = oracle.expand(E, ids)
    assert bad == 0
    lhs = float((X.double() * dX.double()).sum())
    rhs = float((E.double() * oracle.expand_bwd(dX, ids, n, V)).sum())
    assert abs(lhs - rhs) <= 1e-12 * max(1.0, abs(lhs))


def test_expand_bwd_matches_index_add():
    B, L, n, V, D = 3, 17, 4, 11, 5
    g = torch.Generator().manual_seed(330)
    ids = torch.randint(0, V, (B, L), generator=g, dtype=torch.int32)
    dX = _bf16_rand((B, n * L, D), 331)
    ref = torch.zeros(n, V, D, dtype=torch.float64)
    per_stream = dX.double().view(B, L, n, D)
    for s in range(n):
        ref[s].index_add_(0, ids.reshape(-1).long(), per_stream[:, :, s].reshape(-1, D))
    assert torch.equal(oracle.expand_bwd(dX, ids, n, V), ref)


def test_expand_bwd_repeated_id_and_accumulation():
    # every token the same id: that row receives the sum over all tokens of its stream;
    # an existing dE is added to, not replaced; other rows keep their values
    B, L, n, V, D = 2, 7, 3, 5, 4
    ids = torch.full((B, L), 2, dtype=torch.int32)
    dX = _bf16_rand((B, n * L, D), 340)
    dE0 = _rand((n, V, D), 341)
    got = oracle.expand_bwd(dX, ids, n, V, dE=dE0)
    want = dE0.clone()
    want[:, 2] += dX.double().view(B, L, n, D).sum(dim=(0, 1))
    assert torch.allclose(got, want, rtol=0, atol=1e-12)


def test_expand_bwd_out_of_range_ids_contribute_nothing():
    B, L, n, V, D = 1, 6, 2, 4, 3
    ids = torch.tensor([[0, -1, 3, 4, 1, 1000]], dtype=torch.int32)
    dX = _bf16_rand((B, n * L, D), 350)
    got = oracle.expand_bwd(dX, ids, n, V)
    keep = torch.tensor([0, 2, 4])  # tokens whose id is in range
    ref = oracle.expand_bwd(dX.view(B, L, n, D)[:, keep].reshape(B, -1, D), ids[:, keep], n, V)
    assert torch.equal(got, ref)


@pytest.mark.parametrize("n", [1, 2, 4])
def test_select_final_is_last_stream_rows(n):
    # Eq. 2: the loss reads 1-indexed positions t = i n, i.e. stream n of every token
    B, L, D = 2, 5, 6
    X = _bf16_rand((B, n * L, D), 360 + n)
    Y = oracle.select_final(X, n)
    assert torch.equal(Y.view(torch.int16), X.view(B, L, n, D)[:, :, n - 1].contiguous().view(torch.int16))
    rows = [i * n - 1 for i in range(1, L + 1)]  # 0-indexed positions t - 1 = i n - 1
    assert torch.equal(Y.view(torch.int16), X[:, rows].contiguous().view(torch.int16))


@pytest.mark.parametrize("n", [1, 3])
def test_select_final_bwd_is_adjoint(n):
    B, L, D = 2, 4, 5
    X = _bf16_rand((B, n * L, D), 370 + n)
    dY = _bf16_rand((B, L, D), 375 + n)
    dX = oracle.select_final_bwd(dY, n)
    lhs = float((oracle.select_final(X, n).double() * dY.double()).sum())
    rhs = float((X.double() * dX.double()).sum())
    assert abs(lhs - rhs) <= 1e-12 * max(1.0, abs(lhs))
    # every position that is not a final stream receives zero
    mask = torch.ones(B, L, n, dtype=torch.bool)
    mask[:, :, n - 1] = False
    assert not dX.view(B, L, n, D)[mask].any()


# ------------------------------------------------------------------ masks
def _brute_visible(t, tk, n, mode, w):
    """Independent characterisation on (token, stream) pairs, 1-indexed."""
    i, s = (t - 1) // n + 1, (t - 1) % n + 1
    j, r = (tk - 1) // n + 1, (tk - 1) % n + 1
    if mode == oracle.WITHIN:   # Fig. 2c: streams invisible to each other, causal within a stream
        return r == s and j <= i
    if mode == oracle.CROSS:    # Fig. 2a: lower-triangular over positions = earlier token, or same token & earlier-or-same stream
        return j < i or (j == i and r <= s)
    # Fig. 2b: causal window of w positions ending at the query (inclusive)
    return tk <= t and t - tk < w


@pytest.mark.parametrize("n", range(1, 9))
def test_masks_brute_force(n):
    for nL in range(n, 65, n):
        for mode, w in [(oracle.WITHIN, 0), (oracle.CROSS, 0), (oracle.LOCAL, 1), (oracle.LOCAL, 5)]:
            for t in range(1, nL + 1):
                for tk in range(1, nL + 1):
                    assert oracle.visible(t, tk, n, mode, w) == _brute_visible(t, tk, n, mode, w)


@pytest.mark.parametrize("n,L", [(1, 7), (2, 9), (4, 16), (8, 5)])
def test_visible_pair_counts_closed_form(n, L):
    nL = n * L
    cnt = {m: 0 for m in (oracle.WITHIN, oracle.CROSS)}
    for t in range(1, nL + 1):
        for tk in range(1, nL + 1):
            for m in cnt:
                cnt[m] += oracle.visible(t, tk, n, m)
    assert cnt[oracle.WITHIN] == n * L * (L + 1) // 2       # O(nL^2), Eq. 4
    assert cnt[oracle.CROSS] == nL * (nL + 1) // 2          # O(n^2 L^2), Fig. 2a


# ------------------------------------------------------------------ forward
def _sdpa_causal(q, k, v, scale):
    """torch fp64 causal SDPA on [B][S][H][Dh] with K/V heads repeated per group."""
    Hq, Hkv = q.shape[2], k.shape[2]
    qh = q.permute(0, 2, 1, 3)
    kh = k.permute(0, 2, 1, 3).repeat_interleave(Hq // Hkv, dim=1)
    vh = v.permute(0, 2, 1, 3).repeat_interleave(Hq // Hkv, dim=1)
    o = F.scaled_dot_product_attention(qh, kh, vh, is_causal=True, scale=scale)
    return o.permute(0, 2, 1, 3)


def _lse_causal(q, k, scale):
    Hq, Hkv = q.shape[2], k.shape[2]
    qh = q.permute(0, 2, 1, 3)
    kh = k.permute(0, 2, 1, 3).repeat_interleave(Hq // Hkv, dim=1)
    s = torch.einsum("bhpd,bhkd->bhpk", qh, kh) * scale
    S = s.shape[-1]
    s = s.masked_fill(~torch.tril(torch.ones(S, S, dtype=torch.bool)), -math.inf)
    return torch.logsumexp(s, dim=-1)


@pytest.mark.parametrize("Hq,Hkv", [(4, 4), (4, 2), (6, 1)])
def test_fwd_n1_is_causal_sdpa(Hq, Hkv):
    B, L, Dh = 2, 23, 16
    q, k, v = _rand((B, L, Hq, Dh), 1), _rand((B, L, Hkv, Dh), 2), _rand((B, L, Hkv, Dh), 3)
    scale = 0.3
    ref = _sdpa_causal(q, k, v, scale)
    for mode in (oracle.WITHIN, oracle.CROSS):
        o, lse = oracle.sfa_fwd(q, k, v, 1, mode, scale)
        torch.testing.assert_close(o, ref, rtol=1e-12, atol=1e-12)
        torch.testing.assert_close(lse, _lse_causal(q, k, scale), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("n", [2, 3, 4])
def test_fwd_within_is_n_independent_causal_attentions(n):
    B, L, Hq, Hkv, Dh = 2, 11, 4, 2, 8
    q, k, v = _rand((B, n * L, Hq, Dh), 4), _rand((B, n * L, Hkv, Dh), 5), _rand((B, n * L, Hkv, Dh), 6)
    o, lse = oracle.sfa_fwd(q, k, v, n, oracle.WITHIN, 0.25)
    for s in range(n):
        ref = _sdpa_causal(q[:, s::n], k[:, s::n], v[:, s::n], 0.25)
        torch.testing.assert_close(o[:, s::n], ref, rtol=1e-12, atol=1e-12)
        torch.testing.assert_close(lse[:, :, s::n], _lse_causal(q[:, s::n], k[:, s::n], 0.25),
                                   rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("n", [2, 4])
def test_fwd_cross_is_causal_over_expanded_sequence(n):
    B, L, Hq, Hkv, Dh = 1, 9, 4, 1, 8
    q, k, v = _rand((B, n * L, Hq, Dh), 7), _rand((B, n * L, Hkv, Dh), 8), _rand((B, n * L, Hkv, Dh), 9)
    o, lse = oracle.sfa_fwd(q, k, v, n, oracle.CROSS, 0.4)
    torch.testing.assert_close(o, _sdpa_causal(q, k, v, 0.4), rtol=1e-12, atol=1e-12)
    torch.testing.assert_close(lse, _lse_causal(q, k, 0.4), rtol=1e-12, atol=1e-12)


def test_fwd_local_is_banded_sdpa():
    B, n, L, H, Dh, w = 1, 2, 12, 2, 8, 5
    q, k, v = _rand((B, n * L, H, Dh), 10), _rand((B, n * L, H, Dh), 11), _rand((B, n * L, H, Dh), 12)
    o, _ = oracle.sfa_fwd(q, k, v, n, oracle.LOCAL, 0.5, window=w)
    S = n * L
    i = torch.arange(S)
    band = (i[None, :] <= i[:, None]) & (i[:, None] - i[None, :] < w)
    ref = F.scaled_dot_product_attention(q.permute(0, 2, 1, 3), k.permute(0, 2, 1, 3),
                                         v.permute(0, 2, 1, 3), attn_mask=band, scale=0.5)
    torch.testing.assert_close(o, ref.permute(0, 2, 1, 3), rtol=1e-12, atol=1e-12)


def test_fwd_first_rows_exact():
    # A row that sees only itself: O = V of that row, LSE = scale * q.k.
    n, L, Dh = 4, 6, 16
    q, k, v = _rand((1, n * L, 2, Dh), 13), _rand((1, n * L, 2, Dh), 14), _rand((1, n * L, 2, Dh), 15)
    o, lse = oracle.sfa_fwd(q, k, v, n, oracle.WITHIN, 0.2)
    for p in range(n):
        assert torch.equal(o[0, p], v[0, p])
        for h in range(2):
            assert abs(lse[0, h, p].item() - 0.2 * float(q[0, p, h] @ k[0, p, h])) < 1e-14
    o, lse = oracle.sfa_fwd(q, k, v, n, oracle.CROSS, 0.2)
    assert torch.equal(o[0, 0], v[0, 0])


@pytest.mark.parametrize("mode", [oracle.WITHIN, oracle.CROSS])
def test_fwd_probability_rows(mode):
    # With V the identity (Dh >= nL), O row p is the softmax row P[p, :].
    n, L, Dh = 2, 8, 16
    q, k = _rand((1, n * L, 1, Dh), 16), _rand((1, n * L, 1, Dh), 17)
    v = torch.eye(Dh, dtype=torch.float64)[: n * L].reshape(1, n * L, 1, Dh)
    o, lse = oracle.sfa_fwd(q, k, v, n, mode, 0.3)
    P = o[0, :, 0, : n * L]
    z = 0.3 * (q[0, :, 0] @ k[0, :, 0].T)
    for p in range(n * L):
        vis = torch.tensor([oracle.visible(p + 1, j + 1, n, mode) for j in range(n * L)])
        assert torch.all(P[p, ~vis] == 0) and torch.all(P[p, vis] > 0)
        assert abs(P[p].sum().item() - 1.0) < 1e-13
        torch.testing.assert_close(P[p, vis], torch.exp(z[p, vis] - lse[0, 0, p]), rtol=1e-13, atol=0)
        assert lse[0, 0, p] >= z[p, vis].max() - 1e-14


def test_fwd_rows_match_full():
    s = inputs.AttnShape(1, 16, 4, 4, 2, 16)
    q, k, v = inputs.attn_inputs(s, seed=3, with_grad=False)
    for mode in (oracle.WITHIN, oracle.CROSS):
        o, lse = oracle.sfa_fwd(q, k, v, s.n, mode)
        rows = np.array([[0, 0, 0], [0, 3, 63], [0, 1, 17], [0, 2, 5]])
        orow, lrow = oracle.sfa_fwd_rows(q, k, v, s.n, mode, rows)
        for r, (b, h, p) in enumerate(rows):
            assert torch.equal(orow[r], o[b, p, h]) and lrow[r].item() == lse[b, h, p].item()


# ------------------------------------------------------------------ backward
def _fd_check(mode, n, window=0):
    B, L, Hq, Hkv, Dh = 1, 5, 4, 2, 6
    S = n * L
    q, k, v, do = (_rand((B, S, Hq, Dh), 20), _rand((B, S, Hkv, Dh), 21),
                   _rand((B, S, Hkv, Dh), 22), _rand((B, S, Hq, Dh), 23))
    scale = 0.45
    dq, dk, dv = oracle.sfa_bwd(q, k, v, do, n, mode, scale, window)
    def f(args):
        o, _ = oracle.sfa_fwd(args["q"], args["k"], args["v"], n, mode, scale, window)
        return float((o * do).sum())

    h = 1e-6
    g = torch.Generator().manual_seed(0)
    for name, t, grad in (("q", q, dq), ("k", k, dk), ("v", v, dv)):
        for _ in range(12):
            idx = tuple(int(torch.randint(0, m, (1,), generator=g)) for m in t.shape)
            tp, tm = t.clone(), t.clone()
            tp[idx] += h
            tm[idx] -= h
            args_p = {"q": q, "k": k, "v": v}
            args_m = dict(args_p)
            args_p[name], args_m[name] = tp, tm
            num = (f(args_p) - f(args_m)) / (2 * h)
            assert abs(num - grad[idx].item()) <= 1e-6 * max(1.0, abs(num)), (name, idx, num, grad[idx])


@pytest.mark.parametrize("mode,n", [(oracle.WITHIN, 2), (oracle.WITHIN, 3), (oracle.CROSS, 2), (oracle.LOCAL, 2)])
def test_bwd_finite_differences(mode, n):
    _fd_check(mode, n, window=3 if mode == oracle.LOCAL else 0)


@pytest.mark.parametrize("mode", [oracle.WITHIN, oracle.CROSS])
def test_bwd_explicit_jacobian_equals_reduced(mode):
    s = inputs.AttnShape(1, 8, 2, 4, 2, 16)
    q, k, v, do = inputs.attn_inputs(s, seed=5)
    a = oracle.sfa_bwd(q, k, v, do, s.n, mode)
    b = oracle.sfa_bwd_jacobian(q, k, v, do, s.n, mode)
    for x, y in zip(a, b):
        torch.testing.assert_close(x, y, rtol=1e-11, atol=1e-12)


def test_bwd_delta_identity():
    # D = sum_p' P dP (Jacobian form) equals rowsum(dO * O).
    s = inputs.AttnShape(1, 12, 4, 4, 2, 16)
    q, k, v, do = inputs.attn_inputs(s, seed=6)
    for mode in (oracle.WITHIN, oracle.CROSS):
        o, lse = oracle.sfa_fwd(q, k, v, s.n, mode)
        rows = np.array([[0, h, p] for h in range(s.Hq) for p in range(0, s.nL, 5)])
        _, lrow, drow = oracle.sfa_bwd_q_rows(q, k, v, do, s.n, mode, rows)
        for r, (b, h, p) in enumerate(rows):
            ref = float((do[b, p, h].double() * o[b, p, h]).sum())
            assert abs(drow[r].item() - ref) < 1e-12
            assert abs(lrow[r].item() - lse[b, h, p].item()) < 1e-13


@pytest.mark.parametrize("Hq,Hkv", [(2, 2), (4, 2)])
def test_bwd_cross_is_sdpa_autograd(Hq, Hkv):
    n, L, Dh = 3, 6, 8
    S = n * L
    q, k, v, do = (_rand((1, S, Hq, Dh), 30), _rand((1, S, Hkv, Dh), 31),
                   _rand((1, S, Hkv, Dh), 32), _rand((1, S, Hq, Dh), 33))
    qq, kk, vv = (t.clone().requires_grad_() for t in (q, k, v))
    _sdpa_causal(qq, kk, vv, 0.35).backward(do)
    dq, dk, dv = oracle.sfa_bwd(q, k, v, do, n, oracle.CROSS, 0.35)
    for a, b in ((dq, qq.grad), (dk, kk.grad), (dv, vv.grad)):
        torch.testing.assert_close(a, b, rtol=1e-11, atol=1e-12)


def test_bwd_within_is_per_stream_sdpa_autograd():
    n, L, Hq, Hkv, Dh = 4, 7, 4, 2, 8
    S = n * L
    q, k, v, do = (_rand((2, S, Hq, Dh), 40), _rand((2, S, Hkv, Dh), 41),
                   _rand((2, S, Hkv, Dh), 42), _rand((2, S, Hq, Dh), 43))
    dq, dk, dv = oracle.sfa_bwd(q, k, v, do, n, oracle.WITHIN, 0.3)
    for s in range(n):
        qq, kk, vv = (t[:, s::n].clone().requires_grad_() for t in (q, k, v))
        _sdpa_causal(qq, kk, vv, 0.3).backward(do[:, s::n])
        torch.testing.assert_close(dq[:, s::n], qq.grad, rtol=1e-11, atol=1e-12)
        torch.testing.assert_close(dk[:, s::n], kk.grad, rtol=1e-11, atol=1e-12)
        torch.testing.assert_close(dv[:, s::n], vv.grad, rtol=1e-11, atol=1e-12)


def test_bwd_row_functions_match_full():
    s = inputs.AttnShape(1, 16, 2, 4, 2, 16)
    q, k, v, do = inputs.attn_inputs(s, seed=7)
    for mode in (oracle.WITHIN, oracle.CROSS):
        dq, dk, dv = oracle.sfa_bwd(q, k, v, do, s.n, mode)
        qrows = np.array([[0, 0, 0], [0, 3, 31], [0, 1, 10]])
        dqr, _, _ = oracle.sfa_bwd_q_rows(q, k, v, do, s.n, mode, qrows)
        for r, (b, h, p) in enumerate(qrows):
            torch.testing.assert_close(dqr[r], dq[b, p, h], rtol=1e-12, atol=1e-13)
        kvrows = np.array([[0, 0, 0], [0, 1, 31], [0, 1, 9], [0, 0, 20]])
        dkr, dvr = oracle.sfa_bwd_kv_rows(q, k, v, do, s.n, mode, kvrows)
        for r, (b, g, p) in enumerate(kvrows):
            torch.testing.assert_close(dkr[r], dk[b, p, g], rtol=1e-12, atol=1e-13)
            torch.testing.assert_close(dvr[r], dv[b, p, g], rtol=1e-12, atol=1e-13)


# ------------------------------------------------------------------ decoding (Sec. 3.2)
@pytest.mark.parametrize("n", [1, 2, 4])
@pytest.mark.parametrize("mode,w", [(oracle.WITHIN, 0), (oracle.CROSS, 0), (oracle.LOCAL, 5)])
def test_decode_is_forward_rows_of_the_last_token(n, mode, w):
    # decoding token i with the cache holding tokens 1..i equals the forward pass's rows
    # of token i; a shorter sequence (lens < Lcap) equals the forward over its prefix
    B, L, Hq, Hkv, Dh, scale = 2, 7, 4, 2, 16, 0.35
    q, k, v = _rand((B, n * L, Hq, Dh), 40), _rand((B, n * L, Hkv, Dh), 41), _rand((B, n * L, Hkv, Dh), 42)
    lens = torch.tensor([L, 3], dtype=torch.int32)
    qn = torch.stack([q[b, (int(lens[b]) - 1) * n:int(lens[b]) * n] for b in range(B)])
    o, lse, bad = oracle.decode(qn, k, v, lens, n, mode, scale, window=w)
    assert bad == 0
    for b in range(B):
        i = int(lens[b])
        of, lf = oracle.sfa_fwd(q[b:b + 1, :i * n], k[b:b + 1, :i * n], v[b:b + 1, :i * n], n, mode, scale,
                                window=w)
        torch.testing.assert_close(o[b], of[0, (i - 1) * n:i * n], rtol=1e-12, atol=1e-12)
        torch.testing.assert_close(lse[b], lf[0, :, (i - 1) * n:i * n], rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("mode", [oracle.WITHIN, oracle.CROSS])
def test_decode_matches_masked_sdpa(mode):
    # torch fp64 SDPA of the new token's n query rows against all cached rows under an
    # explicit boolean mask (0-indexed: key p' visible from p = (i-1)n + s iff p' <= p,
    # and for the intra-stream layer p' = s mod n)
    B, n, Lcap, Hq, Hkv, Dh, scale = 1, 3, 10, 6, 2, 8, 0.5
    i = 8
    kc, vc = _rand((B, n * Lcap, Hkv, Dh), 43), _rand((B, n * Lcap, Hkv, Dh), 44)
    qn = _rand((B, n, Hq, Dh), 45)
    o, _, _ = oracle.decode(qn, kc, vc, torch.tensor([i], dtype=torch.int32), n, mode, scale)
    p = (i - 1) * n + torch.arange(n)
    pk = torch.arange(i * n)
    mask = pk[None, :] <= p[:, None]
    if mode == oracle.WITHIN:
        mask &= (pk[None, :] % n) == (p[:, None] % n)
    qh = qn.permute(0, 2, 1, 3)
    kh = kc[:, :i * n].permute(0, 2, 1, 3).repeat_interleave(Hq // Hkv, dim=1)
    vh = vc[:, :i * n].permute(0, 2, 1, 3).repeat_interleave(Hq // Hkv, dim=1)
    ref = F.scaled_dot_product_attention(qh, kh, vh, attn_mask=mask, scale=scale).permute(0, 2, 1, 3)
    torch.testing.assert_close(o, ref, rtol=1e-12, atol=1e-12)


def test_decode_n1_is_single_query_attention():
    # n = 1: one query per step attending to every cached token (closed form softmax(qK^T)V)
    B, Lcap, Hq, Hkv, Dh, scale = 2, 9, 2, 1, 8, 0.7
    kc, vc, qn = _rand((B, Lcap, Hkv, Dh), 46), _rand((B, Lcap, Hkv, Dh), 47), _rand((B, 1, Hq, Dh), 48)
    lens = torch.tensor([9, 4], dtype=torch.int32)
    o, lse, _ = oracle.decode(qn, kc, vc, lens, 1, oracle.CROSS, scale)
    for b in range(B):
        i = int(lens[b])
        z = scale * torch.einsum("hd,kd->hk", qn[b, 0], kc[b, :i, 0])
        P = torch.softmax(z, dim=-1)
        torch.testing.assert_close(o[b, 0], P @ vc[b, :i, 0], rtol=1e-12, atol=1e-12)
        torch.testing.assert_close(lse[b, :, 0], torch.logsumexp(z, dim=-1), rtol=1e-12, atol=1e-12)


def test_decode_bad_lens_zero_rows():
    B, n, Lcap, H, Dh = 3, 2, 4, 2, 8
    kc, vc, qn = _rand((B, n * Lcap, H, Dh), 49), _rand((B, n * Lcap, H, Dh), 50), _rand((B, n, H, Dh), 51)
    lens = torch.tensor([0, 4, 5], dtype=torch.int32)
    o, lse, bad = oracle.decode(qn, kc, vc, lens, n, oracle.CROSS)
    assert bad == 2
    assert torch.count_nonzero(o[0]) == 0 and torch.count_nonzero(o[2]) == 0
    assert torch.isinf(lse[0]).all() and torch.isinf(lse[2]).all() and torch.isfinite(lse[1]).all()


def test_kv_append_matches_indexing():
    B, n, Lcap, Hkv, Dh = 3, 4, 5, 2, 8
    cache = _rand((B, n * Lcap, Hkv, Dh), 52, torch.bfloat16)
    new = _rand((B, n, Hkv, Dh), 53, torch.bfloat16)
    lens = torch.tensor([1, 5, 7], dtype=torch.int32)     # the last is out of range
    got, bad = oracle.kv_append(new, cache, lens, n)
    assert bad == 1
    ref = cache.clone()
    for b in range(2):
        i = int(lens[b])
        ref[b, (i - 1) * n:i * n] = new[b]
    assert torch.equal(got.view(torch.int16), ref.view(torch.int16))


# ------------------------------------------------------------------ final-stream problems (Eq. 2, Sec. 3.1)
def _final_mask(L, n, mode, w=0):
    """[L][nL] boolean: final-stream query t (position t*n + n-1) sees key p'."""
    pq = torch.arange(L)[:, None] * n + n - 1
    pk = torch.arange(n * L)[None, :]
    m = pk <= pq
    if mode == oracle.WITHIN:
        m &= (pk % n) == (n - 1)
    if mode == oracle.LOCAL:
        m &= (pq - pk) < w
    return m


@pytest.mark.parametrize("n", [1, 2, 4])
@pytest.mark.parametrize("mode,w", [(oracle.WITHIN, 0), (oracle.CROSS, 0), (oracle.LOCAL, 6)])
def test_final_stream_is_masked_sdpa_with_gradients(n, mode, w):
    # torch fp64 SDPA of the L final-stream queries against the nL keys under an explicit
    # boolean mask, and its autograd gradients
    B, L, Hq, Hkv, Dh, scale = 2, 9, 4, 2, 8, 0.45
    q = _rand((B, L, Hq, Dh), 60).requires_grad_()
    k = _rand((B, n * L, Hkv, Dh), 61).requires_grad_()
    v = _rand((B, n * L, Hkv, Dh), 62).requires_grad_()
    do = _rand((B, L, Hq, Dh), 63)
    mask = _final_mask(L, n, mode, w)
    qh = q.permute(0, 2, 1, 3)
    kh = k.permute(0, 2, 1, 3).repeat_interleave(Hq // Hkv, dim=1)
    vh = v.permute(0, 2, 1, 3).repeat_interleave(Hq // Hkv, dim=1)
    ref = F.scaled_dot_product_attention(qh, kh, vh, attn_mask=mask, scale=scale).permute(0, 2, 1, 3)
    ref.backward(do)
    z = torch.einsum("bhqd,bhkd->bhqk", qh, kh).detach() * scale
    lse_ref = torch.logsumexp(z.masked_fill(~mask, -math.inf), dim=-1)
    o, lse = oracle.sfa_fwd_final(q.detach(), k.detach(), v.detach(), n, mode, scale, window=w)
    torch.testing.assert_close(o, ref.detach(), rtol=1e-12, atol=1e-12)
    torch.testing.assert_close(lse, lse_ref, rtol=1e-12, atol=1e-12)
    dq, dk, dv = oracle.sfa_bwd_final(q.detach(), k.detach(), v.detach(), do, n, mode, scale, window=w)
    torch.testing.assert_close(dq, q.grad, rtol=1e-10, atol=1e-12)
    torch.testing.assert_close(dk, k.grad, rtol=1e-10, atol=1e-12)
    torch.testing.assert_close(dv, v.grad, rtol=1e-10, atol=1e-12)


def test_final_stream_within_reads_only_the_last_stream():
    # intra-stream layer: perturbing keys/values of streams 0..n-2 changes nothing
    B, L, n, H, Dh = 1, 6, 3, 2, 8
    q, k, v = _rand((B, L, H, Dh), 64), _rand((B, n * L, H, Dh), 65), _rand((B, n * L, H, Dh), 66)
    o1, _ = oracle.sfa_fwd_final(q, k, v, n, oracle.WITHIN)
    k2, v2 = k.clone(), v.clone()
    for s in range(n - 1):
        k2[:, s::n] += 3.0
        v2[:, s::n] -= 2.0
    o2, _ = oracle.sfa_fwd_final(q, k2, v2, n, oracle.WITHIN)
    torch.testing.assert_close(o1, o2, rtol=0, atol=0)
    _, dk, dv = oracle.sfa_bwd_final(q, k, v, _rand((B, L, H, Dh), 67), n, oracle.WITHIN)
    for s in range(n - 1):
        assert torch.count_nonzero(dk[:, s::n]) == 0 and torch.count_nonzero(dv[:, s::n]) == 0
