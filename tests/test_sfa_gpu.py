"""GPU parity: the CUDA SFA forward/backward (through the C ABI) against the fp64 oracle.

Small shapes compare every element; they span several 64/128-row tiles and end
in ragged tails.  Full-size shapes (the Qwen3-8B-class and large-MoE-class
layers, in the launch configuration the benchmark times) compare sampled rows
the oracle computes one by one.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_08186_gb300 import binding, build, inputs
from paper_2607_08186_gb300.inputs import AttnShape, CROSS, LOCAL, WITHIN, WITHIN_NAIVE

import guards
from parity import (assert_fwd_close, assert_grads_close, gpu_fwd, gpu_fwd_bwd, group_slices,
                    kv_sample_positions, max_abs, sample_rows, TOL_LSE, TOL_O)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()
    binding.lib()


def _full_case(s: AttnShape, mode, seed, window=0, scale=0.0):
    q, k, v, do = inputs.attn_inputs(s, seed=seed)
    o, lse, dq, dk, dv = gpu_fwd_bwd(q, k, v, do, s.n, mode, scale, window)
    om = WITHIN if mode == WITHIN_NAIVE else mode  # the naive schedule computes the WITHIN result
    o_ref, lse_ref = oracle.sfa_fwd(q, k, v, s.n, om, scale or None, window)
    assert_fwd_close(o, lse, o_ref, lse_ref)
    dq_r, dk_r, dv_r = oracle.sfa_bwd(q, k, v, do, s.n, om, scale or None, window)
    assert_grads_close([("dq", dq, dq_r), ("dk", dk, dk_r), ("dv", dv, dv_r)])


@pytest.mark.parametrize("mode", [WITHIN, CROSS])
def test_tiny_config(mode):
    # B=1, L=64, n=2 (128 positions), Hq=Hkv=4, Dh=64, N(0,1) from seed 0.
    _full_case(inputs.SHAPES["tiny"], mode, seed=0)


SWEEP = [
    # (B, L, n, Hq, Hkv, Dh)
    (1, 100, 1, 4, 2, 128),
    (2, 37, 2, 4, 4, 64),
    (1, 130, 4, 4, 1, 128),
    (1, 70, 8, 2, 2, 64),
    (1, 200, 4, 4, 2, 128),
]


@pytest.mark.parametrize("shape", SWEEP)
@pytest.mark.parametrize("mode", [WITHIN, CROSS])
def test_sweep(shape, mode):
    _full_case(AttnShape(*shape), mode, seed=11 + sum(shape))


@pytest.mark.parametrize("mode,window", [(WITHIN, 0), (CROSS, 0), (LOCAL, 77)])
def test_wide_gqa_groups(mode, window):
    # the paper's 617B head layout (96 query heads over 8 K/V heads: 12 per group) and
    # a 3-head group (Hq=6, Hkv=2), B=2, ragged nL = 4 * 150 = 600
    _full_case(AttnShape(1, 150, 4, 96, 8, 128), mode, seed=21, window=window)
    _full_case(AttnShape(2, 150, 4, 6, 2, 128), mode, seed=22, window=window)


@pytest.mark.parametrize("mode,window", [(WITHIN, 0), (CROSS, 0), (LOCAL, 40)])
def test_head_dim_256(mode, window):
    # head dim 256 (the paper's 80B configuration, 24 query over 2 K/V heads, Table 6):
    # the forward on its own tcgen05 kernel, the backward on the tcgen05 kernel with two
    # CTAs per key tile over halves of the head dim and 64-row query tiles
    _full_case(AttnShape(1, 70, 4, 24, 2, 256), mode, seed=31, window=window)
    _full_case(AttnShape(2, 33, 2, 4, 4, 256), mode, seed=32, window=window)


@pytest.mark.parametrize("mode,window", [(WITHIN, 0), (CROSS, 0), (LOCAL, 333)])
def test_head_dim_256_many_key_tiles(mode, window):
    # 1200 positions: up to 10 key tiles per query tile, so the head-dim-256 forward's
    # five-slot K/V ring wraps several times; ragged last tiles (1200 = 9*128 + 48)
    _full_case(AttnShape(1, 300, 4, 4, 2, 256), mode, seed=33, window=window)


@pytest.mark.parametrize("mode,window", [(WITHIN, 0), (CROSS, 0), (LOCAL, 60)])
@pytest.mark.parametrize("Dh", [64, 128, 256])
def test_uneven_head_chunks(mode, window, Dh):
    # 11 query heads per K/V head on a backward grid of 64 CTAs (128 at head dim 256):
    # each group splits into head chunks of 2 (3) heads with a smaller last one, whose
    # fp32 dK / dV partial sums the finalize pass adds in chunk order; against the
    # oracle, and dK / dV bit-identical on a rerun (dQ's fp32 reduce-adds from many CTAs
    # arrive in a run-dependent order: it agrees to rounding only)
    s = AttnShape(4, 256, 4, 22, 2, Dh)
    _full_case(s, mode, seed=41 + Dh, window=window)
    q, k, v, do = inputs.attn_inputs(s, seed=41 + Dh)
    runs = [gpu_fwd_bwd(q, k, v, do, s.n, mode, 0.0, window)[3:] for _ in range(2)]
    for a, b in zip(*runs):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))


@pytest.mark.parametrize("shape", [(1, 100, 1, 4, 2, 128), (1, 130, 4, 4, 1, 128), (2, 77, 3, 4, 2, 128),
                                   (1, 70, 8, 2, 2, 128)])
def test_naive_within_schedule(shape):
    # WITHIN's mask applied per pair over the full causal tile schedule of nL positions
    # (no stream-tile skipping): the WITHIN oracle's result, forward and backward
    _full_case(AttnShape(*shape), WITHIN_NAIVE, seed=61 + sum(shape))


@pytest.mark.parametrize("window", [1, 50, 200])
def test_local_window(window):
    _full_case(AttnShape(1, 96, 4, 4, 2, 128), LOCAL, seed=5, window=window)


@pytest.mark.parametrize("L,n", [(1, 1), (1, 4), (2, 3), (63, 1), (65, 1), (64, 2)])
def test_edge_sizes(L, n):
    for mode in (WITHIN, CROSS):
        _full_case(AttnShape(1, L, n, 2, 1, 64), mode, seed=3)


def test_explicit_scale_and_first_rows():
    s = AttnShape(1, 40, 4, 2, 2, 128)
    _full_case(s, WITHIN, seed=8, scale=0.05)
    q, k, v = inputs.attn_inputs(s, seed=9, with_grad=False)
    _, _, _, o, lse = gpu_fwd(q, k, v, s.n, WITHIN)
    # the first position of each stream sees only itself: O = V exactly (bf16 round trip)
    for p in range(s.n):
        assert torch.equal(o[0, p].cpu(), v[0, p])


def test_deterministic_forward():
    s = AttnShape(1, 300, 4, 4, 2, 128)
    q, k, v = inputs.attn_inputs(s, seed=12, with_grad=False)
    a = gpu_fwd(q, k, v, s.n, CROSS)
    b = gpu_fwd(q, k, v, s.n, CROSS)
    assert torch.equal(a[3], b[3]) and torch.equal(a[4], b[4])


@pytest.mark.parametrize("mode", [WITHIN, CROSS])
def test_prep_halves_with_the_clear_on_a_side_stream(mode):
    # sfa_bwd_row_terms on the main stream, sfa_bwd_clear on another (workspace filled
    # with NaN bytes first), then main + finalize: the oracle's gradients, and dK / dV
    # bit-identical to the one-call sfa_bwd
    s = AttnShape(1, 300, 4, 8, 2, 128)
    q, k, v, do = inputs.attn_inputs(s, seed=14)
    qd, kd, vd, dod = q.cuda(), k.cuda(), v.cuda(), do.cuda()
    o = guards.like(qd)
    lse = guards.empty((s.B, s.Hq, s.nL), torch.float32)
    binding.sfa_fwd(qd, kd, vd, o, lse, s.n, mode)
    ws = guards.empty((binding.sfa_bwd_workspace_bytes(s.B, s.L, s.n, s.Hq, s.Hkv, s.Dh, mode),), torch.uint8, 255)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        binding.sfa_bwd_clear(s.B, s.L, s.n, s.Hq, s.Hkv, s.Dh, mode, ws, stream=side)
        cleared = torch.cuda.Event()
        cleared.record(side)
    binding.sfa_bwd_row_terms(o, dod, lse, s.n, mode, ws, s.Hkv)
    torch.cuda.current_stream().wait_event(cleared)
    dq, dk, dv = guards.like(qd), guards.like(kd), guards.like(vd)
    binding.sfa_bwd_main(qd, kd, vd, dod, dk, dv, s.n, mode, ws)
    binding.sfa_bwd_finalize(dq, s.n, mode, ws, s.Hkv)
    dq1, dk1, dv1 = guards.like(qd), guards.like(kd), guards.like(vd)
    ws1 = guards.like(ws)
    binding.sfa_bwd(qd, kd, vd, o, lse, dod, dq1, dk1, dv1, s.n, mode, ws1)
    torch.cuda.synchronize()
    dq_r, dk_r, dv_r = oracle.sfa_bwd(q, k, v, do, s.n, mode)
    assert_grads_close([("dq", dq.cpu(), dq_r), ("dk", dk.cpu(), dk_r), ("dv", dv.cpu(), dv_r)])
    assert torch.equal(dk.view(torch.int16), dk1.view(torch.int16))
    assert torch.equal(dv.view(torch.int16), dv1.view(torch.int16))


# ------------------------------------------------------------ full-size layers
def _sampled_parity(s: AttnShape, mode, seed, n_rows=192, n_kv=48, repeat=False):
    q, k, v, do = inputs.attn_inputs(s, seed=seed)
    o, lse, dq, dk, dv = gpu_fwd_bwd(q, k, v, do, s.n, mode)
    if repeat:
        # dK and dV are summed in a fixed order inside one CTA: a second run gives the
        # same bits (an operand read before its load has landed would not)
        _, _, _, dk2, dv2 = gpu_fwd_bwd(q, k, v, do, s.n, mode)
        assert torch.equal(dk.view(torch.int16), dk2.view(torch.int16))
        assert torch.equal(dv.view(torch.int16), dv2.view(torch.int16))
    if mode == WITHIN_NAIVE:  # checked against the WITHIN oracle
        mode = WITHIN
    grp = s.Hq // s.Hkv
    edges = [0, 1, 63, 64, 127, 128, s.nL // 2, s.nL - 129, s.nL - 2, s.nL - 1]
    rows = sample_rows(s.B, s.Hq, s.nL, n_rows, seed, edges)
    # forward rows and dQ rows, oracle per K/V group
    for g in range(s.Hkv):
        sel = rows[(rows[:, 1] // grp) == g]
        if not len(sel):
            continue
        qg, kg, vg, dog = group_slices(q, k, v, do, g, grp)
        loc = sel.copy()
        loc[:, 1] -= g * grp
        o_r, l_r = oracle.sfa_fwd_rows(qg, kg, vg, s.n, mode, loc)
        dq_r, _, _ = oracle.sfa_bwd_q_rows(qg, kg, vg, dog, s.n, mode, loc)
        o_g = o[sel[:, 0], sel[:, 2], sel[:, 1]]
        l_g = lse[sel[:, 0], sel[:, 1], sel[:, 2]]
        assert max_abs(o_g, o_r) <= TOL_O
        assert max_abs(l_g, l_r) <= TOL_LSE
        assert_grads_close([("dq rows", dq[sel[:, 0], sel[:, 2], sel[:, 1]], dq_r)])
    # dK / dV rows of one group, complete sums over every query row and head of the
    # group that sees them: keys from the first 128 positions (the longest sums: every
    # later query tile of the problem, all heads of the group), a band in the middle and
    # the last 384 positions
    g = s.Hkv - 1
    ps = kv_sample_positions(s.nL, n_kv, seed + 1)
    kvrows = np.array([[0, 0, p] for p in ps], dtype=np.int64)
    qg, kg, vg, dog = group_slices(q, k, v, do, g, grp)
    dk_r, dv_r = oracle.sfa_bwd_kv_rows(qg, kg, vg, dog, s.n, mode, kvrows)
    assert_grads_close([("dk rows", dk[0, ps, g], dk_r), ("dv rows", dv[0, ps, g], dv_r)])


@pytest.mark.parametrize("mode", [WITHIN, CROSS, WITHIN_NAIVE])
def test_qwen3_8b_class_layer(mode):
    # B=1, L=4096, n=4 (16384 positions), Hq=32, Hkv=8, Dh=128
    _sampled_parity(inputs.SHAPES["qwen3_8b_n4"], mode, seed=1, repeat=True)


@pytest.mark.parametrize("mode", [WITHIN, CROSS])
def test_qwen3_8b_class_layer_one_group_complete(mode):
    # the benchmark layer (B=1, L=4096, n=4, Hq=32, Hkv=8, Dh=128) with one K/V head group
    # checked whole: O and LSE of its 4 query heads at every position, dQ of those heads
    # and dK, dV of its K/V head at every position, against the oracle over the group
    s = inputs.SHAPES["qwen3_8b_n4"]
    q, k, v, do = inputs.attn_inputs(s, seed=1)
    o, lse, dq, dk, dv = gpu_fwd_bwd(q, k, v, do, s.n, mode)
    grp, g = s.Hq // s.Hkv, 5
    hs = slice(g * grp, (g + 1) * grp)
    qg, kg, vg, dog = group_slices(q, k, v, do, g, grp)
    o_r, l_r = oracle.sfa_fwd(qg, kg, vg, s.n, mode)
    assert_fwd_close(o[:, :, hs], lse[:, hs], o_r, l_r)
    dq_r, dk_r, dv_r = oracle.sfa_bwd(qg, kg, vg, dog, s.n, mode)
    assert_grads_close([("dq", dq[:, :, hs], dq_r), ("dk", dk[:, :, g:g + 1], dk_r), ("dv", dv[:, :, g:g + 1], dv_r)])


@pytest.mark.parametrize("mode", [WITHIN, CROSS])
def test_large_moe_class_layer(mode):
    # B=1, L=8192, n=4 (32768 positions), Hq=64, Hkv=8, Dh=128
    _sampled_parity(inputs.SHAPES["moe_large_n4"], mode, seed=21, n_rows=96, n_kv=24, repeat=True)


@pytest.mark.parametrize("mode", [WITHIN, CROSS])
def test_80b_class_layer(mode):
    # B=1, L=4096, n=4 (16384 positions), Hq=24, Hkv=2, Dh=256 (Table 6's 80B heads)
    _sampled_parity(AttnShape(1, 4096, 4, 24, 2, 256), mode, seed=51, n_rows=64, n_kv=16, repeat=True)


@pytest.mark.parametrize("n", [1, 2, 8])
def test_expansion_sweep_layers(n):
    # the n sweep at L=4096, Hq=32, Hkv=8, Dh=128 (WITHIN; CROSS at n=8 is the largest)
    s = AttnShape(1, 4096, n, 32, 8, 128)
    _sampled_parity(s, WITHIN, seed=31 + n, n_rows=64, n_kv=16)
    if n == 8:
        _sampled_parity(s, CROSS, seed=41, n_rows=32, n_kv=8)
