"""GPU parity of decoding over the expanded KV cache (Sec. 3.2 "Inference Cost") and
of the cache append, against the oracle, through the C ABI.

Tolerances as for the forward: max|dO| <= 2e-2, max|dLSE| <= 1e-3 (bf16 inputs, fp32
accumulation, P rounded to bf16 for its MMA); the append is bit-exact."""
import pytest
import torch

import guards
import oracle
from paper_2607_08186_gb300 import binding, build, inputs

pytestmark = pytest.mark.gpu

WITHIN, CROSS, LOCAL = inputs.WITHIN, inputs.CROSS, inputs.LOCAL


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def _case(B, Lcap, n, Hq, Hkv, Dh, seed):
    q = inputs.normal_bf16((B, n, Hq, Dh), seed)
    kc = inputs.normal_bf16((B, Lcap * n, Hkv, Dh), seed + 1)
    vc = inputs.normal_bf16((B, Lcap * n, Hkv, Dh), seed + 2)
    return q, kc, vc


def _gpu_decode(q, kc, vc, lens, n, mode, window=0, max_tokens=None, status=None, reps=1):
    B, _, Hq, Dh = q.shape
    Lcap, Hkv = kc.shape[1] // n, kc.shape[2]
    T = Lcap if max_tokens is None else max_tokens
    ws = guards.empty((binding.sfa_decode_workspace_bytes(B, T, n, Hq, Hkv, Dh, mode, window),), torch.uint8,
                      what="decode workspace")
    qd, kd, vd, ld = q.cuda(), kc.cuda(), vc.cuda(), lens.cuda()
    outs = []
    for _ in range(reps):
        o = guards.empty((B, n, Hq, Dh), torch.bfloat16, 7.0)
        lse = guards.empty((B, Hq, n), torch.float32, 7.0)
        binding.sfa_decode(qd, kd, vd, ld, o, n, mode, ws, max_tokens=T, lse=lse, window=window,
                           dev_status=status)
        torch.cuda.synchronize()
        outs.append((o.cpu(), lse.cpu()))
    return outs if reps > 1 else outs[0]


def _check(q, kc, vc, lens, n, mode, window=0, max_tokens=None):
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    o, lse = _gpu_decode(q, kc, vc, lens, n, mode, window, max_tokens, st)
    o_r, lse_r, bad = oracle.decode(q, kc, vc, lens, n, mode, window=window)
    assert bad == 0 and int(st.item()) == 0
    eo = float((o.double() - o_r).abs().max())
    el = float((lse.double() - lse_r).abs().max())
    assert eo <= 2e-2 and el <= 1e-3, (eo, el)


@pytest.mark.parametrize("mode,w", [(WITHIN, 0), (CROSS, 0), (LOCAL, 7)])
def test_tiny(mode, w):
    # B=2, n=2, Hq=4, Hkv=2 (8 query rows of 16), Dh=64, ragged lengths 40 and 17
    q, kc, vc = _case(2, 40, 2, 4, 2, 64, 1)
    _check(q, kc, vc, torch.tensor([40, 17], dtype=torch.int32), 2, mode, w)


@pytest.mark.parametrize("mode,w", [(WITHIN, 0), (CROSS, 0), (LOCAL, 1), (LOCAL, 100)])
@pytest.mark.parametrize("n,Hq,Hkv", [(4, 32, 8), (8, 32, 8), (8, 64, 8), (1, 8, 8), (3, 6, 2), (4, 96, 8),
                                     (8, 128, 8)])
def test_shapes_ragged(mode, w, n, Hq, Hkv):
    # query rows per K/V head: 16 (one m16 tile), 32 (two), 64 and 128 (two and four CTAs
    # per head), 48 (Table 6's 617B layout: 96 query over 8 K/V heads), 1 and 9; lengths
    # 1, 129 and the full capacity in one batch
    Lcap = 300
    q, kc, vc = _case(3, Lcap, n, Hq, Hkv, 128, n + Hq)
    _check(q, kc, vc, torch.tensor([Lcap, 1, 129], dtype=torch.int32), n, mode, w)


@pytest.mark.parametrize("mode,w", [(WITHIN, 0), (CROSS, 0), (LOCAL, 1), (LOCAL, 100)])
@pytest.mark.parametrize("n,Hq,Hkv", [(4, 24, 2), (4, 4, 1), (3, 6, 2), (8, 32, 2), (8, 64, 2)])
def test_head_dim_256_ragged(mode, w, n, Hq, Hkv):
    # head dim 256: Table 6's 80B heads (24 query over 2 K/V heads: 48 query rows per K/V
    # head), 16, 9 and exactly 128 rows (one tcgen05 tile, rows padded to 128), and 256 rows
    # (the mma.sync kernel's row groups); lengths 1, 129 and the capacity
    Lcap = 300
    q, kc, vc = _case(3, Lcap, n, Hq, Hkv, 256, 40 + n + Hq)
    _check(q, kc, vc, torch.tensor([Lcap, 1, 129], dtype=torch.int32), n, mode, w)


@pytest.mark.parametrize("Hq,Hkv,Dh", [(8, 2, 128), (24, 2, 256)])
def test_max_tokens_below_capacity(Hq, Hkv, Dh):
    q, kc, vc = _case(2, 500, 4, Hq, Hkv, Dh, 5)
    _check(q, kc, vc, torch.tensor([200, 77], dtype=torch.int32), 4, CROSS, max_tokens=200)


def test_bad_lengths_zero_rows_and_flag():
    q, kc, vc = _case(3, 50, 2, 4, 2, 128, 6)
    lens = torch.tensor([0, 50, 51], dtype=torch.int32)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    o, lse = _gpu_decode(q, kc, vc, lens, 2, CROSS, status=st)
    assert int(st.item()) & binding.HD_DEVBIT_INDEX
    o_r, lse_r, bad = oracle.decode(q, kc, vc, lens, 2, CROSS)
    assert bad == 2
    assert torch.count_nonzero(o[0]) == 0 and torch.count_nonzero(o[2]) == 0
    assert torch.isinf(lse[0]).all() and torch.isinf(lse[2]).all()
    assert float((o[1].double() - o_r[1]).abs().max()) <= 2e-2


def test_deterministic():
    q, kc, vc = _case(2, 700, 4, 32, 8, 128, 7)
    runs = _gpu_decode(q, kc, vc, torch.tensor([700, 350], dtype=torch.int32), 4, CROSS, reps=3)
    for o, lse in runs[1:]:
        assert torch.equal(o.view(torch.int16), runs[0][0].view(torch.int16))
        assert torch.equal(lse, runs[0][1])


@pytest.mark.parametrize("mode", [WITHIN, CROSS])
def test_full_size(mode):
    # Qwen3-8B-class heads, n = 4, an 8192-token context (32768 cached positions), B = 2
    # with one shorter sequence; every output row checked against the oracle
    q, kc, vc = _case(2, 8192, 4, 32, 8, 128, 8)
    _check(q, kc, vc, torch.tensor([8192, 5000], dtype=torch.int32), 4, mode)


@pytest.mark.parametrize("mode", [WITHIN, CROSS])
def test_full_size_head_dim_256(mode):
    # 80B-class heads (Hq=24, Hkv=2, Dh=256), n = 4, an 8192-token context, B = 2 with one
    # shorter sequence; every output row checked against the oracle
    q, kc, vc = _case(2, 8192, 4, 24, 2, 256, 18)
    _check(q, kc, vc, torch.tensor([8192, 3001], dtype=torch.int32), 4, mode)


@pytest.mark.parametrize("mode", [WITHIN, CROSS])
def test_full_size_617b_heads(mode):
    # the 617B configuration's head layout (96 query over 8 K/V heads, Dh=128: 48 query
    # rows per K/V head, two row groups), n = 4, an 8192-token context, B = 2
    q, kc, vc = _case(2, 8192, 4, 96, 8, 128, 28)
    _check(q, kc, vc, torch.tensor([8192, 4321], dtype=torch.int32), 4, mode)


def test_kv_append_bit_exact_and_flag():
    B, n, Lcap, Hkv, Dh = 4, 4, 33, 8, 128
    kc = inputs.normal_bf16((B, Lcap * n, Hkv, Dh), 9)
    vc = inputs.normal_bf16((B, Lcap * n, Hkv, Dh), 10)
    kn = inputs.normal_bf16((B, n, Hkv, Dh), 11)
    vn = inputs.normal_bf16((B, n, Hkv, Dh), 12)
    lens = torch.tensor([1, 33, 17, 34], dtype=torch.int32)        # the last is out of range
    kd, vd = kc.cuda(), vc.cuda()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    binding.sfa_kv_append(kn.cuda(), vn.cuda(), kd, vd, lens.cuda(), n, dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & binding.HD_DEVBIT_INDEX
    k_ref, bad = oracle.kv_append(kn, kc, lens, n)
    v_ref, _ = oracle.kv_append(vn, vc, lens, n)
    assert bad == 1
    assert torch.equal(kd.cpu().view(torch.int16), k_ref.view(torch.int16))
    assert torch.equal(vd.cpu().view(torch.int16), v_ref.view(torch.int16))


@pytest.mark.parametrize("Hq,Hkv,Dh", [(8, 2, 128), (24, 2, 256)])
def test_append_then_decode_equals_forward_rows(Hq, Hkv, Dh):
    # a prefilled cache (the forward's K/V) plus one appended token decodes to the
    # forward's rows of that token, for every mask
    B, L, n = 1, 50, 4
    q, k, v = inputs.attn_inputs(inputs.AttnShape(B, L, n, Hq, Hkv, Dh), seed=13, with_grad=False)
    kd = torch.zeros(B, L * n, Hkv, Dh, dtype=torch.bfloat16, device="cuda")
    vd = torch.zeros_like(kd)
    kd[:, :(L - 1) * n] = k[:, :(L - 1) * n].cuda()
    vd[:, :(L - 1) * n] = v[:, :(L - 1) * n].cuda()
    lens = torch.tensor([L], dtype=torch.int32)
    binding.sfa_kv_append(k[:, (L - 1) * n:].contiguous().cuda(), v[:, (L - 1) * n:].contiguous().cuda(), kd, vd,
                          lens.cuda(), n)
    torch.cuda.synchronize()
    qn = q[:, (L - 1) * n:].contiguous()
    for mode, w in ((WITHIN, 0), (CROSS, 0), (LOCAL, 9)):
        o, lse = _gpu_decode(qn, kd.cpu(), vd.cpu(), lens, n, mode, w)
        rows = [(0, h, p) for h in range(Hq) for p in range((L - 1) * n, L * n)]
        o_r, lse_r = oracle.sfa_fwd_rows(q, k, v, n, mode, rows, window=w)
        got = torch.stack([o[0, p - (L - 1) * n, h] for (_, h, p) in rows]).double()
        assert float((got - o_r).abs().max()) <= 2e-2
        got_l = torch.tensor([float(lse[0, h, p - (L - 1) * n]) for (_, h, p) in rows], dtype=torch.float64)
        assert float((got_l - lse_r).abs().max()) <= 1e-3


@pytest.mark.parametrize("Hq,Hkv,Dh", [(8, 2, 128), (24, 2, 256)])
def test_serving_loop_in_a_cuda_graph(Hq, Hkv, Dh):
    # one step of a serving loop (append the new token's n K/V rows, then an intra-stream
    # and a cross-stream decode over the cache) captured once as a CUDA graph and replayed
    # while the sequences grow; every replay equals the oracle on the cache as it stands
    # (head dim 256 with 24 over 2 heads: the tcgen05 decode kernel)
    B, n, Lcap = 2, 4, 64
    lens0 = [20, 33]
    kc = guards.zeros((B, Lcap * n, Hkv, Dh), torch.bfloat16)
    vc = guards.like(kc, 0)
    for b, t in enumerate(lens0):
        kc[b, :t * n] = inputs.normal_bf16((t * n, Hkv, Dh), 20 + b).cuda()
        vc[b, :t * n] = inputs.normal_bf16((t * n, Hkv, Dh), 30 + b).cuda()
    lens = torch.tensor(lens0, dtype=torch.int32, device="cuda")
    qs = torch.zeros(B, n, Hq, Dh, dtype=torch.bfloat16, device="cuda")
    kn, vn = torch.zeros(B, n, Hkv, Dh, dtype=torch.bfloat16, device="cuda"), torch.zeros(B, n, Hkv, Dh,
                                                                                          dtype=torch.bfloat16,
                                                                                          device="cuda")
    outs = {m: (guards.empty((B, n, Hq, Dh), torch.bfloat16), guards.empty((B, Hq, n), torch.float32))
            for m in (WITHIN, CROSS)}
    wss = {m: guards.empty((binding.sfa_decode_workspace_bytes(B, Lcap, n, Hq, Hkv, Dh, m),), torch.uint8)
           for m in (WITHIN, CROSS)}
    st = torch.zeros(1, dtype=torch.int32, device="cuda")

    def step():
        binding.sfa_kv_append(kn, vn, kc, vc, lens, n, dev_status=st)
        for m in (WITHIN, CROSS):
            binding.sfa_decode(qs, kc, vc, lens, outs[m][0], n, m, wss[m], max_tokens=Lcap, lse=outs[m][1],
                               dev_status=st)

    lens += 1
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()  # warm-up outside the capture (also the first step of the loop)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    for it in range(3):
        if it > 0:  # the captured step reads these buffers: refill them, grow the sequences
            lens += 1
            qs.copy_(inputs.normal_bf16((B, n, Hq, Dh), 100 + it).cuda())
            kn.copy_(inputs.normal_bf16((B, n, Hkv, Dh), 200 + it).cuda())
            vn.copy_(inputs.normal_bf16((B, n, Hkv, Dh), 300 + it).cuda())
            graph.replay()
        else:  # the warm-up already ran step 0 on zero q / K / V rows: run it again with data
            qs.copy_(inputs.normal_bf16((B, n, Hq, Dh), 100).cuda())
            kn.copy_(inputs.normal_bf16((B, n, Hkv, Dh), 200).cuda())
            vn.copy_(inputs.normal_bf16((B, n, Hkv, Dh), 300).cuda())
            graph.replay()
        torch.cuda.synchronize()
        assert int(st.item()) == 0
        lh = lens.cpu()
        for m in (WITHIN, CROSS):
            o_r, lse_r, bad = oracle.decode(qs.cpu(), kc.cpu(), vc.cpu(), lh, n, m)
            assert bad == 0
            assert float((outs[m][0].cpu().double() - o_r).abs().max()) <= 2e-2
            assert float((outs[m][1].cpu().double() - lse_r).abs().max()) <= 1e-3
    assert lens.cpu().tolist() == [t + 3 for t in lens0]
