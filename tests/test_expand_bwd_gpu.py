"""GPU parity of the expansion backward (adjoint of Eq. 1) and of the final-stream
selection the loss reads (Eq. 2) with its adjoint, against the oracle.

Selection and its adjoint are bit copies: bit-exact.  The expansion backward sums
bf16 rows in fp32; the fp64 oracle differs from it only by rounding, bounded per
element by (m + 1) * 2^-24 * (sum of |terms| + |initial value|) with m the largest
number of occurrences of one id (the bound of sequential fp32 summation, which also
covers the kernel's blocked order for long runs).  The kernel's sums are also
checked bitwise for repeatability."""
import pytest
import torch

import guards
import oracle
from paper_2607_08186_gb300 import binding, build, inputs

pytestmark = pytest.mark.gpu

U32 = 2.0 ** -24


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def _gpu_expand_bwd(dX, ids, n, V, dE0=None, status=None, reps=1):
    B, nL, D = dX.shape
    L = nL // n
    ws = guards.empty((binding.hd_expand_embed_bwd_workspace_bytes(B, L),), torch.uint8, what="expand bwd ws")
    xd, idd = dX.cuda(), ids.cuda()
    outs = []
    for _ in range(reps):
        dE = guards.zeros((n, V, D), torch.float32)
        if dE0 is not None:
            dE.copy_(dE0)
        binding.hd_expand_embed_bwd(xd, idd, dE, ws, dev_status=status)
        torch.cuda.synchronize()
        outs.append(dE.cpu())
    return outs if reps > 1 else outs[0]


def _max_run(ids, V):
    valid = ids[(ids >= 0) & (ids < V)].to(torch.int64)
    return int(torch.bincount(valid).max()) if valid.numel() else 0


def _check_sum(got, dX, ids, n, V, dE0=None):
    ref = oracle.expand_bwd(dX, ids, n, V, dE0)
    mag = oracle.expand_bwd(dX.float().abs(), ids, n, V, None if dE0 is None else dE0.abs())
    tol = (_max_run(ids, V) + 1) * U32 * mag
    err = (got.double() - ref).abs()
    bad = err > tol
    assert not bool(bad.any()), f"{int(bad.sum())} elements off, max err {float(err.max()):.3e}"


def test_tiny_config():
    # L = 64 tokens, n = 2 streams, V = 512, D = 256; ids ~ U[0, 512) with repeats by chance
    B, L, n, V, D = 1, 64, 2, 512, 256
    dX = inputs.normal_bf16((B, n * L, D), seed=3)
    ids = inputs.token_ids(B, L, V, seed=3)
    _check_sum(_gpu_expand_bwd(dX, ids, n, V), dX, ids, n, V)


@pytest.mark.parametrize("B,L,n,V,D,zipf", [
    (3, 77, 1, 1000, 8, 0.0),        # n = 1, the smallest row (one 16-byte chunk)
    (2, 129, 3, 300, 136, 0.0),      # odd n, ragged slice of chunks
    (1, 1, 8, 5, 64, 0.0),           # one token
    (2, 513, 4, 64, 1024, 0.0),      # ~16 occurrences of every id
    (1, 5000, 2, 37, 64, 0.0),       # 5000 tokens: sorted by rank count (20 x 20 tiles)
    (4, 4500, 1, 3000, 64, 1.0),     # 18000 tokens: bitonic sort, global steps past 4096 keys
    (1, 16384, 1, 700, 16, 0.0),     # the largest batch sorted by rank count
    (4, 1500, 4, 20000, 512, 1.1),   # Zipf ids: long runs of the frequent ids
])
def test_shapes_accumulate(B, L, n, V, D, zipf):
    dX = inputs.normal_bf16((B, n * L, D), seed=B + L + n)
    ids = inputs.token_ids(B, L, V, seed=L, zipf=zipf)
    dE0 = inputs.normal_bf16((n, V, D), seed=77, std=0.5).float()   # accumulate into existing values
    _check_sum(_gpu_expand_bwd(dX, ids, n, V, dE0), dX, ids, n, V, dE0)


def test_single_id_repeated_everywhere():
    # every token has the same id: one run of B*L tokens, summed in token order
    B, L, n, V, D = 2, 1700, 4, 9, 256
    dX = inputs.normal_bf16((B, n * L, D), seed=11)
    ids = torch.full((B, L), 7, dtype=torch.int32)
    got = _gpu_expand_bwd(dX, ids, n, V)
    _check_sum(got, dX, ids, n, V)
    assert torch.count_nonzero(got[:, :7]) == 0 and torch.count_nonzero(got[:, 8:]) == 0


def test_run_lengths_around_the_split():
    # ids occurring 31, 32, 33, 64 and 257 times (runs up to 32 tokens are summed in token
    # order, longer ones in eight token blocks), plus 100 other tokens, shuffled
    counts = {5: 31, 6: 32, 7: 33, 8: 64, 9: 257}
    gen = torch.Generator().manual_seed(4)
    rest = torch.randint(10, 500, (100,), generator=gen)
    flat = torch.cat([torch.full((c,), v) for v, c in counts.items()] + [rest])
    flat = flat[torch.randperm(flat.numel(), generator=gen)]
    B, n, V, D = 1, 2, 500, 128
    ids = flat.view(B, -1).to(torch.int32)
    L = ids.shape[1]
    dX = inputs.normal_bf16((B, n * L, D), seed=13)
    dE0 = inputs.normal_bf16((n, V, D), seed=14).float()
    _check_sum(_gpu_expand_bwd(dX, ids, n, V, dE0), dX, ids, n, V, dE0)


def test_plan_once_apply_twice_on_another_stream():
    # a plan built on a side stream, applied (after an event) to two different gradients
    B, L, n, V, D = 2, 700, 4, 300, 256
    ids = inputs.token_ids(B, L, V, seed=15, zipf=1.0)
    dX1 = inputs.normal_bf16((B, n * L, D), seed=16)
    dX2 = inputs.normal_bf16((B, n * L, D), seed=17)
    ws = guards.empty((binding.hd_expand_embed_bwd_workspace_bytes(B, L),), torch.uint8, what="expand bwd ws")
    side = torch.cuda.Stream()
    idd = ids.cuda()
    torch.cuda.synchronize()
    with torch.cuda.stream(side):
        binding.hd_expand_embed_bwd_plan(idd, V, ws, stream=side)
        done = torch.cuda.Event()
        done.record(side)
    torch.cuda.current_stream().wait_event(done)
    dE = guards.zeros((n, V, D), torch.float32)
    binding.hd_expand_embed_bwd_apply(dX1.cuda(), dE, ws, L)
    torch.cuda.synchronize()
    _check_sum(dE.cpu(), dX1, ids, n, V)
    dE2 = guards.zeros((n, V, D), torch.float32)
    binding.hd_expand_embed_bwd_apply(dX2.cuda(), dE2, ws, L)
    torch.cuda.synchronize()
    _check_sum(dE2.cpu(), dX2, ids, n, V)
    # plan + apply gives the one-call result bit for bit
    one = _gpu_expand_bwd(dX2, ids, n, V)
    assert torch.equal(one.view(torch.int32), dE2.cpu().view(torch.int32))


def test_apply_skips_what_the_plan_does_not_cover():
    # a plan for V = 300 applied to tables of V = 150 rows: ids >= 150 contribute nothing
    # and the rest sum as usual; a workspace of random bytes (no plan at all) gives
    # meaningless sums but every access stays inside the buffers
    B, L, n, V, D = 2, 700, 4, 300, 128
    ids = inputs.token_ids(B, L, V, seed=18, zipf=1.0)
    dX = inputs.normal_bf16((B, n * L, D), seed=19)
    ws = guards.empty((binding.hd_expand_embed_bwd_workspace_bytes(B, L),), torch.uint8, what="expand bwd ws")
    binding.hd_expand_embed_bwd_plan(ids.cuda(), V, ws)
    dE = guards.zeros((n, 150, D), torch.float32)
    binding.hd_expand_embed_bwd_apply(dX.cuda(), dE, ws, L)
    torch.cuda.synchronize()
    _check_sum(dE.cpu(), dX, ids, n, 150)
    g = torch.Generator().manual_seed(20)
    ws.copy_(torch.randint(0, 256, (ws.numel(),), dtype=torch.uint8, generator=g))
    dE.zero_()
    binding.hd_expand_embed_bwd_apply(dX.cuda(), dE, ws, L)
    torch.cuda.synchronize()
    assert bool(torch.isfinite(dE).all())


def test_deterministic_bits():
    B, L, n, V, D = 2, 3000, 4, 50, 512
    dX = inputs.normal_bf16((B, n * L, D), seed=12)
    ids = inputs.token_ids(B, L, V, seed=12, zipf=1.0)
    a, b, c = _gpu_expand_bwd(dX, ids, n, V, reps=3)
    assert torch.equal(a.view(torch.int32), b.view(torch.int32))
    assert torch.equal(a.view(torch.int32), c.view(torch.int32))


def test_out_of_range_ids_flag_and_contribute_nothing():
    B, L, n, V, D = 2, 50, 4, 100, 64
    dX = inputs.normal_bf16((B, n * L, D), seed=9)
    ids = inputs.token_ids(B, L, V, seed=9)
    ids[0, 5] = 100
    ids[1, 49] = -3
    ids[1, 0] = 2 ** 31 - 1
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    got = _gpu_expand_bwd(dX, ids, n, V, status=st)
    assert int(st.item()) & binding.HD_DEVBIT_INDEX
    _check_sum(got, dX, ids, n, V)
    st.zero_()
    ids2 = inputs.token_ids(B, L, V, seed=10)
    _gpu_expand_bwd(dX, ids2, n, V, status=st)
    assert int(st.item()) == 0


def test_full_size_sampled_ids():
    # the training step's shapes: L = 4096 tokens, n = 4, D = 4096, V = 151936 (Qwen3-8B-sized
    # tables, 10 GB of fp32 gradient); Zipf ids.  Rows of sampled ids are checked against the
    # oracle on the sub-problem of the tokens that carry them; an id that does not occur
    # keeps its rows untouched.
    B, L, n, V, D = 1, 4096, 4, 151936, 4096
    dX = inputs.normal_bf16((B, n * L, D), seed=21)
    ids = inputs.token_ids(B, L, V, seed=21, zipf=1.0)
    ws = guards.empty((binding.hd_expand_embed_bwd_workspace_bytes(B, L),), torch.uint8, what="expand bwd ws")
    dE = guards.zeros((n, V, D), torch.float32)
    xd = dX.cuda()
    binding.hd_expand_embed_bwd(xd, ids.cuda(), dE, ws)
    torch.cuda.synchronize()
    present = torch.unique(ids).tolist()
    gen = torch.Generator().manual_seed(0)
    pick = sorted({present[int(i)] for i in torch.randint(0, len(present), (40,), generator=gen)} |
                  {present[0], present[-1]})
    seen = set(present)
    absent = next(v for v in range(V) if v not in seen)
    sel = torch.tensor(pick, dtype=torch.int32)
    tok_mask = torch.isin(ids[0], sel)
    toks = torch.nonzero(tok_mask).flatten()
    sub_ids = torch.searchsorted(sel, ids[0, toks]).to(torch.int32).view(1, -1)
    rows = (toks.view(-1, 1) * n + torch.arange(n).view(1, -1)).flatten()
    sub_dX = dX[0, rows].view(1, -1, D)
    got = torch.stack([dE[:, v].cpu() for v in pick], dim=1)           # [n][len(pick)][D]
    _check_sum(got, sub_dX, sub_ids, n, len(pick))
    assert torch.count_nonzero(dE[:, absent]).item() == 0


def _gpu_select(X, n):
    B, nL, D = X.shape
    y = guards.empty((B, nL // n, D), torch.bfloat16, 7.0)
    binding.hd_select_final_stream(X.cuda(), y, n)
    torch.cuda.synchronize()
    return y.cpu()


def _gpu_select_bwd(dY, n):
    B, L, D = dY.shape
    dx = guards.empty((B, n * L, D), torch.bfloat16, 7.0)
    binding.hd_select_final_stream_bwd(dY.cuda(), dx, n)
    torch.cuda.synchronize()
    return dx.cpu()


def _bits(t):
    return t.contiguous().view(torch.int16)


@pytest.mark.parametrize("B,L,n,D", [(1, 64, 2, 256), (3, 77, 1, 8), (2, 129, 3, 136), (1, 1, 8, 64),
                                     (1, 4096, 4, 4096)])
def test_select_final_and_adjoint_bit_exact(B, L, n, D):
    X = inputs.normal_bf16((B, n * L, D), seed=L + n)
    assert torch.equal(_bits(_gpu_select(X, n)), _bits(oracle.select_final(X, n)))
    dY = inputs.normal_bf16((B, L, D), seed=L + n + 1)
    assert torch.equal(_bits(_gpu_select_bwd(dY, n)), _bits(oracle.select_final_bwd(dY, n)))
