"""GPU parity of the expansion gather (Eq. 1): bit-exact against the oracle."""
import numpy as np
import pytest
import torch

import guards
import oracle
from paper_2607_08186_gb300 import binding, build, inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def _gpu_expand(tables, ids, status=None):
    n, V, D = tables.shape
    B, L = ids.shape
    td, idd = tables.cuda(), ids.cuda()
    out = guards.empty((B, n * L, D), torch.bfloat16, 7.0)
    binding.hd_expand_embed(td, idd, out, dev_status=status)
    torch.cuda.synchronize()
    return out.cpu()


def _bits(t):
    return t.contiguous().view(torch.int16)


def test_tiny_config():
    # n = 2 tables 512 x 256 ~ N(0, 0.02), ids ~ U[0, 512), L = 64
    tables, ids = inputs.embed_inputs(1, 64, 2, 512, 256, seed=0)
    ref, bad = oracle.expand(tables, ids)
    assert bad == 0
    assert torch.equal(_bits(_gpu_expand(tables, ids)), _bits(ref))


@pytest.mark.parametrize("B,L,n,V,D", [(3, 77, 1, 1000, 8), (2, 129, 3, 300, 136), (1, 1, 8, 5, 64),
                                       (2, 513, 4, 4096, 1024)])
def test_shapes(B, L, n, V, D):
    tables, ids = inputs.embed_inputs(B, L, n, V, D, seed=B + L + n)
    ref, _ = oracle.expand(tables, ids)
    assert torch.equal(_bits(_gpu_expand(tables, ids)), _bits(ref))


def test_out_of_range_ids_flag_and_zero_rows():
    tables, ids = inputs.embed_inputs(2, 50, 4, 100, 64, seed=9)
    ids[0, 5] = 100
    ids[1, 49] = -3
    ids[1, 0] = 2 ** 31 - 1
    ref, bad = oracle.expand(tables, ids)
    assert bad == 3
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = _gpu_expand(tables, ids, st)
    assert int(st.item()) & binding.HD_DEVBIT_INDEX
    assert torch.equal(_bits(out), _bits(ref))
    st.zero_()
    tables2, ids2 = inputs.embed_inputs(1, 10, 2, 100, 64, seed=1)
    _gpu_expand(tables2, ids2, st)
    assert int(st.item()) == 0


def test_full_size_sampled_tokens():
    # the benchmark's gather: L = 4096 tokens, n = 4, D = 4096, V = 151936 (Qwen3-8B-sized tables)
    B, L, n, V, D = 1, 4096, 4, 151936, 4096
    tables, ids = inputs.embed_inputs(B, L, n, V, D, seed=5)
    out = _gpu_expand(tables, ids)
    gen = torch.Generator().manual_seed(0)
    toks = sorted({int(t) for t in torch.randint(0, L, (64,), generator=gen)} | {0, L - 1})
    sub_ids = ids[:, toks]
    ref, _ = oracle.expand(tables, sub_ids)            # oracle on the sampled tokens
    got = torch.stack([out[:, t * n:(t + 1) * n] for t in toks], dim=1).reshape(B, len(toks) * n, D)
    assert torch.equal(_bits(got), _bits(ref))
