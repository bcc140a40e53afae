"""The failure path of the tensor-core kernels, exercised without a fault: a bounded
mbarrier wait (the one every tcgen05 kernel uses) on a barrier nothing arrives on runs
out after about a second, reports HD_DEVBIT_TIMEOUT through the device status word and
returns; the context stays usable (a forward right after it matches the oracle)."""
import time

import pytest
import torch

import oracle
from paper_2607_08186_gb300 import binding, build, inputs

from parity import assert_fwd_close, gpu_fwd

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def test_bounded_wait_runs_out_and_reports():
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    res = torch.full((1,), 7, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    binding.hd_selftest_bounded_wait(st, res)
    torch.cuda.synchronize()
    waited = time.perf_counter() - t0
    assert int(res.item()) == 0                          # the wait gave up
    assert int(st.item()) & binding.HD_DEVBIT_TIMEOUT    # and said so
    assert 0.2 < waited < 20.0, waited                   # after its bound, not at once
    # the context is intact: a forward right after matches the oracle
    s = inputs.SHAPES["tiny"]
    q, k, v, _ = inputs.attn_inputs(s, seed=0)
    _, _, _, o, lse = gpu_fwd(q, k, v, s.n, inputs.WITHIN)
    o_r, lse_r = oracle.sfa_fwd(q, k, v, s.n, inputs.WITHIN)
    assert_fwd_close(o.cpu(), lse.cpu(), o_r, lse_r)
