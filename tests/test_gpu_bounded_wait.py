"""The bounded waits of the tcgen05 kernels run out without hanging.

optr_selftest_wait_timeout runs the cache write's exit path against an
mbarrier phase that nothing completes, with a short limit: the wait gives
up, OPTR_DEVERR_TIMEOUT reaches the host, the tensor-memory columns are
freed (a tensor-core cache write afterwards, which allocates the same
columns, runs and matches its own earlier result bit for bit), and the
context stays usable.  No GPU fault is involved: the wait simply ends.
"""
import time

import numpy as np
import pytest
import torch

from paper_2608_02691_gb300 import optr, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02691_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def _tensor_append(p, c, dev):
    pool = optr.new_pool(p, c["num_pages"], device=dev)
    optr.optr_kv_append(p, c["k_ctx"].to(dev), c["v_ctx"].to(dev),
                        c["cu_ctx"].to(dev), c["pos0_ctx"].to(dev),
                        c["block_table"].to(dev), pool)
    torch.cuda.synchronize()
    return pool


def test_wait_runs_out_and_frees_tensor_memory():
    dev = "cuda"
    c = synth.build_case(synth.workload("decode8k", 0, 1 / 32), 0)  # 16 x 256 tokens
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"],
                                append_variant=optr.OPTR_VARIANT_TENSOR)
    before = _tensor_append(p, c, dev)
    assert optr.optr_device_error(p) == 0
    limit_ns = 200_000_000  # 0.2 s
    t0 = time.perf_counter()
    optr.optr_selftest_wait_timeout(p, limit_ns)
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    assert optr.optr_device_error(p) == optr.OPTR_DEVERR_TIMEOUT
    assert dt >= 0.9 * limit_ns * 1e-9, f"the wait ended after {dt:.3f} s"
    assert dt < 10.0
    # the columns are free again and the context is usable
    after = _tensor_append(p, c, dev)
    assert optr.optr_device_error(p) == 0
    assert torch.equal(before, after)


def test_limit_out_of_range_is_refused():
    c = synth.build_case(synth.workload("tiny", 0, 1 / 8), 0)
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"])
    for bad in (0, 999_999, 2_000_000_001):
        with pytest.raises(optr.OptrError):
            optr.optr_selftest_wait_timeout(p, bad)
