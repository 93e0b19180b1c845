"""The decode entry point for callers that cannot allocate device memory.

Some callers of this library have no way to allocate device memory at
decode time (an engine plugin handed only tensors, or a decode loop that
must never call cudaMalloc).  optr_decode_attention_noalloc serves them
from a fixed scratch array inside the library; this test checks, through
the C ABI, that it returns what the workspace entry point returns, on two
calls in a row (the second call reuses the scratch the first one left), and
that a batch too large for the scratch is refused.  The file name makes
pytest collect it last.
"""
import ctypes

import pytest
import torch

from paper_2608_02691_gb300 import optr, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02691_gb300 import build
    build.build()
    torch.cuda.set_device(0)
    return torch.device("cuda", 0)


@pytest.mark.parametrize("name,scale", [("decode8k", 1 / 16), ("ragged", 1 / 32)])
def test_noalloc_matches_workspace_entry_point(dev, name, scale):
    c = synth.build_case(synth.workload(name, 0, scale), 0)
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"])
    pool = optr.new_pool(p, c["num_pages"], device=dev)
    bt = c["block_table"].to(dev)
    optr.optr_kv_append(p, c["k_ctx"].to(dev), c["v_ctx"].to(dev),
                        c["cu_ctx"].to(dev), c["pos0_ctx"].to(dev), bt, pool)
    q, lens = c["q"].to(dev), c["seq_lens_ctx"].to(dev)
    ref = torch.empty(c["B"], c["h_q"], 128, device=dev)
    ws = optr.new_workspace(p, c["B"], bt.shape[1], device=dev)
    optr.optr_decode_attention(p, q, bt, lens, pool, ref, ws)
    for call in range(2):
        out = torch.full_like(ref, float("nan"))
        optr.optr_decode_attention_noalloc(p, q, bt, lens, pool, out)
        torch.cuda.synchronize()
        # the same kernels with the same plan: bit-identical to the
        # workspace call
        assert torch.equal(out, ref), f"{name} noalloc call {call}"
    assert optr.optr_device_error(p) == 0


def test_noalloc_rejects_batches_beyond_the_scratch(dev):
    c = synth.build_case(synth.workload("tiny", 0, 1 / 64), 0)
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"])
    B, max_pages = 4096, 64
    assert optr.optr_decode_workspace_size(p, B, max_pages) > optr.NOALLOC_SCRATCH_BYTES
    bt = torch.zeros(B, max_pages, dtype=torch.int32, device=dev)
    lens = torch.ones(B, dtype=torch.int32, device=dev)
    q = torch.zeros(B, c["h_q"], 128, dtype=torch.bfloat16, device=dev)
    out = torch.empty(B, c["h_q"], 128, device=dev)
    pool = optr.new_pool(p, 1, device=dev)
    with pytest.raises(optr.OptrError) as e:
        optr.optr_decode_attention_noalloc(p, q, bt, lens, pool, out)
    assert e.value.status == -4


def test_noalloc_errors_follow_the_workspace_entry_point(dev):
    """Argument and range errors come out as optr_decode_attention returns
    them, before the scratch-size check: an oversized batch is out of range
    (not a workspace error), a null query with a batch too large for the
    scratch is an invalid argument, and params with BF16 windows are
    refused.  Every case returns before any launch, so the (aligned,
    non-null) device pointers below are never dereferenced."""
    lib = optr.lib()
    c = synth.build_case(synth.workload("tiny", 0, 1 / 64), 0)
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"])
    buf = torch.zeros(1 << 16, dtype=torch.uint8, device=dev)
    a = ctypes.c_void_p(buf.data_ptr())
    ws = ctypes.c_void_p(buf.data_ptr())
    for B, max_pages, q, want in (((1 << 24) + 1, 1, a, -3),
                                  (64, (1 << 26) + 1, a, -3),
                                  (4096, 64, None, -1)):
        got_ws = lib.optr_decode_attention(p.handle, q, a, a, B, max_pages, a, 1,
                                           a, ws, 1 << 16, None)
        got_na = lib.optr_decode_attention_noalloc(p.handle, q, a, a, B,
                                                   max_pages, a, 1, a, None)
        assert got_ws == want and got_na == want, (B, max_pages, got_ws, got_na)
    pw = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"],
                                 sink=64, recent=256)
    assert lib.optr_decode_attention_noalloc(pw.handle, a, a, a, 1, 1, a, 1, a,
                                             None) == -1
