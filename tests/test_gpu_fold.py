"""Value-rotation folding (Appendix "Equivalent Inference Implementation":
R_V folded into W_V and W_O): optr_params_create with R_v = NULL quantizes
values as given and returns the decode output in that basis.  The oracle
runs the same inputs with R_v = I; both append variants, both decode
variants and the fused decode step must match it as the unfolded path does.
"""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_02691_gb300 import optr, synth

import parity_helpers as ph

pytestmark = pytest.mark.gpu

VARIANTS = [optr.OPTR_VARIANT_CUDA_CORE, optr.OPTR_VARIANT_TENSOR]


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02691_gb300 import build
    build.build()
    oracle.build()
    torch.cuda.set_device(0)


def _folded_case(name, scale):
    c = synth.build_case(synth.workload(name, 0, scale), 0)
    eye = torch.eye(128).expand(c["h_kv"], 128, 128).contiguous()
    ref = dict(c)
    ref["R_v"] = eye  # what the oracle sees
    return c, ref


@pytest.mark.parametrize("name,scale", [("tiny", 1.0), ("decode8k", 1 / 32),
                                        ("ragged", 1 / 64)])
@pytest.mark.parametrize("avar", VARIANTS)
@pytest.mark.parametrize("dvar", VARIANTS)
def test_folded_value_rotation(name, scale, avar, dvar):
    c, ref = _folded_case(name, scale)
    pool_ref, u_ctx, u_new = ph.oracle_case(ref)
    dev = "cuda"
    p = optr.optr_params_create(c["R_k"], None, c["mu"], c["h_q"],
                                append_variant=avar, decode_variant=dvar)
    pool = optr.new_pool(p, c["num_pages"], device=dev)
    bt = c["block_table"].to(dev)
    optr.optr_kv_append(p, c["k_ctx"].to(dev), c["v_ctx"].to(dev),
                        c["cu_ctx"].to(dev), c["pos0_ctx"].to(dev), bt, pool)
    out = torch.empty(c["B"], c["h_q"], 128, dtype=torch.float32, device=dev)
    ws = optr.new_workspace(p, c["B"], bt.shape[1], device=dev)
    # the step's new tokens and the decode through the fused step
    optr.optr_decode_step(p, c["q"].to(dev), c["k_new"].to(dev),
                          c["v_new"].to(dev), c["cu_new"].to(dev),
                          c["pos0_new"].to(dev), bt, c["seq_lens"].to(dev),
                          pool, out, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    pg = pool.cpu().numpy()
    for cu, pos0, u in ((c["cu_ctx"], c["pos0_ctx"], u_ctx),
                        (c["cu_new"], c["pos0_new"], u_new)):
        if u is None:
            continue
        pages, slots = ph.token_slots(cu, pos0, c["block_table"])
        ph.compare_append(pg, pool_ref, u, pages, slots)
    # decode of the oracle-written cache with the folded handle (isolates
    # the decode error)
    pool.copy_(torch.from_numpy(pool_ref))
    optr.optr_decode_attention(p, c["q"].to(dev), bt, c["seq_lens"].to(dev),
                               pool, out, ws)
    torch.cuda.synchronize()
    got = out.cpu().double().numpy()
    want = ph.oracle_decode(ref, pool_ref)
    rms = float(np.sqrt(np.mean(want ** 2)))
    err = float(np.abs(got - want).max())
    assert err <= ph.OUT_TOL * rms, (err / rms)


def test_folding_equals_identity_rotation():
    """R_v = NULL and R_v = I give the same bytes and the same output."""
    c, ref = _folded_case("tiny", 1.0)
    outs, pools = [], []
    for R_v in (None, ref["R_v"]):
        p = optr.optr_params_create(c["R_k"], R_v, c["mu"], c["h_q"])
        pool = optr.new_pool(p, c["num_pages"], device="cuda")
        bt = c["block_table"].cuda()
        optr.optr_kv_append(p, c["k_ctx"].cuda(), c["v_ctx"].cuda(),
                            c["cu_ctx"].cuda(), c["pos0_ctx"].cuda(), bt, pool)
        out = torch.empty(c["B"], c["h_q"], 128, dtype=torch.float32, device="cuda")
        ws = optr.new_workspace(p, c["B"], bt.shape[1], device="cuda")
        optr.optr_decode_step(p, c["q"].cuda(), c["k_new"].cuda(), c["v_new"].cuda(),
                              c["cu_new"].cuda(), c["pos0_new"].cuda(), bt,
                              c["seq_lens"].cuda(), pool, out, ws)
        torch.cuda.synchronize()
        outs.append(out.cpu())
        pools.append(pool.cpu())
    assert torch.equal(pools[0], pools[1])
    assert torch.equal(outs[0], outs[1])


def test_decode_step_replays_from_a_cuda_graph():
    """The fused decode step (single-token cache write, query rotation,
    partial, combine; programmatic dependent launches) captured once in a
    CUDA graph and replayed gives the bytes and output of a direct call."""
    c = synth.build_case(synth.workload("decode8k", 0, 1 / 32), 0)
    dev = "cuda"
    res = []
    for use_graph in (False, True):
        p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"])
        pool = optr.new_pool(p, c["num_pages"], device=dev)
        bt = c["block_table"].to(dev)
        optr.optr_kv_append(p, c["k_ctx"].to(dev), c["v_ctx"].to(dev),
                            c["cu_ctx"].to(dev), c["pos0_ctx"].to(dev), bt, pool)
        args = [c["q"].to(dev), c["k_new"].to(dev), c["v_new"].to(dev),
                c["cu_new"].to(dev), c["pos0_new"].to(dev), bt,
                c["seq_lens"].to(dev)]
        out = torch.empty(c["B"], c["h_q"], 128, dtype=torch.float32, device=dev)
        ws = optr.new_workspace(p, c["B"], bt.shape[1], device=dev)
        torch.cuda.synchronize()
        if use_graph:
            s = torch.cuda.Stream()
            s.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(s):  # warm-up outside the capture
                optr.optr_decode_step(p, *args, pool, out, ws)
            torch.cuda.current_stream().wait_stream(s)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                optr.optr_decode_step(p, *args, pool, out, ws)
            out.zero_()
            g.replay()
        else:
            optr.optr_decode_step(p, *args, pool, out, ws)
            optr.optr_decode_step(p, *args, pool, out, ws)
        torch.cuda.synchronize()
        assert optr.optr_device_error(p) == 0
        res.append((pool.cpu(), out.cpu()))
    assert torch.equal(res[0][0], res[1][0])
    assert torch.equal(res[0][1], res[1][1])
