"""GPU: a bounded device wait that expires reports SSM_ERR_TIMEOUT and leaves the context usable.

Every mbarrier wait of the attention forward gives up after the library's wait limit
(ssm_set_wait_limit_ns), records SSM_ERR_TIMEOUT in the device error word and leaves its
loop; the TMA producers then wait (under their own fixed 200 ms bound, not the shortened
limit) for the copies they issued, the MMA warp for every MMA it issued, and the CTA frees
its tensor memory before it exits.  A limit below 20 us launches the forward's polling form
(non-blocking probes, the limit checked between them), so with a 100 ns limit every wait
that is not complete at its first probe within 100 ns expires -- the MMA warp's wait for
the first P of a unit takes a softmax pass, about a microsecond.  The test checks the status
and then that a launch at the default limit gives the same output as before.
Nothing faults or hangs: the failure is a wait that runs out, read back by the host.
"""
import pytest
import torch

from paper_2608_23167_gb300 import workloads as W
from tests.gpu_helpers import check_device_error, cuda_or_skip

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return cuda_or_skip()


@pytest.mark.parametrize("shape", ["two_tiles", "dual_heads", "split_keys"])
def test_attention_wait_timeout_reports_and_recovers(dev, shape):
    """two_tiles: one 589-row problem without cache (units of two query tiles, 32 heads);
    dual_heads: 8 sequences x 101 rows over 512-row caches, 32 heads (units of two kv heads,
    one query tile each); split_keys: the same with 8 heads (one query tile per unit: the two
    softmax slots split the key tiles and meet at the merge wait)."""
    from paper_2608_23167_gb300 import ssm
    h, d = (8 if shape == "split_keys" else 32), 128
    sizes = [(589, 0)] if shape == "two_tiles" else [(101, 512)] * 8
    rows, new_row = [], 0
    for i, (n, c) in enumerate(sizes):
        rows.append((new_row, i * c, n, c))
        new_row += n
    cache_rows = sum(c for _, c in sizes)
    q = W.draw_normal_bf16((new_row, h, d), 1.0, 91).to(dev)
    k = W.draw_normal_bf16((new_row, h, d), 1.0, 92).to(dev)
    v = W.draw_normal_bf16((new_row, h, d), 1.0, 93).to(dev)
    kc = W.draw_normal_bf16((cache_rows, h, d), 1.0, 94).to(dev) if cache_rows else None
    vc = W.draw_normal_bf16((cache_rows, h, d), 1.0, 95).to(dev) if cache_rows else None
    pos = torch.arange(new_row, dtype=torch.int32).to(dev) % 1500 + 512
    probs = ssm.attn_problems_tensor(rows, dev)
    ws = torch.empty(ssm.ssm_attention_workspace_size(new_row, h, h, d), dtype=torch.uint8, device=dev)
    args = (q, k, v, pos, kc, vc, probs, len(rows), max(r[2] for r in rows), max(r[3] for r in rows))
    ref = torch.empty_like(q)
    ssm.ssm_attention_varlen(*args, ref, 5e5, workspace=ws)
    torch.cuda.synchronize()
    check_device_error()
    out = torch.zeros_like(q)
    ssm.ssm_set_wait_limit_ns(100)
    try:
        ssm.ssm_attention_varlen(*args, out, 5e5, workspace=ws)
        torch.cuda.synchronize()
        assert ssm.ssm_get_device_error() == ssm.SSM_ERR_TIMEOUT
    finally:
        ssm.ssm_set_wait_limit_ns(0)
    # the context is intact: the next launch at the default limit completes and matches
    out.zero_()
    ssm.ssm_attention_varlen(*args, out, 5e5, workspace=ws)
    torch.cuda.synchronize()
    check_device_error()
    assert torch.equal(out, ref)
