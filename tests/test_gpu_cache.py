"""GPU parity: prefix-cache append (prefix caching, Sec. 4.8 "+PC.") against the fp64 oracle.

Bar: appended values bit-exact; appended keys within one bfloat16 spacing of the
oracle's fp64 rotation (the kernel rotates in fp32 with fp32 sin/cos of an angle
reduced in fp64, then rounds once); every other cache row bit-exactly unchanged.
A key appended here and the same key rotated by the attention's pre-pass give
the same attention output as the oracle within the attention tolerance.
"""
import numpy as np
import pytest
import torch

from oracle import ssm_oracle as O
from paper_2608_23167_gb300 import workloads as W
from tests.gpu_helpers import assert_attention_close, bf16_ulp, check_device_error, cuda_or_skip, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return cuda_or_skip()


def _append(dev, batch, cache_rows, n, h_kv, d, theta, start, seed, pos=None):
    from paper_2608_23167_gb300 import ssm
    kc = W.draw_normal_bf16((batch, cache_rows, h_kv, d), 1.0, seed)
    vc = W.draw_normal_bf16((batch, cache_rows, h_kv, d), 1.0, seed + 1)
    kn = W.draw_normal_bf16((batch, n, h_kv, d), 1.0, seed + 2)
    vn = W.draw_normal_bf16((batch, n, h_kv, d), 1.0, seed + 3)
    if pos is None:
        g = torch.Generator().manual_seed(seed + 4)
        pos = (start + torch.randperm(8 * n + 3, generator=g)[:n]).to(torch.int32)
    kc_d, vc_d = kc.to(dev), vc.to(dev)
    ssm.ssm_cache_append(kn.to(dev), vn.to(dev), pos.to(dev), kc_d, vc_d, start, theta)
    torch.cuda.synchronize()
    check_device_error()
    ref_k, ref_v = O.cache_append(f64(kc), f64(vc), f64(kn), f64(vn), pos.numpy(), theta, start)
    return kc_d.cpu(), vc_d.cpu(), kc, vc, ref_k, ref_v


@pytest.mark.parametrize("batch,cache_rows,n,h_kv,d,theta,start", [
    (1, 96, 32, 4, 64, 1e4, 64),       # tiny: one 32-token block after a 64-token prompt
    (2, 3072, 32, 32, 128, 5e5, 1024),  # long-sequence shape: block 0 appended after the prompt
    (3, 700, 37, 2, 128, 1e6, 663),    # ragged row count, block ends exactly at the cache end
    (1, 50, 1, 8, 64, 0.0, 0),         # one row, no rotation, at row 0
])
def test_cache_append_parity(dev, batch, cache_rows, n, h_kv, d, theta, start):
    got_k, got_v, kc, vc, ref_k, ref_v = _append(dev, batch, cache_rows, n, h_kv, d, theta, start, seed=31)
    rows = slice(start, start + n)
    # values: a copy
    assert torch.equal(got_v[:, rows], torch.from_numpy(ref_v[:, rows]).to(torch.bfloat16))
    # keys: within one bf16 spacing of the fp64 rotation
    gk = f64(got_k[:, rows])
    rk = ref_k[:, rows]
    assert np.all(np.abs(gk - rk) <= bf16_ulp(rk) + 1e-30), float(np.max(np.abs(gk - rk) / bf16_ulp(rk)))
    # nothing else moved
    keep = torch.ones(cache_rows, dtype=torch.bool)
    keep[rows] = False
    assert torch.equal(got_k[:, keep], kc[:, keep]) and torch.equal(got_v[:, keep], vc[:, keep])


def test_cache_append_then_attention_matches_oracle(dev):
    """A block appended to the cache is read by the attention like any cached key."""
    from paper_2608_23167_gb300 import ssm
    batch, P, Bk, h, d, theta = 1, 256, 32, 4, 128, 5e5
    got_k, got_v, _, _, ref_k, ref_v = _append(dev, batch, P + Bk, Bk, h, d, theta, P, seed=41,
                                              pos=torch.arange(P, P + Bk, dtype=torch.int32))
    n_q = 48
    q = W.draw_normal_bf16((batch, n_q, h, d), 1.0, 51)
    k = W.draw_normal_bf16((batch, n_q, h, d), 1.0, 52)
    v = W.draw_normal_bf16((batch, n_q, h, d), 1.0, 53)
    pos = torch.arange(P + Bk, P + Bk + n_q, dtype=torch.int32)
    out = torch.empty((batch, n_q, h, d), dtype=torch.bfloat16, device=dev)
    ssm.ssm_attention(q.to(dev), k.to(dev), v.to(dev), pos.to(dev), got_k.to(dev), got_v.to(dev), out, theta)
    torch.cuda.synchronize()
    check_device_error()
    # the oracle reads its own appended cache (fp64 keys rounded to the bf16 the cache stores)
    ref, _ = O.attention(f64(q), f64(k), f64(v), pos.numpy(), O.bf16_round(ref_k), ref_v, theta)
    assert_attention_close(f64(out), ref, "attention over the appended cache")


def test_cache_append_errors(dev):
    from paper_2608_23167_gb300 import ssm
    kn = torch.zeros((1, 8, 2, 64), dtype=torch.bfloat16, device=dev)
    kc = torch.zeros((1, 16, 2, 64), dtype=torch.bfloat16, device=dev)
    pos = torch.arange(8, dtype=torch.int32, device=dev)
    with pytest.raises(ssm.SSMError) as e:
        ssm.ssm_cache_append(kn, kn, pos, kc, kc.clone(), 9, 1e4)   # rows 9..16 do not fit in 16
    assert e.value.status == ssm.SSM_ERR_CAPACITY
    bad = torch.zeros((1, 8, 2, 48), dtype=torch.bfloat16, device=dev)
    with pytest.raises(ssm.SSMError) as e:
        ssm.ssm_cache_append(bad, bad, pos, torch.zeros((1, 16, 2, 48), dtype=torch.bfloat16, device=dev),
                             torch.zeros((1, 16, 2, 48), dtype=torch.bfloat16, device=dev), 0, 1e4)
    assert e.value.status == ssm.SSM_ERR_UNSUPPORTED
    # zero rows: nothing to do
    ssm.ssm_cache_append(kn[:, :0], kn[:, :0], pos[:0], kc, kc.clone(), 16, 1e4)
    check_device_error()
