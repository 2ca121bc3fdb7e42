"""GPU parity: the retained suffix positions' top-k candidates (Sec. 3.2, the set and
probabilities Eq. 6 renormalizes) against the fp64 oracle.

Bar: ids bit-exact (the ranking compares the exact bf16/fp32 logits on both sides,
ties to the lower id); probabilities within 1e-5 relative of the fp64 softmax (the
kernel sums exp in fp32 with ex2.approx over up to 126464 entries).
"""
import numpy as np
import pytest
import torch

from oracle import ssm_oracle as O
from paper_2608_23167_gb300 import workloads as W
from tests.gpu_helpers import check_device_error, cuda_or_skip, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return cuda_or_skip()


def _run(dev, logits, k):
    from paper_2608_23167_gb300 import ssm
    n = logits.shape[0]
    ids = torch.full((n, k), -7, dtype=torch.int32, device=dev)
    probs = torch.full((n, k), float("nan"), dtype=torch.float32, device=dev)
    ssm.ssm_suffix_topk(logits.to(dev), k, ids, probs)
    torch.cuda.synchronize()
    check_device_error()
    return ids.cpu().numpy(), probs.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("n,V,dtype,sigma,k", [
    (37, 126464, torch.bfloat16, 4.0, 5),     # serving vocabulary, N(0, 4) stand-in logits
    (9, 126464, torch.bfloat16, 4.0, 8),      # the longest list
    (64, 4096, torch.float32, 3.0, 5),        # tiny workload vocabulary, fp32
    (5, 40, torch.float32, 1.0, 1),           # a single chunk, k = 1
    (3, 65544, torch.bfloat16, 2.0, 3),       # two segments plus a ragged one
])
def test_topk_parity(dev, n, V, dtype, sigma, k):
    g = torch.Generator().manual_seed(n * 1000 + k)
    logits = (torch.randn((n, V), generator=g) * sigma).to(dtype)
    ids, probs = _run(dev, logits, k)
    ref_ids, ref_probs = O.suffix_topk(f64(logits), k)
    assert np.array_equal(ids, ref_ids)
    assert np.allclose(probs, ref_probs, rtol=1e-5, atol=0)


def test_topk_ties_planted_and_order(dev):
    V = 126464
    # integer-valued logits in [-3, 3]: many exact ties, broken by the lower id
    g = torch.Generator().manual_seed(5)
    logits = torch.randint(-3, 4, (6, V), generator=g).to(torch.bfloat16)
    # plant: row 0 one dominant token, row 1 two equal maxima far apart, row 2 the best tokens at the row's end
    logits[0, 99999] = 12.0
    logits[1, 7] = 9.0
    logits[1, 126000] = 9.0
    logits[2, V - 3:] = torch.tensor([8.0, 10.0, 9.0], dtype=torch.bfloat16)
    ids, probs = _run(dev, logits, 8)
    ref_ids, ref_probs = O.suffix_topk(f64(logits), 8)
    assert np.array_equal(ids, ref_ids)
    assert np.allclose(probs, ref_probs, rtol=1e-5)
    assert ids[0, 0] == 99999 and ids[1, :2].tolist() == [7, 126000] and ids[2, :3].tolist() == [V - 2, V - 1, V - 3]
    assert np.all(np.diff(probs, axis=1) <= 0)


def test_topk_top1_matches_unmask(dev):
    """The first candidate is the unmasking pass's argmax and confidence on the same rows."""
    from paper_2608_23167_gb300 import ssm
    B, V = 32, 126464
    logits = W.draw_logits((1, B, V), "bf16", 4.0, 77)
    ids, probs = _run(dev, logits.reshape(B, V), 5)
    conf = torch.empty((1, B), dtype=torch.float32, device=dev)
    arg = torch.empty((1, B), dtype=torch.int32, device=dev)
    commit = torch.empty((1, B), dtype=torch.uint8, device=dev)
    ssm.ssm_unmask(logits.to(dev), torch.ones((1, B), dtype=torch.uint8, device=dev), conf, arg, commit)
    torch.cuda.synchronize()
    assert np.array_equal(ids[:, 0], arg.cpu().numpy()[0])
    assert np.allclose(probs[:, 0], conf.cpu().numpy()[0].astype(np.float64), rtol=1e-5)


def test_topk_errors(dev):
    from paper_2608_23167_gb300 import ssm
    x = torch.zeros((2, 4096), dtype=torch.bfloat16, device=dev)
    ids = torch.empty((2, 9), dtype=torch.int32, device=dev)
    pr = torch.empty((2, 9), dtype=torch.float32, device=dev)
    with pytest.raises(ssm.SSMError) as e:
        ssm.ssm_suffix_topk(x, 9, ids, pr)                      # k above 8
    assert e.value.status == ssm.SSM_ERR_UNSUPPORTED
    with pytest.raises(ssm.SSMError) as e:
        ssm.ssm_suffix_topk(torch.zeros((2, 4099), dtype=torch.bfloat16, device=dev), 5, ids, pr)
    assert e.value.status == ssm.SSM_ERR_UNSUPPORTED          # rows not 16-byte multiples
    with pytest.raises(ssm.SSMError) as e:
        ssm.ssm_suffix_topk(torch.zeros((2, 3 << 20), dtype=torch.bfloat16, device=dev), 5, ids, pr)
    assert e.value.status == ssm.SSM_ERR_UNSUPPORTED          # a row's slice maxima exceed shared memory
    ssm.ssm_suffix_topk(x[:0], 5, ids, pr)                      # no rows: nothing to do
    check_device_error()
