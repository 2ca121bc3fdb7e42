"""GPU parity: vocabulary softmax, confidence, argmax and the commit rules.

Bars: argmax bit-exact (it compares input values only, so it is exact even
where probabilities are close); conf and p2 within 1e-5 relative of the fp64
oracle; commits bit-exact for every position whose decision is not within
rounding of the threshold (|score - threshold| > 1e-5) and, for the
confidence ranking, where the competing confidences differ by more than 1e-3.
"""
import numpy as np
import pytest
import torch

from oracle import ssm_oracle as O
from paper_2608_23167_gb300 import workloads as W
from tests.gpu_helpers import check_device_error, cuda_or_skip, f64

pytestmark = pytest.mark.gpu

MODES = {"threshold": O.MODE_THRESHOLD, "topk": O.MODE_TOPK, "margin": O.MODE_MARGIN}


@pytest.fixture(scope="module")
def dev():
    return cuda_or_skip()


def _gpu_unmask(dev, logits, masked, mode, threshold, topk, min_commit):
    from paper_2608_23167_gb300 import ssm
    batch, B, V = logits.shape
    conf = torch.full((batch, B), -1.0, device=dev)
    p2 = torch.full((batch, B), -1.0, device=dev)
    arg = torch.full((batch, B), -5, dtype=torch.int32, device=dev)
    commit = torch.full((batch, B), 9, dtype=torch.uint8, device=dev)
    ssm.ssm_unmask(logits.to(dev), masked.to(dev), conf, arg, commit, p2=p2, mode=mode, threshold=threshold,
                   topk=topk, min_commit=min_commit)
    torch.cuda.synchronize()
    check_device_error()
    return conf.cpu().double().numpy(), arg.cpu().numpy(), p2.cpu().double().numpy(), commit.cpu().numpy()


def _check_commits(conf_r, p2_r, masked, commit_g, commit_r, mode, threshold, topk, min_commit):
    batch, B = conf_r.shape
    for b in range(batch):
        cand = [j for j in range(B) if masked[b, j]]
        score = conf_r[b] if mode != O.MODE_MARGIN else conf_r[b] - p2_r[b]
        ambiguous = False
        if mode != O.MODE_TOPK:
            ambiguous = any(abs(score[j] - threshold) <= 1e-5 for j in cand)
        confs = sorted((conf_r[b, j] for j in cand), reverse=True)
        if any(abs(confs[i] - confs[i + 1]) <= 1e-3 for i in range(len(confs) - 1)):
            # the ranking part of the rule is not unique at this precision: check validity only
            if mode == O.MODE_TOPK:
                assert commit_g[b].sum() == min(topk, len(cand))
                continue
            ambiguous_rank = True
        else:
            ambiguous_rank = False
        if ambiguous:
            continue
        passing = {j for j in cand if score[j] > threshold}
        if mode != O.MODE_TOPK and not ambiguous_rank:
            assert commit_g[b].tolist() == commit_r[b].tolist(), b
        elif mode != O.MODE_TOPK:
            # every passing position committed; the count follows the min-commit rule
            assert all(commit_g[b, j] for j in passing)
            assert commit_g[b].sum() == max(len(passing), min(min_commit, len(cand)))
        else:
            assert commit_g[b].tolist() == commit_r[b].tolist(), b
        assert all(commit_g[b, j] == 0 for j in range(B) if not masked[b, j])


@pytest.mark.parametrize("dtype,V,batch,sigma,planted,masked_frac", [
    ("f32", 4096, 1, 3.0, 0.0, 1.0),          # tiny workload
    ("f32", 4096, 2, 3.0, 0.3, 0.5),
    ("bf16", 126464, 8, 4.0, 0.25, 1.0),      # serving workload, planted confident rows
    ("bf16", 126464, 2, 4.0, 0.0, 0.5),
    ("bf16", 50001, 2, 2.0, 0.5, 0.7),        # odd vocabulary: unaligned rows take the scalar path
    ("f32", 3, 1, 1.0, 0.0, 1.0),             # vocabulary smaller than a vector
])
@pytest.mark.parametrize("mode,threshold,topk,min_commit", [
    ("threshold", 0.9, 1, 1), ("topk", 0.0, 3, 0), ("margin", 0.5, 1, 1), ("threshold", 0.999, 1, 2)])
def test_unmask_matches_oracle(dev, dtype, V, batch, sigma, planted, masked_frac, mode, threshold, topk,
                               min_commit):
    B = 32
    logits = W.draw_logits((batch, B, V), dtype, sigma, seed=V + batch, planted_frac=planted)
    g = torch.Generator().manual_seed(V)
    masked = (torch.rand((batch, B), generator=g) < masked_frac).to(torch.uint8)
    masked[0, 0] = 1
    md = MODES[mode]
    conf, arg, p2, commit = _gpu_unmask(dev, logits, masked, md, threshold, topk, min_commit)
    conf_r, arg_r, p2_r, commit_r = O.unmask(f64(logits), masked.numpy(), md, threshold, topk, min_commit)
    m = masked.numpy().astype(bool)
    assert np.array_equal(arg[m], arg_r[m])
    assert np.all(arg[~m] == -1) and np.all(conf[~m] == 0) and np.all(commit[~m] == 0)
    assert np.allclose(conf[m], conf_r[m], rtol=1e-5, atol=0)
    assert np.allclose(p2[m], p2_r[m], rtol=1e-5, atol=1e-30)
    _check_commits(conf_r, p2_r, masked.numpy(), commit, commit_r, md, threshold, topk, min_commit)


def test_unmask_ties_and_uniform_rows(dev):
    V = 4096
    logits = torch.zeros((1, 32, V), dtype=torch.float32)
    logits[0, 1, [7, 3000]] = 5.0          # tied maximum: lowest id, p2 == conf
    logits[0, 2, V - 1] = 1.0              # maximum in the last element
    masked = torch.ones((1, 32), dtype=torch.uint8)
    conf, arg, p2, commit = _gpu_unmask(dev, logits, masked, O.MODE_THRESHOLD, 0.9, 1, 1)
    assert arg[0, 0] == 0 and abs(conf[0, 0] - 1 / V) < 1e-9
    assert arg[0, 1] == 7 and abs(p2[0, 1] - conf[0, 1]) < 1e-9
    assert arg[0, 2] == V - 1
    assert commit[0].sum() == 1 and commit[0, 1] == 1      # min-1: the most confident row
