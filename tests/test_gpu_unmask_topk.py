"""GPU parity: ssm_unmask_topk (everything a step takes from its logits in one call) and two
denoising steps chained through it.

ssm_unmask_topk serves the block rows' logits (confidence, argmax, p2, commit) and the
retained suffix rows' logits (top-k ids and probabilities, the Eq. 6 input of the next
step).  Bars as the separate passes: argmax and ids bit-exact, conf / p2 / probs within
1e-5 relative of the fp64 oracle, commits position by position (see
test_gpu_unmask._check_commits); and the call's outputs equal the two separate calls'.

The chained test runs step t (selection, sparse input with no previous prediction, the
logits pass over stand-in logits) and then step t + 1 of the same block, whose sparse
input mixes the top-k that step t produced (Sec. 3.2 "Soft Suffix Embedding Mixing",
Eqs. 6-8) and whose block tokens carry step t's commits.  Every stage is compared with
the oracle run on the oracle's own outputs of the previous stage.
"""
import numpy as np
import pytest
import torch

from oracle import ssm_oracle as O
from paper_2608_23167_gb300 import workloads as W
from tests.gpu_helpers import bf16_ulp, check_device_error, cuda_or_skip, f64
from tests.test_gpu_unmask import MODES, _check_commits

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return cuda_or_skip()


def _outputs(dev, batch, B, n, k):
    return dict(conf=torch.full((batch, B), -1.0, device=dev), argmax=torch.full((batch, B), -5, dtype=torch.int32,
                device=dev), p2=torch.full((batch, B), -1.0, device=dev),
                commit=torch.full((batch, B), 9, dtype=torch.uint8, device=dev),
                ids=torch.full((max(n, 1), k), -7, dtype=torch.int32, device=dev),
                probs=torch.full((max(n, 1), k), float("nan"), device=dev))


def _fused(dev, logits, masked, suffix, k, mode, threshold, topk, min_commit):
    from paper_2608_23167_gb300 import ssm
    batch, B, _ = logits.shape
    o = _outputs(dev, batch, B, suffix.shape[0], k)
    ssm.ssm_unmask_topk(logits.to(dev), masked.to(dev), o["conf"], o["argmax"], o["commit"], suffix.to(dev), k,
                        o["ids"], o["probs"], p2=o["p2"], mode=mode, threshold=threshold, topk=topk,
                        min_commit=min_commit)
    torch.cuda.synchronize()
    check_device_error()
    return {key: v.cpu() for key, v in o.items()}


@pytest.mark.parametrize("dtype,V,batch,n_suffix,k,sigma,planted", [
    ("bf16", 126464, 8, 69, 5, 4.0, 0.25),   # serving batch: 8 x 32 block rows, one sequence's retained suffix
    ("bf16", 126464, 2, 300, 8, 4.0, 0.0),   # more suffix rows than CTAs of one wave; the longest list
    ("f32", 4096, 1, 41, 5, 3.0, 0.25),      # tiny workload (fp32, 4096 entries)
    ("bf16", 65544, 3, 7, 3, 2.0, 0.5),      # ragged last chunk
])
@pytest.mark.parametrize("mode,threshold,topk,min_commit", [("threshold", 0.9, 1, 1), ("topk", 0.0, 3, 0),
                                                           ("margin", 0.5, 1, 1)])
def test_unmask_topk_matches_oracle_and_separate_calls(dev, dtype, V, batch, n_suffix, k, sigma, planted, mode,
                                                       threshold, topk, min_commit):
    from paper_2608_23167_gb300 import ssm
    B = 32
    logits = W.draw_logits((batch, B, V), dtype, sigma, seed=V + batch + 11, planted_frac=planted)
    suffix = W.draw_logits((n_suffix, V), dtype, sigma, seed=V + n_suffix + 13)
    g = torch.Generator().manual_seed(V + 3)
    masked = (torch.rand((batch, B), generator=g) < 0.7).to(torch.uint8)
    masked[0, 0] = 1
    md = MODES[mode]
    got = _fused(dev, logits, masked, suffix, k, md, threshold, topk, min_commit)
    # the oracle
    conf_r, arg_r, p2_r, commit_r = O.unmask(f64(logits), masked.numpy(), md, threshold, topk, min_commit)
    ids_r, probs_r = O.suffix_topk(f64(suffix), k)
    m = masked.numpy().astype(bool)
    conf, arg, p2 = got["conf"].double().numpy(), got["argmax"].numpy(), got["p2"].double().numpy()
    assert np.array_equal(arg[m], arg_r[m])
    assert np.all(arg[~m] == -1) and np.all(conf[~m] == 0) and np.all(got["commit"].numpy()[~m] == 0)
    assert np.allclose(conf[m], conf_r[m], rtol=1e-5, atol=0)
    assert np.allclose(p2[m], p2_r[m], rtol=1e-5, atol=1e-30)
    _check_commits(conf_r, p2_r, masked.numpy(), got["commit"].numpy(), commit_r, md, threshold, topk, min_commit)
    assert np.array_equal(got["ids"].numpy(), ids_r)
    assert np.allclose(got["probs"].double().numpy(), probs_r, rtol=1e-5, atol=0)
    # the two separate calls give the same bits
    sep = _outputs(dev, batch, B, n_suffix, k)
    ssm.ssm_unmask(logits.to(dev), masked.to(dev), sep["conf"], sep["argmax"], sep["commit"], p2=sep["p2"], mode=md,
                   threshold=threshold, topk=topk, min_commit=min_commit)
    ssm.ssm_suffix_topk(suffix.to(dev), k, sep["ids"], sep["probs"])
    torch.cuda.synchronize()
    check_device_error()
    for key in ("conf", "argmax", "p2", "commit", "ids"):
        assert torch.equal(got[key], sep[key].cpu()), key
    assert np.allclose(got["probs"].numpy(), sep["probs"].cpu().numpy(), rtol=1e-6, atol=0)


def test_unmask_topk_edge_cases(dev):
    """A sequence with no masked position (its outputs are still written), a fully masked one,
    no suffix rows (= ssm_unmask), and argument errors."""
    from paper_2608_23167_gb300 import ssm
    V, B = 126464, 32
    logits = W.draw_logits((3, B, V), "bf16", 4.0, seed=5, planted_frac=0.3)
    masked = torch.ones((3, B), dtype=torch.uint8)
    masked[1] = 0
    suffix = W.draw_logits((4, V), "bf16", 4.0, seed=6)
    got = _fused(dev, logits, masked, suffix, 5, O.MODE_THRESHOLD, 0.9, 1, 1)
    conf_r, arg_r, p2_r, commit_r = O.unmask(f64(logits), masked.numpy(), O.MODE_THRESHOLD, 0.9, 1, 1)
    assert np.array_equal(got["argmax"].numpy(), np.where(masked.numpy() > 0, arg_r, -1))
    assert np.all(got["conf"].numpy()[1] == 0) and np.all(got["commit"].numpy()[1] == 0)
    assert np.all(got["p2"].numpy()[1] == 0)
    o = _outputs(dev, 3, B, 0, 5)
    ssm.ssm_unmask_topk(logits.to(dev), masked.to(dev), o["conf"], o["argmax"], o["commit"], None, 5, None, None)
    torch.cuda.synchronize()
    check_device_error()
    assert torch.equal(o["argmax"].cpu(), got["argmax"])
    with pytest.raises(ssm.SSMError) as e:
        ssm.ssm_unmask_topk(logits.to(dev), masked.to(dev), o["conf"], o["argmax"], o["commit"], suffix.to(dev), 9,
                            o["ids"], o["probs"])
    assert e.value.status == ssm.SSM_ERR_UNSUPPORTED


def test_two_steps_chained_through_the_suffix_topk(dev):
    """Step t and step t + 1 of one block of the Dream-shaped serving layout (prompt 512,
    gen 1024, block 32, budgets 64/32/8), batch 2: step t's logits call produces the commits
    and the retained suffix positions' top-k that step t + 1's sparse input consumes."""
    from paper_2608_23167_gb300 import ssm
    P, G, B, L, M, T = 512, 1024, 32, 64, 32, 8
    b, batch, V, H, k, alpha = 3, 2, 126464, 256, 5, 0.4
    mask_id = V - 1
    cfg = (P, G, B, b, L, M, T)
    # step t: selection and the sparse input (first step of the block: no previous prediction)
    pos_buf = torch.zeros(G, dtype=torch.int32, device=dev)
    R = ssm.ssm_select_suffix(pos_buf, *cfg)
    r_ref, *_ = O.select_suffix(*cfg)
    assert pos_buf[:R].cpu().tolist() == r_ref
    spos = pos_buf[:R]
    embed = W.draw_normal_bf16((V, H), 1.0, 301)
    embed_d = embed.to(dev)
    e64 = f64(embed)
    blk = torch.full((batch, B), mask_id, dtype=torch.int32)
    x = torch.empty((batch, B + R, H), dtype=torch.bfloat16, device=dev)
    xpos = torch.empty(B + R, dtype=torch.int32, device=dev)
    start = P + b * B
    ssm.ssm_build_step_input(blk.to(dev), spos, embed_d, mask_id, None, None, alpha, x, xpos, block_start=start)
    x_ref, pos_ref = O.build_step_input(e64, mask_id, blk.numpy(), start, r_ref, None, None, alpha)
    assert np.array_equal(xpos.cpu().numpy(), pos_ref)
    assert np.array_equal(f64(x), x_ref)          # no mixing at the first step: exact embedding rows
    # step t's logits (stand-ins for the model's): block rows and retained suffix rows
    logits = W.draw_logits((batch, B, V), "bf16", 4.0, seed=302, planted_frac=0.3)
    suffix = W.draw_logits((batch * R, V), "bf16", 4.0, seed=303)
    masked = (blk == mask_id).to(torch.uint8)
    got = _fused(dev, logits, masked, suffix, k, O.MODE_THRESHOLD, 0.9, 1, 1)
    conf_r, arg_r, p2_r, commit_r = O.unmask(f64(logits), masked.numpy(), O.MODE_THRESHOLD, 0.9, 1, 1)
    ids_r, probs_r = O.suffix_topk(f64(suffix), k)
    _check_commits(conf_r, p2_r, masked.numpy(), got["commit"].numpy(), commit_r, O.MODE_THRESHOLD, 0.9, 1, 1)
    assert np.array_equal(got["commit"].numpy(), commit_r)
    assert np.array_equal(got["ids"].numpy(), ids_r)
    assert np.allclose(got["probs"].double().numpy(), probs_r, rtol=1e-5, atol=0)
    # step t + 1: committed positions take their argmax token; the suffix mixes step t's top-k
    blk1 = torch.where(got["commit"] > 0, got["argmax"], blk)
    blk1_ref = np.where(commit_r > 0, arg_r, blk.numpy())
    assert np.array_equal(blk1.numpy(), blk1_ref)
    R1 = ssm.ssm_select_suffix(pos_buf, *cfg)    # same block: the same retained positions
    assert R1 == R
    ids_d = got["ids"].reshape(batch, R, k).to(dev)
    probs_d = got["probs"].reshape(batch, R, k).to(dev)
    x1 = torch.empty_like(x)
    ssm.ssm_build_step_input(blk1.to(dev), spos, embed_d, mask_id, ids_d, probs_d, alpha, x1, xpos, block_start=start)
    torch.cuda.synchronize()
    check_device_error()
    x1_ref, _ = O.build_step_input(e64, mask_id, blk1_ref, start, r_ref, ids_r.reshape(batch, R, k),
                                   probs_r.reshape(batch, R, k), alpha)
    got1 = f64(x1)
    assert np.array_equal(got1[:, :B], x1_ref[:, :B])                    # block rows: embedding rows
    ref_s = x1_ref[:, B:]
    assert np.all(np.abs(got1[:, B:] - ref_s) <= bf16_ulp(ref_s) + 2.0 ** -20)   # mixed suffix rows: 1 ulp
    assert not np.array_equal(got1[:, B:], f64(x)[:, B:])                # step t + 1 really mixed something
