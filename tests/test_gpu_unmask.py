"""GPU parity: vocabulary softmax, confidence, argmax and the commit rules.

Bars: argmax bit-exact (it compares input values only, so it is exact even
where probabilities are close); conf and p2 within 1e-5 relative of the fp64
oracle; commits compared position by position with the oracle's, except for a
score within 1e-5 of the threshold and for swaps among positions whose
confidences lie within 1e-3 of the ranking boundary (top-k, min-commit
fallback) -- see _check_commits.  The separated-confidence cases leave no such
ambiguity and are compared exactly in every row.
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


RANK_TOL = 1e-3      # confidences closer than this may rank either way at fp32
THRESH_TOL = 1e-5    # a score this close to the threshold may pass either way at fp32


def _check_commits(conf_r, p2_r, masked, commit_g, commit_r, mode, threshold, topk, min_commit):
    """Element-wise commit parity against the oracle, one batch row at a time.

    The rule has two decisions.  (1) Threshold / margin: position j passes if its score
    (conf, or conf - p2) is above the threshold; GPU and oracle must agree on every
    position except those whose score is within THRESH_TOL of the threshold.  (2) The
    ranking: top-k mode commits the k most confident masked positions, and the min-commit
    fallback adds the most confident non-passing positions.  The GPU's pick must equal the
    oracle's except for swaps among positions whose oracle confidence lies within RANK_TOL
    of the decision boundary: no position the GPU left out may be more than RANK_TOL more
    confident than a position it picked.  Where the boundary pair (the last picked and the
    first left out) is more than RANK_TOL apart, that makes the pick exactly the oracle's.
    Returns the number of rows whose commits were compared exactly."""
    batch, B = conf_r.shape
    exact_rows = 0
    for b in range(batch):
        cand = [j for j in range(B) if masked[b, j]]
        got = {j for j in range(B) if commit_g[b, j]}
        assert got <= set(cand), f"row {b}: commit outside the masked positions"
        if mode == O.MODE_TOPK:
            passing, undecided, short = set(), set(), topk
        else:
            score = conf_r[b] if mode == O.MODE_THRESHOLD else conf_r[b] - p2_r[b]
            passing = {j for j in cand if score[j] > threshold + THRESH_TOL}
            undecided = {j for j in cand if abs(score[j] - threshold) <= THRESH_TOL}
            short = min_commit - len(passing)
        assert passing <= got, f"row {b}: a passing position was not committed"
        if undecided:
            # the GPU's passing set is one of the sets between `passing` and `passing | undecided`:
            # every clearly failing position it commits must come from the fallback
            extra = got - passing - undecided
            assert len(extra) <= max(0, min_commit - len(passing)), f"row {b}"
            continue
        rest = [j for j in cand if j not in passing]
        want = max(0, min(short, len(rest)))
        picked = got - passing
        assert len(picked) == want, f"row {b}: {len(picked)} picked by rank, expected {want}"
        left = [j for j in rest if j not in picked]
        if picked and left:
            worst_in = min(conf_r[b, j] for j in picked)
            best_out = max(conf_r[b, j] for j in left)
            assert best_out <= worst_in + RANK_TOL, f"row {b}: skipped a position {best_out - worst_in:.2e} more confident"
        ranked = sorted(rest, key=lambda j: (-conf_r[b, j], j))
        separated = want == 0 or want == len(ranked) or conf_r[b, ranked[want - 1]] - conf_r[b, ranked[want]] > RANK_TOL
        if separated:
            assert commit_g[b].tolist() == commit_r[b].tolist(), f"row {b}"
            exact_rows += 1
    return exact_rows


@pytest.mark.parametrize("dtype,V,batch,sigma,planted,masked_frac", [
    ("f32", 4096, 1, 3.0, 0.0, 1.0),          # tiny workload
    ("f32", 4096, 2, 3.0, 0.3, 0.5),
    ("bf16", 126464, 8, 4.0, 0.25, 1.0),      # serving workload, planted confident rows
    ("bf16", 126464, 2, 4.0, 0.0, 0.5),
    ("f32", 126464, 2, 4.0, 0.25, 0.8),       # fp32 rows of 31 stages, the last one partial
    ("bf16", 126464, 24, 4.0, 0.25, 0.9),     # 768 rows: a CTA's stage range ends inside rows and spans several
    ("bf16", 8192, 64, 4.0, 0.25, 0.6),       # one-stage rows: a range holds whole rows, masked and not
    ("bf16", 50001, 2, 2.0, 0.5, 0.7),        # odd vocabulary: unaligned rows take the scalar path
    ("f32", 50001, 24, 2.0, 0.25, 0.8),       # scalar path with ranges that span rows
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


def _separated_logits(batch, B, V, dtype, seed, conf_lo, conf_hi):
    """N(0, 1) logits in which every position's top id is planted so that its confidence is a
    target from linspace(conf_lo, conf_hi, B), permuted per row: the confidences of one row are
    ~(conf_hi - conf_lo) / B apart, far more than RANK_TOL, so every ranking decision is exact."""
    x = W.draw_logits((batch, B, V), dtype, 1.0, seed)
    g = torch.Generator().manual_seed(seed + 1)
    xd = f64(x)
    targets = np.linspace(conf_lo, conf_hi, B)
    for b in range(batch):
        perm = torch.randperm(B, generator=g).numpy()
        ids = torch.randint(0, V, (B,), generator=g).numpy()
        for j in range(B):
            row = xd[b, j]
            z_rest = np.exp(row).sum() - np.exp(row[ids[j]])
            c = targets[perm[j]]
            x[b, j, ids[j]] = float(np.log(c / (1.0 - c) * z_rest))
    return x


@pytest.mark.parametrize("mode,threshold,topk,min_commit", [
    ("topk", 0.0, 1, 0),            # Vanilla top-1
    ("topk", 0.0, 3, 0),
    ("threshold", 0.9, 1, 1),       # nothing above the threshold: the min-1 fallback picks one position
    ("threshold", 0.9, 1, 2),
    ("margin", 0.9, 1, 1),
    ("threshold", 0.5, 1, 1),       # some positions pass, the fallback does not fire
])
def test_unmask_commit_positions_separated(dev, mode, threshold, topk, min_commit):
    """LLaDA vocabulary (126464, bf16), four sequences, confidences planted well apart (0.05 ..
    0.85): the committed positions are compared with the oracle's in every row, so a kernel that
    commits the wrong positions (top-k, or the fallback's choice) fails."""
    batch, B, V = 4, 32, W.LLADA_VOCAB
    logits = _separated_logits(batch, B, V, "bf16", 31 + topk + min_commit, 0.05, 0.85)
    g = torch.Generator().manual_seed(5)
    masked = (torch.rand((batch, B), generator=g) < 0.75).to(torch.uint8)
    masked[:, 0] = 1
    md = MODES[mode]
    conf, arg, p2, commit = _gpu_unmask(dev, logits, masked, md, threshold, topk, min_commit)
    conf_r, arg_r, p2_r, commit_r = O.unmask(f64(logits), masked.numpy(), md, threshold, topk, min_commit)
    m = masked.numpy().astype(bool)
    assert np.array_equal(arg[m], arg_r[m])
    assert np.allclose(conf[m], conf_r[m], rtol=1e-5, atol=0)
    exact = _check_commits(conf_r, p2_r, masked.numpy(), commit, commit_r, md, threshold, topk, min_commit)
    assert exact == batch
    assert np.array_equal(commit, commit_r)


@pytest.mark.parametrize("mode,threshold,want_p2", [("threshold", 0.9, False), ("margin", 0.5, True)])
def test_unmask_long_sweep_full_size_sampled(dev, mode, threshold, want_p2):
    """The long-sequence sweep's unmasking at full size, in the launch configuration the bench
    times: 64 sequences x 32 masked positions x 126464 bf16 logits ~ N(0, 4^2) (518 MB, CTA
    stage ranges that span several rows; the threshold rule without p2, as the bench calls it).
    The oracle checks four sampled sequences (their commits depend only on their own 32
    positions)."""
    from paper_2608_23167_gb300 import ssm
    batch, B, V = 64, 32, W.LLADA_VOCAB
    logits = W.draw_logits((batch, B, V), "bf16", 4.0, seed=64, planted_frac=0.1)
    masked = torch.ones((batch, B), dtype=torch.uint8)
    md = MODES[mode]
    conf = torch.full((batch, B), -1.0, device=dev)
    arg = torch.full((batch, B), -5, dtype=torch.int32, device=dev)
    commit = torch.full((batch, B), 9, dtype=torch.uint8, device=dev)
    p2 = torch.full((batch, B), -1.0, device=dev) if want_p2 else None
    ssm.ssm_unmask(logits.to(dev), masked.to(dev), conf, arg, commit, p2=p2, mode=md, threshold=threshold,
                   topk=1, min_commit=1)
    torch.cuda.synchronize()
    check_device_error()
    conf, arg, commit = conf.cpu().double().numpy(), arg.cpu().numpy(), commit.cpu().numpy()
    for s in (0, 21, 42, 63):
        conf_r, arg_r, p2_r, commit_r = O.unmask(f64(logits[s:s + 1]), masked[s:s + 1].numpy(), md, threshold, 1, 1)
        assert np.array_equal(arg[s:s + 1], arg_r), f"sequence {s}"
        assert np.allclose(conf[s:s + 1], conf_r, rtol=1e-5, atol=0), f"sequence {s}"
        if want_p2:
            assert np.allclose(p2[s:s + 1].cpu().double().numpy(), p2_r, rtol=1e-5, atol=1e-30), f"sequence {s}"
        _check_commits(conf_r, p2_r, masked[s:s + 1].numpy(), commit[s:s + 1], commit_r, md, threshold, 1, 1)


@pytest.mark.parametrize("B,mode,threshold,topk,min_commit", [
    (64, "threshold", 0.5, 1, 3),     # two warps of positions per sequence
    (200, "topk", 0.0, 17, 0),        # a ragged last warp
    (1000, "margin", 0.3, 1, 2),      # close to the 1024-position limit of a block
])
def test_unmask_long_blocks(dev, B, mode, threshold, topk, min_commit):
    """Blocks longer than 32 positions: the commit kernel's CTA has one thread per position
    (up to 1024), and its ranking runs over every position of the block.  Confidences are
    planted from 0.02 to 0.95 (at 64 and 200 positions far more than the 1e-3 ranking band
    apart, so every position is compared exactly; at 1000 positions 9e-4 apart, so the
    ranking boundary's neighbours are checked as a valid commit set)."""
    batch, V = 2, 512
    logits = _separated_logits(batch, B, V, "f32", 7 + B, 0.02, 0.95)
    g = torch.Generator().manual_seed(B)
    masked = (torch.rand((batch, B), generator=g) < 0.7).to(torch.uint8)
    md = MODES[mode]
    conf, arg, p2, commit = _gpu_unmask(dev, logits, masked, md, threshold, topk, min_commit)
    conf_r, arg_r, p2_r, commit_r = O.unmask(f64(logits), masked.numpy(), md, threshold, topk, min_commit)
    m = masked.numpy().astype(bool)
    assert np.array_equal(arg[m], arg_r[m])
    assert np.allclose(conf[m], conf_r[m], rtol=1e-5, atol=0)
    assert np.allclose(p2[m], p2_r[m], rtol=1e-5, atol=1e-30)
    _check_commits(conf_r, p2_r, masked.numpy(), commit, commit_r, md, threshold, topk, min_commit)
