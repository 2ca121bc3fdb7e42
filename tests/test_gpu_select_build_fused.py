"""GPU parity: selection and sparse input in one launch (ssm_select_build_step_input_varlen).

Each retained suffix row places itself at the position of its rank in R_t (the closed form
of Eqs. 2-5); the positions must equal the oracle's set construction bit for bit over every
block index of the five workloads and a grid of edge layouts (budgets not multiples of the
block, a local region reaching into the tail block, more middle blocks than the middle
budget, T = 0 / 1 / 3 / >= B), and the whole output must equal the two-launch path
(ssm_select_suffix_batch, then ssm_build_step_input_varlen) bit for bit.
"""
import numpy as np
import pytest
import torch

from oracle import ssm_oracle as O
from paper_2608_23167_gb300 import workloads as W
from tests.gpu_helpers import check_device_error, cuda_or_skip

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return cuda_or_skip()


def _cases():
    out = []
    for name, w in W.WORKLOADS.items():
        out.append((name, [(w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail) for b in range(w.n_blocks)]))
    for B in (8, 32):       # one launch takes one block length
        grid = []
        for G in (B, 3 * B, 12 * B):
            for L in (0, B // 2, B + 3, 3 * B):
                for M in (0, 1, 5):
                    for T in (0, 1, 3, B, B + 2):
                        for b in sorted({0, (G // B) // 2, G // B - 1}):
                            grid.append((5, G, B, b, L, M, T))
        out.append((f"edge_grid_B{B}", grid))
    return out


@pytest.mark.parametrize("name,cfgs", _cases(), ids=[c[0] for c in _cases()])
def test_select_build_fused_equals_oracle_and_two_launches(dev, name, cfgs):
    from paper_2608_23167_gb300 import ssm
    V, H, k = 3000, 256, 3
    embed = W.draw_normal_bf16((V, H), 1.0, 21).to(dev)
    mask_id = V - 1
    rows, expect_pos = [], []
    out_row = suf_off = 0
    n = len(cfgs)
    B = cfgs[0][2]
    assert all(c[2] == B for c in cfgs)
    for i, c in enumerate(cfgs):
        r, *_ = O.select_suffix(*c)
        rows.append((i * B, 0, suf_off, out_row, 0, len(r), c[0] + c[3] * B))
        expect_pos.append((suf_off, r))
        out_row += B + len(r)
        suf_off += len(r)
    toks = W.draw_block_tokens(n, B, V, mask_id, 0.5, 22).to(dev)
    ids, probs = W.draw_prev_topk(max(suf_off, 1), k, V - 1, 23)
    ids, probs = ids.to(dev), probs.to(dev)
    tab = ssm.step_problems_tensor(rows, dev)
    cfg_t = ssm.suffix_cfgs_tensor(cfgs, dev)
    max_rows = max(B + r[5] for r in rows)
    x1 = torch.full((max(out_row, 1), H), 7.0, dtype=torch.bfloat16, device=dev)
    pos1 = torch.full((max(out_row, 1),), -9, dtype=torch.int32, device=dev)
    spos1 = torch.full((max(suf_off, 1),), -9, dtype=torch.int32, device=dev)
    ssm.ssm_select_build_step_input_varlen(tab, cfg_t, n, max_rows, B, toks, embed, mask_id, ids, probs, k, 0.4, x1,
                                           pos1, spos1)
    torch.cuda.synchronize()
    check_device_error()
    sp = spos1.cpu().numpy()
    for off, r in expect_pos:
        assert sp[off:off + len(r)].tolist() == r
    # the two-launch path
    spos2 = torch.zeros(max(suf_off, 1), dtype=torch.int32, device=dev)
    ssm.ssm_select_suffix_batch(spos2, cfgs)
    x2 = torch.full_like(x1, 7.0)
    pos2 = torch.full_like(pos1, -9)
    ssm.ssm_build_step_input_varlen(tab, n, max_rows, B, toks, spos2, embed, mask_id, ids, probs, k, 0.4, x2, pos2)
    torch.cuda.synchronize()
    check_device_error()
    assert torch.equal(spos1, spos2)
    assert torch.equal(pos1, pos2)
    assert torch.equal(x1, x2)


def test_select_build_fused_rejects_a_mismatched_table(dev):
    """A problem whose n_suffix disagrees with its selection: the device error is recorded and
    that problem's suffix rows are zeroed."""
    from paper_2608_23167_gb300 import ssm
    V, H = 3000, 256
    embed = W.draw_normal_bf16((V, H), 1.0, 31).to(dev)
    c = (64, 256, 32, 0, 32, 8, 4)
    r, *_ = O.select_suffix(*c)
    tab = ssm.step_problems_tensor([(0, 0, 0, 0, 0, len(r) - 1, 96)], dev)
    toks = torch.full((1, 32), V - 1, dtype=torch.int32, device=dev)
    x = torch.full((32 + len(r), H), 7.0, dtype=torch.bfloat16, device=dev)
    ssm.ssm_select_build_step_input_varlen(tab, ssm.suffix_cfgs_tensor([c], dev), 1, 32 + len(r), 32, toks, embed,
                                           V - 1, None, None, 0, 0.4, x)
    torch.cuda.synchronize()
    assert ssm.ssm_get_device_error() == ssm.SSM_ERR_DEVICE_INPUT
    assert torch.all(x[32:32 + len(r) - 1] == 0)
