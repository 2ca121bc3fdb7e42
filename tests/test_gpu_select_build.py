"""GPU parity: structured suffix selection and the sparse step input against the oracle."""
import numpy as np
import pytest
import torch

from oracle import ssm_oracle as O
from paper_2608_23167_gb300 import workloads as W
from tests.gpu_helpers import bf16_ulp, check_device_error, cuda_or_skip, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return cuda_or_skip()


def _gpu_select(dev, P, G, B, b, L, M, T):
    from paper_2608_23167_gb300 import ssm
    buf = torch.full((G + 8,), -7, dtype=torch.int32, device=dev)
    n = ssm.ssm_select_suffix(buf, P, G, B, b, L, M, T)
    torch.cuda.synchronize()
    out = buf.cpu().tolist()
    assert all(v == -7 for v in out[n:]), "wrote past |R_t|"
    return out[:n]


@pytest.mark.parametrize("name", list(W.WORKLOADS))
def test_select_every_block_index_bit_exact(dev, name):
    w = W.WORKLOADS[name]
    for b in range(w.n_blocks):
        r, *_ = O.select_suffix(w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail)
        assert _gpu_select(dev, w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail) == r, (name, b)
    check_device_error()


@pytest.mark.parametrize("cfg", [
    (16, 256, 32, 48, 1000, 2),     # fractional local region
    (0, 320, 32, 32, 3, 2),         # middle cap binds
    (16, 256, 32, 0, 1000, 2),      # no local region
    (16, 256, 32, 64, 0, 0),        # no middle, no tail
    (16, 256, 32, 64, 1000, 3),     # start + mid + end tail
    (16, 256, 32, 64, 1000, 40),    # tail budget beyond the block
    (3, 96, 8, 12, 1, 9),           # small blocks
    (5, 8192, 32, 96, 7, 5),        # long generation, several selection loop trips
])
def test_select_edge_cases_bit_exact(dev, cfg):
    P, G, B, L, M, T = cfg
    for b in range(G // B):
        r, *_ = O.select_suffix(P, G, B, b, L, M, T)
        assert _gpu_select(dev, P, G, B, b, L, M, T) == r, (cfg, b)


def test_select_batch_concatenates(dev):
    from paper_2608_23167_gb300 import ssm
    w = W.WORKLOADS["long"]
    cfgs = [(w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail) for b in range(w.n_blocks)]
    cfgs += [(7, 256, 32, b, 48, 2, 3) for b in range(8)]     # > 64 configurations: two launches
    buf = torch.zeros(20000, dtype=torch.int32, device=dev)
    off = ssm.ssm_select_suffix_batch(buf, cfgs)
    torch.cuda.synchronize()
    got = buf.cpu().tolist()
    for i, c in enumerate(cfgs):
        r, *_ = O.select_suffix(*c)
        assert got[off[i]:off[i + 1]] == r


def _build_case(dev, V, H, batch, B, R, k, alpha, seed, masked_frac=1.0, n_prefix=0, no_pred_frac=0.0):
    from paper_2608_23167_gb300 import ssm
    embed = W.draw_normal_bf16((V, H), 1.0, seed)
    mask_id = V - 1
    blk = W.draw_block_tokens(batch, B, V, mask_id, masked_frac, seed + 1)
    pre = W.draw_block_tokens(batch, n_prefix, V, mask_id, 0.0, seed + 2) if n_prefix else None
    spos = torch.arange(R, dtype=torch.int32) * 3 + 1000
    ids, probs = W.draw_prev_topk(batch * R, k, V - 1, seed + 3, no_pred_frac=no_pred_frac)
    ids = ids.reshape(batch, R, k)
    probs = probs.reshape(batch, R, k)
    rows = n_prefix + B + R
    x = torch.full((batch, rows, H), float("nan"), dtype=torch.bfloat16, device=dev)
    pos = torch.zeros(rows, dtype=torch.int32, device=dev)
    ssm.ssm_build_step_input(blk.to(dev), spos.to(dev), embed.to(dev), mask_id, ids.to(dev), probs.to(dev), alpha,
                             x, pos, block_start=700, prefix_tokens=None if pre is None else pre.to(dev))
    torch.cuda.synchronize()
    xr, pr = O.build_step_input(f64(embed), mask_id, blk.numpy(), 700, spos.tolist(), ids.numpy(),
                                probs.to(torch.float64).numpy(), alpha,
                                prefix_tokens=None if pre is None else pre.numpy())
    return f64(x), pos.cpu().numpy(), xr, pr, n_prefix + B


def _assert_build_close(x, xr, n_exact):
    assert np.array_equal(x[:, :n_exact], xr[:, :n_exact]), "prompt/block rows must be exact copies"
    d = np.abs(x[:, n_exact:] - xr[:, n_exact:])
    tol = bf16_ulp(xr[:, n_exact:]) + 2.0 ** -20
    assert np.all(d <= tol), f"suffix rows: worst excess {np.max(d - tol):.3e}"
    return float((d > 0).mean())


@pytest.mark.parametrize("V,H,batch,R,k,alpha", [
    (4096, 256, 1, 41, 5, 0.4),        # tiny workload
    (126464, 4096, 1, 45, 5, 0.4),     # LLaDA-shaped
    (126464, 3584, 4, 100, 7, 0.3),    # Dream-shaped, batch 4
    (5000, 1024, 3, 17, 3, 0.2),       # odd sizes
])
def test_build_step_input_matches_oracle(dev, V, H, batch, R, k, alpha):
    x, pos, xr, pr, n_exact = _build_case(dev, V, H, batch, 32, R, k, alpha, seed=R)
    assert np.array_equal(pos, pr)
    _assert_build_close(x, xr, n_exact)
    check_device_error()


def test_build_step_input_special_cases(dev):
    # alpha = 0: every suffix row is e_mask exactly
    x, pos, xr, pr, n = _build_case(dev, 2048, 256, 2, 32, 20, 5, 0.0, seed=5)
    assert np.array_equal(x, xr)
    assert np.all(x[:, n:] == x[:, n:n + 1])
    # alpha = 1, k = 1: the suffix row is the candidate's embedding exactly
    x, pos, xr, pr, n = _build_case(dev, 2048, 256, 2, 32, 20, 1, 1.0, seed=6)
    assert np.array_equal(x, xr)
    # rows without a previous-step prediction keep e_mask; half-masked block; recomputed prompt
    x, pos, xr, pr, n = _build_case(dev, 3000, 512, 2, 32, 33, 5, 0.4, seed=7, masked_frac=0.5, n_prefix=45,
                                    no_pred_frac=0.3)
    assert np.array_equal(pos, pr)
    _assert_build_close(x, xr, n)
    check_device_error()


def test_build_step_input_bad_token_is_reported(dev):
    from paper_2608_23167_gb300 import ssm
    V, H = 512, 64
    embed = W.draw_normal_bf16((V, H), 1.0, 3).to(dev)
    blk = torch.full((1, 32), V - 1, dtype=torch.int32, device=dev)
    blk[0, 5] = V + 3
    spos = torch.arange(4, dtype=torch.int32, device=dev)
    x = torch.ones((1, 36, H), dtype=torch.bfloat16, device=dev)
    ssm.ssm_build_step_input(blk, spos, embed, V - 1, None, None, 0.4, x)
    assert ssm.ssm_get_device_error() == 7
    assert float(x[0, 5].abs().sum()) == 0.0
    assert ssm.ssm_get_device_error() == 0


def test_build_step_input_varlen(dev):
    """Problems at different block indices packed in one launch (the block-index sweep)."""
    from paper_2608_23167_gb300 import ssm
    w = W.WORKLOADS["long"]
    V, H, k = 6000, 512, 5
    embed = W.draw_normal_bf16((V, H), 1.0, 11)
    mask_id = V - 1
    blocks = [0, 17, 61, 62, 63]
    rows = []
    toks, sufs, ids_all, pr_all = [], [], [], []
    out_row = suf_off = 0
    expect = []
    for i, b in enumerate(blocks):
        r, *_ = O.select_suffix(w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail)
        blk = W.draw_block_tokens(1, w.block, V, mask_id, 0.6, 100 + i)
        ids, probs = W.draw_prev_topk(max(len(r), 1), k, V - 1, 200 + i)
        ids, probs = ids[:len(r)], probs[:len(r)]
        bs = W.block_start(w, b)
        rows.append((i * w.block, 0, suf_off, out_row, 0, len(r), bs))
        xr, pr = O.build_step_input(f64(embed), mask_id, blk.numpy(), bs, r, ids.numpy()[None],
                                    probs.to(torch.float64).numpy()[None], 0.4)
        expect.append((out_row, xr[0], pr))
        toks.append(blk.flatten())
        sufs.append(torch.tensor(r, dtype=torch.int32))
        ids_all.append(ids)
        pr_all.append(probs)
        out_row += w.block + len(r)
        suf_off += len(r)
    probs_t = ssm.step_problems_tensor(rows, dev)
    x = torch.zeros((out_row, H), dtype=torch.bfloat16, device=dev)
    pos = torch.zeros(out_row, dtype=torch.int32, device=dev)
    max_rows = max(w.block + len(s) for s in sufs)
    ssm.ssm_build_step_input_varlen(probs_t, len(blocks), max_rows, w.block, torch.cat(toks).to(dev),
                                    torch.cat(sufs).to(dev), embed.to(dev), mask_id, torch.cat(ids_all).to(dev),
                                    torch.cat(pr_all).to(dev), k, 0.4, x, pos)
    torch.cuda.synchronize()
    xg, pg = f64(x), pos.cpu().numpy()
    for (o, xr, pr) in expect:
        n = len(pr)
        assert np.array_equal(pg[o:o + n], pr)
        _assert_build_close(xg[None, o:o + n], xr[None], w.block)
    check_device_error()
