"""GPU parity: tcgen05 bidirectional attention against the fp64 oracle.

Tolerance (attention): max-abs error <= 2e-2 and mean-abs error <= 2e-3 on the
outputs; the natural-log LSE within 2e-2 absolute.
"""
import math

import numpy as np
import pytest
import torch

from oracle import ssm_oracle as O
from paper_2608_23167_gb300 import workloads as W
from tests.gpu_helpers import assert_attention_close, check_device_error, cuda_or_skip, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return cuda_or_skip()


def _ramp(t: torch.Tensor, top: float) -> torch.Tensor:
    """Scales row i of [batch, rows, h, d] by 1 + (top - 1) i / rows: later keys score higher,
    so the running maximum keeps growing past the first key tile (the lazy rescale path)."""
    n = t.shape[1]
    f = 1.0 + (top - 1.0) * torch.arange(n, dtype=torch.float32) / max(n, 1)
    return (t.float() * f[None, :, None, None]).to(torch.bfloat16)


def _run(dev, batch, n_new, n_cache, h_q, h_kv, d, theta, seed, pos=None, with_lse=True, ramp=0.0):
    from paper_2608_23167_gb300 import ssm
    q = W.draw_normal_bf16((batch, n_new, h_q, d), 1.0, seed)
    k = W.draw_normal_bf16((batch, n_new, h_kv, d), 1.0, seed + 1)
    v = W.draw_normal_bf16((batch, n_new, h_kv, d), 1.0, seed + 2)
    kc = W.draw_normal_bf16((batch, n_cache, h_kv, d), 1.0, seed + 3) if n_cache else None
    vc = W.draw_normal_bf16((batch, n_cache, h_kv, d), 1.0, seed + 4) if n_cache else None
    if ramp and kc is not None:
        kc = _ramp(kc, ramp)
        k = (k.float() * ramp).to(torch.bfloat16)  # the new keys come after the cache: the largest
    if pos is None:
        g = torch.Generator().manual_seed(seed + 5)
        pos = (n_cache + torch.randperm(4 * n_new + 7, generator=g)[:n_new]).to(torch.int32)
    out = torch.full((batch, n_new, h_q, d), float("nan"), dtype=torch.bfloat16, device=dev)
    lse = torch.full((batch, n_new, h_q), float("nan"), dtype=torch.float32, device=dev) if with_lse else None
    ssm.ssm_attention(q.to(dev), k.to(dev), v.to(dev), pos.to(dev), None if kc is None else kc.to(dev),
                      None if vc is None else vc.to(dev), out, theta, lse=lse)
    torch.cuda.synchronize()
    check_device_error()
    ref, ref_lse = O.attention(f64(q), f64(k), f64(v), pos.numpy(), None if kc is None else f64(kc),
                               None if vc is None else f64(vc), theta)
    return f64(out), ref, (None if lse is None else f64(lse)), ref_lse


@pytest.mark.parametrize("batch,n_new,n_cache,h_q,h_kv,d,theta,ramp", [
    (1, 73, 64, 4, 4, 64, 1e4, 0),          # tiny workload (b = 0)
    (1, 589, 0, 8, 8, 128, 5e5, 0),         # LLaDA no-cache shape (8 of 32 heads), 5 query tiles
    (2, 132, 512, 14, 2, 128, 1e6, 0),      # Dream GQA, 7 query heads per kv head
    (2, 101, 512, 8, 8, 128, 5e5, 0),       # serving shape (8 of 32 heads): one query tile, keys split
    (1, 1, 0, 2, 1, 64, 1e4, 0),            # a single key
    (3, 37, 100, 4, 2, 128, 0.0, 0),        # ragged cache (100 = 3*32 + 4), no rotary encoding
    (1, 200, 1000, 2, 2, 64, 1e4, 0),       # cache and new segments both ragged
    (1, 129, 31, 4, 4, 128, 5e5, 0),        # one row past a query tile: a second tile of one row
    (1, 172, 1024, 4, 4, 128, 5e5, 0),      # long sweep at block 0
    (1, 96, 65, 4, 2, 128, 1e4, 0),         # GQA, 192 rows in two query tiles
    (1, 128, 77, 2, 2, 128, 1e4, 0),        # 128 rows: the largest keys-split unit
    (2, 16, 300, 2, 1, 128, 1e4, 0),        # 32 rows
    (1, 5, 0, 2, 2, 128, 1e4, 0),           # one key tile: slot B of a keys-split unit has no work
    (1, 150, 900, 2, 2, 128, 0.0, 4.0),     # cache keys ramped x1..x4: maxima grow past the first tile
    (1, 100, 900, 2, 2, 128, 0.0, 4.0),     # the same with the keys split between the slots
    (1, 150, 900, 2, 2, 128, 0.0, 16.0),    # x1..x16: later tiles' p reach 2^50 against the first tile's
    (1, 100, 900, 2, 2, 128, 0.0, 16.0),    #   maximum, so the exact (rescaling) path runs, both layouts
])
def test_attention_matches_oracle(dev, batch, n_new, n_cache, h_q, h_kv, d, theta, ramp):
    from paper_2608_23167_gb300 import ssm
    out, ref, lse, ref_lse = _run(dev, batch, n_new, n_cache, h_q, h_kv, d, theta, seed=n_new + n_cache, ramp=ramp)
    assert_attention_close(out, ref, f"b{batch} n{n_new} c{n_cache} h{h_q}/{h_kv} d{d}")
    assert np.abs(lse - ref_lse).max() <= 2e-2


def test_attention_full_workloads_sampled(dev):
    """Full-size serving, Dream and LLaDA launches (the serving batch's one-tile problems, Dream's
    single-tile units, LLaDA's pairs of query tiles over 32 heads without a cache); the oracle
    checks a sample of heads."""
    from paper_2608_23167_gb300 import ssm
    for name in ("serve", "dream", "llada"):
        w = W.WORKLOADS[name]
        r, *_ = O.select_suffix(w.prompt, w.gen, w.block, 0, w.local, w.middle, w.tail)
        n_cache = w.prompt if w.prefix_cached else 0
        # without a cache the step recomputes the prompt: its rows come first, at positions 0..P-1
        prefix = [] if w.prefix_cached else list(range(w.prompt))
        bs = W.block_start(w, 0)
        plist = prefix + list(range(bs, bs + w.block)) + r
        n_new = len(plist)
        pos = torch.tensor(plist, dtype=torch.int32)
        q = W.draw_normal_bf16((w.batch, n_new, w.h_q, w.head_dim), 1.0, 31)
        k = W.draw_normal_bf16((w.batch, n_new, w.h_kv, w.head_dim), 1.0, 32)
        v = W.draw_normal_bf16((w.batch, n_new, w.h_kv, w.head_dim), 1.0, 33)
        kc = vc = None
        if n_cache:
            kc = W.draw_normal_bf16((w.batch, n_cache, w.h_kv, w.head_dim), 1.0, 34)
            vc = W.draw_normal_bf16((w.batch, n_cache, w.h_kv, w.head_dim), 1.0, 35)
        o = torch.empty((w.batch, n_new, w.h_q, w.head_dim), dtype=torch.bfloat16, device=dev)
        ssm.ssm_attention(q.to(dev), k.to(dev), v.to(dev), pos.to(dev), kc.to(dev) if n_cache else None,
                          vc.to(dev) if n_cache else None, o, w.rope_theta)
        torch.cuda.synchronize()
        check_device_error()
        grp = w.h_q // w.h_kv
        for b in sorted({0, w.batch - 1}):
            for g in sorted({0, w.h_kv - 1}):
                hs = list(range(g * grp, (g + 1) * grp))
                ref, _ = O.attention(f64(q[b:b + 1, :, hs]), f64(k[b:b + 1, :, g:g + 1]), f64(v[b:b + 1, :, g:g + 1]),
                                     pos.numpy(), f64(kc[b:b + 1, :, g:g + 1]) if n_cache else None,
                                     f64(vc[b:b + 1, :, g:g + 1]) if n_cache else None, w.rope_theta)
                assert_attention_close(f64(o[b:b + 1, :, hs]), ref, f"{name} batch {b} kv head {g}")


def test_attention_long_sweep_full_size_sampled(dev):
    """The long-sequence sweep at full size, in the launch configuration the bench times: the
    64 block indices over one shared 32-head prefix cache as one ragged launch (packed units
    over 32 kv heads, rotate and core as two calls); the oracle checks three block indices on
    three heads."""
    from paper_2608_23167_gb300 import ssm
    w = W.WORKLOADS["long"]
    H, d = w.h_q, w.head_dim
    total_pos = w.prompt + w.gen
    kc = W.draw_normal_bf16((total_pos, H, d), 1.0, 51)
    vc = W.draw_normal_bf16((total_pos, H, d), 1.0, 52)
    rows, poss, new_row = [], [], 0
    for b in range(w.n_blocks):
        r, *_ = O.select_suffix(w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail)
        bs = W.block_start(w, b)
        p = list(range(bs, bs + w.block)) + r
        rows.append((new_row, 0, len(p), bs))
        poss.extend(p)
        new_row += len(p)
    q = W.draw_normal_bf16((new_row, H, d), 1.0, 53)
    k = W.draw_normal_bf16((new_row, H, d), 1.0, 54)
    v = W.draw_normal_bf16((new_row, H, d), 1.0, 55)
    pos = torch.tensor(poss, dtype=torch.int32)
    probs = ssm.attn_problems_tensor(rows, dev)
    out = torch.full((new_row, H, d), float("nan"), dtype=torch.bfloat16, device=dev)
    ws = torch.empty(ssm.ssm_attention_workspace_size(new_row, H, H, d), dtype=torch.uint8, device=dev)
    args = (q.to(dev), k.to(dev), v.to(dev), pos.to(dev), kc.to(dev), vc.to(dev), probs, len(rows),
            max(r[2] for r in rows), max(r[3] for r in rows), out, w.rope_theta)
    ssm.ssm_attention_varlen_rotate(*args, workspace=ws)
    ssm.ssm_attention_varlen_core(*args, workspace=ws)
    torch.cuda.synchronize()
    check_device_error()
    for b in (0, 31, 63):
        nr, _, n, nc = rows[b]
        sl = slice(nr, nr + n)
        for h in (0, 17, 31):
            ref, _ = O.attention(f64(q[None, sl, h:h + 1]), f64(k[None, sl, h:h + 1]), f64(v[None, sl, h:h + 1]),
                                 pos[sl].numpy(), f64(kc[None, :nc, h:h + 1]), f64(vc[None, :nc, h:h + 1]),
                                 w.rope_theta)
            assert_attention_close(f64(out[sl, h:h + 1])[None], ref, f"block {b} head {h}")


def test_attention_varlen_block_sweep(dev):
    """The long-sequence sweep: every block index 0..63 as one ragged launch over a
    shared prefix cache; the oracle checks several block indices on a few heads."""
    from paper_2608_23167_gb300 import ssm
    w = W.WORKLOADS["long"]
    H, d = 4, w.head_dim                     # heads are independent in MHA: 4 of 32 suffice here
    total_pos = w.prompt + w.gen
    kc = W.draw_normal_bf16((total_pos, H, d), 1.0, 41)
    vc = W.draw_normal_bf16((total_pos, H, d), 1.0, 42)
    rows, poss, new_row = [], [], 0
    for b in range(w.n_blocks):
        r, *_ = O.select_suffix(w.prompt, w.gen, w.block, b, w.local, w.middle, w.tail)
        bs = W.block_start(w, b)
        p = list(range(bs, bs + w.block)) + r
        rows.append((new_row, 0, len(p), bs))
        poss.extend(p)
        new_row += len(p)
    q = W.draw_normal_bf16((new_row, H, d), 1.0, 43)
    k = W.draw_normal_bf16((new_row, H, d), 1.0, 44)
    v = W.draw_normal_bf16((new_row, H, d), 1.0, 45)
    pos = torch.tensor(poss, dtype=torch.int32)
    probs = ssm.attn_problems_tensor(rows, dev)
    out = torch.full((new_row, H, d), float("nan"), dtype=torch.bfloat16, device=dev)
    lse = torch.empty((new_row, H), dtype=torch.float32, device=dev)
    ssm.ssm_attention_varlen(q.to(dev), k.to(dev), v.to(dev), pos.to(dev), kc.to(dev), vc.to(dev), probs,
                             len(rows), max(r[2] for r in rows), max(r[3] for r in rows), out, w.rope_theta,
                             lse=lse)
    torch.cuda.synchronize()
    check_device_error()
    og, lg = f64(out), f64(lse)
    for b in (0, 1, 31, 43, 44, 60, 62, 63):
        nr, _, n, nc = rows[b]
        sl = slice(nr, nr + n)
        ref, ref_lse = O.attention(f64(q[None, sl]), f64(k[None, sl]), f64(v[None, sl]), pos[sl].numpy(),
                                   f64(kc[None, :nc]), f64(vc[None, :nc]), w.rope_theta)
        assert_attention_close(og[sl][None], ref, f"block {b}")
        assert np.abs(lg[sl][None] - ref_lse).max() <= 2e-2


def test_attention_key_permutation_invariance(dev):
    """Permuting the new rows together with their positions permutes the output rows."""
    from paper_2608_23167_gb300 import ssm
    n, c, h, d = 150, 70, 4, 128
    q = W.draw_normal_bf16((1, n, h, d), 1.0, 51).to(dev)
    k = W.draw_normal_bf16((1, n, h, d), 1.0, 52).to(dev)
    v = W.draw_normal_bf16((1, n, h, d), 1.0, 53).to(dev)
    kc = W.draw_normal_bf16((1, c, h, d), 1.0, 54).to(dev)
    vc = W.draw_normal_bf16((1, c, h, d), 1.0, 55).to(dev)
    pos = (c + torch.randperm(n)).to(torch.int32).to(dev)
    perm = torch.randperm(n).to(dev)
    o1 = torch.empty_like(q)
    o2 = torch.empty_like(q)
    ssm.ssm_attention(q, k, v, pos, kc, vc, o1, 1e4)
    ssm.ssm_attention(q[:, perm].contiguous(), k[:, perm].contiguous(), v[:, perm].contiguous(),
                      pos[perm].contiguous(), kc, vc, o2, 1e4)
    torch.cuda.synchronize()
    assert_attention_close(f64(o2), f64(o1[:, perm]), "permuted")


def test_attention_varlen_rotate_then_core_equals_one_call(dev):
    """ssm_attention_varlen_rotate followed by ssm_attention_varlen_core gives exactly the
    outputs of ssm_attention_varlen (the same two launches, made as two calls)."""
    from paper_2608_23167_gb300 import ssm
    h, d = 4, 128
    cache_rows = 700
    kc = W.draw_normal_bf16((cache_rows, h, d), 1.0, 61).to(dev)
    vc = W.draw_normal_bf16((cache_rows, h, d), 1.0, 62).to(dev)
    sizes = [(150, 600), (37, 700), (90, 0), (1, 33)]
    rows, new_row = [], 0
    for n, c in sizes:
        rows.append((new_row, 0, n, c))
        new_row += n
    q = W.draw_normal_bf16((new_row, h, d), 1.0, 63).to(dev)
    k = W.draw_normal_bf16((new_row, h, d), 1.0, 64).to(dev)
    v = W.draw_normal_bf16((new_row, h, d), 1.0, 65).to(dev)
    pos = (cache_rows + torch.randperm(new_row)).to(torch.int32).to(dev)
    probs = ssm.attn_problems_tensor(rows, dev)
    args = (q, k, v, pos, kc, vc, probs, len(rows), max(r[2] for r in rows), max(r[3] for r in rows))
    o1 = torch.empty_like(q)
    o2 = torch.empty_like(q)
    l1 = torch.empty((new_row, h), dtype=torch.float32, device=dev)
    l2 = torch.empty_like(l1)
    ssm.ssm_attention_varlen(*args, o1, 5e5, lse=l1)
    ws = torch.empty(ssm.ssm_attention_workspace_size(new_row, h, h, d), dtype=torch.uint8, device=dev)
    ssm.ssm_attention_varlen_rotate(*args, o2, 5e5, lse=l2, workspace=ws)
    ssm.ssm_attention_varlen_core(*args, o2, 5e5, lse=l2, workspace=ws)
    torch.cuda.synchronize()
    check_device_error()
    assert torch.equal(o1, o2)
    assert torch.equal(l1, l2)


def test_attention_varlen_serving_batch(dev):
    """The serving batch through the ragged entry point: 8 sequences of 101 new rows, each with
    its own 512-row prefix cache (cache_row = 512 s), 32 heads: every work unit is one query
    tile whose key tiles the two softmax slots split.  This launch once ended with an
    unspecified launch failure (a warp reaching a tcgen05.ld before it had reconverged)."""
    from paper_2608_23167_gb300 import ssm
    w = W.WORKLOADS["serve"]
    r, *_ = O.select_suffix(w.prompt, w.gen, w.block, 0, w.local, w.middle, w.tail)
    n_new = w.block + len(r)
    p1 = list(range(W.block_start(w, 0), W.block_start(w, 0) + w.block)) + r
    H, d = w.h_q, w.head_dim
    rows = [(s * n_new, s * w.prompt, n_new, w.prompt) for s in range(w.batch)]
    total = w.batch * n_new
    q = W.draw_normal_bf16((total, H, d), 1.0, 71)
    k = W.draw_normal_bf16((total, H, d), 1.0, 72)
    v = W.draw_normal_bf16((total, H, d), 1.0, 73)
    kc = W.draw_normal_bf16((w.batch * w.prompt, H, d), 1.0, 74)
    vc = W.draw_normal_bf16((w.batch * w.prompt, H, d), 1.0, 75)
    pos = torch.tensor(p1 * w.batch, dtype=torch.int32)
    out = torch.full((total, H, d), float("nan"), dtype=torch.bfloat16, device=dev)
    for rep in range(3):
        ssm.ssm_attention_varlen(q.to(dev), k.to(dev), v.to(dev), pos.to(dev), kc.to(dev), vc.to(dev),
                                 ssm.attn_problems_tensor(rows, dev), w.batch, n_new, w.prompt, out, w.rope_theta)
        torch.cuda.synchronize()
        check_device_error()
    og = f64(out)
    for s in (0, 3, w.batch - 1):
        sl = slice(s * n_new, (s + 1) * n_new)
        cs = slice(s * w.prompt, (s + 1) * w.prompt)
        hs = [0, H - 1]
        ref, _ = O.attention(f64(q[None, sl][:, :, hs]), f64(k[None, sl][:, :, hs]), f64(v[None, sl][:, :, hs]),
                             pos[sl].numpy(), f64(kc[None, cs][:, :, hs]), f64(vc[None, cs][:, :, hs]), w.rope_theta)
        assert_attention_close(og[sl][None][:, :, hs], ref, f"serve sequence {s}")


@pytest.mark.parametrize("shape", ["llada", "serve"])
def test_attention_varlen_cold_l2_and_graph_replay(dev, shape):
    """Pipeline timing edge cases: every launch behind a 256 MB write (cold L2, slow tile loads
    while the producers run ahead), eagerly and as CUDA-graph replays, with a 0.2 s wait limit so
    a stuck barrier wait reports SSM_ERR_TIMEOUT quickly; the outputs must equal a warm launch's.
    Shapes: one 589-row problem without cache (LLaDA: two-query-tile units and a split-key tail
    unit), and 8 x 101 rows with per-sequence 512-row caches (serving: split-key units only)."""
    from paper_2608_23167_gb300 import ssm
    h, d = 32, 128
    if shape == "llada":
        sizes, cache_rows = [(589, 0)], 0
    else:
        sizes, cache_rows = [(101, 512)] * 8, 8 * 512
    rows, new_row = [], 0
    for i, (n, c) in enumerate(sizes):
        rows.append((new_row, i * c, n, c))
        new_row += n
    q = W.draw_normal_bf16((new_row, h, d), 1.0, 81).to(dev)
    k = W.draw_normal_bf16((new_row, h, d), 1.0, 82).to(dev)
    v = W.draw_normal_bf16((new_row, h, d), 1.0, 83).to(dev)
    kc = W.draw_normal_bf16((cache_rows, h, d), 1.0, 84).to(dev) if cache_rows else None
    vc = W.draw_normal_bf16((cache_rows, h, d), 1.0, 85).to(dev) if cache_rows else None
    pos = torch.arange(new_row, dtype=torch.int32).to(dev) % 1500 + 512
    probs = ssm.attn_problems_tensor(rows, dev)
    ws = torch.empty(ssm.ssm_attention_workspace_size(new_row, h, h, d), dtype=torch.uint8, device=dev)
    args = (q, k, v, pos, kc, vc, probs, len(rows), max(r[2] for r in rows), max(r[3] for r in rows))
    ref = torch.empty_like(q)
    ssm.ssm_attention_varlen(*args, ref, 5e5, workspace=ws)
    torch.cuda.synchronize()
    check_device_error()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    out = torch.empty_like(q)
    ssm.ssm_set_wait_limit_ns(200_000_000)
    try:
        for i in range(8):
            flush.fill_(i)
            ssm.ssm_attention_varlen(*args, out, 5e5, workspace=ws)
        torch.cuda.synchronize()
        check_device_error()
        assert torch.equal(out, ref)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            ssm.ssm_attention_varlen(*args, out, 5e5, workspace=ws)
        for i in range(8):
            flush.fill_(i)
            out.zero_()
            g.replay()
        torch.cuda.synchronize()
        check_device_error()
        assert torch.equal(out, ref)
    finally:
        ssm.ssm_set_wait_limit_ns(0)


@pytest.mark.parametrize("case", ["mixed", "gqa", "d64", "one_row"])
def test_attention_varlen_packed_prefix(dev, case):
    """Ragged batches whose problems read prefixes of one shared cache and whose new rows
    follow one another: the kernel packs the rows of consecutive problems into shared query
    tiles (each row masked to its own prefix and its own new rows).  Every problem is checked
    against the oracle: problems without cache rows next to ones with long prefixes, problems
    straddling a tile pair, GQA packing (several query heads per kv head), d = 64, and one-row
    problems (hundreds per tile pair); the last pair has at most 128 rows (split keys)."""
    from paper_2608_23167_gb300 import ssm
    h_q, h_kv, d, theta = 4, 4, 128, 1e4
    if case == "mixed":
        sizes = [(37, 100), (1, 0), (130, 250), (64, 250), (5, 31), (200, 512), (33, 64)]
    elif case == "gqa":
        h_q, h_kv = 8, 2
        sizes = [(50, 300), (70, 320), (20, 0), (90, 400)]
    elif case == "d64":
        d = 64
        sizes = [(37, 100), (1, 0), (130, 250), (64, 250), (5, 31), (200, 512), (33, 64)]
    else:
        sizes = [(1, (7 * i) % 200) for i in range(300)]
    cache_rows = max(c for _, c in sizes) or 1
    rows, new_row = [], 0
    for n, c in sizes:
        rows.append((new_row, 0, n, c))
        new_row += n
    seed = 91 + len(sizes) + d
    q = W.draw_normal_bf16((new_row, h_q, d), 1.0, seed)
    k = W.draw_normal_bf16((new_row, h_kv, d), 1.0, seed + 1)
    v = W.draw_normal_bf16((new_row, h_kv, d), 1.0, seed + 2)
    kc = W.draw_normal_bf16((cache_rows, h_kv, d), 1.0, seed + 3)
    vc = W.draw_normal_bf16((cache_rows, h_kv, d), 1.0, seed + 4)
    g = torch.Generator().manual_seed(seed + 5)
    pos = torch.cat([(c + torch.randperm(2 * n + 3, generator=g)[:n]) for n, c in sizes]).to(torch.int32)
    out = torch.full((new_row, h_q, d), float("nan"), dtype=torch.bfloat16, device=dev)
    lse = torch.full((new_row, h_q), float("nan"), dtype=torch.float32, device=dev)
    ssm.ssm_attention_varlen(q.to(dev), k.to(dev), v.to(dev), pos.to(dev), kc.to(dev), vc.to(dev),
                             ssm.attn_problems_tensor(rows, dev), len(rows), max(n for n, _ in sizes),
                             max(c for _, c in sizes), out, theta, lse=lse)
    torch.cuda.synchronize()
    check_device_error()
    og, lg = f64(out), f64(lse)
    for i, (nr, _, n, c) in enumerate(rows):
        if case == "one_row" and i % 10:
            continue
        sl = slice(nr, nr + n)
        ref, ref_lse = O.attention(f64(q[None, sl]), f64(k[None, sl]), f64(v[None, sl]), pos[sl].numpy(),
                                   f64(kc[None, :c]) if c else None, f64(vc[None, :c]) if c else None, theta)
        assert_attention_close(og[sl][None], ref, f"{case} problem {i} ({n} rows, prefix {c})")
        assert np.abs(lg[sl][None] - ref_lse).max() <= 2e-2, f"{case} problem {i} lse"
