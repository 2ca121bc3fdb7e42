"""Pins for the CPU oracle: checks against what the paper and mathematics fix.

Each test ties the oracle to something other than itself: hand-worked examples
from the paper's definitions (tests/golden/), closed forms, invariants, special
cases that reduce to a library routine, and brute force on tiny inputs.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import ssm_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# ----------------------------------------------------------------------------- bf16


def test_bf16_round_matches_torch_on_float32_values():
    # float32 -> bfloat16 in torch is round-to-nearest-even; on values that are
    # exactly float32 the float64 rounding must agree bit for bit.
    g = torch.Generator().manual_seed(0)
    x = torch.cat([torch.randn(20000, generator=g) * s for s in (1e-3, 1.0, 50.0, 1e20)])
    x = torch.cat([x, torch.tensor([0.0, -0.0, 1.0, -1.0, 3.0e38, 1e-39, -2.5e-40])])
    ref = x.to(torch.bfloat16).to(torch.float64).numpy()
    got = O.bf16_round(x.to(torch.float64).numpy())
    assert np.array_equal(ref, got)


def test_bf16_round_ties_to_even():
    one = 1.0
    assert O.bf16_round(np.array([one + 2.0 ** -8]))[0] == 1.0                 # tie -> even (1.0)
    assert O.bf16_round(np.array([one + 3 * 2.0 ** -8]))[0] == 1.0 + 2.0 ** -6  # tie -> even (odd+1)
    assert O.bf16_round(np.array([one + 2.0 ** -8 + 2.0 ** -30]))[0] == 1.0 + 2.0 ** -7
    assert O.bf16_round(np.array([0.2]))[0] == 0.2001953125
    assert O.bf16_round(np.array([1.4]))[0] == 1.3984375


# ----------------------------------------------------------------------------- selector


def _expand(positions):
    out = []
    for a, b in positions["ranges"]:
        out.extend(range(a, b))
    out.extend(positions["singles"])
    return sorted(out)


@pytest.mark.parametrize("case", _load("selector_cases.json")["cases"], ids=lambda c: c["name"])
def test_selector_golden(case):
    r, nl, nm, nt = O.select_suffix(case["P"], case["G"], case["B"], case["b"],
                                    case["L"], case["M"], case["T"])
    assert r == _expand(case["positions"])
    assert [nl, nm, nt] == case["counts"]


def _classify_bruteforce(P, G, B, b, L, M, T):
    """Per-position classification straight from Eq. 1-5 (independent of the set code)."""
    nb = G // B
    out = []
    n_sb = nb - 1 - b
    for pos in range(P + (b + 1) * B, P + G):
        blk = (pos - P) // B               # block index of this token
        rank = pos - (P + (b + 1) * B)     # index of the token within the suffix
        if n_sb * B <= L:
            out.append(pos)
            continue
        is_local = rank < L
        is_tail_block = blk == nb - 1
        off = (pos - P) % B
        keep = is_local
        if is_tail_block:
            if T >= B:
                keep = True
            elif T == 1:
                keep = keep or off == 0
            elif T >= 2:
                keep = keep or any((j * (B - 1)) // (T - 1) == off for j in range(T))
        else:
            first_block_rank = (blk - (b + 1)) * B
            middle = first_block_rank >= L
            if middle and off == 0:
                mids = [j for j in range(b + 1, nb - 1) if (j - (b + 1)) * B >= L]
                nm = len(mids)
                chosen = mids if nm <= M else [mids[(q * nm) // M] for q in range(M)]
                keep = keep or blk in chosen
        if keep:
            out.append(pos)
    return out


def test_selector_bruteforce_small_grid():
    for P, G, B in [(0, 64, 4), (5, 96, 8), (16, 256, 32)]:
        nb = G // B
        for b in range(nb):
            for L in sorted({0, 1, B // 2, B, B + B // 2, 2 * B, 3 * B, G}):
                for M in (0, 1, 2, 3, 100):
                    for T in (0, 1, 2, 3, B - 1, B, B + 3):
                        r, nl, nm, nt = O.select_suffix(P, G, B, b, L, M, T)
                        assert r == _classify_bruteforce(P, G, B, b, L, M, T)
                        assert nl + nm + nt == len(r)


@pytest.mark.parametrize("P,G,B,L,M,T", [(64, 256, 32, 32, 8, 4), (512, 256, 32, 32, 16, 8),
                                         (512, 1024, 32, 64, 32, 8), (1024, 2048, 32, 64, 64, 16),
                                         (512, 1024, 32, 32, 32, 8)])
def test_selector_region_sizes_equal_budgets(P, G, B, L, M, T):
    """Retained-set sizes equal the region budgets whenever the suffix is longer than L."""
    nb = G // B
    for b in range(nb):
        r, nl, nm, nt = O.select_suffix(P, G, B, b, L, M, T)
        n_sb = nb - 1 - b
        assert r == sorted(set(r))
        assert all(P + (b + 1) * B <= x < P + G for x in r)
        if n_sb == 0:
            assert r == []
        elif n_sb * B <= L:
            assert nl == n_sb * B and nm == 0 and nt == 0
        else:
            n_mid_blocks = len([j for j in range(b + 1, nb - 1) if (j - b - 1) * B >= L])
            assert nl == L and nt == min(T, B) and nm == min(M, n_mid_blocks)


def test_selector_paper_exact_mode_is_eqs_2_to_5():
    """L = wB, uncapped middle, T = 2: R is local blocks + middle starts + {tail start, end}."""
    P, G, B = 7, 512, 32
    nb = G // B
    for w in (1, 2, 3):
        for b in range(nb):
            r, *_ = O.select_suffix(P, G, B, b, w * B, 10 ** 6, 2)
            suffix_blocks = list(range(b + 1, nb))
            if len(suffix_blocks) <= w:
                expect = set(range(P + (b + 1) * B, P + G))
            else:
                local = suffix_blocks[:w]
                tail = suffix_blocks[-1]
                middle = suffix_blocks[w:-1]
                expect = set()
                for j in local:
                    expect |= set(range(P + j * B, P + (j + 1) * B))
                expect |= {P + j * B for j in middle}
                expect |= {P + tail * B, P + tail * B + B - 1}
            assert set(r) == expect


def test_selector_full_retention():
    for b in range(8):
        r, *_ = O.select_suffix(3, 256, 32, b, 256, 0, 0)
        assert r == list(range(3 + (b + 1) * 32, 3 + 256))


def test_selector_rejects_bad_layout():
    with pytest.raises(ValueError):
        O.select_suffix(0, 100, 32, 0, 32, 8, 4)
    with pytest.raises(ValueError):
        O.select_suffix(0, 256, 32, 8, 32, 8, 4)
    with pytest.raises(ValueError):
        O.select_suffix(0, 256, 32, 0, -1, 8, 4)


# ----------------------------------------------------------------------------- soft embedding


@pytest.mark.parametrize("case", _load("soft_embedding_cases.json")["cases"], ids=lambda c: c["why"][:30])
def test_soft_embedding_golden(case):
    d = _load("soft_embedding_cases.json")
    embed = np.array(d["embed"], dtype=np.float64)
    x = O.bf16_round(O.soft_suffix_embedding(embed, d["mask_id"], case["ids"], case["probs"],
                                             case["alpha"]))
    assert x.tolist() == case["x"]


def _rand_embed(V=64, H=16, seed=0):
    rng = np.random.default_rng(seed)
    return O.bf16_round(rng.standard_normal((V, H)))


def test_soft_embedding_special_cases():
    E = _rand_embed()
    mask = 63
    rng = np.random.default_rng(1)
    for _ in range(20):
        ids = rng.choice(63, 5, replace=False)
        probs = rng.random(5)
        # alpha = 0 -> e_mask exactly
        assert np.array_equal(O.soft_suffix_embedding(E, mask, ids, probs, 0.0), E[mask])
        # alpha = 1, k = 1 -> e_u exactly
        assert np.array_equal(O.soft_suffix_embedding(E, mask, ids[:1], probs[:1], 1.0), E[ids[0]])
        # identical ids -> e_u, whatever the probabilities
        same = [ids[0]] * 5
        x = O.soft_suffix_embedding(E, mask, same, probs, 1.0)
        assert np.allclose(x, E[ids[0]], rtol=0, atol=1e-14)
        # linear in alpha
        a0 = O.soft_suffix_embedding(E, mask, ids, probs, 0.25)
        a1 = O.soft_suffix_embedding(E, mask, ids, probs, 0.75)
        am = O.soft_suffix_embedding(E, mask, ids, probs, 0.5)
        assert np.allclose(am, 0.5 * (a0 + a1), atol=1e-13)
        # the mix lies in the convex hull: |x| <= max row norm
        x = O.soft_suffix_embedding(E, mask, ids, probs, 0.4)
        assert np.linalg.norm(x) <= max(np.linalg.norm(E[i]) for i in list(ids) + [mask]) + 1e-12


def test_eq6_renormalisation_equals_softmax_over_topk_logits():
    """Renormalising full-vocabulary probabilities within the top-k set is a softmax
    over the top-k logits; the mixed row must not depend on which form is given."""
    E = _rand_embed(V=50)
    rng = np.random.default_rng(3)
    logits = rng.standard_normal(49) * 3
    p_full = np.exp(logits - logits.max())
    p_full /= p_full.sum()
    top = np.argsort(-p_full)[:5]
    z = logits[top]
    p_soft = np.exp(z - z.max())
    p_soft /= p_soft.sum()
    a = O.soft_suffix_embedding(E, 49, top, p_full[top], 0.4)
    b = O.soft_suffix_embedding(E, 49, top, p_soft, 0.4)
    assert np.allclose(a, b, atol=1e-13)
    # independent of the order of the candidates
    perm = rng.permutation(5)
    c = O.soft_suffix_embedding(E, 49, top[perm], p_full[top][perm], 0.4)
    assert np.allclose(a, c, atol=1e-13)


def test_build_step_input_layout_and_positions():
    E = _rand_embed(V=32, H=8)
    mask = 31
    blk = np.array([[mask, 4, mask, 7]])
    pre = np.array([[1, 2, 3]])
    ids = np.array([[[5, 6], [-1, -1]]])
    probs = np.array([[[0.5, 0.25], [0.1, 0.1]]])
    x, pos = O.build_step_input(E, mask, blk, 40, [50, 63], ids, probs, 0.4, prefix_tokens=pre)
    assert x.shape == (1, 3 + 4 + 2, 8)
    assert pos.tolist() == [0, 1, 2, 40, 41, 42, 43, 50, 63]
    for r, t in enumerate([1, 2, 3, mask, 4, mask, 7]):
        assert np.array_equal(x[0, r], E[t])            # prompt and block rows are lookups
    expect = 0.6 * E[mask] + 0.4 * (2.0 / 3.0 * E[5] + 1.0 / 3.0 * E[6])
    assert np.array_equal(x[0, 7], O.bf16_round(expect))
    assert np.array_equal(x[0, 8], E[mask])


# ----------------------------------------------------------------------------- RoPE / attention


def test_rope_d2_closed_form():
    # d = 2: one pair, inverse frequency theta**0 = 1, so the vector turns by `pos` radians
    pos = np.array([0, 1, 2, 7, 1000])
    x = np.tile(np.array([[[1.0, 0.0]]]), (5, 1, 1))
    y = O.rope(x, pos, 10000.0)
    assert np.allclose(y[:, 0, 0], np.cos(pos), atol=1e-15)
    assert np.allclose(y[:, 0, 1], np.sin(pos), atol=1e-15)


def test_rope_pair_frequencies_and_norm():
    d = 8
    theta = 10000.0
    x = np.zeros((1, 1, d))
    x[0, 0, 1] = 1.0       # pair (1, 5) -> inverse frequency theta**(-2/8)
    y = O.rope(x, np.array([3]), theta)
    ang = 3 * theta ** (-0.25)
    assert np.isclose(y[0, 0, 1], math.cos(ang)) and np.isclose(y[0, 0, 5], math.sin(ang))
    rng = np.random.default_rng(0)
    z = rng.standard_normal((9, 2, 16))
    pz = O.rope(z, rng.integers(0, 5000, 9), 5e5)
    assert np.allclose(np.linalg.norm(pz, axis=-1), np.linalg.norm(z, axis=-1))
    assert np.array_equal(O.rope(z, np.zeros(9, dtype=int), 5e5), z)


def test_rope_relative_position():
    rng = np.random.default_rng(2)
    q = rng.standard_normal((1, 1, 64))
    k = rng.standard_normal((1, 1, 64))
    for m, n, t in [(5, 3, 100), (0, 1000, 17), (2047, 12, 999)]:
        a = np.sum(O.rope(q, np.array([m]), 5e5) * O.rope(k, np.array([n]), 5e5))
        b = np.sum(O.rope(q, np.array([m + t]), 5e5) * O.rope(k, np.array([n + t]), 5e5))
        assert abs(a - b) < 1e-10


# ----------------------------------------------------------------------------- suffix top-k


def test_suffix_topk_bruteforce_and_closed_forms():
    # logits ln(1..6) on V = 6: probabilities are i / 21
    l = np.log(np.array([[3.0, 1.0, 6.0, 2.0, 5.0, 4.0]]))
    ids, probs = O.suffix_topk(l, 3)
    assert ids.tolist() == [[2, 4, 5]]
    assert np.allclose(probs, [[6 / 21, 5 / 21, 4 / 21]])
    # all equal: the k lowest ids, each 1 / V
    ids, probs = O.suffix_topk(np.zeros((2, 50)), 4)
    assert ids.tolist() == [[0, 1, 2, 3]] * 2 and np.allclose(probs, 1 / 50)
    # ties are broken by the lower id, and the order is by probability, not by id
    ids, _ = O.suffix_topk(np.array([[0.0, 2.0, 1.0, 2.0, 1.0]]), 4)
    assert ids.tolist() == [[1, 3, 2, 4]]
    # one planted logit: p = 1 / (1 + (V - 1) e^-d)
    V, d = 1000, 7.0
    l = np.zeros((1, V))
    l[0, 613] = d
    ids, probs = O.suffix_topk(l, 2)
    assert ids[0, 0] == 613 and np.isclose(probs[0, 0], 1 / (1 + (V - 1) * math.exp(-d)))
    assert ids[0, 1] == 0 and np.isclose(probs[0, 1], math.exp(-d) * probs[0, 0])
    with pytest.raises(ValueError):
        O.suffix_topk(np.zeros((1, 3)), 4)


def test_suffix_topk_agrees_with_unmask_confidence_and_sorting():
    rng = np.random.default_rng(31)
    l = np.round(rng.standard_normal((6, 300)) * 4, 2)
    ids, probs = O.suffix_topk(l, 5)
    for r in range(6):
        conf, arg, p2 = O.token_confidence(l[r])
        assert ids[r, 0] == arg and np.isclose(probs[r, 0], conf) and np.isclose(probs[r, 1], p2)
        # against a full sort of the softmax (scipy-free: numpy argsort on (-p, id))
        p = np.exp(l[r] - l[r].max())
        p /= p.sum()
        ref = np.lexsort((np.arange(300), -p))[:5]
        assert ids[r].tolist() == ref.tolist() and np.allclose(probs[r], p[ref])
    assert np.all(np.diff(probs, axis=1) <= 0) and np.all(probs.sum(1) <= 1 + 1e-12)


# ----------------------------------------------------------------------------- early termination


def test_early_stop_hand_cases():
    E = 9
    toks = np.array([[1, 2, 3, 4, 5, 6, 7, 8],     # no EOS in block 1 (positions 4..7): still running
                     [1, 2, 3, 4, 5, E, 7, 8],     # EOS at 5: 6, 7 become EOS
                     [1, E, 3, 4, 5, 6, 7, 8],     # EOS only in block 0, not the checked block: running
                     [1, 2, 3, 4, E, 6, E, 8],     # first EOS of the block at 4 decides
                     [1, 2, 3, 4, 5, 6, 7, E]])    # EOS at the block's last position: nothing to fill
    fin = np.array([0, 0, 0, 0, 0], dtype=np.uint8)
    t, f, n = O.early_stop(toks, 4, 1, E, fin)
    assert f.tolist() == [0, 1, 0, 1, 1] and n == 2
    assert t[0].tolist() == toks[0].tolist() and t[2].tolist() == toks[2].tolist()
    assert t[1].tolist() == [1, 2, 3, 4, 5, E, E, E]
    assert t[3].tolist() == [1, 2, 3, 4, E, E, E, E]
    assert t[4].tolist() == toks[4].tolist()
    # a finished sequence is not touched, even with an EOS in the block
    t2, f2, n2 = O.early_stop(toks, 4, 1, E, np.array([1, 1, 1, 1, 1], dtype=np.uint8))
    assert np.array_equal(t2, toks) and f2.tolist() == [1] * 5 and n2 == 0
    # filling reaches later blocks: block 0 of 3
    t3, f3, _ = O.early_stop(np.array([[E, 5, 5, 5, 5, 5]]), 2, 0, E, np.array([0], dtype=np.uint8))
    assert t3.tolist() == [[E] * 6] and f3.tolist() == [1]


# ----------------------------------------------------------------------------- prefix-cache append


def test_cache_append_places_rotated_rows_and_leaves_the_rest():
    # d = 2: one pair with inverse frequency 1, so a key at position p turns by p radians
    rng = np.random.default_rng(21)
    B, C, n, H = 2, 9, 3, 2
    kc = rng.standard_normal((B, C, H, 2))
    vc = rng.standard_normal((B, C, H, 2))
    kn = rng.standard_normal((B, n, H, 2))
    vn = rng.standard_normal((B, n, H, 2))
    pos = np.array([40, 3, 1000])          # positions need not follow the row order
    k2, v2 = O.cache_append(kc, vc, kn, vn, pos, 5e5, 4)
    c, s_ = np.cos(pos)[None, :, None], np.sin(pos)[None, :, None]
    want0 = kn[..., 0] * c - kn[..., 1] * s_
    want1 = kn[..., 1] * c + kn[..., 0] * s_
    assert np.allclose(k2[:, 4:7, :, 0], want0, atol=1e-12) and np.allclose(k2[:, 4:7, :, 1], want1, atol=1e-12)
    assert np.array_equal(v2[:, 4:7], vn)
    keep = np.r_[0:4, 7:9]
    assert np.array_equal(k2[:, keep], kc[:, keep]) and np.array_equal(v2[:, keep], vc[:, keep])
    # the inputs are not modified
    assert not np.shares_memory(k2, kc)


def test_cache_append_rotation_invariants_and_capacity():
    rng = np.random.default_rng(22)
    kn = rng.standard_normal((1, 6, 4, 64))
    vn = rng.standard_normal((1, 6, 4, 64))
    pos = np.arange(6) + 1024
    kc, vc = O.cache_append(np.zeros((1, 16, 4, 64)), np.zeros((1, 16, 4, 64)), kn, vn, pos, 5e5, 10)
    # a rotation keeps every head vector's norm
    assert np.allclose(np.linalg.norm(kc[:, 10:], axis=-1), np.linalg.norm(kn, axis=-1))
    # scores between two appended keys depend only on their position difference
    kd, _ = O.cache_append(np.zeros((1, 16, 4, 64)), np.zeros((1, 16, 4, 64)), kn, vn, pos + 777, 5e5, 10)
    g1 = np.einsum("nhd,mhd->hnm", kc[0, 10:], kc[0, 10:])
    g2 = np.einsum("nhd,mhd->hnm", kd[0, 10:], kd[0, 10:])
    assert np.allclose(g1, g2, atol=1e-9)
    # theta == 0: no rotation, a plain copy
    k0, _ = O.cache_append(np.zeros((1, 6, 4, 64)), np.zeros((1, 6, 4, 64)), kn, vn, pos, 0.0, 0)
    assert np.array_equal(k0, kn)
    with pytest.raises(ValueError):
        O.cache_append(np.zeros((1, 16, 4, 64)), np.zeros((1, 16, 4, 64)), kn, vn, pos, 5e5, 11)


def _attn_bruteforce(q, keys, vals, scale):
    out = []
    for qi in q:
        s = [scale * sum(a * b for a, b in zip(qi, kj)) for kj in keys]
        m = max(s)
        e = [math.exp(x - m) for x in s]
        z = sum(e)
        out.append([sum(e[j] * vals[j][c] for j in range(len(keys))) / z for c in range(len(vals[0]))])
    return np.array(out)


def test_attention_bruteforce_tiny():
    rng = np.random.default_rng(5)
    n, d = 5, 8
    q = rng.standard_normal((1, n, 1, d))
    k = rng.standard_normal((1, n, 1, d))
    v = rng.standard_normal((1, n, 1, d))
    kc = rng.standard_normal((1, 3, 1, d))
    vc = rng.standard_normal((1, 3, 1, d))
    pos = np.array([10, 11, 12, 40, 77])
    out, _ = O.attention(q, k, v, pos, kc, vc, 0.0, 0.3)
    ref = _attn_bruteforce(q[0, :, 0], list(kc[0, :, 0]) + list(k[0, :, 0]),
                           list(vc[0, :, 0]) + list(v[0, :, 0]), 0.3)
    assert np.allclose(out[0, :, 0], ref, atol=1e-12)


def test_attention_closed_forms():
    # two keys, d = 2: q = (1,0), k = (1,0),(0,0), v = e1, e2 -> out = (e/(e+1), 1/(e+1))
    q = np.array([[[[1.0, 0.0]]]])
    k = np.array([[[[1.0, 0.0]], [[0.0, 0.0]]]]).reshape(1, 2, 1, 2)
    v = np.array([[[[1.0, 0.0]], [[0.0, 1.0]]]]).reshape(1, 2, 1, 2)
    out, lse = O.attention(q, k[:, 1:], v[:, 1:], np.array([0]), k[:, :1], v[:, :1], 0.0, 1.0)
    e = math.e
    assert np.allclose(out[0, 0, 0], [e / (e + 1), 1 / (e + 1)])
    assert np.isclose(lse[0, 0, 0], math.log(e + 1))
    rng = np.random.default_rng(7)
    # one key -> O = v
    q = rng.standard_normal((2, 1, 4, 16))
    kk = rng.standard_normal((2, 1, 2, 16))
    vv = rng.standard_normal((2, 1, 2, 16))
    out, _ = O.attention(q, kk, vv, np.array([5]), None, None, 1e4)
    assert np.allclose(out, np.repeat(vv, 2, axis=2))
    # identical keys -> mean of values
    kc = np.repeat(rng.standard_normal((1, 1, 1, 16)), 6, axis=1)
    vc = rng.standard_normal((1, 6, 1, 16))
    q = rng.standard_normal((1, 1, 1, 16))
    out, _ = O.attention(q, np.zeros((1, 1, 1, 16)), vc[:, :1], np.array([0]), kc[:, 1:], vc[:, 1:], 0.0)
    # new key is zero and differs; use the cache-only identical set via a zero query instead
    out, _ = O.attention(np.zeros((1, 1, 1, 16)), kc[:, :1], vc[:, :1], np.array([3]), kc[:, 1:],
                         vc[:, 1:], 0.0)
    assert np.allclose(out[0, 0, 0], vc[0, :, 0].mean(axis=0))


def test_attention_softmax_rows_sum_to_one_and_permutation_invariance():
    rng = np.random.default_rng(9)
    B, n, nc, hq, hkv, d = 2, 7, 5, 4, 2, 16
    q = rng.standard_normal((B, n, hq, d))
    k = rng.standard_normal((B, n, hkv, d))
    v = rng.standard_normal((B, n, hkv, d))
    kc = rng.standard_normal((B, nc, hkv, d))
    vc = rng.standard_normal((B, nc, hkv, d))
    pos = rng.permutation(100)[:n] + nc
    out, lse = O.attention(q, k, v, pos, kc, vc, 1e4)
    # rows sum to one: sum_k exp(s - lse) == 1 (recomputed from the definition)
    qr, kr = O.rope(q, pos, 1e4), O.rope(k, pos, 1e4)
    keys = np.concatenate([kc, kr], axis=1)
    for b in range(B):
        for h in range(hq):
            s = qr[b, :, h] @ keys[b, :, h // 2].T / math.sqrt(d)
            assert np.allclose(np.exp(s - lse[b, :, h][:, None]).sum(1), 1.0)
    # permuting the new rows together with their positions permutes the output rows
    perm = rng.permutation(n)
    out2, _ = O.attention(q[:, perm], k[:, perm], v[:, perm], pos[perm], kc, vc, 1e4)
    assert np.allclose(out2, out[:, perm])
    # permuting the cache rows does not change anything
    cp = rng.permutation(nc)
    out3, _ = O.attention(q, k, v, pos, kc[:, cp], vc[:, cp], 1e4)
    assert np.allclose(out3, out)
    # GQA: query head h reads kv head h // 2 -- equal to MHA with kv heads repeated
    out4, _ = O.attention(q, np.repeat(k, 2, axis=2), np.repeat(v, 2, axis=2), pos,
                          np.repeat(kc, 2, axis=2), np.repeat(vc, 2, axis=2), 1e4)
    assert np.allclose(out4, out)


def test_full_retention_equals_full_sequence_attention():
    """With budgets that keep the whole suffix, the sparse step is the dense step:
    attention over [cache; block; R_t] equals full-sequence bidirectional attention
    over [P; B_t; S_t] (computed here by brute force over the whole sequence)."""
    rng = np.random.default_rng(11)
    P, G, B, b, d = 6, 32, 8, 1, 8
    r, *_ = O.select_suffix(P, G, B, b, G, 0, 0)
    total = P + G
    seq_q = rng.standard_normal((total, d))
    seq_k = rng.standard_normal((total, d))
    seq_v = rng.standard_normal((total, d))
    theta = 100.0
    # cache holds the rotated keys of the committed prefix [0, P + bB)
    n_cache = P + b * B
    all_pos = np.arange(total)
    kc = O.rope(seq_k[:n_cache, None, :][None], all_pos[:n_cache], theta)
    vc = seq_v[None, :n_cache, None, :]
    rows = list(range(P + b * B, P + (b + 1) * B)) + list(r)
    assert rows == list(range(n_cache, total))
    out, _ = O.attention(seq_q[None, rows, None, :], seq_k[None, rows, None, :],
                         seq_v[None, rows, None, :], np.array(rows), kc, vc, theta)
    qr = O.rope(seq_q[:, None, :], all_pos, theta)[:, 0]
    kr = O.rope(seq_k[:, None, :], all_pos, theta)[:, 0]
    dense = _attn_bruteforce(qr[rows], list(kr), list(seq_v), 1 / math.sqrt(d))
    assert np.allclose(out[0, :, 0], dense, atol=1e-12)


# ----------------------------------------------------------------------------- unmask


def test_unmask_golden():
    d = _load("unmask_cases.json")
    logits = np.log(np.array(d["logits_ln"], dtype=np.float64))[None]
    masked = np.array(d["masked"])[None]
    modes = {"threshold": O.MODE_THRESHOLD, "topk": O.MODE_TOPK, "margin": O.MODE_MARGIN}
    for c in d["commits"]:
        conf, arg, p2, commit = O.unmask(logits, masked, modes[c["mode"]], c["threshold"], c["topk"],
                                         c["min_commit"])
        assert commit[0].tolist() == c["commit"], c
        for j, row in enumerate(d["expect_rows"]):
            assert arg[0, j] == row["argmax"]
            if row["conf"] is None:
                assert conf[0, j] == 0 and p2[0, j] == 0
            else:
                assert np.isclose(conf[0, j], row["conf"][0] / row["conf"][1], rtol=1e-14)
                assert np.isclose(p2[0, j], row["p2"][0] / row["p2"][1], rtol=1e-14)


def test_token_confidence_special_cases():
    V = 4096
    conf, arg, p2 = O.token_confidence(np.zeros(V))
    assert np.isclose(conf, 1.0 / V) and arg == 0 and np.isclose(p2, 1.0 / V)
    x = np.zeros(V)
    x[1234] = 60.0
    conf, arg, p2 = O.token_confidence(x)
    assert conf >= 1 - 1e-12 and arg == 1234 and p2 < 1e-20
    # ties: lowest id wins, p2 equals conf
    x = np.zeros(8)
    x[[3, 6]] = 2.0
    conf, arg, p2 = O.token_confidence(x)
    assert arg == 3 and np.isclose(conf, p2)


def test_token_confidence_bruteforce_v8():
    rng = np.random.default_rng(13)
    for _ in range(200):
        x = rng.standard_normal(8) * 4
        e = [math.exp(v) for v in x]
        z = sum(e)
        p = sorted((v / z for v in e), reverse=True)
        conf, arg, p2 = O.token_confidence(x)
        assert math.isclose(conf, p[0], rel_tol=1e-13) and math.isclose(p2, p[1], rel_tol=1e-13)
        assert arg == max(range(8), key=lambda i: (x[i], -i))


def test_unmask_min_commit_and_ties():
    # every row below the threshold: exactly one commit, at the highest confidence;
    # equal confidences resolve to the lower position
    logits = np.zeros((1, 6, 16))
    logits[0, 2, 0] = 1.0
    logits[0, 4, 0] = 1.0
    masked = np.array([[1, 1, 1, 1, 1, 0]])
    conf, arg, p2, commit = O.unmask(logits, masked, O.MODE_THRESHOLD, 0.9)
    assert commit[0].tolist() == [0, 0, 1, 0, 0, 0]
    conf, arg, p2, commit = O.unmask(logits, masked, O.MODE_TOPK, 0.0, topk=3)
    assert commit[0].tolist() == [1, 0, 1, 0, 1, 0]
    # nothing masked: nothing committed
    conf, arg, p2, commit = O.unmask(logits, np.zeros((1, 6), dtype=int), O.MODE_THRESHOLD, 0.9)
    assert commit.sum() == 0 and (arg == -1).all()


# ----------------------------------------------------------------------------- pins catch mistakes


def test_pins_catch_planted_mistakes(monkeypatch):
    """Plant plausible mistakes in the oracle (on the CPU) and check that a pin fails."""
    d = _load("soft_embedding_cases.json")
    embed = np.array(d["embed"])
    case = d["cases"][0]

    def no_renorm(embed, mask_id, ids, probs, alpha):     # Eq. 6 dropped
        e = sum(p * embed[v] for v, p in zip(ids, probs) if v >= 0)
        return (1 - alpha) * embed[mask_id] + alpha * e

    assert O.bf16_round(no_renorm(embed, 3, case["ids"], case["probs"], case["alpha"])).tolist() != case["x"]

    def swapped_mix(embed, mask_id, ids, probs, alpha):   # alpha on the wrong term
        z = sum(p for v, p in zip(ids, probs) if v >= 0)
        e = sum(p / z * embed[v] for v, p in zip(ids, probs) if v >= 0)
        return alpha * embed[mask_id] + (1 - alpha) * e

    assert O.bf16_round(swapped_mix(embed, 3, [0, 1], [0.3, 0.1], 0.4)).tolist() != \
        O.bf16_round(O.soft_suffix_embedding(embed, 3, [0, 1], [0.3, 0.1], 0.4)).tolist()

    # RoPE with the wrong sign of sin fails the d = 2 closed form
    orig = O.rope

    def bad_rope(x, pos, theta):
        y = orig(x, pos, theta)
        h = y.shape[-1] // 2
        return np.concatenate([y[..., :h], -y[..., h:]], axis=-1)

    monkeypatch.setattr(O, "rope", bad_rope)
    with pytest.raises(AssertionError):
        test_rope_d2_closed_form()
    monkeypatch.setattr(O, "rope", orig)

    # tail spacing that drops the end token fails the golden selector
    cases = _load("selector_cases.json")["cases"]
    c = [c for c in cases if c["name"] == "tiny_workload_b0"][0]
    r, *_ = O.select_suffix(c["P"], c["G"], c["B"], c["b"], c["L"], c["M"], c["T"] + 1)
    assert r != _expand(c["positions"])
