"""CPU oracle for one structured-suffix (SSM) denoising step -- TEST INFRASTRUCTURE.

This module is the plain, slow, fp64 definition that the CUDA path is checked
against.  Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU
baseline leg may import it; the product path never calls it and shares no code
with it.  Every function takes plain numpy arrays (bf16 inputs arrive as the
exact float64 values of the bf16 numbers) and follows the paper's definitions
in the paper's order:

* ``select_suffix``      -- Sec. 3.2 "Suffix Region Partition" (Eq. 1) and
                            "Suffix Token Retention" (Eqs. 2-5).
* ``build_step_input``   -- Sec. 3.2 "Soft Suffix Embedding Mixing" (Eqs. 6-8)
                            and "Sparse Input Construction" (the sparse input
                            X~_t = [P; B_t; R_t] with original positions).
* ``rope`` / ``attention`` -- bidirectional attention of the DLM (Sec. 1,
                            Sec. 2) over the sparse input with rotary position
                            encodings at the retained tokens' original positions
                            (Sec. 3.2, sparse input construction).
* ``unmask``             -- parallel (threshold) decoding and Vanilla top-1
                            decoding (Sec. 4.2 "Baselines"), and the margin rule
                            (Sec. 4.6).
* ``suffix_topk``        -- the top-k candidates of a retained suffix position
                            and their probabilities under the full-vocabulary
                            softmax (Sec. 3.2 "Soft Suffix Embedding Mixing": the
                            set T^i_{t+1} and p^i_{t+1}(v) that Eq. 6 renormalizes
                            at the next step).
* ``early_stop``         -- early termination after a decoded block (Sec. 3.2
                            "Early Termination").
* ``cache_append``       -- the prefix-cache update at a block boundary in the
                            prefix-caching setting ("+PC.", Sec. 4.8, Table 4):
                            the block's keys (rotated at their positions) and
                            values are written into the cache.
* ``bf16_round``         -- round-to-nearest-even to bfloat16 (the storage type
                            of the sparse input).

Readings where the paper is silent (token budgets, tail spacing, RoPE
convention, tie rules, the min-1 commit) are stated in each docstring.
Parity status: every function here is pinned by ``tests/test_oracle_*.py``.
"""
from __future__ import annotations

import math
from typing import Optional, Sequence, Tuple

import numpy as np

# --------------------------------------------------------------------------------------
# bfloat16 rounding
# --------------------------------------------------------------------------------------


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round float64 values to the nearest bfloat16 value, ties to even.

    bfloat16 keeps 8 significant bits and the float32 exponent range.  For a
    normal value x = m * 2**e (0.5 <= |m| < 1) the spacing of bfloat16 numbers
    around x is 2**(e - 8); below 2**-126 the spacing is fixed at 2**-133.
    Values beyond the largest finite bfloat16 become infinities.
    """
    x = np.asarray(x, dtype=np.float64)
    out = np.array(x, copy=True)
    finite = np.isfinite(x) & (x != 0)
    xf = x[finite]
    _, e = np.frexp(xf)
    e = np.maximum(e, -125)           # |x| < 2**-126 -> subnormal spacing 2**-133
    q = np.ldexp(1.0, e - 8)
    r = np.rint(xf / q) * q          # np.rint rounds half to even
    bf16_max = (2.0 - 2.0 ** -7) * 2.0 ** 127
    r = np.where(np.abs(r) > bf16_max, np.sign(r) * np.inf, r)
    out[finite] = r
    return out


# --------------------------------------------------------------------------------------
# Selector: Eqs. 1-5
# --------------------------------------------------------------------------------------


def select_suffix(prompt_len: int, gen_len: int, block_len: int, block_idx: int,
                  local_budget: int, middle_budget: int, tail_budget: int):
    """Retained suffix set R_t for the block being decoded (Sec. 3.2, Eqs. 1-5).

    Layout: the prompt occupies positions [0, P); the generation [P, P+G) is cut
    into nb = G / B blocks; block b is [P + bB, P + (b+1)B) and the suffix S_t is
    every later block.

    Eq. 1 partitions S_t: the first w suffix blocks are local, the last suffix
    block is the tail, the blocks between are middle; with fewer suffix blocks
    than w, all are local.  Readings:
      * the local size is given in tokens, L = w * B (w may be fractional in the
        paper's sweep, so L need not be a multiple of B); when the whole suffix
        fits in L (n_sb * B <= L) every suffix token is local;
      * a block that the local region covers in part yields no middle start
        token (its start is already local);
      * the middle budget M caps the number of middle start tokens; with more
        middle blocks than M, blocks q*nm//M for q = 0..M-1 are kept;
      * the tail budget T keeps T evenly spaced tokens of the tail block,
        offsets (j*(B-1))//(T-1) for j = 0..T-1, which always include start and
        end; T = 2 is exactly Eq. 4, T = 1 keeps the start, T >= B keeps the
        whole block, T = 0 keeps nothing.
    Eq. 2 keeps every local token, Eq. 3 the start token of each middle block,
    Eq. 4 the tail tokens, Eq. 5 takes the union.

    Returns (positions ascending, n_local, n_mid, n_tail) where n_tail counts the
    tail tokens not already local (so the three counts add up to |R_t|).
    """
    P, G, B, b = prompt_len, gen_len, block_len, block_idx
    L, M, T = local_budget, middle_budget, tail_budget
    if B <= 0 or G <= 0 or G % B != 0 or P < 0:
        raise ValueError("invalid layout")
    nb = G // B
    if not (0 <= b < nb) or min(L, M, T) < 0:
        raise ValueError("invalid block index or budget")

    suffix_blocks = [P + j * B for j in range(b + 1, nb)]   # start position of each suffix block
    n_sb = len(suffix_blocks)
    if n_sb == 0:
        return [], 0, 0, 0
    s0 = suffix_blocks[0]
    suffix_tokens = list(range(s0, P + G))

    # Eq. 1 (with the "fewer than w blocks" rule)
    if n_sb * B <= L:
        return suffix_tokens, len(suffix_tokens), 0, 0
    local_region = suffix_tokens[:L]
    tail_block = suffix_blocks[-1]
    middle_blocks = [s for s in suffix_blocks[:-1] if s >= s0 + L]

    # Eq. 2
    r_local = set(local_region)
    # Eq. 3 (capped by M)
    nm = len(middle_blocks)
    if nm <= M:
        kept = middle_blocks
    else:
        kept = [middle_blocks[(q * nm) // M] for q in range(M)]
    r_middle = set(kept)
    # Eq. 4 (T tokens of the tail block)
    if T == 0:
        offsets = []
    elif T >= B:
        offsets = list(range(B))
    elif T == 1:
        offsets = [0]
    else:
        offsets = [(j * (B - 1)) // (T - 1) for j in range(T)]
    r_tail = {tail_block + o for o in offsets}
    # Eq. 5
    r = sorted(r_local | r_middle | r_tail)
    return r, len(r_local), len(r_middle), len(r_tail - r_local)


# --------------------------------------------------------------------------------------
# Sparse input with soft suffix embeddings: Eqs. 6-8 and the sparse input X~_t
# --------------------------------------------------------------------------------------


def soft_suffix_embedding(embed: np.ndarray, mask_id: int, ids: Sequence[int],
                          probs: Sequence[float], alpha: float) -> np.ndarray:
    """One retained suffix row, exact in float64 (not rounded).

    Eq. 6 renormalises the previous step's probabilities within its top-k set
    T (entries with id -1 are absent), Eq. 7 forms the soft decoded embedding
    sum_v p~(v) e_v, Eq. 8 mixes it with the [MASK] embedding:
    (1 - alpha) e_mask + alpha e~.  Reading: a position with no previous-step
    prediction (empty set, or zero retained mass) keeps e_mask.
    """
    e_mask = embed[mask_id]
    cand = [(int(v), float(p)) for v, p in zip(ids, probs) if int(v) >= 0]
    z = sum(p for _, p in cand)
    if not cand or not z > 0.0:
        return e_mask.copy()
    p_tilde = [(v, p / z) for v, p in cand]                       # Eq. 6
    e_soft = np.zeros_like(e_mask)
    for v, pt in p_tilde:                                         # Eq. 7
        e_soft = e_soft + pt * embed[v]
    return (1.0 - alpha) * e_mask + alpha * e_soft                # Eq. 8


def build_step_input(embed: np.ndarray, mask_id: int, block_tokens: np.ndarray,
                     block_start: int, suffix_pos: Sequence[int], topk_ids: Optional[np.ndarray],
                     topk_prob: Optional[np.ndarray], alpha: float,
                     prefix_tokens: Optional[np.ndarray] = None):
    """Sparse step input X~_t = [P; B_t; R_t] and its position ids (Sec. 3.2).

    embed:        [V, hidden] float64 (bf16 values)
    block_tokens: [batch, B] token ids of the current block (mask_id where still masked)
    suffix_pos:   [R] retained suffix positions (ascending)
    topk_ids/prob:[batch, R, k] previous-step candidates (None: no prediction anywhere)
    prefix_tokens:[batch, n_prefix] prompt ids when the prompt is recomputed, else None

    Prompt and block rows are embedding lookups (a masked block row is e_mask,
    unmixed: the mixing of Eq. 8 applies to retained suffix positions only).
    Suffix rows follow Eqs. 6-8.  Every row is rounded to bf16 (round to nearest
    even) from the exact value.  Positions are the original absolute positions
    (prompt 0..n_prefix-1, block block_start..block_start+B-1, suffix R_t),
    which is what keeps the rotary encodings of the retained tokens intact.
    Returns (x [batch, n_prefix+B+R, hidden] float64, pos [n_prefix+B+R] int64).
    """
    block_tokens = np.asarray(block_tokens)
    batch, B = block_tokens.shape
    n_prefix = 0 if prefix_tokens is None else np.asarray(prefix_tokens).shape[1]
    R = len(suffix_pos)
    hidden = embed.shape[1]
    x = np.zeros((batch, n_prefix + B + R, hidden), dtype=np.float64)
    for bi in range(batch):
        row = 0
        for j in range(n_prefix):
            x[bi, row] = embed[int(prefix_tokens[bi, j])]
            row += 1
        for j in range(B):
            x[bi, row] = embed[int(block_tokens[bi, j])]
            row += 1
        for i in range(R):
            if topk_ids is None:
                x[bi, row] = embed[mask_id]
            else:
                x[bi, row] = bf16_round(soft_suffix_embedding(
                    embed, mask_id, topk_ids[bi, i], topk_prob[bi, i], alpha))
            row += 1
    pos = np.concatenate([np.arange(n_prefix), block_start + np.arange(B),
                          np.asarray(suffix_pos, dtype=np.int64)]).astype(np.int64)
    return x, pos


# --------------------------------------------------------------------------------------
# Rotary position encoding and bidirectional attention
# --------------------------------------------------------------------------------------


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotary position encoding (the rotate-half convention), in float64.

    x: [..., n, heads, d]; pos: [n].  Channel pairs (i, i + d/2), i < d/2, are
    rotated by the angle pos * theta**(-2i/d).  theta == 0 means no encoding.
    Reading: the paper states that retained tokens keep their original rotary
    encodings but not the convention; the convention of LLaDA/Dream-style
    rotary layers (pairs split by halves) is taken.
    """
    if theta == 0:
        return np.array(x, dtype=np.float64)
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    half = d // 2
    inv_freq = theta ** (-(2.0 * np.arange(half)) / d)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv_freq[None, :]     # [n, half]
    cos = np.cos(ang)[:, None, :]
    sin = np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)


def attention(q: np.ndarray, k_new: np.ndarray, v_new: np.ndarray, pos: np.ndarray,
              k_cache: Optional[np.ndarray], v_cache: Optional[np.ndarray],
              theta: float, scale: Optional[float] = None):
    """Bidirectional (non-causal) multi-head / grouped-query attention.

    q:              [batch, n, Hq, d]   queries of the sparse input rows
    k_new, v_new:   [batch, n, Hkv, d]  keys/values of the same rows
    pos:            [n]                 original positions of those rows
    k_cache/v_cache:[batch, nc, Hkv, d] prefix cache (keys already rotated), or None
    Query head h reads key/value head h // (Hq / Hkv).  No mask of any kind:
    every query sees every cached and new key (bidirectional DLM attention).
    Reading: the scale defaults to 1/sqrt(d).
    Returns (out [batch, n, Hq, d], lse [batch, n, Hq]) in float64; lse is the
    natural log of sum_k exp(scale * q.k).
    """
    q = np.asarray(q, dtype=np.float64)
    batch, n, hq, d = q.shape
    hkv = k_new.shape[2]
    grp = hq // hkv
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    qr = rope(q, pos, theta)
    kr = rope(k_new, pos, theta)
    if k_cache is not None and k_cache.shape[1] > 0:
        keys = np.concatenate([np.asarray(k_cache, dtype=np.float64), kr], axis=1)
        vals = np.concatenate([np.asarray(v_cache, dtype=np.float64),
                               np.asarray(v_new, dtype=np.float64)], axis=1)
    else:
        keys, vals = kr, np.asarray(v_new, dtype=np.float64)
    out = np.zeros((batch, n, hq, d), dtype=np.float64)
    lse = np.zeros((batch, n, hq), dtype=np.float64)
    for bi in range(batch):
        for h in range(hq):
            g = h // grp
            s = (qr[bi, :, h, :] @ keys[bi, :, g, :].T) * scale      # [n, nk]
            m = s.max(axis=1, keepdims=True)
            p = np.exp(s - m)
            l = p.sum(axis=1, keepdims=True)
            out[bi, :, h, :] = (p @ vals[bi, :, g, :]) / l
            lse[bi, :, h] = (m + np.log(l))[:, 0]
    return out, lse


def early_stop(tokens: np.ndarray, block_len: int, block_idx: int, eos_id: int, finished: np.ndarray):
    """Early termination after block block_idx is decoded (Sec. 3.2 "Early Termination").

    tokens: int [batch, gen_len], the generated region; finished: bool/uint8 [batch].
    A running sequence whose block holds eos_id stops: it is marked finished and
    every generated position after its first EOS becomes eos_id.  Readings: the
    paper halts generation without saying what the positions after EOS hold; they
    are filled with EOS, so no later block has a masked position left.  Returns
    (tokens, finished, n_active) as new arrays.
    """
    tokens = np.array(tokens, copy=True)
    finished = np.array(finished, dtype=np.uint8, copy=True)
    b0, b1 = block_idx * block_len, (block_idx + 1) * block_len
    for s in range(tokens.shape[0]):
        if finished[s]:
            continue
        hits = [p for p in range(b0, b1) if tokens[s, p] == eos_id]
        if hits:
            finished[s] = 1
            tokens[s, hits[0] + 1:] = eos_id
    return tokens, finished, int(np.sum(finished == 0))


def cache_append(k_cache: np.ndarray, v_cache: np.ndarray, k_new: np.ndarray, v_new: np.ndarray,
                 pos: np.ndarray, theta: float, start_row: int):
    """Prefix-cache append at a block boundary (prefix caching, Sec. 4.8 "+PC.").

    k_cache, v_cache: [batch, cache_rows, Hkv, d]; k_new, v_new: [batch, n, Hkv, d];
    pos: [n] original positions of the new rows (shared by the batch).
    Returns new (k_cache, v_cache) in float64 where rows start_row .. start_row+n-1
    hold rope(k_new, pos) and v_new, and every other row is unchanged.  Reading:
    the cache stores keys already rotated at their own positions, which is how
    ``attention`` consumes it.  Raises ValueError when the rows do not fit.
    """
    k_cache = np.array(k_cache, dtype=np.float64)
    v_cache = np.array(v_cache, dtype=np.float64)
    n = k_new.shape[1]
    if start_row < 0 or start_row + n > k_cache.shape[1]:
        raise ValueError("appended rows do not fit in the cache")
    k_cache[:, start_row:start_row + n] = rope(np.asarray(k_new, dtype=np.float64), pos, theta)
    v_cache[:, start_row:start_row + n] = np.asarray(v_new, dtype=np.float64)
    return k_cache, v_cache


# --------------------------------------------------------------------------------------
# Confidence-based unmasking
# --------------------------------------------------------------------------------------

MODE_THRESHOLD = 0
MODE_TOPK = 1
MODE_MARGIN = 2


def token_confidence(logits_row: np.ndarray):
    """Softmax over the vocabulary of one position, in float64.

    Returns (conf = largest probability, argmax = lowest id among the largest
    logits, p2 = second-largest probability, counting a tied maximum twice).
    """
    l = np.asarray(logits_row, dtype=np.float64)
    m = l.max()
    e = np.exp(l - m)
    p = e / e.sum()
    order = np.sort(p)
    conf = float(order[-1])
    p2 = float(order[-2]) if p.size > 1 else 0.0
    argmax = int(np.flatnonzero(l == m)[0])
    return conf, argmax, p2


def suffix_topk(logits: np.ndarray, k: int):
    """Top-k tokens of each row of logits [n, V] with their softmax probabilities.

    Sec. 3.2 "Soft Suffix Embedding Mixing": for a retained suffix position the
    next step takes the k most probable tokens under the current prediction
    p(v) = softmax(logits)(v) and their probabilities (which Eq. 6 then
    renormalizes within the set).  Returns ids int64 [n, k] in decreasing
    probability and probs float64 [n, k] (full-vocabulary probabilities).
    Readings: ties are broken by the lower token id; k > V is an error.
    """
    l = np.asarray(logits, dtype=np.float64)
    n, V = l.shape
    if not 1 <= k <= V:
        raise ValueError("k must be in [1, V]")
    ids = np.zeros((n, k), dtype=np.int64)
    probs = np.zeros((n, k), dtype=np.float64)
    for r in range(n):
        m = l[r].max()
        e = np.exp(l[r] - m)
        p = e / e.sum()
        order = np.lexsort((np.arange(V), -l[r]))[:k]      # by decreasing logit, then by id
        ids[r] = order
        probs[r] = p[order]
    return ids, probs


def unmask(logits: np.ndarray, masked: np.ndarray, mode: int = MODE_THRESHOLD,
           threshold: float = 0.9, topk: int = 1, min_commit: int = 1):
    """Which masked positions of the current block are decoded this step.

    logits: [batch, B, V]; masked: [batch, B] (nonzero = still [MASK]).
    * threshold ("Par.", Sec. 4.2): commit every masked position whose
      confidence is above the threshold (read as strictly greater);
    * top-k (Vanilla is k = 1, Sec. 4.2): commit the k masked positions of
      highest confidence;
    * margin (Sec. 4.6): commit masked positions whose top-1 minus top-2
      probability is above the threshold.
    Reading (threshold and margin): when fewer than min_commit positions pass,
    the highest-confidence remaining masked positions are added, so that each
    step decodes at least one token.  Ties between positions go to the lower
    position.  Unmasked positions report conf = 0, argmax = -1, p2 = 0, commit = 0.
    Returns conf, argmax, p2 (each [batch, B]) and commit [batch, B] (uint8).
    """
    logits = np.asarray(logits)
    batch, B, _ = logits.shape
    conf = np.zeros((batch, B), dtype=np.float64)
    p2 = np.zeros((batch, B), dtype=np.float64)
    arg = np.full((batch, B), -1, dtype=np.int64)
    commit = np.zeros((batch, B), dtype=np.uint8)
    for bi in range(batch):
        for j in range(B):
            if masked[bi, j]:
                conf[bi, j], arg[bi, j], p2[bi, j] = token_confidence(logits[bi, j])
        cand = [j for j in range(B) if masked[bi, j]]
        # rank by confidence descending, position ascending
        ranked = sorted(cand, key=lambda j: (-conf[bi, j], j))
        if mode == MODE_TOPK:
            for j in ranked[:topk]:
                commit[bi, j] = 1
            continue
        for j in cand:
            score = conf[bi, j] if mode == MODE_THRESHOLD else conf[bi, j] - p2[bi, j]
            if score > threshold:
                commit[bi, j] = 1
        short = min_commit - int(commit[bi].sum())
        for j in ranked:
            if short <= 0:
                break
            if not commit[bi, j]:
                commit[bi, j] = 1
                short -= 1
    return conf, arg, p2, commit
