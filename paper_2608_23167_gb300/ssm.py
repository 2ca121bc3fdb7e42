"""Python binding of libssm (include/ssm.h): argument marshalling only.

Each function takes torch tensors that already live on the current CUDA
device, passes their data pointers and the current stream to the C entry point
of the same name, and raises SSMError on a non-OK status.  Every step of the
path runs in the library's CUDA kernels; there is no fallback: if libssm.so
cannot be loaded the import of this module's functions fails loudly.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_PKG, "libssm.so")

SSM_DTYPE_BF16 = 0
SSM_DTYPE_F32 = 1
SSM_COMMIT_THRESHOLD = 0
SSM_COMMIT_TOPK = 1
SSM_COMMIT_MARGIN = 2

STATUS = {0: "ok", 1: "invalid argument", 2: "inconsistent shapes", 3: "capacity", 4: "CUDA error",
          5: "device wait timed out", 6: "unsupported", 7: "device input out of range"}
SSM_OK, SSM_ERR_INVALID_ARG, SSM_ERR_SHAPE, SSM_ERR_CAPACITY = 0, 1, 2, 3
SSM_ERR_CUDA, SSM_ERR_TIMEOUT, SSM_ERR_UNSUPPORTED, SSM_ERR_DEVICE_INPUT = 4, 5, 6, 7


class SSMError(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn}: {STATUS.get(status, status)} (status {status})")
        self.status = status


class SuffixCfg(ctypes.Structure):
    _fields_ = [("prompt_len", ctypes.c_int32), ("gen_len", ctypes.c_int32),
                ("block_len", ctypes.c_int32), ("block_idx", ctypes.c_int32),
                ("local_budget", ctypes.c_int32), ("middle_budget", ctypes.c_int32),
                ("tail_budget", ctypes.c_int32)]


# ctypes mirrors of the packed problem descriptors (layout must match ssm.h)
STEP_PROBLEM_DTYPE = [("block_tok_off", "i8"), ("prefix_tok_off", "i8"), ("suffix_off", "i8"),
                      ("out_row", "i8"), ("n_prefix", "i4"), ("n_suffix", "i4"),
                      ("block_start", "i4"), ("reserved", "i4")]
ATTN_PROBLEM_DTYPE = [("new_row", "i8"), ("cache_row", "i8"), ("n_new", "i4"), ("n_cache", "i4")]

_lib = None


def lib() -> ctypes.CDLL:
    """Load libssm.so (built by __graft_entry__.build() / build_lib.build())."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"{_LIB_PATH} is missing: build it with paper_2608_23167_gb300.build_lib.build()")
        L = ctypes.CDLL(_LIB_PATH)
        vp, i32, i64, f32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
        P = ctypes.POINTER
        sig = {
            "ssm_status_str": (ctypes.c_char_p, [ctypes.c_int]),
            "ssm_version": (ctypes.c_char_p, []),
            "ssm_get_device_error": (ctypes.c_int, [vp]),
            "ssm_set_wait_limit_ns": (ctypes.c_int, [ctypes.c_uint64]),
            "ssm_suffix_count": (ctypes.c_int, [P(SuffixCfg), P(i32), P(i32), P(i32)]),
            "ssm_select_suffix": (ctypes.c_int, [P(SuffixCfg), vp, i32, P(i32), vp]),
            "ssm_select_suffix_batch": (ctypes.c_int, [P(SuffixCfg), i32, vp, i64, P(i64), vp]),
            "ssm_build_step_input": (ctypes.c_int, [vp, vp, i32, i32, i32, i32, vp, i32, vp, i64, i32, i32,
                                                    vp, vp, i32, f32, vp, vp, vp]),
            "ssm_build_step_input_varlen": (ctypes.c_int, [vp, i32, i32, i32, vp, vp, vp, vp, i64, i32, i32,
                                                           vp, vp, i32, f32, vp, vp, vp]),
            "ssm_select_build_step_input_varlen": (ctypes.c_int, [vp, vp, i32, i32, i32, vp, vp, vp, vp, i64, i32,
                                                                  i32, vp, vp, i32, f32, vp, vp, vp]),
            "ssm_attention_workspace_size": (sz, [i64, i32, i32, i32]),
            "ssm_attention": (ctypes.c_int, [vp, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, i32, f32, f32,
                                             vp, vp, vp, sz, vp]),
            "ssm_attention_varlen": (ctypes.c_int, [vp, vp, vp, vp, vp, vp, i64, i64, vp, i32, i32, i32, i32,
                                                    i32, i32, f32, f32, vp, vp, vp, sz, vp]),
            "ssm_attention_varlen_rotate": (ctypes.c_int, [vp, vp, vp, vp, vp, vp, i64, i64, vp, i32, i32, i32,
                                                           i32, i32, i32, f32, f32, vp, vp, vp, sz, vp]),
            "ssm_attention_varlen_core": (ctypes.c_int, [vp, vp, vp, vp, vp, vp, i64, i64, vp, i32, i32, i32,
                                                         i32, i32, i32, f32, f32, vp, vp, vp, sz, vp]),
            "ssm_unmask_workspace_size": (sz, [i32, i32, i64, ctypes.c_int]),
            "ssm_unmask": (ctypes.c_int, [vp, ctypes.c_int, i32, i32, i64, vp, ctypes.c_int, f32, i32, i32,
                                          vp, vp, vp, vp, vp, sz, vp]),
            "ssm_unmask_noalloc": (ctypes.c_int, [vp, ctypes.c_int, i32, i32, i64, vp, ctypes.c_int, f32, i32,
                                                  i32, vp, vp, vp, vp, vp]),
            "ssm_cache_append": (ctypes.c_int, [vp, vp, vp, i32, i32, i32, i32, f32, vp, vp, i64, i64, vp]),
            "ssm_suffix_topk": (ctypes.c_int, [vp, ctypes.c_int, i64, i64, i32, vp, vp, vp]),
            "ssm_unmask_topk": (ctypes.c_int, [vp, ctypes.c_int, i32, i32, i64, vp, ctypes.c_int, f32, i32, i32,
                                               vp, vp, vp, vp, vp, i64, i32, vp, vp, vp, sz, vp]),
            "ssm_early_stop": (ctypes.c_int, [vp, i32, i32, i32, i32, i32, vp, vp, vp]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def exported_symbols() -> Sequence[str]:
    return ["ssm_status_str", "ssm_version", "ssm_get_device_error", "ssm_set_wait_limit_ns",
            "ssm_suffix_count", "ssm_select_suffix", "ssm_select_suffix_batch", "ssm_build_step_input",
            "ssm_build_step_input_varlen", "ssm_select_build_step_input_varlen", "ssm_attention_workspace_size", "ssm_attention",
            "ssm_attention_varlen", "ssm_attention_varlen_rotate", "ssm_attention_varlen_core",
            "ssm_unmask_workspace_size", "ssm_unmask", "ssm_unmask_topk", "ssm_unmask_noalloc",
            "ssm_cache_append", "ssm_suffix_topk", "ssm_early_stop"]


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libssm takes device tensors")
    if not t.is_contiguous():
        raise ValueError("libssm takes contiguous tensors")
    return t.data_ptr()


def _stream(stream=None) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _check(fn: str, status: int):
    if status != 0:
        raise SSMError(fn, status)


def _cfg(prompt_len, gen_len, block_len, block_idx, local_budget, middle_budget, tail_budget) -> SuffixCfg:
    return SuffixCfg(prompt_len, gen_len, block_len, block_idx, local_budget, middle_budget, tail_budget)


# ------------------------------------------------------------------------------ library-wide


def ssm_get_device_error(stream=None) -> int:
    return lib().ssm_get_device_error(_stream(stream))


def ssm_set_wait_limit_ns(ns: int) -> None:
    _check("ssm_set_wait_limit_ns", lib().ssm_set_wait_limit_ns(int(ns)))


# ------------------------------------------------------------------------------ selector


def ssm_suffix_count(prompt_len, gen_len, block_len, block_idx, local_budget, middle_budget, tail_budget):
    c = _cfg(prompt_len, gen_len, block_len, block_idx, local_budget, middle_budget, tail_budget)
    a, b, d = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
    _check("ssm_suffix_count", lib().ssm_suffix_count(ctypes.byref(c), ctypes.byref(a), ctypes.byref(b),
                                                      ctypes.byref(d)))
    return a.value, b.value, d.value


def ssm_select_suffix(positions: torch.Tensor, prompt_len, gen_len, block_len, block_idx, local_budget,
                      middle_budget, tail_budget, stream=None) -> int:
    """Writes R_t into `positions` (int32, device) and returns |R_t|."""
    assert positions.dtype == torch.int32
    c = _cfg(prompt_len, gen_len, block_len, block_idx, local_budget, middle_budget, tail_budget)
    n = ctypes.c_int32()
    _check("ssm_select_suffix", lib().ssm_select_suffix(ctypes.byref(c), _ptr(positions), positions.numel(),
                                                        ctypes.byref(n), _stream(stream)))
    return n.value


def ssm_select_suffix_batch(positions: torch.Tensor, cfgs, stream=None):
    """cfgs: list of 7-tuples (prompt, gen, block, block_idx, L, M, T).  Returns offsets (n + 1 ints)."""
    assert positions.dtype == torch.int32
    n = len(cfgs)
    arr = (SuffixCfg * max(n, 1))(*[_cfg(*c) for c in cfgs])
    off = (ctypes.c_int64 * (n + 1))()
    _check("ssm_select_suffix_batch", lib().ssm_select_suffix_batch(arr, n, _ptr(positions), positions.numel(),
                                                                    off, _stream(stream)))
    return list(off)


# ------------------------------------------------------------------------------ step input


def ssm_build_step_input(block_tokens, suffix_pos, embed, mask_id: int, prev_topk_ids, prev_topk_prob,
                         alpha: float, x_out, pos_out=None, block_start: int = 0, prefix_tokens=None,
                         stream=None):
    batch, block_len = block_tokens.shape
    n_prefix = 0 if prefix_tokens is None else prefix_tokens.shape[1]
    n_suffix = suffix_pos.numel()
    vocab, hidden = embed.shape
    k = 0 if prev_topk_ids is None else prev_topk_ids.shape[-1]
    assert embed.dtype == torch.bfloat16 and x_out.dtype == torch.bfloat16
    _check("ssm_build_step_input", lib().ssm_build_step_input(
        _ptr(block_tokens), _ptr(prefix_tokens), batch, n_prefix, block_len, block_start, _ptr(suffix_pos),
        n_suffix, _ptr(embed), vocab, hidden, mask_id, _ptr(prev_topk_ids), _ptr(prev_topk_prob), k,
        float(alpha), _ptr(x_out), _ptr(pos_out), _stream(stream)))


def ssm_build_step_input_varlen(problems, n_problems: int, max_rows: int, block_len: int, block_tokens,
                                suffix_pos, embed, mask_id: int, prev_topk_ids, prev_topk_prob, k: int,
                                alpha: float, x_out, pos_out=None, prefix_tokens=None, stream=None):
    """problems: device int64 tensor holding n_problems packed ssm_step_problem records."""
    vocab, hidden = embed.shape
    _check("ssm_build_step_input_varlen", lib().ssm_build_step_input_varlen(
        _ptr(problems), n_problems, max_rows, block_len, _ptr(block_tokens), _ptr(prefix_tokens),
        _ptr(suffix_pos), _ptr(embed), vocab, hidden, mask_id, _ptr(prev_topk_ids), _ptr(prev_topk_prob), k,
        float(alpha), _ptr(x_out), _ptr(pos_out), _stream(stream)))


def step_problems_tensor(rows, device) -> torch.Tensor:
    """Packs (block_tok_off, prefix_tok_off, suffix_off, out_row, n_prefix, n_suffix, block_start)
    tuples into the ssm_step_problem layout (40 bytes each) on `device`."""
    import numpy as np
    a = np.zeros(len(rows), dtype=np.dtype(STEP_PROBLEM_DTYPE))
    for i, r in enumerate(rows):
        a[i] = tuple(r) + (0,)
    return torch.from_numpy(a.view(np.int64).copy()).to(device)


def suffix_cfgs_tensor(cfgs, device) -> torch.Tensor:
    """Packs (prompt, gen, block, block_idx, L, M, T) tuples into ssm_suffix_cfg records (28 bytes)."""
    return torch.tensor([list(c) for c in cfgs], dtype=torch.int32).reshape(-1, 7).to(device)


def ssm_select_build_step_input_varlen(problems, cfgs, n_problems: int, max_rows: int, block_len: int, block_tokens,
                                       embed, mask_id: int, prev_topk_ids, prev_topk_prob, k: int, alpha: float,
                                       x_out, pos_out=None, suffix_pos_out=None, prefix_tokens=None, stream=None):
    """problems: device ssm_step_problem table; cfgs: device ssm_suffix_cfg table (suffix_cfgs_tensor)."""
    vocab, hidden = embed.shape
    _check("ssm_select_build_step_input_varlen", lib().ssm_select_build_step_input_varlen(
        _ptr(problems), _ptr(cfgs), n_problems, max_rows, block_len, _ptr(block_tokens), _ptr(prefix_tokens),
        _ptr(suffix_pos_out), _ptr(embed), vocab, hidden, mask_id, _ptr(prev_topk_ids), _ptr(prev_topk_prob), k,
        float(alpha), _ptr(x_out), _ptr(pos_out), _stream(stream)))


# ------------------------------------------------------------------------------ attention


def ssm_attention_workspace_size(total_new_rows: int, h_q: int, h_kv: int, head_dim: int) -> int:
    return int(lib().ssm_attention_workspace_size(total_new_rows, h_q, h_kv, head_dim))


def ssm_attention(q, k_new, v_new, pos, k_cache, v_cache, out, rope_theta: float, scale: Optional[float] = None,
                  lse=None, workspace=None, stream=None):
    batch, n_new, h_q, d = q.shape
    h_kv = k_new.shape[2]
    n_cache = 0 if k_cache is None else k_cache.shape[1]
    if scale is None:
        scale = d ** -0.5
    need = ssm_attention_workspace_size(batch * n_new, h_q, h_kv, d)
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=q.device)
    _check("ssm_attention", lib().ssm_attention(
        _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(pos), _ptr(k_cache), _ptr(v_cache), batch, n_new, n_cache, h_q,
        h_kv, d, float(rope_theta), float(scale), _ptr(out), _ptr(lse), _ptr(workspace), workspace.numel(),
        _stream(stream)))


def attn_problems_tensor(rows, device) -> torch.Tensor:
    """Packs (new_row, cache_row, n_new, n_cache) tuples into ssm_attn_problem records (24 bytes)."""
    import numpy as np
    a = np.zeros(len(rows), dtype=np.dtype(ATTN_PROBLEM_DTYPE))
    for i, r in enumerate(rows):
        a[i] = tuple(r)
    return torch.from_numpy(a.view(np.uint8).copy()).to(device)


def _attention_varlen(fn: str, q, k_new, v_new, pos, k_cache, v_cache, problems, n_problems, max_n_new,
                      max_n_cache, out, rope_theta, scale, lse, workspace, stream):
    total_new, h_q, d = q.shape
    h_kv = k_new.shape[1]
    total_cache = 0 if k_cache is None else k_cache.shape[0]
    if scale is None:
        scale = d ** -0.5
    need = ssm_attention_workspace_size(total_new, h_q, h_kv, d)
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=q.device)
    _check(fn, getattr(lib(), fn)(
        _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(pos), _ptr(k_cache), _ptr(v_cache), total_new, total_cache,
        _ptr(problems), n_problems, max_n_new, max_n_cache, h_q, h_kv, d, float(rope_theta), float(scale),
        _ptr(out), _ptr(lse), _ptr(workspace), workspace.numel(), _stream(stream)))


def ssm_attention_varlen(q, k_new, v_new, pos, k_cache, v_cache, problems, n_problems: int, max_n_new: int,
                         max_n_cache: int, out, rope_theta: float, scale: Optional[float] = None, lse=None,
                         workspace=None, stream=None):
    _attention_varlen("ssm_attention_varlen", q, k_new, v_new, pos, k_cache, v_cache, problems, n_problems,
                      max_n_new, max_n_cache, out, rope_theta, scale, lse, workspace, stream)


def ssm_attention_varlen_rotate(q, k_new, v_new, pos, k_cache, v_cache, problems, n_problems: int,
                                max_n_new: int, max_n_cache: int, out, rope_theta: float,
                                scale: Optional[float] = None, lse=None, workspace=None, stream=None):
    """The RoPE pre-pass of ssm_attention_varlen alone (writes the workspace)."""
    _attention_varlen("ssm_attention_varlen_rotate", q, k_new, v_new, pos, k_cache, v_cache, problems,
                      n_problems, max_n_new, max_n_cache, out, rope_theta, scale, lse, workspace, stream)


def ssm_attention_varlen_core(q, k_new, v_new, pos, k_cache, v_cache, problems, n_problems: int,
                              max_n_new: int, max_n_cache: int, out, rope_theta: float,
                              scale: Optional[float] = None, lse=None, workspace=None, stream=None):
    """The attention forward of ssm_attention_varlen alone, from a workspace the rotate call wrote."""
    _attention_varlen("ssm_attention_varlen_core", q, k_new, v_new, pos, k_cache, v_cache, problems,
                      n_problems, max_n_new, max_n_cache, out, rope_theta, scale, lse, workspace, stream)


# ------------------------------------------------------------------------------ suffix top-k


def ssm_suffix_topk(logits, k: int, ids, probs, stream=None):
    """logits: bf16/fp32 [n_rows, vocab]; ids int32 [n_rows, k]; probs fp32 [n_rows, k]."""
    n_rows, vocab = logits.shape
    _check("ssm_suffix_topk", lib().ssm_suffix_topk(
        _ptr(logits), _dtype_code(logits), n_rows, vocab, int(k), _ptr(ids), _ptr(probs), _stream(stream)))


# ------------------------------------------------------------------------------ early termination


def ssm_early_stop(tokens, block_len: int, block_idx: int, eos_id: int, finished, n_active=None, stream=None):
    """tokens: int32 [batch, gen_len] (in place); finished: uint8 [batch] (in place); n_active: int32 [1]."""
    batch, gen_len = tokens.shape
    _check("ssm_early_stop", lib().ssm_early_stop(
        _ptr(tokens), batch, gen_len, int(block_len), int(block_idx), int(eos_id), _ptr(finished), _ptr(n_active),
        _stream(stream)))


# ------------------------------------------------------------------------------ prefix-cache append


def ssm_cache_append(k_new, v_new, pos, k_cache, v_cache, start_row: int, rope_theta: float, stream=None):
    """k_new, v_new: bf16 [batch, n_rows, h_kv, d]; k_cache, v_cache: bf16 [batch, cache_rows, h_kv, d],
    written in place at rows start_row .. start_row + n_rows - 1."""
    batch, n_rows, h_kv, d = k_new.shape
    _check("ssm_cache_append", lib().ssm_cache_append(
        _ptr(k_new), _ptr(v_new), _ptr(pos), batch, n_rows, h_kv, d, float(rope_theta), _ptr(k_cache),
        _ptr(v_cache), k_cache.shape[1], int(start_row), _stream(stream)))


# ------------------------------------------------------------------------------ unmask


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return SSM_DTYPE_BF16
    if t.dtype == torch.float32:
        return SSM_DTYPE_F32
    raise ValueError(f"unsupported logits dtype {t.dtype}")


def ssm_unmask_workspace_size(batch: int, block_len: int, vocab: int, dtype: torch.dtype) -> int:
    code = SSM_DTYPE_BF16 if dtype == torch.bfloat16 else SSM_DTYPE_F32
    return int(lib().ssm_unmask_workspace_size(batch, block_len, vocab, code))


def ssm_unmask(logits, masked, conf, argmax, commit, p2=None, mode: int = SSM_COMMIT_THRESHOLD,
               threshold: float = 0.9, topk: int = 1, min_commit: int = 1, workspace=None, stream=None):
    batch, block_len, vocab = logits.shape
    need = ssm_unmask_workspace_size(batch, block_len, vocab, logits.dtype)
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=logits.device)
    _check("ssm_unmask", lib().ssm_unmask(
        _ptr(logits), _dtype_code(logits), batch, block_len, vocab, _ptr(masked), mode, float(threshold), topk,
        min_commit, _ptr(conf), _ptr(argmax), _ptr(p2), _ptr(commit), _ptr(workspace), workspace.numel(),
        _stream(stream)))


def ssm_unmask_topk(logits, masked, conf, argmax, commit, suffix_logits, k: int, ids, probs, p2=None,
                    mode: int = SSM_COMMIT_THRESHOLD, threshold: float = 0.9, topk: int = 1, min_commit: int = 1,
                    workspace=None, stream=None):
    """ssm_unmask of the block rows and ssm_suffix_topk of suffix_logits [n_rows, vocab] in one pass."""
    batch, block_len, vocab = logits.shape
    n_suffix = suffix_logits.shape[0] if suffix_logits is not None else 0
    need = ssm_unmask_workspace_size(batch, block_len, vocab, logits.dtype)
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=logits.device)
    _check("ssm_unmask_topk", lib().ssm_unmask_topk(
        _ptr(logits), _dtype_code(logits), batch, block_len, vocab, _ptr(masked), mode, float(threshold), topk,
        min_commit, _ptr(conf), _ptr(argmax), _ptr(p2), _ptr(commit), _ptr(suffix_logits), n_suffix, int(k),
        _ptr(ids), _ptr(probs), _ptr(workspace), workspace.numel(), _stream(stream)))


def ssm_unmask_noalloc(logits, masked, conf, argmax, commit, p2=None, mode: int = SSM_COMMIT_THRESHOLD,
                       threshold: float = 0.9, topk: int = 1, min_commit: int = 1, stream=None):
    """ssm_unmask without a workspace: for callers that cannot allocate device memory
    (the library's fixed scratch array is used; concurrent calls race)."""
    batch, block_len, vocab = logits.shape
    _check("ssm_unmask_noalloc", lib().ssm_unmask_noalloc(
        _ptr(logits), _dtype_code(logits), batch, block_len, vocab, _ptr(masked), mode, float(threshold), topk,
        min_commit, _ptr(conf), _ptr(argmax), _ptr(p2), _ptr(commit), _stream(stream)))
