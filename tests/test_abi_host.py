"""Host-side checks of the C ABI (no GPU needed): the library loads, exports
every entry point that include/ssm.h declares, and its pure host logic and
argument validation behave as documented."""
import ctypes
import os
import re

import pytest

from oracle import ssm_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_23167_gb300 import build_lib, ssm
    build_lib.build()
    return ssm.lib()


def _declared_functions():
    with open(os.path.join(ROOT, "include", "ssm.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ssm_[a-z_0-9]+)\s*\(", text)))


def test_library_exports_every_declared_symbol(lib):
    names = _declared_functions()
    assert len(names) >= 14
    for n in names:
        assert hasattr(lib, n), n
    from paper_2608_23167_gb300 import ssm
    assert sorted(ssm.exported_symbols()) == names


def test_status_strings_and_version(lib):
    assert lib.ssm_status_str(0) == b"ok"
    assert lib.ssm_status_str(3).startswith(b"output or workspace")
    assert b"sm_103a" in lib.ssm_version()


def test_suffix_count_matches_oracle(lib):
    from paper_2608_23167_gb300 import ssm
    for (P, G, B, L, M, T) in [(64, 256, 32, 32, 8, 4), (512, 1024, 32, 64, 32, 8), (1024, 2048, 32, 64, 64, 16),
                               (0, 320, 32, 32, 3, 2), (16, 256, 32, 48, 1000, 2), (5, 96, 8, 12, 1, 9)]:
        for b in range(G // B):
            r, nl, nm, nt = O.select_suffix(P, G, B, b, L, M, T)
            assert ssm.ssm_suffix_count(P, G, B, b, L, M, T) == (nl, nm, nt)


def test_suffix_count_closed_form_grid(lib):
    """The region sizes in closed form (which the gather that selects as it builds also uses to
    place every retained row) against the oracle's set construction over a grid of layouts:
    budgets not multiples of the block, a local region reaching into the tail block, more middle
    blocks than the middle budget, T = 0 / 1 / 2 / 3 / >= B."""
    from paper_2608_23167_gb300 import ssm
    n = 0
    for B in (4, 8, 32):
        for G in (B, 2 * B, 5 * B, 12 * B):
            for L in (0, 1, B // 2, B, B + 3, 3 * B):
                for M in (0, 1, 2, 5, 100):
                    for T in (0, 1, 2, 3, B - 1, B, B + 2):
                        for b in range(0, G // B, max(1, (G // B) // 4)):
                            r, nl, nm, nt = O.select_suffix(7, G, B, b, L, M, T)
                            assert ssm.ssm_suffix_count(7, G, B, b, L, M, T) == (nl, nm, nt), (G, B, b, L, M, T)
                            n += 1
    assert n > 2000


def test_argument_validation_without_device(lib):
    from paper_2608_23167_gb300 import ssm
    cfg = ssm.SuffixCfg(0, 100, 32, 0, 32, 8, 4)          # G % B != 0
    n = ctypes.c_int32()
    assert lib.ssm_select_suffix(ctypes.byref(cfg), None, 0, ctypes.byref(n), None) == 2
    cfg = ssm.SuffixCfg(0, 256, 32, 8, 32, 8, 4)          # block index out of range
    assert lib.ssm_select_suffix(ctypes.byref(cfg), None, 0, ctypes.byref(n), None) == 1
    cfg = ssm.SuffixCfg(64, 256, 32, 0, 32, 8, 4)         # capacity too small: count reported
    assert lib.ssm_select_suffix(ctypes.byref(cfg), None, 10, ctypes.byref(n), None) == 3
    assert n.value == 41
    # attention: h_q % h_kv != 0, unsupported head_dim
    fake = 1 << 20
    assert lib.ssm_attention(fake, fake, fake, fake, None, None, 1, 8, 0, 6, 4, 128, 0.0, 0.1, fake, None,
                             fake, 1 << 30, None) == 2
    assert lib.ssm_attention(fake, fake, fake, fake, None, None, 1, 8, 0, 4, 4, 96, 0.0, 0.1, fake, None,
                             fake, 1 << 30, None) == 6
    assert lib.ssm_attention(fake, fake, fake, fake, None, None, 1, 8, 0, 4, 4, 128, 0.0, 0.1, fake, None,
                             fake, 16, None) == 3
    # unmask: bad dtype, block too long, workspace too small
    assert lib.ssm_unmask(fake, 7, 1, 32, 4096, fake, 0, 0.9, 1, 1, fake, fake, fake, fake, fake, 1 << 20,
                          None) == 6
    assert lib.ssm_unmask(fake, 0, 1, 2048, 4096, fake, 0, 0.9, 1, 1, fake, fake, fake, fake, fake, 1 << 20,
                          None) == 6
    assert lib.ssm_unmask(fake, 0, 8, 32, 126464, fake, 0, 0.9, 1, 1, fake, fake, fake, fake, fake, 256,
                          None) == 3
    # build_step_input: alpha outside [0, 1], hidden not a multiple of 8
    assert lib.ssm_build_step_input(fake, None, 1, 0, 32, 0, fake, 4, fake, 100, 64, 99, fake, fake, 5, 1.5,
                                    fake, None, None) == 1
    assert lib.ssm_build_step_input(fake, None, 1, 0, 32, 0, fake, 4, fake, 100, 60, 99, fake, fake, 5, 0.4,
                                    fake, None, None) == 6
    # cache append: rows past the cache end, unsupported head_dim, negative start; zero rows is a no-op
    assert lib.ssm_cache_append(fake, fake, fake, 1, 32, 4, 128, 1e4, fake, fake, 64, 40, None) == 3
    assert lib.ssm_cache_append(fake, fake, fake, 1, 32, 4, 96, 1e4, fake, fake, 64, 0, None) == 6
    assert lib.ssm_cache_append(fake, fake, fake, 1, 32, 4, 128, 1e4, fake, fake, 64, -1, None) == 1
    assert lib.ssm_cache_append(None, None, None, 1, 0, 4, 128, 1e4, None, None, 64, 64, None) == 0


def test_workspace_sizes(lib):
    from paper_2608_23167_gb300 import ssm
    import torch
    # rotated queries and keys, then the unit plan (32-byte header, 32 bytes per packed unit of
    # 256 query rows of a kv head) and the problem index of every new row, each region 256-aligned
    up = lambda x: (x + 255) // 256 * 256
    rows, pairs = 101 * 8, (101 * 8 + 255) // 256
    assert ssm.ssm_attention_workspace_size(rows, 32, 32, 128) == (
        2 * rows * 32 * 128 * 2 + up(32 + 32 * pairs) + up(16 * rows))
    rows, pairs = 8854, (8854 * 7 + 255) // 256    # GQA: 7 query heads per kv head pack 7 rows per query
    assert ssm.ssm_attention_workspace_size(rows, 28, 4, 128) == (
        up(rows * 28 * 256) + up(rows * 4 * 256) + up(32 + 32 * pairs) + up(16 * rows))
    # 126464 bf16 entries are 16 stages of 8192; sized at the grid cap of 768 CTAs, each taking
    # per = ceil(stages / 768) consecutive stages, a row meets at most ceil(15 / per) + 1 CTA
    # ranges (at most 16), one 16-byte partial each
    ws = ssm.ssm_unmask_workspace_size(8, 32, 126464, torch.bfloat16)
    assert ws == 8 * 32 * 4 * 16   # 4096 stages: per = 6, four ranges per row
    assert ssm.ssm_unmask_workspace_size(64, 32, 126464, torch.bfloat16) == 64 * 32 * 2 * 16   # per = 43: two
    assert ssm.ssm_unmask_workspace_size(1, 4, 126464, torch.bfloat16) == 4 * 16 * 16      # per = 1: sixteen
    # fp32 rows of 4096 entries are one stage: one partial per row
    assert ssm.ssm_unmask_workspace_size(1, 32, 4096, torch.float32) == 32 * 16


def test_attention_digest_covers_its_includes():
    """The bench trusts a recorded DRAM-traffic figure only while its source digest matches the
    attention forward's sources; every local header attention.cu includes (transitively) must be
    part of that digest, or a change to it would leave a stale figure in use."""
    import os
    import re
    from paper_2608_23167_gb300 import build_lib
    seen, todo = set(), ["attention.cu"]
    while todo:
        name = todo.pop()
        if name in seen:
            continue
        seen.add(name)
        with open(build_lib.source_path(name)) as f:
            for inc in re.findall(r'^#include "([^"]+)"', f.read(), flags=re.M):
                # every quoted include is a local file of the package or of include/: fail on any
                # the digest could not read
                assert os.path.exists(build_lib.source_path(inc)), f"{name} includes unknown {inc}"
                todo.append(inc)
    assert seen <= set(build_lib.ATTENTION_SOURCES), seen - set(build_lib.ATTENTION_SOURCES)
