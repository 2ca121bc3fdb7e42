"""ssm_unmask_noalloc: the unmask entry point for callers that cannot allocate
device memory (its scratch is the library's fixed device array).  Called through
the C ABI and compared with ssm_unmask on two calls in a row.  Collected last so
that a run stopping at the first failure has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _inputs(seed, batch, V, dtype):
    from paper_2608_23167_gb300 import workloads as W
    logits = W.draw_logits((batch, 32, V), dtype, 4.0, seed, planted_frac=0.25).cuda()
    g = torch.Generator().manual_seed(seed)
    masked = (torch.rand((batch, 32), generator=g) < 0.8).to(torch.uint8).cuda()
    return logits, masked


def _outputs(batch):
    return (torch.full((batch, 32), -1.0, device="cuda"), torch.full((batch, 32), -9, dtype=torch.int32, device="cuda"),
            torch.full((batch, 32), -1.0, device="cuda"), torch.full((batch, 32), 7, dtype=torch.uint8, device="cuda"))


def test_unmask_noalloc_matches_workspace_version_twice():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2608_23167_gb300 import build_lib, ssm
    build_lib.build()
    lib = ssm.lib()
    stream = torch.cuda.current_stream().cuda_stream
    for call, (seed, batch, V, dtype, mode) in enumerate([(1, 8, 126464, "bf16", ssm.SSM_COMMIT_THRESHOLD),
                                                          (2, 3, 4096, "f32", ssm.SSM_COMMIT_MARGIN)]):
        logits, masked = _inputs(seed, batch, V, dtype)
        code = ssm.SSM_DTYPE_BF16 if dtype == "bf16" else ssm.SSM_DTYPE_F32
        c0, a0, p0, k0 = _outputs(batch)
        ssm.ssm_unmask(logits, masked, c0, a0, k0, p2=p0, mode=mode, threshold=0.5)
        c1, a1, p1, k1 = _outputs(batch)
        st = lib.ssm_unmask_noalloc(logits.data_ptr(), code, batch, 32, V, masked.data_ptr(), mode,
                                    ctypes.c_float(0.5), 1, 1, c1.data_ptr(), a1.data_ptr(), p1.data_ptr(),
                                    k1.data_ptr(), stream)
        assert st == 0, f"call {call}: status {st}"
        torch.cuda.synchronize()
        assert ssm.ssm_get_device_error() == 0
        assert torch.equal(a1, a0) and torch.equal(k1, k0), f"call {call}"
        assert np.allclose(c1.cpu().numpy(), c0.cpu().numpy(), rtol=1e-5, atol=0)
        assert np.allclose(p1.cpu().numpy(), p0.cpu().numpy(), rtol=1e-5, atol=0)


def test_unmask_noalloc_rejects_sizes_beyond_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2608_23167_gb300 import build_lib, ssm
    build_lib.build()
    lib = ssm.lib()
    fake = 1 << 20
    # with this many positions every streaming range covers more than a row of a 126464-entry
    # bf16 vocabulary, so a row meets at most two ranges (two 16-byte partials): 65536
    # positions fill 2 MiB exactly, one sequence more does not fit (and nothing is enqueued)
    assert lib.ssm_unmask_workspace_size(2048, 32, 126464, 0) == 2 << 20
    assert lib.ssm_unmask_noalloc(fake, 0, 2049, 32, 126464, fake, 0, ctypes.c_float(0.9), 1, 1, fake, fake,
                                  fake, fake, None) == 3
