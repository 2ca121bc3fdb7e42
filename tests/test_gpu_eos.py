"""GPU parity: early termination after a decoded block (Sec. 3.2 "Early Termination")
against the oracle.  Bar: tokens, finished flags and the running count bit-exact."""
import numpy as np
import pytest
import torch

from oracle import ssm_oracle as O
from tests.gpu_helpers import check_device_error, cuda_or_skip

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return cuda_or_skip()


@pytest.mark.parametrize("batch,gen,B,b,p_eos", [
    (64, 2048, 32, 0, 0.01),      # long generation, first block, sparse EOS
    (8, 256, 32, 7, 0.05),        # last block: nothing after it to fill
    (5, 96, 32, 1, 0.0),          # no EOS anywhere
    (300, 1024, 32, 13, 0.02),    # many sequences, a middle block
])
def test_early_stop_parity(dev, batch, gen, B, b, p_eos):
    from paper_2608_23167_gb300 import ssm
    g = torch.Generator().manual_seed(batch + gen + b)
    eos = 126081
    toks = torch.randint(0, 126464, (batch, gen), generator=g, dtype=torch.int32)
    toks[toks == eos] = 0
    toks[torch.rand((batch, gen), generator=g) < p_eos] = eos
    fin = (torch.rand(batch, generator=g) < 0.2).to(torch.uint8)
    t_d, f_d = toks.to(dev), fin.to(dev)
    n_d = torch.full((1,), -5, dtype=torch.int32, device=dev)
    ssm.ssm_early_stop(t_d, B, b, eos, f_d, n_d)
    torch.cuda.synchronize()
    check_device_error()
    rt, rf, rn = O.early_stop(toks.numpy(), B, b, eos, fin.numpy())
    assert np.array_equal(t_d.cpu().numpy(), rt)
    assert np.array_equal(f_d.cpu().numpy(), rf)
    assert int(n_d.item()) == rn


def test_early_stop_errors(dev):
    from paper_2608_23167_gb300 import ssm
    toks = torch.zeros((2, 100), dtype=torch.int32, device=dev)
    fin = torch.zeros(2, dtype=torch.uint8, device=dev)
    with pytest.raises(ssm.SSMError) as e:
        ssm.ssm_early_stop(toks, 32, 0, 5, fin)          # 100 is not a multiple of 32
    assert e.value.status == ssm.SSM_ERR_SHAPE
    toks = torch.zeros((2, 96), dtype=torch.int32, device=dev)
    with pytest.raises(ssm.SSMError) as e:
        ssm.ssm_early_stop(toks, 32, 3, 5, fin)          # block 3 of 3 does not exist
    assert e.value.status == ssm.SSM_ERR_INVALID_ARG
