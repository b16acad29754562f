"""Host-side checks of the torch.optim wrapper (no GPU needed)."""
import pytest
import torch

from paper_2606_13894_gb300.optim import Gefen


def test_cpu_parameters_are_refused():
    with pytest.raises(ValueError, match="CUDA fp32"):
        Gefen([torch.nn.Parameter(torch.zeros(4))])


def test_argument_checks():
    p = [torch.nn.Parameter(torch.zeros(4))]
    with pytest.raises(ValueError):
        Gefen(p, betas=(1.0, 0.9))
    with pytest.raises(ValueError):
        Gefen(p, levels=1)
    with pytest.raises(ValueError):
        Gefen(p, levels=16, bins=8)
