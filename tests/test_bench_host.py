"""Host-side formulas of the benchmark (CPU only).

The roofline lines of the PPO update divide an algorithmic FLOP count by the
measured time.  That count, bench.ppo_flops_per_sample, is pinned here to
PyTorch's own count of the matrix products in one forward and backward pass
of the policy and the value network (tanh MLPs D-H-H, heads of A and 1
outputs; the input needs no gradient, so the first layer has no
data-gradient product)."""
import pytest
import torch
from torch.utils.flop_counter import FlopCounterMode

import bench


def _mlp(D, H, out):
    return torch.nn.Sequential(torch.nn.Linear(D, H), torch.nn.Tanh(), torch.nn.Linear(H, H), torch.nn.Tanh(),
                               torch.nn.Linear(H, out))


@pytest.mark.parametrize("D,H,A", [(8, 64, 3), (16, 128, 5), (32, 256, 16), (64, 512, 16)])
def test_ppo_flops_per_sample_matches_autograd_count(D, H, A):
    B = 32
    torch.manual_seed(0)
    x = torch.randn(B, D)
    total = 0
    for out in (A, 1):
        net = _mlp(D, H, out)
        with FlopCounterMode(display=False) as fc:
            net(x).sum().backward()
        total += fc.get_total_flops()
    assert total == bench.ppo_flops_per_sample(D, H, A) * B


def test_ppo_flops_per_sample_7b_figure():
    """The 7B and 72B counts quoted in the roofline lines and the design notes."""
    assert bench.ppo_flops_per_sample(16, 128, 5) == 217_600
    assert bench.ppo_flops_per_sample(32, 256, 16) == 878_080
