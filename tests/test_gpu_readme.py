"""The README's PyTorch example runs as written.

The code block is executed against a small model whose logits require grad:
the backward pass with the library's dlogits must reach the model's weights,
the statistics must be consistent, and the EWMA update must move theta_prox.
"""

import os
import re

import pytest
import torch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_readme_example_runs():
    text = open(os.path.join(ROOT, "README.md")).read()
    code = re.search(r"```python\n(.*?)```", text, re.S).group(1)
    from paper_2605_12070_gb300.workloads import make_loss_batch
    b = make_loss_batch("tight_f32_v151936", T=256, V=4096, seed=2, device="cuda")
    hidden = torch.randn(b.T, 64, device="cuda")
    W = torch.randn(64, b.V, device="cuda", requires_grad=True)
    # the current policy a small step away from the old one (tight thresholds)
    z_theta = b.z_old + hidden @ W * 1e-4
    # two 128-token sequences form one GRPO group whose rewards can tie (A = 0):
    # give every token an advantage of its own so that the gradient is not empty
    adv = torch.randn(b.T, device="cuda")
    mask = torch.ones(b.T, dtype=torch.uint8, device="cuda")
    ns = {"z_theta": z_theta, "z_old": b.z_old, "ids": b.ids, "logp_mu": b.logp_mu,
          "adv": adv, "mask": mask,
          "theta": torch.randn(10_000, device="cuda"), "theta_prox": torch.zeros(10_000, device="cuda")}
    exec(compile(code, "README.md", "exec"), ns)
    torch.cuda.synchronize()
    st = ns["stats"]
    assert st.n_valid > 0 and st.n_rd_out + st.n_active <= st.n_valid and st.n_active > 0
    assert W.grad is not None and torch.isfinite(W.grad).all() and W.grad.abs().sum() > 0
    assert torch.equal(ns["theta_prox"], ns["theta"])  # an empty history: the first step copies theta
