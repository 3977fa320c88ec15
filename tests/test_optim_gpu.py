"""The torch.optim interface on the GPU: equal to the plan it wraps, and a
small training loop that learns (App. E diagnostics read back)."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _mats(seed, shapes, dtype):
    import torch
    g = torch.Generator().manual_seed(seed)
    return [(torch.randn(r, c, generator=g) * 0.05).to(dtype).cuda() for r, c in shapes]


@pytest.mark.parametrize("variant", ["G", "L"])
def test_optimizer_equals_plan(variant):
    import torch
    from paper_2609_36692_gb300.optim import NormPre, NormPreOptimizer
    shapes = [(64, 96), (96, 64), (64, 96)]
    W0 = _mats(1, shapes, torch.float32)
    G = [[x * 10 for x in _mats(2 + s, shapes, torch.float32)] for s in range(3)]
    params = [torch.nn.Parameter(w.clone()) for w in W0]
    opt = NormPreOptimizer(params, lr=0.05, variant=variant, rank=8, oversample=8, precision=1, seed=3)
    plan = NormPre(shapes, ["f32"] * 3, ["f32"] * 3, variant={"G": 0, "L": 1}[variant], rank=8, oversample=8,
                   precision=1, seed=3, momentum=0.95, weight_decay=0.1, target_rms=0.2)
    W = [w.clone() for w in W0]
    M = [torch.zeros_like(w) for w in W0]
    for t in range(3):
        for p, g in zip(params, G[t]):
            p.grad = g.clone()
        opt.step()
        plan.step(t, 0.05, W, G[t], M)
    torch.cuda.synchronize()
    for p, w, m in zip(params, W, M):
        assert torch.equal(p.detach(), w)
        assert torch.equal(opt.state[p]["momentum_buffer"], m)
    assert opt.param_groups[0]["t"] == 3


@pytest.mark.parametrize("variant", ["G", "L", "L_exact"])
def test_small_training_loop_learns(variant):
    """A two-layer ReLU network fit to a random teacher on seeded synthetic
    data: the hidden matrices under NormPreOptimizer (with a cosine learning-
    rate schedule), no biases.  The loss falls and the diagnostics read back."""
    import torch
    torch.manual_seed(0)
    d_in, d_h, d_out, n = 64, 128, 32, 2048
    g = torch.Generator(device="cuda").manual_seed(11)
    X = torch.randn(n, d_in, device="cuda", generator=g)
    teacher = torch.randn(d_in, d_out, device="cuda", generator=g) / d_in ** 0.5
    Y = torch.tanh(X @ teacher) * 2
    l1 = torch.nn.Linear(d_in, d_h, bias=False).cuda()
    l2 = torch.nn.Linear(d_h, d_out, bias=False).cuda()
    from paper_2609_36692_gb300.optim import NormPreOptimizer
    opt = NormPreOptimizer([l1.weight, l2.weight], lr=0.05, variant=variant, rank=16, oversample=8,
                           diagnostics=1, check_status=True)
    sched = torch.optim.lr_scheduler.CosineAnnealingLR(opt, T_max=60)
    losses = []
    for step in range(60):
        idx = torch.randint(0, n, (256,), device="cuda", generator=g)
        loss = torch.nn.functional.mse_loss(l2(torch.relu(l1(X[idx]))), Y[idx])
        opt.zero_grad(set_to_none=True)
        loss.backward()
        opt.step()
        sched.step()
        losses.append(float(loss.detach()))
    first, last = np.mean(losses[:5]), np.mean(losses[-5:])
    assert last < 0.5 * first, (variant, first, last)
    diag, mean_align = opt.diagnostics()
    assert np.isfinite(mean_align) and -1.0 <= mean_align <= 1.0
    for rec in diag.values():
        assert rec["grad_norm"] > 0 and rec["update_norm"] > 0
        if variant == "L_exact":
            assert rec["E_global"] >= rec["E_top"] >= 0
        else:
            assert np.isnan(rec["E_top"])
