"""GPU acceptance kernel (sd2_accept_logits) against the oracle: emitted tokens bit-exact.

Both sides see the same logits and the same Philox stream; every decision (accept/reject, the
replacement drawn from the residual, the bonus token, greedy matches) must be identical.
"""
import numpy as np
import pytest
import torch

from oracle import sampling
from paper_2511_09844_gb300 import sd2
from paper_2511_09844_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _oracle(target, draft, xhat, temps, seed, step):
    t = target.float().cpu().numpy()
    d = draft.float().cpu().numpy()
    x = xhat.cpu().numpy()
    out = []
    for b in range(t.shape[0]):
        out.append(sampling.accept_block(t[b], d[b], list(x[b]), float(temps[b]), seed, b, step))
    return out


def _compare(target, draft, xhat, temps, seed, step):
    tt = torch.tensor(temps, dtype=torch.float32, device="cuda")
    tok, n = sd2.accept_logits(target.cuda(), draft.cuda(), xhat.cuda(), tt, seed, step)
    torch.cuda.synchronize()
    tok, n = tok.cpu(), n.cpu()
    ref = _oracle(target, draft, xhat, temps, seed, step)
    js = []
    for b, (emitted, j) in enumerate(ref):
        assert int(n[b]) == j + 1, (b, int(n[b]), j)
        assert tok[b, :j + 1].tolist() == emitted, (b, tok[b].tolist(), emitted)
        js.append(j)
    return js


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("V,B,k", [(4096, 8, 4), (32000, 4, 8), (1000, 16, 1)])
def test_sweep_logits_bit_exact(dtype, V, B, k):
    target, draft, xhat = W.make_sweep_logits(B, k, V, seed=V + B + k)
    temps = [[0.0, 0.7, 1.0][b % 3] for b in range(B)]
    _compare(target.to(dtype), draft.to(dtype), xhat, temps, seed=99, step=3)


def test_high_acceptance_reaches_bonus_and_residual_paths():
    """Draft rows close to the target rows: many accepts, full blocks (bonus), and rejections."""
    B, k, V = 32, 6, 2048
    g = torch.Generator().manual_seed(5)
    target = torch.randn(B, k + 1, V, generator=g) * 2
    noise = torch.randn(B, k, V, generator=g) * torch.linspace(0.0, 1.5, B)[:, None, None]
    draft = target[:, :k] + noise
    # drafts: the draft row's most likely token (what a sampler would usually pick)
    xhat = draft.argmax(-1).to(torch.int32)
    temps = [1.0 if b % 4 else 0.7 for b in range(B)]
    js = _compare(target, draft, xhat, temps, seed=2024, step=11)
    assert max(js) == k and min(js) < k and len(set(js)) >= 3


def test_identical_rows_always_accept():
    B, k, V = 4, 5, 512
    g = torch.Generator().manual_seed(6)
    target = torch.randn(B, k + 1, V, generator=g)
    draft = target[:, :k].clone()
    xhat = torch.randint(0, V, (B, k), generator=g, dtype=torch.int32)
    js = _compare(target, draft, xhat, [1.0] * B, seed=3, step=1)
    assert js == [k] * B          # u*q <= p with q == p and u < 1


def test_greedy_prefix_match():
    B, k, V = 6, 4, 300
    g = torch.Generator().manual_seed(7)
    target = torch.randn(B, k + 1, V, generator=g)
    am = target.argmax(-1)
    xhat = am[:, :k].clone().to(torch.int32)
    for b in range(B):                 # sequence b mismatches at draft b (none for b >= k)
        if b < k:
            xhat[b, b] = (xhat[b, b] + 1) % V
    draft = torch.randn(B, k, V, generator=g)
    js = _compare(target, draft, xhat, [0.0] * B, seed=1, step=1)
    assert js == [min(b, k) for b in range(B)]


def test_step_and_seed_change_the_stream():
    B, k, V = 16, 4, 4096
    target, draft, xhat = W.make_sweep_logits(B, k, V, seed=8, std=0.5, boost=1.0)   # flat rows
    tt = torch.ones(B, device="cuda")

    def emitted(step):
        tok, n = sd2.accept_logits(target.cuda(), draft.cuda(), xhat.cuda(), tt, 1, step)
        tok, n = tok.cpu(), n.cpu()
        return [tok[b, :n[b]].tolist() for b in range(B)]        # entries past n are not written

    a, b, c = emitted(1), emitted(2), emitted(1)
    assert a == c and a != b


def test_nonfinite_logits_are_reported_not_trapped():
    """A NaN logit is latched in the error word; the context stays usable."""
    B, k, V = 2, 2, 256
    target = torch.randn(B, k + 1, V)
    target[1, 0, 7] = float("nan")
    draft = torch.randn(B, k, V)
    xhat = torch.zeros(B, k, dtype=torch.int32)
    L = sd2.load_library()
    ws = torch.zeros(L.sd2_accept_workspace_bytes(B, k), dtype=torch.uint8, device="cuda")
    sd2.accept_logits(target.cuda(), draft.cuda(), xhat.cuda(), torch.ones(B, device="cuda"), 1, 1, workspace=ws)
    torch.cuda.synchronize()
    # the error word sits right after the scratch tables
    R = B * (2 * k + 1)
    off = 8 * 2 * R + 8 * 2 * B + 4 * B + 8 * B
    word = int(ws[off:off + 4].cpu().view(torch.int32)[0])
    assert word & 1
    torch.cuda.synchronize()                      # no sticky error
