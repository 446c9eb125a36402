"""Teacher-forced parity between the CUDA engine and the CPU oracle.

The engine runs free; after each call the oracle recomputes the same quantities on the engine's
committed prefix and its drafted tokens (random-weight near-ties make free-running bf16 and fp32
trajectories diverge, so the oracle follows the GPU's decisions):
  * logits, verifier taps, steering vector and biases agree within the float tolerance;
  * every integer decision (first token, each draft token, the accepted prefix and the replacement
    or bonus token) is recomputed by the oracle from the engine's own logits and must be equal.
Float tolerance: per row, max|gpu - ref| / max|ref| <= 2e-2 (bf16 GPU against fp32 oracle).
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List

import numpy as np
import torch

from oracle import sampling
from oracle.sd import OracleSD
from paper_2511_09844_gb300 import sd2
from paper_2511_09844_gb300 import workloads as W

TOL = 2e-2


def row_rel_err(gpu: torch.Tensor, ref: torch.Tensor) -> float:
    """max over rows of max|gpu - ref| / max|ref| (last dim = row)."""
    g = gpu.detach().float().cpu().reshape(-1, gpu.shape[-1])
    r = ref.detach().float().cpu().reshape(-1, ref.shape[-1])
    den = r.abs().amax(dim=1).clamp_min(1e-30)
    return float(((g - r).abs().amax(dim=1) / den).max())


def to_device(w, device="cuda"):
    if isinstance(w, dict):
        return {k: to_device(v, device) for k, v in w.items()}
    if isinstance(w, list):
        return [to_device(v, device) for v in w]
    return w.to(device)


@dataclasses.dataclass
class ParityReport:
    steps: int = 0
    blocks: int = 0
    accepted: int = 0
    max_err: Dict[str, float] = dataclasses.field(default_factory=dict)
    decisions: int = 0

    def note(self, name, err):
        self.max_err[name] = max(self.max_err.get(name, 0.0), err)


def run(work, vw, dw, st, prompts, temps, seed, n_steps, max_ctx=None, graphs=True, tol=TOL,
        check_taps=True, gemm_impl=0, steering=True, chain=False, fused_attention=False,
        max_batch=None) -> ParityReport:
    """Run prefill + n_steps iterations on the GPU and check each against the oracle.

    steering=False runs the engine's pretrained-drafter mode (no steering stage, no bias); the
    oracle then needs W_s = 0 (its biases are exactly zero, the unsteered drafter)."""
    B, k, V = len(prompts), work.k, work.verifier.vocab
    if max_ctx is None:
        max_ctx = max(len(p) for p in prompts) + n_steps * (k + 1) + k + 4
    dev = (to_device(vw), to_device(dw), to_device(st))
    eng = sd2.SD2Engine(work, *dev, max_batch=B if max_batch is None else max_batch, max_ctx=max_ctx,
                        max_prefill_tokens=sum(len(p) for p in prompts), steering=steering)
    eng.set_graphs(graphs)
    eng.set_gemm_impl(gemm_impl)
    eng.set_drafter_chain(chain)
    eng.set_fused_attention(fused_attention)
    rep = ParityReport()
    try:
        first = eng.prefill(prompts, temps, seed).cpu().tolist()
        ora = OracleSD(work, vw, dw, st, seed)
        ora.prefill(prompts, temps, forced_first=first)
        tgt = eng.buffer(sd2.BUF_TARGET).view(B, k + 1, V)
        taps = eng.buffer(sd2.BUF_TAPS).view(B, k + 1, 3, -1)
        for b in range(B):
            rep.note("prefill_logits", row_rel_err(tgt[b, 0], ora.prefill_logits[b]))
            if check_taps:
                rep.note("prefill_taps", row_rel_err(taps[b, 0], ora.prefill_taps[b]))
            y = sampling.sample_from_target(tgt[b, 0].cpu().numpy(), temps[b], seed, b, 0, 0)
            assert y == first[b], f"first token of sequence {b}: oracle {y}, gpu {first[b]}"
            rep.decisions += 1
        g0 = eng.buffer(sd2.BUF_G).view(B, -1)
        b0 = eng.buffer(sd2.BUF_BIAS).view(B, -1)
        stage_biases = work.steering_site != "cond_mlp"    # cond: per-row biases, checked via the logits
        for b in range(B if steering else 0):
            rep.note("g", row_rel_err(g0[b], ora.gs[ora.seqs[b].cur_bias]))
            if stage_biases:
                rep.note("bias", row_rel_err(b0[b], ora.biases[ora.seqs[b].cur_bias].reshape(-1)))
        for step in range(1, n_steps + 1):
            state_before = eng.buffer(sd2.BUF_STATE).view(4, -1)[:, :B].cpu()
            eng.step()
            tokens, n = eng.accept()
            torch.cuda.synchronize()
            tgt = eng.buffer(sd2.BUF_TARGET).view(B, k + 1, V).cpu()
            drf = eng.buffer(sd2.BUF_DRAFT).view(B, k, V).cpu()
            xh = eng.buffer(sd2.BUF_XHAT).view(B, k).cpu()
            tp = eng.buffer(sd2.BUF_TAPS).view(B, k + 1, 3, -1).cpu()
            gg = eng.buffer(sd2.BUF_G).view(B, -1).cpu()
            bb = eng.buffer(sd2.BUF_BIAS).view(B, -1).cpu()
            tokens, n = tokens.cpu(), n.cpu()
            rep.steps += 1
            for b in range(B):
                if int(state_before[3, b]):
                    assert int(n[b]) == 0
                    continue
                s = ora.seqs[b]
                assert int(state_before[0, b]) == len(s.tokens)
                if steering:
                    rep.note("g", row_rel_err(gg[b], ora.gs[s.cur_bias]))
                    if stage_biases:
                        rep.note("bias", row_rel_err(bb[b], ora.biases[s.cur_bias].reshape(-1)))
                xb = [int(x) for x in xh[b]]
                out = ora.stage(b, step, forced_xhat=xb)
                rep.note("draft_logits", row_rel_err(drf[b], out["draft"]))
                rep.note("target_logits", row_rel_err(tgt[b], out["target"]))
                if check_taps:
                    rep.note("taps", row_rel_err(tp[b], out["taps"]))
                for i in range(1, k + 1):
                    x = sampling.sample_draft(drf[b, i - 1].numpy(), s.temp, seed, b, step, i)
                    assert x == xb[i - 1], f"draft {i} of seq {b} at step {step}: oracle {x}, gpu {xb[i - 1]}"
                    rep.decisions += 1
                emitted, j = sampling.accept_block(tgt[b].numpy(), drf[b].numpy(), xb, s.temp, seed, b, step)
                got = [int(t) for t in tokens[b, :int(n[b])]]
                assert got == emitted, f"acceptance of seq {b} at step {step}: oracle {emitted}, gpu {got}"
                rep.decisions += 1
                rep.blocks += 1
                rep.accepted += j
                ora.commit(b, got, len(got) - 1, out["taps"])
            committed = eng.buffer(sd2.BUF_COMMITTED).view(B, -1).cpu()
            state = eng.buffer(sd2.BUF_STATE).view(4, -1)[:, :B].cpu()
            for b in range(B):
                s = ora.seqs[b]
                if int(state[3, b]) and int(state_before[3, b]):
                    continue
                assert int(state[0, b]) == len(s.tokens)
                assert committed[b, :len(s.tokens)].tolist() == s.tokens
                assert int(state[1, b]) == s.d_cached
        eng.check()
    finally:
        eng.close()
    for name, e in rep.max_err.items():
        assert e <= tol, f"{name}: relative error {e:.3g} > {tol}"
    return rep


def tiny_work(**kw):
    return dataclasses.replace(W.WORKLOADS["tiny"], **kw)


def tiny_weights(work, seed=1, std=0.02, jitter=0.1):
    vw = W.make_lm_weights(work.verifier, seed, std=std, norm_jitter=jitter)
    dw = W.make_lm_weights(work.drafter, seed + 1, std=std, norm_jitter=jitter)
    st = W.make_steering_weights(work, seed + 2, std=std, ln_jitter=jitter)
    return vw, dw, st
