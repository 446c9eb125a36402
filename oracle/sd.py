"""The SD^2 draft-and-verify loop (oracle; test infrastructure only).

Restates Sec. 3 with the bookkeeping the paper leaves implicit. Per sequence, with n committed
tokens x_0..x_{n-1} (prompt plus emitted):

  prefill   The verifier reads the prompt; its last row gives the first new token (sampled as a
            bonus token at step 0). The steering vector g comes from the verifier's taps at the
            last prompt position, and the drafter reads the whole prompt under the biases of g.
  stage     (step s >= 1) With biases b = W_s g (Eq. 2, computed once per stage, Sec. 3.2):
            the drafter reads its pending committed tokens (1, or 2 after a full accept), then
            drafts x^_1..x^_k autoregressively (x^_k itself is not fed). The verifier reads
            [x_{n-1}, x^_1..x^_k] at positions n-1..n+k-1: row i is p_i (Sec. 3.1).
  accept    Speculative acceptance (sampling.accept_block) keeps j drafts and adds one token y.
  commit    n += j + 1. Verifier cache: positions 0..n-2 (y not yet read). Drafter cache keeps the
            positions whose inputs were accepted, each with the biases it was computed under
            (Sec. 3.2, last sentence: keys/values carry the prior steering vectors): positions
            0..min(n_old + j, n_old + k - 1) - 1. The next g is read at position n - 2, the
            position whose distribution produced y ("the last token returned", Sec. 3.1).

The decoder is evaluated from scratch over each prefix (no cache), which is the definition the
GPU's cached computation must reproduce. With exact_rows=True every verifier row is its own
forward over exactly its prefix, so greedy SD can be compared bit for bit with greedy decoding.

Pinned in tests/test_oracle_sd.py: greedy SD equals greedy decoding of the verifier; with the
drafter equal to the verifier and W_s = 0, every greedy block is fully accepted (tau = k + 1,
Sec. 4 "Metrics"); W_s = 0 leaves the drafter exactly unsteered (App. A.2); rollback keeps the
cached drafter positions consistent with a fresh recomputation.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

from . import model, sampling, steering


@dataclass
class SeqState:
    tokens: List[int]
    prompt_len: int
    temp: float
    d_cached: int = 0
    bias_ids: List[int] = field(default_factory=list)   # per cached drafter position
    cur_bias: int = -1                                  # stage biases for the next stage
    blocks: int = 0
    accepted: int = 0


class OracleSD:
    def __init__(self, work, verifier_w: Dict, drafter_w: Dict, steer_w: Dict, seed: int,
                 exact_rows: bool = False):
        self.work = work
        self.vs, self.ds = work.verifier, work.drafter
        self.vw, self.dw, self.st = verifier_w, drafter_w, steer_w
        self.k = work.k
        self.taps = tuple(work.tap_layers)
        self.seed = int(seed)
        self.exact_rows = exact_rows
        self.biases: List[torch.Tensor] = []              # [L_D, F_D] per stage
        self.gs: List[torch.Tensor] = []                  # the steering vector g of each stage
        self.seqs: List[SeqState] = []

    # -- model evaluations --------------------------------------------------------------------
    def verifier_rows(self, tokens: Sequence[int], first: int, last: int):
        """Verifier logits and taps at positions first..last of `tokens` (inclusive)."""
        if self.exact_rows:
            outs, taps = [], []
            for t in range(first, last + 1):
                z, tp = model.forward(self.vs, self.vw, tokens[:t + 1], tap_layers=self.taps,
                                      logit_rows=[t])
                outs.append(z[0])
                taps.append(tp[t])
            return torch.stack(outs), torch.stack(taps)
        z, tp = model.forward(self.vs, self.vw, tokens[:last + 1], tap_layers=self.taps,
                              logit_rows=list(range(first, last + 1)))
        return z, tp[first:last + 1]

    def drafter_last(self, tokens: Sequence[int], bias_ids: Sequence[int]) -> torch.Tensor:
        """Drafter logits at the last position; position t computed under the steering of stage
        bias_ids[t] (its biases, or for "cond_mlp" its g)."""
        if self.work.steering_site == "cond_mlp":
            g_rows = torch.stack([self.gs[i] for i in bias_ids])
            z, _ = model.forward(self.ds, self.dw, tokens, logit_rows=[len(tokens) - 1], bias_site="cond_mlp",
                                 cond=(g_rows, self.st))
            return z[0]
        bias = torch.stack([self.biases[i] for i in bias_ids])
        z, _ = model.forward(self.ds, self.dw, tokens, bias=bias, logit_rows=[len(tokens) - 1],
                             bias_site=self.work.steering_site)
        return z[0]

    def _new_bias(self, taps_hml: torch.Tensor) -> int:
        g = steering.steering_vector(taps_hml, self.st, self.work.steer_ln_eps)
        self.gs.append(g)
        if self.work.steering_site == "cond_mlp":     # the biases depend on each position's input
            self.biases.append(torch.zeros(0))
        else:
            self.biases.append(steering.steering_bias(g, self.st, self.ds.n_layers, self.work.bias_width))
        return len(self.biases) - 1

    # -- the loop -------------------------------------------------------------------------------
    def prefill(self, prompts: Sequence[Sequence[int]], temps: Sequence[float],
                forced_first: Optional[Sequence[int]] = None) -> List[int]:
        """Start every sequence; forced_first replaces the sampled first tokens (teacher forcing)."""
        firsts = []
        self.prefill_logits, self.prefill_taps = [], []
        for b, (prompt, temp) in enumerate(zip(prompts, temps)):
            n0 = len(prompt)
            z, tp = self.verifier_rows(list(prompt), n0 - 1, n0 - 1)
            self.prefill_logits.append(z[0])
            self.prefill_taps.append(tp[0])
            if forced_first is not None:
                y = int(forced_first[b])
            else:
                y = sampling.sample_from_target(z[0].numpy(), temp, self.seed, b, 0, 0)
            s = SeqState(tokens=list(prompt) + [y], prompt_len=n0, temp=float(temp))
            s.cur_bias = self._new_bias(tp[0])
            s.bias_ids = [s.cur_bias] * n0          # drafter prefill under the first g
            s.d_cached = n0
            self.seqs.append(s)
            firsts.append(y)
        return firsts

    def stage(self, b: int, step: int, forced_xhat: Optional[Sequence[int]] = None):
        """Draft k tokens and verify them. Returns dict(xhat, draft [k,V], target [k+1,V], taps)."""
        s = self.seqs[b]
        n = len(s.tokens)
        ids = s.bias_ids[:s.d_cached] + [s.cur_bias] * (n - s.d_cached)
        xhat, drafts = [], []
        for i in range(1, self.k + 1):
            seq = s.tokens + xhat
            z = self.drafter_last(seq, ids + [s.cur_bias] * (len(seq) - n))
            drafts.append(z)
            if forced_xhat is not None:
                x = int(forced_xhat[i - 1])
            else:
                x = sampling.sample_draft(z.numpy(), s.temp, self.seed, b, step, i)
            xhat.append(x)
        target, taps = self.verifier_rows(s.tokens + xhat, n - 1, n - 1 + self.k)
        return {"xhat": xhat, "draft": torch.stack(drafts), "target": target, "taps": taps}

    def accept(self, b: int, step: int, out: dict):
        s = self.seqs[b]
        return sampling.accept_block(out["target"].numpy(), out["draft"].numpy(), out["xhat"],
                                     s.temp, self.seed, b, step)

    def commit(self, b: int, emitted: Sequence[int], j: int, taps_block: torch.Tensor):
        """Append the emitted tokens, roll back both caches, and set the next stage's biases."""
        s = self.seqs[b]
        n_old = len(s.tokens)
        ids = s.bias_ids[:s.d_cached] + [s.cur_bias] * (n_old + self.k - 1 - s.d_cached)
        s.tokens = s.tokens + [int(t) for t in emitted]
        s.d_cached = min(n_old + j, n_old + self.k - 1)
        s.bias_ids = ids[:s.d_cached]
        s.blocks += 1
        s.accepted += j
        if self.exact_rows:
            _, tp = self.verifier_rows(s.tokens, len(s.tokens) - 2, len(s.tokens) - 2)
            s.cur_bias = self._new_bias(tp[0])
        else:
            s.cur_bias = self._new_bias(taps_block[j])

    def generate(self, prompts, temps, n_new: int, max_steps: int = 10 ** 6):
        """Free-running SD^2 until every sequence has at least n_new new tokens."""
        self.prefill(prompts, temps)
        step = 0
        while any(len(s.tokens) - s.prompt_len < n_new for s in self.seqs) and step < max_steps:
            step += 1
            for b, s in enumerate(self.seqs):
                if len(s.tokens) - s.prompt_len >= n_new:
                    continue
                out = self.stage(b, step)
                emitted, j = self.accept(b, step, out)
                self.commit(b, emitted, j, out["taps"])
        return [s.tokens[s.prompt_len:] for s in self.seqs]


def greedy_decode(shape, w: Dict, prompt: Sequence[int], n_new: int) -> List[int]:
    """Plain autoregressive greedy decoding of one model (each step a forward over its prefix)."""
    tokens = list(prompt)
    for _ in range(n_new):
        z, _ = model.forward(shape, w, tokens, logit_rows=[len(tokens) - 1])
        tokens.append(sampling.argmax(z[0].numpy()))
    return tokens[len(prompt):]
