"""Pins for the oracle's draft-and-verify loop (CPU only).

O2: greedy SD^2 equals greedy decoding of the verifier, token for token.
O4: W_s = 0 leaves the drafter exactly unsteered (App. A.2: "initially unchanged").
O5: drafter = verifier and W_s = 0 at T = 0 -> every block keeps all k drafts (tau = k + 1).
Rollback: the cached drafter positions always number n-1 or n-2 and keep their stage's biases.
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import model, sampling
from oracle.sd import OracleSD, greedy_decode
from paper_2511_09844_gb300 import workloads as W


def _tiny(**kw):
    work = W.WORKLOADS["tiny"]
    vs = W.shrink(work.verifier, n_layers=4, d_model=64, n_heads=4, n_kv_heads=2, head_dim=16,
                  d_ffn=128, vocab=61)
    ds = W.shrink(work.drafter, n_layers=2, d_model=32, n_heads=2, n_kv_heads=1, head_dim=16,
                  d_ffn=64, vocab=61)
    return dataclasses.replace(work, verifier=vs, drafter=ds, d_steer=32, **kw)


def _weights(work, seed=1, zero_ws=False, same=False):
    vw = W.make_lm_weights(work.verifier, seed, norm_jitter=0.1, std=0.2)
    dw = vw if same else W.make_lm_weights(work.drafter, seed + 1, norm_jitter=0.1, std=0.2)
    st = W.make_steering_weights(work, seed + 2, std=0.2, ln_jitter=0.1, zero_ws=zero_ws)
    return vw, dw, st


def test_greedy_sd_equals_greedy_decoding():
    work = _tiny(k=3)
    vw, dw, st = _weights(work)
    prompt = W.make_prompts(work.verifier.vocab, 1, (6, 6), seed=3)[0]
    sd = OracleSD(work, vw, dw, st, seed=5, exact_rows=True)
    out = sd.generate([prompt], [0.0], n_new=20)[0]
    ref = greedy_decode(work.verifier, vw, prompt, len(out))
    assert out == ref
    s = sd.seqs[0]
    assert s.blocks >= 1 and len(out) == 1 + s.blocks + s.accepted   # + the prefill token


def test_self_drafting_accepts_everything():
    work = _tiny(k=4)
    work = dataclasses.replace(work, drafter=work.verifier)
    vw, _, st = _weights(work, zero_ws=True)
    prompt = W.make_prompts(work.verifier.vocab, 1, (5, 5), seed=4)[0]
    sd = OracleSD(work, vw, vw, st, seed=6, exact_rows=True)
    out = sd.generate([prompt], [0.0], n_new=15)[0]
    s = sd.seqs[0]
    assert s.accepted == s.blocks * work.k          # tau = k + 1 in every block
    assert out == greedy_decode(work.verifier, vw, prompt, len(out))


def test_zero_ws_is_unsteered_and_nonzero_ws_steers():
    work = _tiny(k=3)
    vw, dw, st0 = _weights(work, zero_ws=True)
    prompt = W.make_prompts(work.verifier.vocab, 1, (7, 7), seed=8)[0]
    sd = OracleSD(work, vw, dw, st0, seed=1)
    sd.prefill([prompt], [1.0])
    out = sd.stage(0, 1)
    seq = sd.seqs[0].tokens + out["xhat"]
    for i in range(work.k):
        ref, _ = model.forward(work.drafter, dw, seq[:len(sd.seqs[0].tokens) + i],
                               logit_rows=[len(sd.seqs[0].tokens) + i - 1])
        assert torch.equal(out["draft"][i], ref[0])
    _, _, st1 = _weights(work, zero_ws=False)
    sd1 = OracleSD(work, vw, dw, st1, seed=1)
    sd1.prefill([prompt], [1.0])
    out1 = sd1.stage(0, 1, forced_xhat=out["xhat"])
    assert (out1["draft"] - out["draft"]).abs().max() > 1e-3
    assert torch.equal(out1["target"], out["target"])      # the verifier is never steered


@pytest.mark.parametrize("temp", [0.0, 1.0])
def test_rollback_bookkeeping(temp):
    work = _tiny(k=3)
    vw, dw, st = _weights(work)
    prompts = W.make_prompts(work.verifier.vocab, 2, (4, 9), seed=11)
    sd = OracleSD(work, vw, dw, st, seed=2)
    sd.prefill(prompts, [temp, temp])
    for step in range(1, 6):
        for b, s in enumerate(sd.seqs):
            n = len(s.tokens)
            assert s.d_cached in (n - 1, n - 2) and len(s.bias_ids) == s.d_cached
            out = sd.stage(b, step)
            emitted, j = sd.accept(b, step, out)
            assert 0 <= j <= work.k and len(emitted) == j + 1 and emitted[:j] == out["xhat"][:j]
            old_ids = list(s.bias_ids)
            stage_bias = s.cur_bias
            sd.commit(b, emitted, j, out["taps"])
            assert len(s.tokens) == n + j + 1
            assert s.d_cached == min(n + j, n + work.k - 1)
            assert s.bias_ids[:len(old_ids)] == old_ids                 # kept entries keep their g
            assert all(i == stage_bias for i in s.bias_ids[len(old_ids):])
            assert s.cur_bias != stage_bias


def test_cached_drafter_matches_recomputation_under_recorded_biases():
    """Each drafter row equals a fresh forward over its prefix with the per-position biases."""
    work = _tiny(k=3)
    vw, dw, st = _weights(work)
    prompt = W.make_prompts(work.verifier.vocab, 1, (6, 6), seed=12)[0]
    sd = OracleSD(work, vw, dw, st, seed=3)
    sd.prefill([prompt], [1.0])
    for step in range(1, 4):
        out = sd.stage(0, step)
        emitted, j = sd.accept(0, step, out)
        sd.commit(0, emitted, j, out["taps"])
    s = sd.seqs[0]
    toks = s.tokens[:s.d_cached]
    bias = torch.stack([sd.biases[i] for i in s.bias_ids])
    z, _ = model.forward(work.drafter, dw, toks, bias=bias, logit_rows=[len(toks) - 1])
    assert torch.equal(sd.drafter_last(toks, s.bias_ids), z[0])
    # the steering row of the next stage is position n-2 of the committed sequence
    _, tp = model.forward(work.verifier, vw, s.tokens, tap_layers=work.tap_layers)
    from oracle import steering
    g = steering.steering_vector(tp[len(s.tokens) - 2], st, work.steer_ln_eps)
    b = steering.steering_bias(g, st, work.drafter.n_layers, work.drafter.d_ffn)
    assert torch.allclose(sd.biases[s.cur_bias], b, atol=1e-5, rtol=1e-4)


def test_sampled_sd_runs_and_tau_in_range():
    work = _tiny(k=4)
    vw, dw, st = _weights(work)
    prompts = W.make_prompts(work.verifier.vocab, 2, (5, 8), seed=13)
    sd = OracleSD(work, vw, dw, st, seed=4)
    outs = sd.generate(prompts, [1.0, 0.7], n_new=16)
    for o, s in zip(outs, sd.seqs):
        assert len(o) >= 16 and all(0 <= t < work.verifier.vocab for t in o)
        tau = (s.accepted + s.blocks) / s.blocks
        assert 1.0 <= tau <= work.k + 1
