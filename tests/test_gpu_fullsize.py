"""Parity at the benchmark workloads' full widths, batch shapes and context lengths.

The oracle cannot run 32 to 64 decoder layers of these widths in seconds, so the engine runs
one-layer slices of each workload's models (every width, the vocabulary, the batch, the prompt
lengths, k and the temperatures are the workload's own) teacher-forced against the oracle (see
parity.py). The full-depth 8B/1B pair, in the launch configuration the benchmark times, is checked
on what needs no oracle forward: every draft sample and every acceptance decision, recomputed by
the oracle from the engine's own logits, must be bit-exact, and the committed state must follow.
"""
import dataclasses

import pytest
import torch

import parity
from oracle import sampling
from paper_2511_09844_gb300 import sd2
from paper_2511_09844_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _host(w):
    if isinstance(w, dict):
        return {k: _host(v) for k, v in w.items()}
    if isinstance(w, list):
        return [_host(v) for v in w]
    return w.cpu()


def _one_layer(work, **kw):
    return dataclasses.replace(work, verifier=dataclasses.replace(work.verifier, n_layers=1),
                               drafter=dataclasses.replace(work.drafter, n_layers=1), **kw)


def _weights(work, seed):
    """Workload-shaped random weights, drawn on the GPU (fast at these sizes), host copies."""
    vw = W.make_lm_weights(work.verifier, seed, device="cuda", norm_jitter=0.1)
    dw = W.make_lm_weights(work.drafter, seed + 1, device="cuda", norm_jitter=0.1)
    st = W.make_steering_weights(work, seed + 2, device="cuda", ln_jitter=0.1)
    return _host(vw), _host(dw), _host(st)


def _temps(work):
    return [work.temperatures[b % len(work.temperatures)] for b in range(work.batch)]


@pytest.mark.parametrize("name,n_steps", [("llama8b_1b", 2), ("llama8b_1b_b16", 1), ("qwen32b_05b", 1)])
def test_full_width_one_layer_slices(name, n_steps):
    """Logits, taps, g, biases within 2e-2 and every decision bit-exact at the workload's shapes."""
    work = _one_layer(W.WORKLOADS[name])
    vw, dw, st = _weights(work, 21)
    prompts = W.make_prompts(work.verifier.vocab, work.batch, work.prompt_len, seed=17)
    rep = parity.run(work, vw, dw, st, prompts, _temps(work), seed=5, n_steps=n_steps)
    assert rep.blocks == work.batch * n_steps


def test_full_width_slice_drafter_chain():
    """The drafter steps as one persistent kernel (chain.cu) at the 8B/1B pair's widths."""
    work = _one_layer(W.WORKLOADS["llama8b_1b"])
    work = dataclasses.replace(work, drafter=dataclasses.replace(W.WORKLOADS["llama8b_1b"].drafter, n_layers=2))
    vw, dw, st = _weights(work, 23)
    prompts = W.make_prompts(work.verifier.vocab, work.batch, work.prompt_len, seed=18)
    rep = parity.run(work, vw, dw, st, prompts, _temps(work), seed=7, n_steps=2, chain=True)
    assert rep.blocks == 2


def test_full_width_slice_attention_in_o_projection():
    """The 1B drafter's decode attention inside its O projection (16 tiles x 8 KV heads) at the 8B/1B
    pair's widths; the 8B verifier (hd 128) keeps the attention kernel."""
    work = _one_layer(W.WORKLOADS["llama8b_1b"])
    work = dataclasses.replace(work, drafter=dataclasses.replace(W.WORKLOADS["llama8b_1b"].drafter, n_layers=2))
    vw, dw, st = _weights(work, 29)
    prompts = W.make_prompts(work.verifier.vocab, work.batch, work.prompt_len, seed=20)
    rep = parity.run(work, vw, dw, st, prompts, _temps(work), seed=8, n_steps=2, fused_attention=True)
    assert rep.blocks == 2


def test_long_context_verify_16k():
    """8B-shaped verify at a 16384-token context, batch 1 (one-layer slice, k = 1)."""
    work = _one_layer(W.WORKLOADS["llama8b_1b"], k=1, prompt_len=(16384, 16384))
    vw, dw, st = _weights(work, 31)
    prompts = W.make_prompts(work.verifier.vocab, 1, work.prompt_len, seed=19)
    rep = parity.run(work, vw, dw, st, prompts, [1.0], seed=6, n_steps=1)
    assert rep.blocks == 1


def test_long_context_two_ragged_sequences():
    """Two sequences of 12000 and 16384 tokens (8B/1B one-layer slices, k = 2): at this context the
    drafter's decode attention spreads each sequence over two clusters of context splits whose
    partials meet in global scratch, and the two sequences split their own contexts differently."""
    work = _one_layer(W.WORKLOADS["llama8b_1b"], k=2, batch=2, prompt_len=(12000, 16384))
    vw, dw, st = _weights(work, 37)
    V = work.verifier.vocab
    prompts = W.make_prompts(V, 1, (12000, 12000), seed=23) + W.make_prompts(V, 1, (16384, 16384), seed=24)
    rep = parity.run(work, vw, dw, st, prompts, [1.0, 0.0], seed=9, n_steps=2)
    assert rep.blocks == 4


def test_full_depth_decisions_bit_exact():
    """Full 32-layer / 16-layer models at the benchmark's shape: the oracle's draft samples and
    acceptance on the engine's logits equal the engine's tokens; committed state follows."""
    work = W.WORKLOADS["llama8b_1b"]
    B, k, V = work.batch, work.k, work.verifier.vocab
    vw = W.make_lm_weights(work.verifier, 1, device="cuda")
    dw = W.make_lm_weights(work.drafter, 2, device="cuda")
    st = W.make_steering_weights(work, 3, device="cuda")
    prompts = W.make_prompts(V, B, work.prompt_len, seed=7)
    seed, temp = 1234, work.temperatures[-1]
    eng = sd2.SD2Engine(work, vw, dw, st, max_batch=B, max_ctx=len(prompts[0]) + 8 * (k + 1) + k + 8,
                        max_prefill_tokens=sum(len(p) for p in prompts))
    try:
        first = eng.prefill(prompts, [temp] * B, seed).cpu().tolist()
        tgt = eng.buffer(sd2.BUF_TARGET).view(B, k + 1, V)
        assert sampling.sample_from_target(tgt[0, 0].cpu().numpy(), temp, seed, 0, 0, 0) == first[0]
        committed = list(prompts[0]) + first
        for step in range(1, 5):
            eng.step()
            tokens, n = eng.accept()
            torch.cuda.synchronize()
            tgt = eng.buffer(sd2.BUF_TARGET).view(B, k + 1, V)[0].cpu().numpy()
            drf = eng.buffer(sd2.BUF_DRAFT).view(B, k, V)[0].cpu().numpy()
            xh = [int(x) for x in eng.buffer(sd2.BUF_XHAT).view(B, k)[0].cpu()]
            for i in range(1, k + 1):
                assert sampling.sample_draft(drf[i - 1], temp, seed, 0, step, i) == xh[i - 1]
            emitted, _ = sampling.accept_block(tgt, drf, xh, temp, seed, 0, step)
            got = [int(t) for t in tokens[0, :int(n[0])].cpu()]
            assert got == emitted
            committed += got
            state = eng.buffer(sd2.BUF_STATE).view(4, -1)[:, 0].cpu()
            assert int(state[0]) == len(committed)
            assert eng.buffer(sd2.BUF_COMMITTED).view(B, -1)[0, :len(committed)].cpu().tolist() == committed
        eng.check()
    finally:
        eng.close()
