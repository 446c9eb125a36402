"""End-to-end GPU parity of the SD^2 engine against the oracle (teacher-forced, see parity.py)."""
import dataclasses

import pytest
import torch

import parity
from oracle import steering
from oracle import model as omodel
from paper_2511_09844_gb300 import sd2
from paper_2511_09844_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("gemm_impl,chain,fused", [(0, True, False), (0, False, False), (0, False, True), (1, False, False)])
@pytest.mark.parametrize("temp", [0.0, 1.0])
def test_tiny_single_sequence(temp, gemm_impl, chain, fused):
    """gemm_impl 0: tensor-core GEMM with fused epilogues, the drafter steps as one persistent
    kernel (chain) or one kernel per projection, the decode attention in its own kernel or inside
    the O projection (fused: both tiny models take it, hd 64); 1: CUDA-core GEMM + separate kernels."""
    work = parity.tiny_work()
    vw, dw, st = parity.tiny_weights(work)
    prompts = W.make_prompts(work.verifier.vocab, 1, (32, 32), seed=7)
    rep = parity.run(work, vw, dw, st, prompts, [temp], seed=1234, n_steps=8, gemm_impl=gemm_impl, chain=chain,
                     fused_attention=fused)
    assert rep.blocks == 8 and rep.decisions > 8 * work.k


def test_tiny_ragged_batch_mixed_temperatures_gqa():
    """Ragged prompts, per-sequence temperatures, grouped KV heads, block-crossing lengths."""
    base = parity.tiny_work()
    vs = W.shrink(base.verifier, n_kv_heads=2)
    ds = W.shrink(base.drafter, n_kv_heads=1)
    work = dataclasses.replace(base, verifier=vs, drafter=ds, k=5, batch=3)
    vw, dw, st = parity.tiny_weights(work, seed=3)
    prompts = W.make_prompts(vs.vocab, 3, (15, 49), seed=8)
    rep = parity.run(work, vw, dw, st, prompts, [0.0, 0.7, 1.0], seed=77, n_steps=6)
    assert rep.blocks == 18


def test_tiny_longest_draft_and_wider_batch():
    """k = 16 (the largest draft length: 17 verify rows per sequence) over 8 ragged sequences with
    mixed temperatures: wide token tiles, many attention groups, long acceptance blocks."""
    base = parity.tiny_work()
    work = dataclasses.replace(base, k=16, batch=8)
    vw, dw, st = parity.tiny_weights(work, seed=5)
    prompts = W.make_prompts(base.verifier.vocab, 8, (9, 70), seed=11)
    temps = [0.0, 1.0, 0.7, 1.0, 0.0, 0.5, 1.0, 0.9]
    rep = parity.run(work, vw, dw, st, prompts, temps, seed=91, n_steps=3)
    assert rep.blocks == 24


def test_flat_attention_ragged_batch():
    """Eight sequences, one of 2100 tokens among seven of 9-40: the verify steps' attention runs in
    flat mode (every resident CTA a slot, shared out on the device by length). The long sequence's
    33 tiles spread over 17 slots (the per-sequence cap of 32 raises the tiles per slot to 2), each
    short one takes one slot, most slots have nothing to do; every decision matches the oracle."""
    work = dataclasses.replace(parity.tiny_work(), batch=8)
    vw, dw, st = parity.tiny_weights(work, seed=31)
    V = work.verifier.vocab
    long_prompt = W.make_prompts(V, 1, (2100, 2100), seed=32)[0]
    short = W.make_prompts(V, 7, (9, 40), seed=33)
    prompts = [short[0], short[1], long_prompt, *short[2:]]
    temps = [1.0, 0.0, 1.0, 0.7, 1.0, 0.0, 1.0, 0.5]
    rep = parity.run(work, vw, dw, st, prompts, temps, seed=93, n_steps=3)
    assert rep.blocks == 24


def test_batch_below_context_capacity():
    """A context built for 5 sequences serving 2: the per-row scratch of the acceptance pass is laid
    out for the capacity, and every decision still matches the oracle."""
    work = dataclasses.replace(parity.tiny_work(), k=4)
    vw, dw, st = parity.tiny_weights(work, seed=12)
    prompts = W.make_prompts(work.verifier.vocab, 2, (17, 38), seed=13)
    rep = parity.run(work, vw, dw, st, prompts, [1.0, 0.7], seed=55, n_steps=6, max_batch=5)
    assert rep.blocks == 12


def test_single_draft_token():
    """k = 1: one draft, two verify rows per sequence, at mixed temperatures."""
    work = dataclasses.replace(parity.tiny_work(), k=1, batch=2)
    vw, dw, st = parity.tiny_weights(work, seed=14)
    prompts = W.make_prompts(work.verifier.vocab, 2, (21, 44), seed=15)
    rep = parity.run(work, vw, dw, st, prompts, [1.0, 0.0], seed=61, n_steps=8)
    assert rep.blocks == 16


def test_prompts_at_block_and_tile_boundaries():
    """Prompts of 1, 16, 64 and 65 tokens: a lone token, one full 16-position cache block, one full
    64-position attention tile, and one position past it."""
    work = dataclasses.replace(parity.tiny_work(), batch=4)
    vw, dw, st = parity.tiny_weights(work, seed=16)
    V = work.verifier.vocab
    prompts = [p[:n] for p, n in zip(W.make_prompts(V, 4, (65, 65), seed=17), (1, 16, 64, 65))]
    rep = parity.run(work, vw, dw, st, prompts, [1.0, 0.7, 0.0, 1.0], seed=62, n_steps=5)
    assert rep.blocks == 20


def test_long_context_many_tiles_grouped_heads():
    """A 300-token prompt (five attention tiles) with 4 query heads per KV head on both models, and
    a capacity far above the context (empty context splits)."""
    base = parity.tiny_work()
    vs = W.shrink(base.verifier, n_kv_heads=1)
    ds = W.shrink(base.drafter, n_kv_heads=1, n_heads=2)
    work = dataclasses.replace(base, verifier=vs, drafter=ds, batch=1)
    vw, dw, st = parity.tiny_weights(work, seed=18)
    prompts = W.make_prompts(vs.vocab, 1, (300, 300), seed=19)
    rep = parity.run(work, vw, dw, st, prompts, [1.0], seed=63, n_steps=4, max_ctx=2048)
    assert rep.blocks == 4


def test_high_acceptance_with_self_drafting():
    """Drafter = verifier with W_s = 0 at T = 0: every block is fully accepted (tau = k + 1)."""
    base = parity.tiny_work()
    work = dataclasses.replace(base, drafter=base.verifier)
    vw = W.make_lm_weights(work.verifier, 11, norm_jitter=0.1)
    st = W.make_steering_weights(work, 12, zero_ws=True)
    prompts = W.make_prompts(work.verifier.vocab, 2, (20, 33), seed=9)
    rep = parity.run(work, vw, vw, st, prompts, [0.0, 0.0], seed=5, n_steps=5)
    assert rep.accepted >= 0.8 * rep.blocks * work.k     # bf16 near-ties may cut a block short


def test_graphs_and_direct_launches_agree():
    work = parity.tiny_work()
    vw, dw, st = parity.tiny_weights(work, seed=4)
    prompts = W.make_prompts(work.verifier.vocab, 2, (30, 40), seed=10)
    outs = []
    for graphs in (True, False):
        dev = [parity.to_device(x) for x in (vw, dw, st)]
        eng = sd2.SD2Engine(work, *dev, max_batch=2, max_ctx=120, max_prefill_tokens=80)
        eng.set_graphs(graphs)
        eng.prefill(prompts, [1.0, 0.0], seed=42)
        toks = []
        for _ in range(6):
            eng.step()
            t, n = eng.accept()
            toks.append((t.cpu().clone(), n.cpu().clone()))
        outs.append(toks)
        eng.close()
    for (ta, na), (tb, nb) in zip(*outs):
        assert torch.equal(na, nb)
        for b in range(2):
            assert torch.equal(ta[b, :na[b]], tb[b, :nb[b]])


def _step_loop(eng, prompts, temps, seed, max_new):
    """One request by sd2_prefill and sd2_step/sd2_accept pairs, tokens gathered on the host."""
    out = [[f] for f in eng.prefill(prompts, temps, seed=seed).cpu().tolist()]
    while any(len(o) < max_new for o in out):
        eng.step()
        t, n = eng.accept()
        t, n = t.cpu(), n.cpu()
        assert int(n.min()) > 0
        for b, o in enumerate(out):
            o.extend(t[b, :n[b]].tolist())
    return [o[:max_new] for o in out]


def test_generate_and_graphs_across_requests():
    """sd2_generate on host buffers equals the prefill/step/accept loop, and a context serving a
    run of requests (same batch with other prompt lengths and seeds, then another batch size, then
    back) gives every request the tokens a fresh context without graphs gives it."""
    work = parity.tiny_work()
    vw, dw, st = parity.tiny_weights(work, seed=6)
    dev = [parity.to_device(x) for x in (vw, dw, st)]
    V = work.verifier.vocab
    requests = [
        (W.make_prompts(V, 2, (30, 40), seed=20), [1.0, 0.0], 101, "generate"),
        (W.make_prompts(V, 2, (12, 47), seed=21), [0.7, 1.0], 102, "loop"),
        (W.make_prompts(V, 1, (25, 25), seed=22), [1.0], 103, "generate"),
        (W.make_prompts(V, 2, (8, 33), seed=23), [1.0, 1.0], 104, "generate"),
    ]
    max_new = 24
    eng = sd2.SD2Engine(work, *dev, max_batch=2, max_ctx=160, max_prefill_tokens=100)
    served = []
    for prompts, temps, seed, how in requests:
        if how == "generate":
            served.append(eng.generate(prompts, temps, seed=seed, max_new=max_new))
        else:
            served.append(_step_loop(eng, prompts, temps, seed, max_new))
    eng.check()
    eng.close()
    for (prompts, temps, seed, _), got in zip(requests, served):
        ref = sd2.SD2Engine(work, *dev, max_batch=2, max_ctx=160, max_prefill_tokens=100)
        ref.set_graphs(False)
        want = _step_loop(ref, prompts, temps, seed, max_new)
        ref.close()
        assert got == want


@pytest.mark.parametrize("temp", [0.0, 1.0])
def test_pretrained_drafter_mode(temp):
    """no_steering: the drafter runs without the steering stage and biases; the oracle with W_s = 0
    (biases exactly zero) is the unsteered drafter, so every logit and decision must match it."""
    work = parity.tiny_work()
    vw, dw, _ = parity.tiny_weights(work, seed=6)
    st0 = W.make_steering_weights(work, 8, std=0.02, ln_jitter=0.1, zero_ws=True)
    prompts = W.make_prompts(work.verifier.vocab, 1, (32, 32), seed=12)
    rep = parity.run(work, vw, dw, st0, prompts, [temp], seed=99, n_steps=6, steering=False)
    assert rep.blocks == 6


@pytest.mark.parametrize("gemm_impl", [0, 1])
def test_after_mlp_steering_site(gemm_impl):
    """The "Inv. Bias after MLP" ablation (Sec. 5): W_s g (d_D wide) added to each drafter layer's
    output, through the residual-adding GEMM epilogue; parity with the oracle's same site."""
    work = parity.tiny_work(steering_site="after_mlp")
    vw, dw, st = parity.tiny_weights(work, seed=9)
    assert st["w_s"].shape[0] == work.drafter.n_layers * work.drafter.d_model
    prompts = W.make_prompts(work.verifier.vocab, 2, (20, 33), seed=13)
    rep = parity.run(work, vw, dw, st, prompts, [1.0, 0.0], seed=17, n_steps=5, gemm_impl=gemm_impl)
    assert rep.blocks == 10


@pytest.mark.parametrize("gemm_impl", [0, 1])
def test_cond_bias_steering_site(gemm_impl):
    """The "Cond. Bias in MLP" ablation (Sec. 5): per row and layer b = W_c2 SiLU(W_c1x f^(l-1) +
    W_c1g g), added as in Eq. 2; parity with the oracle's same site."""
    work = parity.tiny_work(steering_site="cond_mlp")
    vw, dw, st = parity.tiny_weights(work, seed=12)
    assert "w_s" not in st and st["w_c2"].shape[0] == work.drafter.n_layers * work.drafter.d_ffn
    prompts = W.make_prompts(work.verifier.vocab, 2, (18, 30), seed=14)
    rep = parity.run(work, vw, dw, st, prompts, [1.0, 0.0], seed=19, n_steps=5, gemm_impl=gemm_impl)
    assert rep.blocks == 10


def test_stage_timing_keeps_results():
    """Stage event nodes in the captured step change no output; the stage times are positive."""
    work = parity.tiny_work()
    vw, dw, st = parity.tiny_weights(work, seed=5)
    prompts = W.make_prompts(work.verifier.vocab, 2, (30, 40), seed=11)
    outs = []
    for timed in (False, True):
        dev = [parity.to_device(x) for x in (vw, dw, st)]
        eng = sd2.SD2Engine(work, *dev, max_batch=2, max_ctx=120, max_prefill_tokens=80)
        eng.prefill(prompts, [1.0, 0.0], seed=9)
        if timed:
            with pytest.raises(sd2.SD2Error):
                eng.stage_read()                       # nothing timed yet
            eng.stage_timing(True)
        toks = []
        for _ in range(5):
            eng.step()
            t, n = eng.accept()
            toks.append((t.cpu().clone(), n.cpu().clone()))
            if timed:
                ms = eng.stage_read()
                assert ms["steer"] > 0 and ms["draft"] > 0 and ms["verify"] > 0
        outs.append(toks)
        eng.close()
    for (ta, na), (tb, nb) in zip(*outs):
        assert torch.equal(na, nb)
        for b in range(2):
            assert torch.equal(ta[b, :na[b]], tb[b, :nb[b]])


def test_capacity_stop_and_call_order():
    work = parity.tiny_work()
    vw, dw, st = parity.tiny_weights(work)
    dev = [parity.to_device(x) for x in (vw, dw, st)]
    eng = sd2.SD2Engine(work, *dev, max_batch=1, max_ctx=48, max_prefill_tokens=64)
    with pytest.raises(sd2.SD2Error, match="ESTATE"):
        eng.step()
    with pytest.raises(sd2.SD2Error, match="ECAPACITY"):
        eng.prefill([list(range(60))], [1.0], seed=1)
    eng.prefill([list(range(30))], [1.0], seed=1)
    with pytest.raises(sd2.SD2Error, match="ESTATE"):
        eng.accept()
    total = 0
    stopped = False
    for _ in range(24):
        eng.step()
        _, n = eng.accept()
        m = int(n.cpu()[0])
        total += m
        if m == 0:
            stopped = True
            break
    assert stopped
    state = eng.buffer(sd2.BUF_STATE).view(4, -1)[:, 0].cpu()
    assert int(state[3]) == 1 and int(state[0]) + work.k + 1 > 48 and int(state[0]) <= 48
    eng.check()
    eng.close()


def test_standalone_steering_and_swiglu():
    work = W.WORKLOADS["tiny"]
    st = W.make_steering_weights(work, 3, ln_jitter=0.2)
    taps = W.make_taps(5, work.verifier.d_model, seed=4)
    nb = work.drafter.n_layers * work.drafter.d_ffn
    g, bias = sd2.steer(taps.cuda(), parity.to_device(st), work.steer_ln_eps, nb)
    g_ref = steering.steering_vector(taps, st, work.steer_ln_eps)
    b_ref = steering.steering_bias(g_ref, st, work.drafter.n_layers, work.drafter.d_ffn).reshape(5, -1)
    assert parity.row_rel_err(g, g_ref) < parity.TOL
    assert parity.row_rel_err(bias, b_ref) < parity.TOL
    gen = torch.Generator().manual_seed(1)
    gate, up = torch.randn(7, 96, generator=gen), torch.randn(7, 96, generator=gen)
    bb = torch.randn(3, 96, generator=gen)
    seq = torch.tensor([0, 1, 2, 0, 1, 2, 2], dtype=torch.int32)
    h = sd2.swiglu_steered(gate.cuda(), up.cuda(), bb.cuda(), seq.cuda())
    ref = (up + bb[seq.long()]) * omodel.silu(gate)
    assert parity.row_rel_err(h, ref) < 1e-2


@pytest.mark.parametrize("B", [37, 256])
def test_standalone_steering_full_width(B):
    """The steering step at the Qwen pair's widths (d_v 5120 -> d_g 896, 24 x 4864 biases) for 37 and
    256 sequences: both projections on the tensor cores, with ragged and full-width token tiles."""
    work = W.WORKLOADS["qwen32b_05b"]
    st = W.make_steering_weights(work, 5)
    taps = W.make_taps(B, work.verifier.d_model, seed=6)
    nb = work.drafter.n_layers * work.drafter.d_ffn
    g, bias = sd2.steer(taps.cuda(), parity.to_device(st), work.steer_ln_eps, nb)
    g_ref = steering.steering_vector(taps, st, work.steer_ln_eps)
    b_ref = steering.steering_bias(g_ref, st, work.drafter.n_layers, work.drafter.d_ffn).reshape(B, -1)
    assert parity.row_rel_err(g, g_ref) < parity.TOL
    assert parity.row_rel_err(bias, b_ref) < parity.TOL
