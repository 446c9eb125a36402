"""Failure detection on the GPU without a fault (nothing traps, hangs or touches bad memory):

* an allocation failure injected at several points of sd2_init returns SD2_ENOMEM and leaves no
  device memory behind; a context made afterwards works;
* a bounded device wait that nothing satisfies, with a short budget set by the test, gives up,
  latches the time-out and returns: sd2_check reports SD2_ETIMEOUT, and the context goes on to
  produce exactly the tokens of a context that never saw it.
"""
import pytest
import torch

import parity
from paper_2511_09844_gb300 import sd2
from paper_2511_09844_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _engine(work, dev_w, max_ctx=256):
    return sd2.SD2Engine(work, *dev_w, max_batch=2, max_ctx=max_ctx, max_prefill_tokens=64)


def test_injected_allocation_failures_leave_nothing_allocated():
    lib = sd2.load_library()
    work = parity.tiny_work()
    dev_w = [parity.to_device(w) for w in parity.tiny_weights(work)]
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for after in (1, 4, 11, 23, 37):
        lib.sd2_debug_fail_alloc(after)
        try:
            with pytest.raises(sd2.SD2Error) as e:
                _engine(work, dev_w, max_ctx=4096)      # 16 MB of verifier KV pool: a leak would show
        finally:
            lib.sd2_debug_fail_alloc(-1)
        assert e.value.status == sd2.SD2_ENOMEM and "injected" in str(e.value)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free0 - free1 < 8 * 2 ** 20, (free0, free1)
    eng = _engine(work, dev_w)
    prompts = W.make_prompts(work.verifier.vocab, 2, (20, 30), seed=3)
    eng.prefill(prompts, [1.0, 0.0], seed=5)
    eng.step()
    eng.accept()
    eng.check()
    eng.close()


def _tokens(eng, n_steps, probe_after=None):
    lib = sd2.load_library()
    out = []
    for i in range(n_steps):
        if i == probe_after:
            assert lib.sd2_debug_expire_wait(eng.ctx, 200000) == sd2.SD2_OK      # ~0.1 ms budget
            with pytest.raises(sd2.SD2Error) as e:
                eng.check()
            assert e.value.status == sd2.SD2_ETIMEOUT
            eng.check()                                                       # the word was cleared
        eng.step()
        tok, n = eng.accept()
        tok, n = tok.cpu(), n.cpu()
        out.append([tok[b, :int(n[b])].tolist() for b in range(tok.shape[0])])
    eng.check()
    return out


def test_bounded_wait_expiry_is_reported_and_the_context_stays_usable():
    work = parity.tiny_work()
    dev_w = [parity.to_device(w) for w in parity.tiny_weights(work)]
    prompts = W.make_prompts(work.verifier.vocab, 2, (20, 30), seed=4)
    runs = []
    for probe in (None, 1):
        eng = _engine(work, dev_w)
        eng.prefill(prompts, [1.0, 0.7], seed=6)
        runs.append(_tokens(eng, 4, probe))
        eng.close()
    assert runs[0] == runs[1]
