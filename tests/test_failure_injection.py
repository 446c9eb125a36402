"""Failure detection without a GPU fault, host side: an allocation failure injected into the
context's device-allocation wrapper surfaces as SD2_ENOMEM from sd2_init, with nothing left
allocated. The first allocation is the one made to fail here, so no CUDA call is reached and the
test runs on a machine without a GPU."""
import pytest

import parity
from paper_2511_09844_gb300 import sd2


class _NoStream:
    cuda_stream = 0


def test_injected_allocation_failure_returns_enomem_on_the_host():
    lib = sd2.load_library()
    work = parity.tiny_work()
    vw, dw, st = parity.tiny_weights(work)          # host tensors: only their addresses are read
    lib.sd2_debug_fail_alloc(0)
    try:
        with pytest.raises(sd2.SD2Error) as e:
            sd2.SD2Engine(work, vw, dw, st, max_batch=1, max_ctx=64, max_prefill_tokens=32, stream=_NoStream())
    finally:
        lib.sd2_debug_fail_alloc(-1)
    assert e.value.status == sd2.SD2_ENOMEM
    assert "injected" in str(e.value)
    assert b"injected" in lib.sd2_last_error(None)


def test_hook_disarms_after_firing():
    lib = sd2.load_library()
    work = parity.tiny_work()
    vw, dw, st = parity.tiny_weights(work)
    lib.sd2_debug_fail_alloc(0)
    for _ in range(2):     # first: the injected failure; second: nothing injected (the host checks pass,
        try:               # then the real allocation needs a device, which this machine may not have)
            sd2.SD2Engine(work, vw, dw, st, max_batch=1, max_ctx=64, max_prefill_tokens=32, stream=_NoStream())
        except sd2.SD2Error as e:
            msg = str(e)
        else:
            msg = ""
        if _ == 0:
            assert "injected" in msg
        else:
            assert "injected" not in msg
