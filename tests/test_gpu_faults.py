"""Fault reporting of the bounded in-kernel waits, without any fault.

Every wait in the kernels is bounded; one that gives up is counted on the
states object it worked for (psc_state_faults).  psc_check_wait runs the same
bounded wait on an mbarrier phase that nothing completes, so the wait gives up
after its limit: the count rises, the device stays usable, and the process-wide
pipeline-fault count (psc_info().device_timeouts) is untouched.  Decoding on a
healthy device records no fault.
"""
from __future__ import annotations

import numpy as np
import pytest

from workloads import configs

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def psc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_03065_gb300 import build, psc as mod
    build.build()
    mod.load()
    return mod


def test_a_wait_that_gives_up_is_counted_on_the_states(psc):
    w = configs.load(2, batch=8)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    st = psc.psc_state_init(h, w.B, 64)
    other = psc.psc_state_init(h, w.B, 64)
    assert psc.psc_state_faults(st) == 0
    timeouts0 = h.info().device_timeouts
    psc.psc_check_wait(st, 4096)
    assert psc.psc_state_faults(st) == 1
    psc.psc_check_wait(st, 1)
    psc.psc_check_wait(st, 1 << 12)
    assert psc.psc_state_faults(st, reset=True) == 3
    assert psc.psc_state_faults(st) == 0
    assert psc.psc_state_faults(other) == 0            # counted on the states object it worked for
    assert h.info().device_timeouts == timeouts0      # not a pipeline fault of the process
    with pytest.raises(psc.PscError):
        psc.psc_check_wait(st, 0)
    # the device is still usable: a decode step runs and records no fault
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(h, st, tm[:, j].contiguous())
    x = w.logits(1).cuda()
    tok = torch.empty(w.B, dtype=torch.int32, device="cuda")
    psc.psc_decode_step(h, st, x, tok)
    torch.cuda.synchronize()
    assert (tok.cpu().numpy() >= 0).all()
    assert psc.psc_state_faults(st) == 0


def test_decoding_records_no_fault(psc):
    w = configs.load(3, batch=32)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    st = psc.psc_state_init(h, w.B, 256)
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(h, st, tm[:, j].contiguous())
    tok = torch.empty(w.B, dtype=torch.int32, device="cuda")
    for i in range(6):
        psc.psc_decode_step_mask(h, st, w.logits(40 + i).cuda())
        psc.psc_decode_step_advance(h, st, tok)
    torch.cuda.synchronize()
    assert psc.psc_state_faults(st) == 0
    assert np.isin(psc.psc_states_download(st)["status"], [psc.ROW_OK, psc.ROW_DONE]).all()
