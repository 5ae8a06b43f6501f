"""psc_fill_apply_noalloc: the allocation-free variant of psc_fill_apply.

Callers that cannot allocate device memory at the point of the call (inside a
CUDA graph capture, under a framework allocator that owns all memory, or in a
loop where an allocation could synchronise the device) pass their own state
arrays; the per-row scratch lives in a fixed array inside the library.  This
file checks, through the C ABI, that two calls in a row give bit-for-bit the
masked logits and bitmask of psc_fill_apply on the same states.  It is named
to be collected last.
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


def _device_copy_of_states(psc, st):
    d = psc.psc_states_download(st)
    q = torch.from_numpy(d["q"]).cuda()
    depth = torch.from_numpy(d["depth"]).cuda()
    status = torch.from_numpy(d["status"]).cuda()
    stack = torch.from_numpy(d["stack"].view(np.int16)).cuda()
    return q, depth, status, stack


def _bits(t):
    t = t.cpu()
    return t.view(torch.int16 if t.dtype == torch.bfloat16 else torch.int32).numpy()


@pytest.mark.parametrize("cfg_id,pad,with_bitmask", [(2, 0, True), (1, 0, True), (2, 40, False), (1, 7, True)])
def test_noalloc_matches_fill_apply_on_two_calls(psc, cfg_id, pad, with_bitmask):
    """Two calls in a row, each against psc_fill_apply on the same states: bf16
    (config 2) and f32 (config 1) logits, rows padded past V (row stride > V,
    columns >= V untouched), with and without the bitmask copy.  psc_fill_apply
    classifies through the states object's kept bottom-up blocks; the no-alloc
    call has none and walks the classifier DFA from the stack top, so the
    comparison also checks those two classifications against each other."""
    w = configs.load(cfg_id)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    st = psc.psc_state_init(h, w.B, 64)
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(h, st, tm[:, j].contiguous())
    tok = torch.empty(w.B, dtype=torch.int32, device="cuda")
    for call in range(2):
        base = w.logits(call + 20)
        padded = torch.cat([base, base[:, :pad]], dim=1) if pad else base
        logits = padded.cuda()
        a, b = logits.clone(), logits.clone()
        av, bv = a[:, :w.V], b[:, :w.V]          # row stride V + pad
        bm_a = torch.zeros(w.B, h.W, dtype=torch.int32, device="cuda")
        bm_b = torch.full((w.B, h.W), -1, dtype=torch.int32, device="cuda") if with_bitmask else None
        q, depth, status, stack = _device_copy_of_states(psc, st)
        psc.psc_fill_apply(h, st, av, bm_a)
        psc.psc_fill_apply_noalloc(h, q, depth, status, stack, bv, bm_b)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(_bits(b), _bits(a))
        np.testing.assert_array_equal(_bits(b)[:, w.V:], _bits(logits)[:, w.V:])
        if with_bitmask:
            np.testing.assert_array_equal(bm_b.cpu().numpy(), bm_a.cpu().numpy())
        # move the batch on by one greedy step before the second call
        psc.psc_argmax_masked(h, st, av, tok)
        psc.psc_advance(h, st, tok)
    torch.cuda.synchronize()


def test_noalloc_rejects_batches_above_the_scratch_size(psc):
    w = configs.load(1)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    B = psc.NOALLOC_MAX_ROWS + 1
    q = torch.zeros(B, dtype=torch.int32, device="cuda")
    stack = torch.zeros(B, 4, dtype=torch.int16, device="cuda")
    x = torch.zeros(1, w.V, device="cuda").expand(B, w.V)   # row stride 0: nothing is read
    with pytest.raises(psc.PscError) as e:
        psc.psc_fill_apply_noalloc(h, q, q, q, stack, x)
    assert e.value.code == 5 and "PSC_NOALLOC_MAX_ROWS" in str(e.value)
