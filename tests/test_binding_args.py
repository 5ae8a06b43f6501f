"""The Python binding refuses wrongly shaped arguments before any call reaches
the library (so before any kernel launch): no GPU is needed to check it."""
from __future__ import annotations

import pytest

torch = pytest.importorskip("torch")


@pytest.fixture()
def psc():
    from paper_2608_03065_gb300 import psc as mod
    return mod


def _states(B=4, cap=8):
    q = torch.zeros(B, dtype=torch.int32)
    stack = torch.zeros(B, cap, dtype=torch.int16)
    return q, q.clone(), q.clone(), stack


@pytest.mark.parametrize("shape", [(4, 15), (3, 16), (4, 17), (16, 4)])
def test_noalloc_bitmask_of_the_wrong_shape_is_refused(psc, shape):
    h = psc.Handle(0, 512)                       # W = 16; never reaches the library
    q, depth, status, stack = _states()
    logits = torch.zeros(4, 512)
    with pytest.raises(ValueError, match="bitmask_out"):
        psc.psc_fill_apply_noalloc(h, q, depth, status, stack, logits, torch.zeros(shape, dtype=torch.int32))


def test_noalloc_non_contiguous_bitmask_is_refused(psc):
    h = psc.Handle(0, 512)
    q, depth, status, stack = _states()
    bm = torch.zeros(16, 4, dtype=torch.int32).t()   # [4, 16] but not contiguous
    with pytest.raises(ValueError, match="bitmask_out"):
        psc.psc_fill_apply_noalloc(h, q, depth, status, stack, torch.zeros(4, 512), bm)


def test_noalloc_stack_and_logits_shapes_are_checked(psc):
    h = psc.Handle(0, 512)
    q, depth, status, stack = _states()
    with pytest.raises(ValueError, match="stack"):
        psc.psc_fill_apply_noalloc(h, q, depth, status, stack[:3], torch.zeros(4, 512))
    with pytest.raises(ValueError, match="logits"):
        psc.psc_fill_apply_noalloc(h, q, depth, status, stack, torch.zeros(4, 511))
    with pytest.raises(ValueError, match="logits"):
        psc.psc_fill_apply_noalloc(h, q, depth, status, stack, torch.zeros(4 * 512))
