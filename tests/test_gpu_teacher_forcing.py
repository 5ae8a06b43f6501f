"""Teacher forcing (the paper's RQ1 method, Section 4): whole sentences of the
workload grammars are fed token by token through the device path (psc_fill_mask
then psc_advance); every token of a sentence must be in the row's mask and the
end-of-sequence token must be allowed at its end.  Sentences with one foreign
token spliced in must be stopped exactly where the oracle stops them."""
from __future__ import annotations

import numpy as np
import pytest

from oracle import Oracle
from workloads import configs, teacher

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


def first_rejection_oracle(o, w, ids):
    """Index of the first token (len(ids) = the end of sequence) the oracle's
    mask excludes, or -1 when the whole sentence and its end are allowed."""
    c = o.initial()
    for i, v in enumerate(ids):
        if not o.allowed(c, w.vocab[v]):
            return i
        o.advance(c, w.vocab[v])
    return -1 if o.allowed(c, None) else len(ids)


def first_rejection_device(psc, h, w, seqs):
    B = len(seqs)
    T = max(len(s) for s in seqs) + 1
    tokm = np.full((B, T), -1, dtype=np.int32)
    for b, s in enumerate(seqs):
        tokm[b, :len(s)] = s
        tokm[b, len(s)] = w.eos_id
    st = psc.psc_state_init(h, B, 256)
    bm = torch.empty(B, h.W, dtype=torch.int32, device="cuda")
    first = np.full(B, -1, dtype=np.int64)
    for j in range(T):
        psc.psc_fill_mask(h, st, bm)
        col = tokm[:, j]
        m = bm.cpu().numpy().view(np.uint32)
        for b in range(B):
            v = int(col[b])
            if v >= 0 and first[b] < 0 and not ((m[b, v >> 5] >> (v & 31)) & 1):
                first[b] = j
        psc.psc_advance(h, st, torch.from_numpy(np.where(first < 0, col, -1).astype(np.int32)).cuda())
    return first


@pytest.mark.parametrize("cfg_id", [2, 3, 4])
def test_teacher_forcing(psc, cfg_id):
    w = configs.load(cfg_id, batch=1)
    ts = teacher.teacher_set(w, 32)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    o = Oracle(w.grammar_text)
    pos = first_rejection_device(psc, h, w, ts.positives)
    assert (pos == -1).all(), f"valid sentences masked at {np.nonzero(pos >= 0)[0][:8]}"
    neg = first_rejection_device(psc, h, w, ts.negatives)
    want = np.array([first_rejection_oracle(o, w, s) for s in ts.negatives])
    np.testing.assert_array_equal(neg, want)
    # a rejection never comes before the spliced-in token
    assert all(r < 0 or r >= k for r, k in zip(neg, ts.inserted_at))
