"""The seeded input recipe of the five workloads: sizes, vocabulary structure,
prefix lengths and tokenization, logits distribution, and determinism (every
input is a pure function of the config id and its seed streams)."""
from __future__ import annotations

import numpy as np
import pytest

from workloads import configs

torch = pytest.importorskip("torch")

SINGLES = {bytes([b]) for b in list(range(0x20, 0x7F)) + [9, 10, 13]}


@pytest.mark.parametrize("cfg_id,batch", [(1, None), (2, None), (3, 16), (4, 16), (5, 16), (6, 16), (7, 16),
                                          (8, 16)])
def test_vocabulary_and_prefixes(cfg_id, batch):
    w = configs.load(cfg_id, batch=batch)
    s = configs.SPECS[cfg_id]
    assert len(w.vocab) == s.V == w.V
    assert w.eos_id == s.V - 1 and w.vocab[w.eos_id] == b""
    assert len(set(w.vocab)) == s.V                          # unique strings
    assert SINGLES <= set(w.vocab)                           # every prefix is tokenizable
    assert max(len(t) for t in w.vocab) <= s.vocab_max_len
    assert all(len(t) >= 1 for t in w.vocab[:-1])
    assert len(w.prefixes) == len(w.prefix_ids) == w.B == (batch or s.B)
    for p, ids in zip(w.prefixes, w.prefix_ids):
        assert s.prefix_min <= len(p) <= s.prefix_max        # the drawn length, never a shorter sentence
        assert b"".join(w.vocab[i] for i in ids) == p        # greedy tokenization is exact
        assert w.eos_id not in ids
    m = w.token_matrix()
    assert m.shape[0] == w.B and m.dtype == np.int32


def test_pretokenized_vocabulary_follows_the_splitting_rule():
    """Workload 7's tokens are each one pre-token of the byte-level BPE splitting
    rule (single bytes aside): no token mixes letters with punctuation, numbers
    have at most three digits; about 3 % are punctuation runs, the structure
    that makes a token span several grammar symbols."""
    import re
    from workloads import sample
    w = configs.load(7, batch=16)
    toks = [t for t in w.vocab[:-1] if len(t) > 1]
    assert all(sample.PRETOKEN.fullmatch(t) for t in toks)
    assert not any(re.search(rb"[A-Za-z][^A-Za-z]|[0-9][^0-9]", t) for t in toks)
    assert not any(re.fullmatch(rb"[0-9]{4,}", t) for t in toks)
    punct = [t for t in toks if re.fullmatch(rb" ?[!-/:-@\[-`{-~]+\n*", t)]
    assert 0.02 * w.V < len(punct) < 0.06 * w.V
    assert {b");", b"()", b" {"} <= set(toks) | set(w.vocab)
    assert configs.vocab_for(7, 4096)[:-1] != w.vocab[:4095]   # the size is part of the recipe


@pytest.mark.parametrize("cfg_id", [1, 2])
def test_prefix_lengths_are_uniform_over_the_range(cfg_id):
    """Prefix lengths are drawn uniformly in [prefix_min, prefix_max] (a sentence
    that ends before its drawn length is drawn again): the lengths spread over the
    whole range instead of piling up at the short sentences."""
    w = configs.load(cfg_id)
    s = configs.SPECS[cfg_id]
    L = np.array([len(p) for p in w.prefixes])
    lo, hi = s.prefix_min, s.prefix_max
    assert np.quantile(L, 0.75) > lo + 0.5 * (hi - lo)
    assert np.quantile(L, 0.25) < lo + 0.5 * (hi - lo)


def test_inputs_are_deterministic():
    a, b = configs.load(2, batch=8), configs.load(2, batch=8)
    assert a.vocab == b.vocab and a.prefixes == b.prefixes and a.prefix_ids == b.prefix_ids
    x, y = a.logits(3), b.logits(3)
    assert torch.equal(x.view(torch.int16), y.view(torch.int16))
    assert not torch.equal(a.logits(3).float(), a.logits(4).float())   # fresh logits per step


@pytest.mark.parametrize("cfg_id", [1, 2])
def test_logits_distribution(cfg_id):
    """fp32 N(0,1) for config 1; bf16 N(0,2) (variance 2) for the others."""
    w = configs.load(cfg_id, batch=8)
    x = w.logits(0)
    assert tuple(x.shape) == (w.B, w.V)
    assert x.dtype == (torch.float32 if cfg_id == 1 else torch.bfloat16)
    v = x.float().var().item()
    want = 1.0 if cfg_id == 1 else 2.0
    assert abs(v - want) < 0.1 * want
    assert abs(x.float().mean().item()) < 0.05 * want ** 0.5
