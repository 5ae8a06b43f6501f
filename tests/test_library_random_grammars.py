"""Differential test of the whole offline construction on seeded random small
grammars: the library's compiled tables (its own grammar reader, lexer DFA,
LALR(1) tables, classifier and bottom-up classifier) against the oracle (its
own reader, Thompson-NFA lexer, canonical LR(1) parser and per-token brute
force), on the configurations a random vocabulary reaches in up to 5 tokens
(small grammars) or 6 tokens (the larger variant), at most 200 / 400 of them.

Grammars mix literals with two regex terminals that collide with them (so
lexemes form classes), ignored whitespace, empty alternatives and recursion,
in both lexer modes.  Grammars with an LALR(1) conflict are refused by the
library (PSC_ERR_CONFLICT) and skipped.
"""
from __future__ import annotations

import numpy as np
import pytest

from oracle import ST_OK, Oracle, Vocab

from ._random_grammars import random_grammar, random_vocab


@pytest.fixture(scope="module")
def psc():
    from paper_2608_03065_gb300 import build, psc as mod
    build.build()
    mod.load()
    return mod


@pytest.mark.parametrize("large,draws,depth,keep", [(False, 600, 5, 200), (True, 1500, 6, 400)])
def test_random_grammars_compiled_tables_match_the_oracle(psc, large, draws, depth, keep):
    rng = np.random.default_rng(20261202 + large)
    compared = configs_checked = 0
    for _ in range(draws):
        text = random_grammar(rng, large)
        vocab = random_vocab(rng, large)
        if text is None:
            continue
        eos = len(vocab) - 1
        try:
            h = psc.psc_compile(text, vocab, eos, host_only=True)
        except psc.PscError as e:
            assert e.code == 3, (text, str(e))   # only LALR(1) conflicts are expected
            continue
        o = Oracle(text)
        voc = Vocab.from_list(vocab, eos)
        seen = {}
        frontier = [((), h.host_initial())]
        for _ in range(depth):
            nxt = []
            for seq, c in frontier:
                for v in range(eos):
                    c2 = h.host_advance(c, v, cap=256)
                    key = (c2["q"], tuple(c2["stack"]))
                    if c2["status"] == psc.ROW_OK and key not in seen and len(seen) < keep:
                        seen[key] = seq + (v,)
                        nxt.append((seq + (v,), c2))
            frontier = nxt
        cfgs, ocs = [h.host_initial()], [o.initial()]
        for (q, stack), seq in seen.items():
            oc = o.initial()
            assert o.advance_tokens(oc, voc, seq) == ST_OK, (text, seq)   # same reachable prefixes
            cfgs.append({"q": q, "stack": list(stack), "status": psc.ROW_OK})
            ocs.append(oc)
        om = o.masks(ocs, voc, threads=1)
        for c, m in zip(cfgs, om):
            mid = h.host_classify(c["q"], c["stack"])
            np.testing.assert_array_equal(h.host_mask_row(mid), m, err_msg=f"{text}\n{c}")
            assert h.host_classify_bottom_up(c["q"], c["stack"]) == mid, (text, c)
        compared += 1
        configs_checked += len(cfgs)
    assert compared > 200 and configs_checked > 2000
