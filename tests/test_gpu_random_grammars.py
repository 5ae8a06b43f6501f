"""Device path against the oracle on seeded random small grammars (shapes the
five workloads lack: literals colliding with regex terminals, ignored
whitespace, empty alternatives, recursion, both lexer modes).

For every grammar the library compiles, a batch of rows is driven on the
device by psc_advance with tokens drawn from the oracle's masks (so rows walk
through the configurations the grammar reaches), and after every step:
psc_fill_mask equals the oracle's masks, psc_fill_apply masks seeded logits
exactly as the oracle's masks say (with the bitmask copy), and the statuses
psc_advance reports equal the oracle's.  Every advance table path runs: dense
tables staged in shared memory, packed tables staged in shared memory, tables
read from global memory.
"""
from __future__ import annotations

import numpy as np
import pytest

from oracle import Oracle, Vocab

from ._random_grammars import random_grammar, random_vocab

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


def _masked(raw, allowed):
    out = raw.copy()
    out[~allowed] = np.int32(-8388608)    # f32 -inf
    return out


def _drive(psc, h, text, vocab, rng, seed, B=16, steps=6):
    """Rows driven by psc_advance with tokens drawn from the oracle's masks; after
    every step the device masks, masked logits and statuses equal the oracle's.
    Returns the number of configurations compared."""
    eos = len(vocab) - 1
    o = Oracle(text)
    voc = Vocab.from_list(vocab, eos)
    V = len(vocab)
    st = psc.psc_state_init(h, B, 64)
    ocs = [o.initial() for _ in range(B)]
    bm = torch.empty(B, h.W, dtype=torch.int32, device="cuda")
    bm2 = torch.empty_like(bm)
    stat = torch.empty(B, dtype=torch.int32, device="cuda")
    seen = 0
    for step in range(steps):
        want = o.masks(ocs, voc, threads=1)
        psc.psc_fill_mask(h, st, bm)
        np.testing.assert_array_equal(bm.cpu().numpy().view(np.uint32), want, err_msg=text)
        allowed = np.unpackbits(want.view(np.uint8), axis=-1, bitorder="little")[:, :V].astype(bool)
        logits = torch.randn(B, V, generator=torch.Generator().manual_seed(seed * 100 + step))
        x = logits.cuda()
        psc.psc_fill_apply(h, st, x, bm2)
        np.testing.assert_array_equal(x.cpu().view(torch.int32).numpy(),
                                      _masked(logits.view(torch.int32).numpy(), allowed), err_msg=text)
        np.testing.assert_array_equal(bm2.cpu().numpy().view(np.uint32), want, err_msg=text)
        seen += B
        tok = np.full(B, -1, dtype=np.int32)
        for r in range(B):
            idx = np.nonzero(allowed[r])[0]
            if len(idx):
                tok[r] = int(rng.choice(idx))
        psc.psc_advance(h, st, torch.from_numpy(tok).cuda(), stat)
        s = stat.cpu().numpy()
        for r in range(B):
            if tok[r] >= 0:
                ost = o.advance(ocs[r], None if tok[r] == eos else vocab[tok[r]])
                assert s[r] == {0: psc.ROW_OK, 1: psc.ROW_DONE, 2: psc.ROW_REJECTED}[ost], (text, r)
    return seen


@pytest.mark.parametrize("tables", ["staged", "global", "packed"])
def test_random_grammars_device_matches_the_oracle(psc, tables):
    rng = np.random.default_rng({"staged": 77, "global": 78, "packed": 79}[tables])
    done, modes, configs_seen = 0, set(), 0
    while done < 40:
        text, vocab = random_grammar(rng, True), random_vocab(rng, True)
        if text is None:
            continue
        eos = len(vocab) - 1
        try:
            h = psc.psc_compile(text, vocab, eos, global_tables=tables == "global",
                                packed_tables=tables == "packed")
        except psc.PscError as e:
            assert e.code == 3, (text, str(e))        # only LALR(1) conflicts are expected
            continue
        assert (h.info().advance_table_bytes > 0) == (tables != "global")
        assert h.info().advance_tables_packed == (tables == "packed")
        modes.add("contextual" if "%lexer contextual" in text else "basic")
        configs_seen += _drive(psc, h, text, vocab, rng, done)
        done += 1
    assert modes == {"basic", "contextual"} and configs_seen >= 40 * 16 * 6


# a rule of 19 symbols: too long for reduce entries that carry the rule's length in 4 bits,
# so the staged advance reads rule lengths and left-hand sides from their own tables
LONG_SEQ = b"()[]+-*/%&|^!~?:<>;"
LONG_RULE = ('start: | start stmt\n'
             'stmt: ' + " ".join(f'"{chr(c)}"' for c in LONG_SEQ) + ' | ID "=" NUM ";" | "{" start "}"\n'
             'ID: /[a-z]+/\nNUM: /[0-9]+/\nWS: / +/\n%ignore WS\n%lexer contextual\n')


@pytest.mark.parametrize("tables", ["staged", "global", "packed"])
def test_long_rules_without_packed_reduce_entries(psc, tables):
    """A grammar with a 19-symbol rule through every advance table path; rows are
    driven by the oracle's masks through many reductions of the long rule (its
    symbols come one or a few per token, in order)."""
    rng = np.random.default_rng(4242)
    vocab = {bytes([c]) for c in LONG_SEQ + b"xyz=019{} "}
    for n in (2, 3, 5):
        vocab |= {LONG_SEQ[i:i + n] for i in range(len(LONG_SEQ) - n + 1)}
    vocab |= {b"x = 1;", b"= 12;", b"}{", b"{(", b";{", b";}", b"  "}
    vocab = sorted(vocab) + [b""]
    h = psc.psc_compile(LONG_RULE, vocab, len(vocab) - 1, global_tables=tables == "global",
                        packed_tables=tables == "packed")
    assert h.info().advance_tables_packed == (tables == "packed")
    assert _drive(psc, h, LONG_RULE, vocab, rng, 7, B=32, steps=40) == 32 * 40
