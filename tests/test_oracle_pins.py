"""Pins for the CPU oracle: it is checked against things other than itself.

* hand-enumerated masks (tests/golden/arith_micro_masks.txt, json_micro_masks.txt);
* closed forms: balanced parentheses, a single literal, any byte string;
* Eq. (1) by brute force: search for completions y with x v y in the language;
* an independent parser: Python lexer + Earley recognizer vs the C lexer + LR(1);
* the regex reader against Python's ``re``;
* the contextual-lexer reading (keywords usable as names where only a name fits;
  resolution by the LALR(1) state's action set);
* invariants: teacher-forced prefixes are never masked, allowed tokens are
  prefix-closed, reachable states have non-empty masks, rows are independent.
"""
from __future__ import annotations

import itertools
import os
import re

import numpy as np
import pytest

from oracle import ST_DONE, ST_ERROR, ST_OK, Oracle, Vocab
from oracle.grammar_spec import GrammarError, parse_grammar
from oracle.regex_thompson import build_lexer_nfa, matches
from workloads import configs, grammars
from workloads.sample import SentenceSampler, TrieTokenizer

from ._lexref import PyCheck

HERE = os.path.dirname(os.path.abspath(__file__))
ARITH = grammars.arithmetic().text()
MICRO = [b"1", b"12", b"a", b"ab", b"+", b"(", b")", b" ", b"+(", b"a1", b""]


def _cfg(o: Oracle, vocab: Vocab, prefix: bytes):
    cf = o.initial()
    toks = [vocab.token(v) for v in range(vocab.V) if v != vocab.eos_id]
    ids = TrieTokenizer(toks + [b""]).encode(prefix) if prefix else []
    st = o.advance_tokens(cf, vocab, ids)
    return cf, st


def _bits(row: np.ndarray, V: int) -> set[int]:
    return {v for v in range(V) if (int(row[v >> 5]) >> (v & 31)) & 1}


# ------------------------------------------------------------------ golden
def test_golden_hand_enumerated_masks():
    o = Oracle(ARITH)
    voc = Vocab.from_list(MICRO, eos_id=10)
    n = 0
    with open(os.path.join(HERE, "golden", "arith_micro_masks.txt")) as f:
        for line in f:
            if not line.strip() or line.startswith("#"):
                continue
            m = re.match(r'"(.*)"\s+([\d,]+)', line.strip())
            prefix, allowed = m.group(1).encode(), {int(x) for x in m.group(2).split(",")}
            cf, st = _cfg(o, voc, prefix)
            assert st == ST_OK
            assert o.mask_set(cf, voc) == allowed, prefix
            n += 1
    assert n == 7


JSON_MICRO = [b"{", b"}", b'"a"', b'"', b":", b"1", b"0", b".5", b"-", b"e", b"tr", b"true", b",", b" ", b"\\",
              b"]", b"[", b'"a":', b""]


def test_golden_json_micro_masks():
    """Hand-enumerated masks on the JSON grammar: number lexing with one byte of
    lookahead, string escapes, ignored whitespace, the end-of-sequence rule."""
    o = Oracle(grammars.json_grammar().text())
    voc = Vocab.from_list(JSON_MICRO, eos_id=18)
    n = 0
    with open(os.path.join(HERE, "golden", "json_micro_masks.txt")) as f:
        for line in f:
            if not line.strip() or line.startswith("#"):
                continue
            m = re.match(r'"(.*)"\s+([\d,]+)$', line.strip())
            prefix, allowed = m.group(1).encode(), {int(x) for x in m.group(2).split(",")}
            cf, st = _cfg(o, voc, prefix)
            assert st == ST_OK, prefix
            assert o.mask_set(cf, voc) == allowed, (prefix, sorted(o.mask_set(cf, voc)))
            n += 1
    assert n == 13


# -------------------------------------------------------------- closed forms
DYCK = 'start: s\ns: | s "(" s ")"\n'


def test_closed_form_balanced_parentheses_deep():
    """Tokens over ( and ): allowed iff the running depth never drops below 0;
    end of sequence iff the depth is 0.  Depths up to 300 exercise deep stacks."""
    o = Oracle(DYCK)
    toks = [bytes(p) for n in range(1, 5) for p in itertools.product(b"()", repeat=n)]
    voc = Vocab.from_list(toks + [b""], eos_id=len(toks))
    rng = np.random.default_rng(0)
    for depth_target in [0, 1, 2, 7, 64, 300]:
        # a prefix of the given final depth with some balanced noise in it
        parts = []
        for _ in range(depth_target):
            parts.append(b"(" + (b"()" if rng.random() < 0.3 else b""))
        prefix = b"".join(parts)
        cf = o.initial()
        for ch in prefix:
            assert o.advance(cf, bytes([ch])) == ST_OK
        d = depth_target
        expect = set()
        for v, t in enumerate(toks):
            run, ok = d, True
            for ch in t:
                run += 1 if ch == ord("(") else -1
                ok &= run >= 0
            if ok:
                expect.add(v)
        if d == 0:
            expect.add(voc.eos_id)
        assert o.mask_set(cf, voc) == expect, depth_target


def test_closed_form_single_literal():
    """One literal S: after S[:i], v is allowed iff S[i:] starts with v; EOS iff i = |S|."""
    S = b"hello world"
    o = Oracle('start: "hello world"\n')
    subs = sorted({S[i:j] for i in range(len(S)) for j in range(i + 1, len(S) + 1)})
    toks = subs + [b"x", b"hello world!", b"dd", b"oo"]
    voc = Vocab.from_list(toks + [b""], eos_id=len(toks))
    for i in range(len(S) + 1):
        cf = o.initial()
        if i:
            assert o.advance(cf, S[:i]) == ST_OK
        expect = {v for v, t in enumerate(toks) if S[i:].startswith(t)}
        if i == len(S):
            expect.add(voc.eos_id)
        assert o.mask_set(cf, voc) == expect, i


def test_closed_form_any_bytes():
    o = Oracle("start: | start ANY\nANY: /[\\x00-\\xff]/\n")
    rng = np.random.default_rng(1)
    toks = list({bytes(rng.integers(0, 256, int(rng.integers(1, 6))).astype(np.uint8)) for _ in range(300)})
    voc = Vocab.from_list(toks + [b""], eos_id=len(toks))
    cf = o.initial()
    for t in toks[:20]:
        assert o.advance(cf, t) == ST_OK
        assert o.mask_set(cf, voc) == set(range(voc.V))


# --------------------------------------------------------- Eq. (1) brute force
def test_eq1_completion_search_arithmetic():
    """c(x) = {v : exists y, x v y in L} (Eq. 1), searched over y in an alphabet
    of 7 single-byte strings up to length 5 on shallow prefixes (a branch stops
    once the terminals already emitted are no prefix of any sentence).  A witness
    y for a disallowed token is a completeness failure; an allowed token without
    a witness would be a soundness failure within the bound."""
    o = Oracle(ARITH)
    voc = Vocab.from_list(MICRO, eos_id=10)
    py = PyCheck(parse_grammar(ARITH))
    alphabet = [b"1", b"a", b"+", b"*", b"(", b")", b" "]

    def witness(s: bytes, budget: int) -> bool:
        r = py.lex(s)
        if r is None or not py.earley.viable(r[0]):
            return False
        if py.sentence(s):
            return True
        return budget > 0 and any(witness(s + c, budget - 1) for c in alphabet)

    for prefix in [b"", b"(", b"(1", b"1", b"a", b"1 +", b"(a)", b"((", b"a*", b"12+(a"]:
        cf = o.initial()
        for ch in prefix:
            assert o.advance(cf, bytes([ch])) == ST_OK
        got = o.mask_set(cf, voc)
        for v, t in enumerate(MICRO):
            brute = py.sentence(prefix) if v == voc.eos_id else witness(prefix + t, 5)
            assert (v in got) == brute, (prefix, t)


def test_eq1_completion_search_json():
    """Eq. (1) by search on the JSON grammar with the JSON micro vocabulary:
    completions y over 9 single bytes up to length 4 (memoised; a branch stops
    once its terminals are no prefix of a sentence), on prefixes inside numbers,
    strings, escapes, objects and arrays."""
    text = grammars.json_grammar().text()
    o = Oracle(text)
    voc = Vocab.from_list(JSON_MICRO, eos_id=18)
    py = PyCheck(parse_grammar(text))
    alphabet = [b'"', b"a", b"1", b"}", b"]", b":", b",", b"u", b"e"]
    memo = {}

    def witness(s: bytes, budget: int) -> bool:
        if (s, budget) not in memo:
            r = py.lex(s)
            if r is None or not py.earley.viable(r[0]):
                memo[s, budget] = False
            elif py.sentence(s):
                memo[s, budget] = True
            else:
                memo[s, budget] = budget > 0 and any(witness(s + c, budget - 1) for c in alphabet)
        return memo[s, budget]

    for prefix in [b"", b"{", b'{"a":', b"[1", b"[1e", b"[1,", b'"', b'"\\', b"0", b"-", b"[", b'{"a"']:
        cf = o.initial()
        for ch in prefix:
            assert o.advance(cf, bytes([ch])) == ST_OK
        got = o.mask_set(cf, voc)
        for v, t in enumerate(JSON_MICRO):
            brute = py.sentence(prefix) if v == voc.eos_id else witness(prefix + t, 4)
            assert (v in got) == brute, (prefix, t)


# ------------------------------------------------------ independent parser
@pytest.mark.parametrize("cfg_id", [1, 2])
def test_earley_cross_check_workload(cfg_id):
    """Mask bits of the C lexer + canonical LR(1) equal a Python lexer + Earley
    recognizer on workload prefixes (basic-lexer grammars)."""
    w = configs.load(cfg_id, batch=6)
    o = Oracle(w.grammar_text)
    voc = Vocab.from_list(w.vocab, w.eos_id)
    py = PyCheck(parse_grammar(w.grammar_text))
    rng = np.random.default_rng(cfg_id)
    sample = sorted(set(rng.integers(0, voc.V, 160).tolist()) | {w.eos_id} | set(range(0, 98, 7)))
    cfgs = []
    for ids in w.prefix_ids:
        cf = o.initial()
        assert o.advance_tokens(cf, voc, ids) == ST_OK
        cfgs.append(cf)
    m = o.masks(cfgs, voc)
    for b, prefix in enumerate(w.prefixes):
        for v in sample:
            got = (int(m[b, v >> 5]) >> (v & 31)) & 1
            want = py.allowed(prefix, None if v == w.eos_id else w.vocab[v])
            assert got == want, (b, prefix[-40:], w.vocab[v])


def test_earley_cross_check_random_grammars(n: int = 150):
    """The same cross-check on seeded random small grammars (basic lexer;
    literals colliding with regex terminals, ignored whitespace, empty
    alternatives, recursion): the oracle's mask of every token after random
    reachable prefixes equals the Python lexer + Earley recognizer's answer.
    Grammars that are not LR(1) are refused by the oracle and skipped."""
    from ._random_grammars import random_grammar, random_vocab
    rng = np.random.default_rng(8)
    done = 0
    while done < n:
        text, vocab = random_grammar(rng), random_vocab(rng)
        if text is None or "contextual" in text:
            continue
        try:
            o = Oracle(text)
        except GrammarError:
            continue
        py = PyCheck(parse_grammar(text))
        voc = Vocab.from_list(vocab, len(vocab) - 1)
        prefixes = [b""]
        for _ in range(4):
            cf, p = o.initial(), b""
            for _ in range(int(rng.integers(1, 6))):
                allowed = sorted(o.mask_set(cf, voc) - {voc.eos_id})
                if not allowed:
                    break
                v = int(rng.choice(allowed))
                p += vocab[v]
                o.advance(cf, vocab[v])
            prefixes.append(p)
        for p in prefixes:
            cf = o.initial()
            if p:
                assert o.advance(cf, p) == ST_OK
            got = o.mask_set(cf, voc)
            for v, t in enumerate(vocab):
                assert (v in got) == py.allowed(p, None if v == voc.eos_id else t), (text, p, t)
        done += 1


# ------------------------------------------------------------ regex reader
def _regex_cases():
    out = []
    for cfg_id in (1, 2, 3, 4):
        spec = configs.grammar_spec(cfg_id)
        for name, t in spec.terminals.items():
            if t.pattern.startswith("/"):
                out.append((cfg_id, name, t))
    return out


@pytest.mark.parametrize("cfg_id,name,term", _regex_cases(), ids=lambda x: str(x) if not hasattr(x, "pattern") else "")
def test_regex_nfa_agrees_with_python_re(cfg_id, name, term):
    g = parse_grammar(configs.grammar_spec(cfg_id).text())
    t_idx = g.term_index[name]
    nfa, start = build_lexer_nfa(g)
    pat = re.compile(g.terminals[t_idx].pattern, re.DOTALL if False else 0)
    rng = np.random.default_rng(hash(name) % 1000)
    alphabet = sorted(set(b"\"\\/*'0123456789abcdefxXeE.+-_ \n\tuAZ{}") | {0x01, 0x7f, 0xc3})
    cases = []
    for _ in range(300):
        s = term.sample(rng)
        cases.append(s)
        if s:
            i = int(rng.integers(0, len(s)))
            cases.append(s[:i] + bytes([alphabet[int(rng.integers(0, len(alphabet)))]]) + s[i:])
            cases.append(s[:i] + s[i + 1:])
    for _ in range(300):
        cases.append(bytes(alphabet[int(k)] for k in rng.integers(0, len(alphabet), int(rng.integers(0, 7)))))
    for s in cases:
        assert (t_idx in matches(nfa, start, s)) == bool(pat.fullmatch(s)), (name, s)


# ---------------------------------------------------------- contextual lexer
KW = '''
start: | start stmt
stmt: "if" NAME ";" | NAME "=" NAME ";"
NAME: /[a-z]+/
WS: /[ ]+/
%ignore WS
%lexer contextual
'''


def test_contextual_keyword_resolution():
    """A lexeme matching a keyword and NAME is the keyword where the parser has an
    action on it, otherwise NAME; with the basic lexer it is always the keyword."""
    toks = [b"if", b"x", b"=", b";", b" ", b"i", b"if "]
    voc = Vocab.from_list(toks + [b""], eos_id=len(toks))
    o = Oracle(KW)
    basic = Oracle(KW.replace("%lexer contextual", "%lexer basic"))
    # "if" alone is allowed wherever a name fits in both modes (it may grow into
    # "ifx"); "if " ends the lexeme, so only the contextual lexer accepts it there.
    for prefix, want_ctx, want_basic in [
        (b"", {0, 1, 4, 5, 6, 7}, {0, 1, 4, 5, 6, 7}),
        (b"x = ", {0, 1, 4, 5, 6}, {0, 1, 4, 5}),
        (b"if ", {0, 1, 4, 5, 6}, {0, 1, 4, 5}),
        (b"if x", {0, 1, 3, 4, 5, 6}, {0, 1, 3, 4, 5, 6}),
    ]:
        for orc, want in ((o, want_ctx), (basic, want_basic)):
            cf = orc.initial()
            for ch in prefix:
                assert orc.advance(cf, bytes([ch])) == ST_OK
            assert orc.mask_set(cf, voc) == want, (prefix, orc.grammar.lexer_mode)


PRIO = '''
start: A "+" B
A: /[0-9]+/
B.2: /[0-9a-z]+/
WS: /[ ]+/
%ignore WS
%lexer basic
'''

TIE = '''
start: AA "+" BB
AA: /[0-9]+/
BB: /[0-9]+/
WS: /[ ]+/
%ignore WS
%lexer basic
'''


def test_terminal_rank_priority_then_name():
    """Hand-derived: with the basic lexer a lexeme matching several terminals is
    the highest-ranked one, by priority first (B.2 over A, so no digit string
    can be the A the grammar starts with), then by name (AA over BB, so after
    "1+" no digit string can be the BB the grammar wants); the contextual lexer
    picks, among them, one the parser can take."""
    toks = [b"12", b"12 ", b"x", b"+", b" ", b"1", b"2"]
    voc = Vocab.from_list(toks + [b""], eos_id=len(toks))
    cases = [   # (grammar, prefix, basic mask, contextual mask); None: the prefix is not reachable
        (PRIO, b"", {4}, {0, 1, 4, 5, 6}),
        (TIE, b"", {0, 1, 4, 5, 6}, {0, 1, 4, 5, 6}),
        (TIE, b"1+", {4}, {0, 1, 4, 5, 6}),
        (TIE, b"1+2", None, {0, 1, 4, 5, 6, 7}),
    ]
    for text, prefix, want_basic, want_ctx in cases:
        for mode, want in (("basic", want_basic), ("contextual", want_ctx)):
            if want is None:
                continue
            o = Oracle(text.replace("%lexer basic", "%lexer " + mode))
            cf = o.initial()
            for ch in prefix:
                assert o.advance(cf, bytes([ch])) == ST_OK
            assert o.mask_set(cf, voc) == want, (text.split()[1], prefix, mode, sorted(o.mask_set(cf, voc)))


LALR_MERGE = '''
start: "a" e "x" | "a" e NAME "z" | "b" e "y"
e: "e"
NAME: /[a-z]+/
WS: /[ ]+/
%ignore WS
%lexer contextual
'''


def test_contextual_uses_lalr_action_set():
    """After "a e" the canonical LR(1) state acts on x and NAME only, but the
    LALR(1) state (merged with the one after "b e") also acts on y.  The lexeme
    "y" therefore resolves to the literal y, which then fails: the token is
    masked out, although NAME would have fitted."""
    o = Oracle(LALR_MERGE)
    toks = [b"y ", b"q", b"x", b" "]      # "y " ends the lexeme "y" at once
    voc = Vocab.from_list(toks + [b""], eos_id=len(toks))
    cf = o.initial()
    for t in (b"a", b" ", b"e", b" "):
        assert o.advance(cf, t) == ST_OK
    assert o.mask_set(cf, voc) == {1, 2, 3}
    cf2 = o.initial()
    for t in (b"b", b" ", b"e", b" "):
        assert o.advance(cf2, t) == ST_OK
    assert o.mask_set(cf2, voc) == {0, 3}              # only y (and space) after "b e"


def test_grammar_errors():
    with pytest.raises(GrammarError):
        parse_grammar("start: FOO\n")
    with pytest.raises(GrammarError):
        Oracle('start: a | b\na: "x"\nb: "x"\n')   # reduce-reduce conflict, not LR(1)


# ---------------------------------------------------------------- invariants
@pytest.mark.parametrize("cfg_id", [1, 2, 3, 6, 8])
def test_invariants_on_workloads(cfg_id):
    w = configs.load(cfg_id, batch=8)
    o = Oracle(w.grammar_text)
    voc = Vocab.from_list(w.vocab, w.eos_id)
    cfgs = []
    for ids in w.prefix_ids:
        cf = o.initial()
        for v in ids:                                  # teacher forcing: never masked
            assert o.allowed(cf, w.vocab[v])
            assert o.advance(cf, w.vocab[v]) == ST_OK
        cfgs.append(cf)
    m = o.masks(cfgs, voc)
    tok = TrieTokenizer(w.vocab)
    index = {t: i for i, t in enumerate(w.vocab)}
    for b in range(len(cfgs)):
        allowed = _bits(m[b], voc.V)
        assert allowed, "reachable state with an empty mask"
        for v in list(allowed)[:400]:                  # prefix-closed
            t = w.vocab[v]
            for k in range(1, len(t)):
                u = index.get(t[:k])
                if u is not None:
                    assert u in allowed, (t, t[:k])
    perm = np.random.default_rng(0).permutation(len(cfgs))
    m2 = o.masks([cfgs[i] for i in perm], voc)
    assert np.array_equal(m2, m[perm])                 # rows are independent


@pytest.mark.parametrize("cfg_id", [1, 2, 3, 6, 8])
def test_tokenwise_equals_bytewise(cfg_id):
    """The configuration (q, alpha) is a function of the bytes consumed (Section
    3.2): a prefix advanced token by token and byte by byte reaches the same
    status, pending lexeme, stack and mask (the lexer looks one byte ahead and
    never backtracks, so where a token boundary falls changes nothing)."""
    w = configs.load(cfg_id, batch=8)
    o = Oracle(w.grammar_text)
    voc = Vocab.from_list(w.vocab, w.eos_id)
    tokwise, bytewise = [], []
    for ids in w.prefix_ids:
        a, b = o.initial(), o.initial()
        for k, v in enumerate(ids):
            t = w.vocab[v]
            assert o.advance(a, t) == ST_OK
            for byte in t:
                assert o.advance(b, bytes([byte])) == ST_OK
            if k % 5 == 0:
                assert a.info() == b.info()
        assert a.info() == b.info()
        tokwise.append(a)
        bytewise.append(b)
    np.testing.assert_array_equal(o.masks(tokwise, voc), o.masks(bytewise, voc))


def test_eos_only_after_complete_sentence():
    o = Oracle(grammars.json_grammar().text())
    voc = Vocab.from_list([b"{", b"}", b"1", b" "] + [b""], eos_id=4)
    cf = o.initial()
    assert o.mask_set(cf, voc) == {0, 2, 3}
    o.advance(cf, b"{")
    assert voc.eos_id not in o.mask_set(cf, voc)
    o.advance(cf, b"}")
    assert voc.eos_id in o.mask_set(cf, voc)
    assert o.advance(cf, None) == ST_DONE
    assert o.mask_set(cf, voc) == {voc.eos_id}
    assert o.advance(cf, b"1") == ST_ERROR
    assert o.mask_set(cf, voc) == set()


def test_sampled_sentences_are_sentences():
    """Complete sentences from the sampler end with EOS allowed (pins that the
    oracle's accept path is reachable on every workload grammar)."""
    for cfg_id in (1, 2, 4):
        spec = configs.grammar_spec(cfg_id)
        o = Oracle(spec.text())
        rng = np.random.default_rng(5)
        s = SentenceSampler(spec, max_depth=12)
        n_done = 0
        for _ in range(20):
            txt, finished = s.text(rng, 10 ** 6)
            if not finished:
                continue
            cf = o.initial()
            for ch in range(0, len(txt), 3):
                assert o.advance(cf, txt[ch:ch + 3]) == ST_OK
            assert o.allowed(cf, None)
            n_done += 1
        assert n_done > 0


@pytest.mark.parametrize("cfg_id", [2, 4])
def test_teacher_forced_sentences_never_masked(cfg_id):
    """RQ1 invariant (Section 4): every token of a whole sentence of the grammar is
    in the oracle's mask when teacher-forced, and the end of sequence is allowed
    after it."""
    from workloads import configs, teacher
    w = configs.load(cfg_id, batch=1)
    ts = teacher.teacher_set(w, 8)
    o = Oracle(w.grammar_text)
    for ids in ts.positives:
        c = o.initial()
        for v in ids:
            assert o.allowed(c, w.vocab[v])
            o.advance(c, w.vocab[v])
        assert o.allowed(c, None)
