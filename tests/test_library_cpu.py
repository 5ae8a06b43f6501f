"""CPU-side tests of the library: it loads, exports every symbol the header
declares, reports grammar errors, and its compiled host tables give the
oracle's masks (a walk of the same flattened tables the GPU reads)."""
from __future__ import annotations

import os
import re
import sys

import numpy as np
import pytest

from oracle import ST_DONE, ST_ERROR, ST_OK, Oracle, Vocab
from workloads import configs, grammars

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="session")
def psc():
    from paper_2608_03065_gb300 import build, psc as mod
    build.build()
    mod.load()
    return mod


def _header_symbols():
    text = open(os.path.join(ROOT, "include", "psc.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(psc_[a-z_]+)\s*\(", text)))


def test_library_exports_every_declared_symbol(psc):
    lib = psc.load()
    syms = _header_symbols()
    assert len(syms) >= 16
    for s in syms:
        assert hasattr(lib, s), s
    assert set(syms) == set(psc.EXPORTED)


def _c_type(decl: str):
    """ctypes type the binding must use for one C parameter or return declaration."""
    import ctypes
    d = " ".join(decl.replace("const ", "").split())
    if "*" in d:
        return (ctypes.c_void_p, ctypes.c_char_p)
    base = d.split()[0]
    return {"int32_t": (ctypes.c_int32,), "psc_dtype": (ctypes.c_int32,), "psc_status": (ctypes.c_int32,),
            "int64_t": (ctypes.c_int64,), "size_t": (ctypes.c_size_t,), "void": (None,)}[base]


def test_binding_signatures_match_the_header(psc):
    """Every prototype of include/psc.h has the same number and kinds of
    parameters (pointer, int32, int64, size_t) and return type in the binding."""
    lib = psc.load()
    text = re.sub(r"/\*.*?\*/", "", open(os.path.join(ROOT, "include", "psc.h")).read(), flags=re.S)
    protos = re.findall(r"([A-Za-z_][\w ]*?\**)\s*\b(psc_[a-z_]+)\s*\(([^)]*)\)\s*;", text)
    assert len(protos) == len(psc.EXPORTED)
    for ret, name, params in protos:
        f = getattr(lib, name)
        args = [] if params.strip() in ("", "void") else [p.strip() for p in params.split(",")]
        assert len(f.argtypes) == len(args), name
        for decl, t in zip(args, f.argtypes):
            want = _c_type(decl.rsplit(" ", 1)[0] if "*" not in decl.split()[-1] else decl)
            assert t in want, (name, decl, t)
        assert f.restype in _c_type(ret), (name, ret, f.restype)


def test_binding_structs_match_the_header(psc):
    """psc_options and psc_info_t: same fields, order and types in the binding."""
    import ctypes
    text = re.sub(r"/\*.*?\*/", "", open(os.path.join(ROOT, "include", "psc.h")).read(), flags=re.S)
    ctype = {"int32_t": ctypes.c_int32, "int64_t": ctypes.c_int64, "double": ctypes.c_double}
    for cname, py in (("psc_options", psc.Options), ("psc_info_t", psc.InfoT)):
        body = re.search(r"typedef struct \{([^}]*)\}\s*" + cname + r"\s*;", text).group(1)
        fields = []
        for decl in body.split(";"):
            decl = decl.strip()
            if not decl:
                continue
            typ, names = decl.split(None, 1)
            fields += [(n.strip(), ctype[typ]) for n in names.split(",")]
        assert [(n, t) for n, t in py._fields_] == fields, cname   # ctypes then lays them out as C does


def _host_cfg(h, ids):
    c = h.host_initial()
    for v in ids:
        c = h.host_advance(c, v)
    return c


def _host_mask(h, c):
    return h.host_mask_row(h.host_classify(c["q"], c["stack"], c["status"]))


_handles = {}


def _handle(psc, cfg_id, batch):
    """Host-only handle of a workload (compiled once per test session)."""
    if cfg_id not in _handles:
        w = configs.load(cfg_id, batch=batch)
        _handles[cfg_id] = (w, psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True))
    return _handles[cfg_id]


@pytest.mark.parametrize("cfg_id,batch", [(1, 8), (2, 24), (3, 6)])
def test_host_tables_match_oracle(psc, cfg_id, batch):
    w, h = _handle(psc, cfg_id, batch)
    o = Oracle(w.grammar_text)
    voc = Vocab.from_list(w.vocab, w.eos_id)
    cfgs, ocs = [], []
    for ids in w.prefix_ids:
        cfgs.append(_host_cfg(h, ids))
        oc = o.initial()
        o.advance_tokens(oc, voc, ids)
        ocs.append(oc)
    om = o.masks(ocs, voc)
    for b, c in enumerate(cfgs):
        assert c["status"] == psc.ROW_OK
        np.testing.assert_array_equal(_host_mask(h, c), om[b], err_msg=f"row {b}")


@pytest.mark.parametrize("cfg_id,batch", [(1, 8), (2, 24), (3, 6)])
def test_bottom_up_classifier_agrees_with_the_walk(psc, cfg_id, batch):
    """The bottom-up classifier (the classifier DFA reversed, reading the stack
    from the bottom; it exists by the regularity theorem of Section 3.5) gives
    the top-down walk's mask id at every token of every prefix, and refuses
    stacks that no parser builds."""
    w, h = _handle(psc, cfg_id, batch)
    assert h.info().bottom_up_states > 0
    n = 0
    for ids in w.prefix_ids:
        c = h.host_initial()
        for v in ids:
            c = h.host_advance(c, v)
            assert c["status"] == psc.ROW_OK
            want = h.host_classify(c["q"], c["stack"])
            assert h.host_classify_bottom_up(c["q"], c["stack"]) == want, (ids, c)
            n += 1
        for st in (psc.ROW_DONE, psc.ROW_REJECTED):   # statuses decide before any table
            assert h.host_classify_bottom_up(c["q"], c["stack"], st) == h.host_classify(c["q"], c["stack"], st)
    assert n > 50
    assert h.host_classify_bottom_up(0, [0, 0]) == -2        # nothing enters the LR start state
    assert h.host_classify_bottom_up(0, [1]) == -2           # every stack starts with state 0


@pytest.mark.parametrize("cfg_id,batch", [(1, 8), (2, 24)])
def test_host_advance_tokenwise_equals_bytewise(psc, cfg_id, batch):
    """The compiled lexer and parser tables keep the state a function of the bytes:
    advancing by the prefix's tokens or by the single-byte tokens of its bytes
    gives the same lexer state, stack and mask id (prefixes whose bytes all have
    single-byte tokens)."""
    w, h = _handle(psc, cfg_id, batch)
    single = {t[0]: i for i, t in enumerate(w.vocab) if len(t) == 1}
    n = 0
    for ids in w.prefix_ids:
        if not all(b in single for v in ids for b in w.vocab[v]):
            continue
        a, b = h.host_initial(), h.host_initial()
        for v in ids:
            a = h.host_advance(a, v)
            for byte in w.vocab[v]:
                b = h.host_advance(b, single[byte])
            assert a == b
        assert h.host_classify(a["q"], a["stack"]) == h.host_classify(b["q"], b["stack"])
        n += 1
    assert n >= 4


def test_bottom_up_classifier_c_like_random_walks(psc):
    """The C-like grammar (150 rules, 15 precedence levels, contextual lexer) with a
    4,000-token slice of its vocabulary: along random decodes that favour opening
    brackets, the bottom-up classifier gives the walk's mask id at every step."""
    w = configs.load(4, batch=1)
    singles = [bytes([b]) for b in list(range(0x20, 0x7F)) + [9, 10, 13]]
    vocab = sorted(set(singles) | {t for t in w.vocab[:4000] if t}) + [b""]
    eos = len(vocab) - 1
    h = psc.psc_compile(w.grammar_text, vocab, eos, host_only=True)
    assert h.info().bottom_up_states > 0
    opens = np.array([t[:1] in (b"(", b"{", b"[") for t in vocab])
    rng = np.random.default_rng(3)
    n = deepest = 0
    for _ in range(12):
        c = h.host_initial()
        for _ in range(200):
            mid = h.host_classify(c["q"], c["stack"])
            assert h.host_classify_bottom_up(c["q"], c["stack"]) == mid
            n += 1
            bits = np.unpackbits(h.host_mask_row(mid).view(np.uint8), bitorder="little")[:len(vocab)].astype(bool)
            bits[eos] = False
            allowed = np.nonzero(bits)[0]
            if len(allowed) == 0:
                break
            deep = allowed[opens[allowed]]
            v = int(rng.choice(deep)) if len(deep) and rng.random() < 0.7 else int(rng.choice(allowed))
            c = h.host_advance(c, v, cap=4096)
            deepest = max(deepest, len(c["stack"]))
            if c["status"] != psc.ROW_OK:
                break
    assert n > 1000 and deepest > 16


@pytest.mark.parametrize("name", ["literal", "any_bytes", "parentheses"])
def test_bottom_up_classifier_small_grammars(psc, name):
    """Degenerate classifiers (a single literal, every byte string, balanced
    parentheses): the bottom-up classifier is built and agrees with the walk
    along random decodes."""
    grammar, toks = {
        "literal": ('start: "hello world"\n', [b"h", b"he", b"hello", b" ", b"world", b"o w", b"d", b"x", b""]),
        "any_bytes": ("start: | start ANY\nANY: /[\\x00-\\xff]/\n", [bytes([b]) for b in range(256)] + [b"ab", b""]),
        "parentheses": ('start: s\ns: | s "(" s ")"\n', [b"(", b")", b"((", b"))", b""]),
    }[name]
    eos = len(toks) - 1
    h = psc.psc_compile(grammar, toks, eos, host_only=True)
    assert h.info().bottom_up_states > 0
    rng = np.random.default_rng(0)
    n = 0
    for _ in range(20):
        c = h.host_initial()
        for _ in range(40):
            mid = h.host_classify(c["q"], c["stack"])
            assert h.host_classify_bottom_up(c["q"], c["stack"]) == mid, c
            n += 1
            bits = np.unpackbits(h.host_mask_row(mid).view(np.uint8), bitorder="little")[:len(toks)].astype(bool)
            bits[eos] = False
            allowed = np.nonzero(bits)[0]
            if len(allowed) == 0:
                break
            c = h.host_advance(c, int(rng.choice(allowed)), cap=512)
            if c["status"] != psc.ROW_OK:
                break
    assert n >= 20


def test_bottom_up_classifier_limits(psc):
    """Not built on request or over its memory limit (compilation still succeeds;
    the device then walks stacks from the top)."""
    w = configs.load(2, batch=2)
    for kw in ({"bottom_up": False}, {"max_bottom_up_bytes": 4096}):
        h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True, **kw)
        assert h.info().bottom_up_states == 0 and h.info().bottom_up_bytes == 0
        c = _host_cfg(h, w.prefix_ids[0])
        assert h.host_classify_bottom_up(c["q"], c["stack"]) == -2
        assert h.host_classify(c["q"], c["stack"]) >= 0


@pytest.mark.parametrize("fixture", ["arith_micro_masks.txt", "json_micro_masks.txt"])
def test_host_tables_match_golden_masks(psc, fixture):
    """The compiled tables give the hand-enumerated masks of the golden fixtures."""
    from workloads.sample import TrieTokenizer
    from .test_oracle_pins import JSON_MICRO, MICRO
    if fixture.startswith("arith"):
        text, vocab = grammars.arithmetic().text(), MICRO
    else:
        text, vocab = grammars.json_grammar().text(), JSON_MICRO
    eos = len(vocab) - 1
    h = psc.psc_compile(text, vocab, eos, host_only=True)
    tok = TrieTokenizer(vocab)
    n = 0
    with open(os.path.join(ROOT, "tests", "golden", fixture)) as f:
        for line in f:
            if not line.strip() or line.startswith("#"):
                continue
            m = re.match(r'"(.*)"\s+([\d,]+)$', line.strip())
            prefix, allowed = m.group(1).encode(), {int(x) for x in m.group(2).split(",")}
            c = _host_cfg(h, tok.encode(prefix) if prefix else [])
            assert c["status"] == psc.ROW_OK
            bits = np.unpackbits(_host_mask(h, c).view(np.uint8), bitorder="little")[:len(vocab)]
            assert set(np.nonzero(bits)[0].tolist()) == allowed, prefix
            n += 1
    assert n >= 7


@pytest.mark.parametrize("which", ["arith", "json"])
def test_host_tables_exhaustive_small_configurations(psc, which):
    """Every configuration the micro vocabularies reach in up to 6 tokens
    (breadth first, deduplicated by lexer state and stack): the compiled tables'
    mask equals the oracle's, and so does the status of every next token."""
    from .test_oracle_pins import JSON_MICRO, MICRO
    text, vocab = ((grammars.arithmetic().text(), MICRO) if which == "arith"
                   else (grammars.json_grammar().text(), JSON_MICRO))
    eos = len(vocab) - 1
    h = psc.psc_compile(text, vocab, eos, host_only=True)
    o = Oracle(text)
    voc = Vocab.from_list(vocab, eos)
    seen = {}
    frontier = [((), h.host_initial())]
    for _ in range(6):
        nxt = []
        for seq, c in frontier:
            for v in range(eos):
                c2 = h.host_advance(c, v, cap=64)
                key = (c2["q"], tuple(c2["stack"]))
                if c2["status"] != psc.ROW_OK or key in seen:
                    continue
                seen[key] = seq + (v,)
                nxt.append((seq + (v,), c2))
        frontier = nxt
    assert len(seen) > 100
    cfgs, ocs = [], []
    for (q, stack), seq in seen.items():
        oc = o.initial()
        assert o.advance_tokens(oc, voc, seq) == ST_OK
        cfgs.append({"q": q, "stack": list(stack), "status": psc.ROW_OK})
        ocs.append(oc)
    om = o.masks(ocs, voc)
    want_status = {ST_OK: psc.ROW_OK, ST_DONE: psc.ROW_DONE, ST_ERROR: psc.ROW_REJECTED}
    for c, oc, m in zip(cfgs, ocs, om):
        np.testing.assert_array_equal(_host_mask(h, c), m, err_msg=str(c))
        for v in range(len(vocab)):
            oc2 = oc.copy()
            st = o.advance(oc2, None if v == eos else vocab[v])
            assert h.host_advance(c, v, cap=64)["status"] == want_status[st], (c, v)


@pytest.mark.parametrize("cfg_id", [1, 2, 3, 4, 6, 8])
def test_host_tables_on_sentences_and_mutations(psc, cfg_id):
    """Whole sentences of each workload grammar and copies with one byte
    inserted, deleted or replaced, fed byte by byte (a vocabulary of the 256
    single bytes): the compiled LALR(1) tables and lexer stop at the same byte
    as the oracle's canonical LR(1) parser and Thompson-NFA lexer, and accept the
    same strings at the end of sequence."""
    from workloads.sample import SentenceSampler
    spec = configs.grammar_spec(cfg_id)
    text = spec.text()
    vocab = [bytes([b]) for b in range(256)] + [b""]
    h = psc.psc_compile(text, vocab, 256, host_only=True, bottom_up=False, **configs.COMPILE_LIMITS.get(cfg_id, {}))
    o = Oracle(text)
    want_status = {ST_OK: psc.ROW_OK, ST_DONE: psc.ROW_DONE, ST_ERROR: psc.ROW_REJECTED}
    rng = np.random.default_rng([cfg_id, 11])
    sampler = SentenceSampler(spec, max_depth=10)
    n = stopped = tries = 0
    while n < 60 and tries < 2000:
        tries += 1
        txt, finished = sampler.text(rng, 4000)
        if not finished or not txt:
            continue
        b = bytearray(txt)
        if n % 4:   # three in four mutated, one in four kept whole
            kind, pos, ch = int(rng.integers(0, 3)), int(rng.integers(0, len(b))), int(rng.integers(0x20, 0x7F))
            if kind == 0:
                b.insert(pos, ch)
            elif kind == 1:
                del b[pos]
            else:
                b[pos] = ch
        c, oc = h.host_initial(), o.initial()
        st = ST_OK
        for byte in bytes(b):
            st = o.advance(oc, bytes([byte]))
            c = h.host_advance(c, byte, cap=1024)
            assert c["status"] == want_status[st], (bytes(b), byte)
            if st != ST_OK:
                break
        if st == ST_OK:
            st = o.advance(oc, None)
            assert h.host_advance(c, 256, cap=1024)["status"] == want_status[st], bytes(b)
        if n % 4 == 0:
            assert st == ST_DONE, bytes(b)   # whole sentences are accepted
        stopped += st != ST_DONE
        n += 1
    assert n == 60 and stopped > 10


@pytest.mark.parametrize("cfg_id", [6, 8])
def test_host_masks_of_the_java_and_sql_grammars(psc, cfg_id):
    """The Java-sized and SQL-like grammars with a 512-token vocabulary of their
    workload's recipe: at every 7th token of sampled sentences, the mask the
    compiled tables give (host classification, host mask rows) equals the
    oracle's over every token, and so does the bottom-up classification."""
    from workloads.sample import SentenceSampler, TrieTokenizer
    spec = configs.grammar_spec(cfg_id)
    text = spec.text()
    toks = configs.vocab_for(cfg_id, 512)
    eos = len(toks) - 1
    h = psc.psc_compile(text, toks, eos, host_only=True, **configs.COMPILE_LIMITS.get(cfg_id, {}))
    o = Oracle(text)
    voc = Vocab.from_list(toks, eos)
    tok = TrieTokenizer(toks)
    rng = np.random.default_rng([cfg_id, 12])
    sampler = SentenceSampler(spec, max_depth=12)
    cfgs, ocs = [], []
    while len(cfgs) < 120:
        txt, _ = sampler.text(rng, 1500)
        c, oc = h.host_initial(), o.initial()
        for i, v in enumerate(tok.encode(txt)):
            c = h.host_advance(c, v, cap=1024)
            assert o.advance(oc, toks[v]) == ST_OK and c["status"] == psc.ROW_OK
            if i % 7 == 6:
                cfgs.append(dict(c))
                ocs.append(oc.copy())
    want = o.masks(ocs, voc, threads=os.cpu_count() or 1)
    for c, m in zip(cfgs, want):
        mid = h.host_classify(c["q"], c["stack"])
        np.testing.assert_array_equal(h.host_mask_row(mid), m)
        if h.info().bottom_up_states:
            assert h.host_classify_bottom_up(c["q"], c["stack"]) == mid
    assert len({bytes(m) for m in want}) > 10   # the configurations are not all alike


def test_host_tables_terminal_rank(psc):
    """The compiled lexer resolves colliding terminals like the hand-derived
    oracle pin: priority first, then name (basic), or the first one the parser
    can take (contextual)."""
    from workloads.sample import TrieTokenizer
    from .test_oracle_pins import PRIO, TIE
    toks = [b"12", b"12 ", b"x", b"+", b" ", b"1", b"2", b""]
    cases = [(PRIO, b"", {4}, {0, 1, 4, 5, 6}), (TIE, b"", {0, 1, 4, 5, 6}, {0, 1, 4, 5, 6}),
             (TIE, b"1+", {4}, {0, 1, 4, 5, 6}), (TIE, b"1+2", None, {0, 1, 4, 5, 6, 7})]
    tok = TrieTokenizer(toks)
    for text, prefix, want_basic, want_ctx in cases:
        for mode, want in (("basic", want_basic), ("contextual", want_ctx)):
            if want is None:
                continue
            h = psc.psc_compile(text.replace("%lexer basic", "%lexer " + mode), toks, 7, host_only=True)
            c = _host_cfg(h, tok.encode(prefix) if prefix else [])
            assert c["status"] == psc.ROW_OK
            bits = np.unpackbits(_host_mask(h, c).view(np.uint8), bitorder="little")[:len(toks)]
            assert set(np.nonzero(bits)[0].tolist()) == want, (prefix, mode)


def test_host_tables_deep_parentheses(psc):
    """Balanced parentheses to depth 200: the classifier walk reads deep stacks."""
    g = 'start: s\ns: | s "(" s ")"\n'
    toks = [b"(", b")", b"((", b"))", b"()", b")(", b"())", b""]
    h = psc.psc_compile(g, toks, 7, host_only=True)
    o = Oracle(g)
    voc = Vocab.from_list(toks, 7)
    c, oc = h.host_initial(), o.initial()
    for d in range(200):
        c = h.host_advance(c, 0, cap=512)       # two stack entries per level
        o.advance(oc, b"(")
        if d % 37 == 0 or d == 199:
            np.testing.assert_array_equal(_host_mask(h, c), o.masks([oc], voc)[0])
        assert h.host_classify_bottom_up(c["q"], c["stack"]) == h.host_classify(c["q"], c["stack"])
    for d in range(200):
        c = h.host_advance(c, 1, cap=512)
        o.advance(oc, b")")
        assert h.host_classify_bottom_up(c["q"], c["stack"]) == h.host_classify(c["q"], c["stack"])
    np.testing.assert_array_equal(_host_mask(h, c), o.masks([oc], voc)[0])
    assert (_host_mask(h, c)[0] >> 7) & 1   # end of sequence allowed at depth 0


def test_host_advance_statuses(psc):
    g = grammars.json_grammar().text()
    toks = [b"{", b"}", b"1", b" ", b'"a"', b":", b""]
    h = psc.psc_compile(g, toks, 6, host_only=True)
    c = h.host_initial()
    c = h.host_advance(c, 0)
    assert c["status"] == psc.ROW_OK
    c2 = h.host_advance(c, 2)                  # "{1" is not JSON
    assert c2["status"] == psc.ROW_REJECTED
    assert h.host_classify(c2["q"], c2["stack"], c2["status"]) == 0
    c = h.host_advance(c, 1)
    c = h.host_advance(c, 6)                   # end of sequence after "{}"
    assert c["status"] == psc.ROW_DONE
    assert h.host_classify(c["q"], c["stack"], c["status"]) == 1
    row = h.host_mask_row(1)
    assert row[0] == 1 << 6
    assert h.host_advance(c, 6)["status"] == psc.ROW_DONE
    assert h.host_advance(c, 0)["status"] == psc.ROW_REJECTED
    # stack overflow at a small capacity
    arr = psc.psc_compile('start: s\ns: | s "(" s ")"\n', [b"(", b")", b""], 2, host_only=True)
    c = arr.host_initial()
    for _ in range(10):
        c = arr.host_advance(c, 0, cap=8)
    assert c["status"] == psc.ROW_OVERFLOW


@pytest.mark.parametrize("text,code", [
    ('start: a | b\na: "x"\nb: "x"\n', 3),                                  # reduce/reduce conflict
    ('start: "x" | "x" "y"\nstart2: FOO\n', 2),                             # unknown terminal
    ('start: NAME\nNAME: /[a-z]+/\nKW: "if"\nWS: /if/\n%ignore WS\n', 4),   # ignored and kept collide
    ('start: A\nA: /x*/\n', 2),                                            # terminal matches empty
    ('nostart: "x"\n', 2),
])
def test_grammar_errors(psc, text, code):
    with pytest.raises(psc.PscError) as e:
        psc.psc_compile(text, [b"x", b""], 1, host_only=True)
    assert e.value.code == code, str(e.value)


def test_state_limit(psc):
    w = configs.load(2, batch=1)
    with pytest.raises(psc.PscError) as e:
        psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True, max_states=50)
    assert e.value.code == 5


def test_host_calls_check_their_arguments(psc):
    """Host inspection calls refuse out-of-range lexer states, stack entries and
    mask ids instead of reading past their tables."""
    w, h = _handle(psc, 1, 8)
    n_lr = h.info().n_parser_states
    assert h.host_classify(0, [0, n_lr]) == -1
    assert h.host_classify_bottom_up(0, [0, n_lr]) == -1
    with pytest.raises(psc.PscError) as e:
        h.host_mask_row(h.info().n_masks)
    assert e.value.code == 1
    for bad in ({"q": h.info().n_lexer_states, "stack": [0], "status": psc.ROW_OK},
                {"q": 0, "stack": [0, n_lr + 3], "status": psc.ROW_OK},
                {"q": 0, "stack": [], "status": psc.ROW_OK}):
        with pytest.raises(psc.PscError) as e:
            h.host_advance(bad, 0)
        assert e.value.code == 1, bad
    c = h.host_advance(h.host_initial(), -1)          # a negative token leaves the row as it is
    assert c == h.host_initial()


def test_binding_refuses_short_or_host_arrays(psc):
    """The binding checks per-row arrays before any launch: fewer elements than
    rows, a non-contiguous view, or host memory are refused with ValueError."""
    torch = pytest.importorskip("torch")
    _, h = _handle(psc, 1, 8)
    st = psc.States(0, h, 4, 16)   # never reaches the library: every call below fails first
    for tokens in (torch.zeros(2, dtype=torch.int32), torch.zeros(8, dtype=torch.int32)[::2],
                   torch.zeros(4, dtype=torch.int32)):
        with pytest.raises(ValueError):
            psc.psc_advance(h, st, tokens)
        with pytest.raises(ValueError):
            psc.psc_decode_step_advance(h, st, tokens)
    with pytest.raises(ValueError):
        psc.psc_state_reset(st, torch.zeros(3, dtype=torch.int64))


def test_binding_fails_loudly_without_the_library(tmp_path):
    """No fallback: a binding that cannot find the compiled library raises."""
    import importlib.util
    spec = importlib.util.spec_from_file_location(
        "psc_fresh", os.path.join(ROOT, "paper_2608_03065_gb300", "psc.py"))
    fresh = importlib.util.module_from_spec(spec)
    sys.modules["psc_fresh"] = fresh   # dataclasses look their module up there
    try:
        spec.loader.exec_module(fresh)
        with pytest.raises(RuntimeError, match="missing"):
            fresh.load(str(tmp_path / "libpsc_gb300.so"))
    finally:
        del sys.modules["psc_fresh"]


def test_c_abi_argument_errors(psc):
    """Calls straight through the C ABI with bad arguments return PSC_ERR_ARG
    (1) and leave a message; nothing is dereferenced."""
    import ctypes
    lib = psc.load()
    g = b'start: "x"\n'
    blob = (ctypes.c_uint8 * 1)(120)
    offs = (ctypes.c_int64 * 3)(0, 1, 1)
    bad_offs = (ctypes.c_int64 * 3)(0, 1, 0)
    out = ctypes.c_void_p()
    cases = [
        lib.psc_compile(g, len(g), blob, offs, 2, 1, None, None),                 # out is NULL
        lib.psc_compile(g, len(g), blob, offs, 0, -1, None, ctypes.byref(out)),   # V = 0
        lib.psc_compile(g, len(g), blob, offs, 2, 2, None, ctypes.byref(out)),    # eos_id >= V
        lib.psc_compile(g, len(g), blob, bad_offs, 2, 1, None, ctypes.byref(out)),  # offsets decrease
        lib.psc_compile(None, 0, blob, offs, 2, 1, None, ctypes.byref(out)),      # no grammar
        lib.psc_info(None, None),
        lib.psc_save(None, b"/nonexistent/x"),
        lib.psc_load(None, None, ctypes.byref(out)),
        lib.psc_host_mask_row(None, 0, None),
        lib.psc_host_advance(None, None, None, None, 2, None, 0),
        lib.psc_state_init(None, 4, 16, None, ctypes.byref(out)),
        lib.psc_state_faults(None, None, 0, None),
        lib.psc_check_wait(None, 1, None),
    ]
    assert cases == [1] * len(cases), cases
    assert lib.psc_last_error()
    assert lib.psc_host_classify(None, 0, None, 0, 0) == -1
    assert lib.psc_host_classify_bottom_up(None, 0, None, 0, 0) == -1


def test_device_calls_refuse_host_only_handle(psc):
    h = psc.psc_compile(grammars.arithmetic().text(), [b"1", b""], 1, host_only=True)
    with pytest.raises(psc.PscError) as e:
        psc.psc_state_init(h, 4, 16, stream=0)
    assert e.value.code == 1


@pytest.mark.parametrize("cfg_id", [1, 2, 3])
def test_sparse_classifier_layout_classifies_like_the_dense_one(psc, cfg_id, tmp_path):
    """The classifier held sparse (a default target and the exceptions to it per
    state) classifies every configuration the workload prefixes pass through
    exactly as the dense table does, its bottom-up form agrees, and a saved and
    loaded sparse handle stays sparse and agrees too."""
    w = configs.load(cfg_id, batch=8)
    hd = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True)
    hs = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True, max_dense_classifier_bytes=-1)
    assert hd.info().classifier_sparse == 0 and hs.info().classifier_sparse == 1
    assert hs.info().n_classifier_states == hd.info().n_classifier_states
    assert hs.info().classifier_bytes < hd.info().classifier_bytes
    path = str(tmp_path / "sparse.psc")
    psc.psc_save(hs, path)
    hl = psc.psc_load(path, host_only=True)
    assert hl.info().classifier_sparse == 1
    n = 0
    for ids in w.prefix_ids:
        c = hd.host_initial()
        for v in ids:
            c = hd.host_advance(c, v)
            if c["status"] != psc.ROW_OK:
                break
            want = hd.host_classify(c["q"], c["stack"])
            assert hs.host_classify(c["q"], c["stack"]) == want
            assert hl.host_classify(c["q"], c["stack"]) == want
            assert hs.host_classify_bottom_up(c["q"], c["stack"]) == want
            n += 1
    assert n > 50


def test_packed_advance_tables(psc):
    """The packed staged parser tables (ACTION and GOTO row-displaced, equal rows
    stored once, lexeme classes resolved by trying candidate terminals in order)
    are what the advance stages for the Java-sized grammar, whose dense compact
    tables pass the shared-memory budget; the library builds them only after
    every lookup of them equals the dense tables' entry and the candidate order
    reproduces the class-resolution table in every parser state, so a packed
    layout on the seeded random grammars (both lexer modes, classes with several
    candidate terminals) means both checks passed.  A host_only handle reports
    what a device upload would stage."""
    from ._random_grammars import random_grammar, random_vocab
    toks = configs.vocab_for(6, 300)
    hj = psc.psc_compile(grammars.java_like().text(), toks, len(toks) - 1, host_only=True, bottom_up=False)
    ij = hj.info()
    assert ij.n_parser_states >= 1000 and ij.advance_tables_packed == 1
    assert 0 < ij.advance_table_bytes <= 200 * 1024
    w = configs.load(2, batch=4)
    for kw, packed in (({}, 0), ({"packed_tables": True}, 1)):
        i = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True, **kw).info()
        assert i.advance_table_bytes > 0 and i.advance_tables_packed == packed
    assert psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True,
                           global_tables=True).info().advance_table_bytes == 0
    with pytest.raises(ValueError):
        psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True, global_tables=True, packed_tables=True)
    import tempfile
    with tempfile.TemporaryDirectory() as d:   # the placement is chosen again when tables are loaded
        path = os.path.join(d, "t.psc")
        psc.psc_save(psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True), path)
        assert psc.psc_load(path, host_only=True).info().advance_tables_packed == 0
        assert psc.psc_load(path, host_only=True, packed_tables=True).info().advance_tables_packed == 1
        assert psc.psc_load(path, host_only=True, global_tables=True).info().advance_table_bytes == 0
    rng = np.random.default_rng(5150)
    modes, multi = set(), 0
    done = 0
    while done < 60:
        text, vocab = random_grammar(rng, True), random_vocab(rng, True)
        if text is None:
            continue
        try:
            h = psc.psc_compile(text, vocab, len(vocab) - 1, host_only=True, packed_tables=True, bottom_up=False)
        except psc.PscError as e:
            assert e.code == 3
            continue
        i = h.info()
        assert i.advance_tables_packed == 1 and i.advance_table_bytes > 0, text
        modes.add("contextual" if "%lexer contextual" in text else "basic")
        multi += "%lexer contextual" in text and re.search(r'"[a-z]+"', text) is not None
        done += 1
    assert modes == {"basic", "contextual"} and multi > 5


def test_table_placement_values_are_checked(psc):
    """psc_options.global_tables takes 0, 1 or 2; anything else is PSC_ERR_ARG."""
    import ctypes
    lib = psc.load()
    g = b'start: "x"\n'
    blob = (ctypes.c_uint8 * 1)(120)
    offs = (ctypes.c_int64 * 3)(0, 1, 1)
    out = ctypes.c_void_p()
    for bad in (3, -1):
        opts = psc.Options(0, 0, 0, 1, bad, 0, 0)
        assert lib.psc_compile(g, len(g), blob, offs, 2, 1, ctypes.byref(opts), ctypes.byref(out)) == 1
        assert b"global_tables" in lib.psc_last_error()
    opts = psc.Options(0, 0, 0, 1, 2, 0, 0)
    assert lib.psc_compile(g, len(g), blob, offs, 2, 1, ctypes.byref(opts), ctypes.byref(out)) == 0
    lib.psc_destroy(out)
