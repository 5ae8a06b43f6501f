"""The oracle never turns a capacity of its checker into "token not allowed".

Each case builds the oracle's C checker with one capacity made tiny (the
ORACLE_* build macros of brute.c), drives a small grammar past it, and expects
OracleLimitError naming that capacity from every call that can reach it (the
masks, a single-token check, an advance; the T_p cache fills only across the
tokens of one mask call).  A grammar whose lexeme is matched by an ignored and
a kept terminal (refused by the library's compiler) raises too.  Each variant
runs in a child process, because the oracle keeps one loaded checker per
process.  The default build decides the same inputs without error.
"""
from __future__ import annotations

import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

ARITH = """start: expr
expr: expr "+" term | expr "-" term | term
term: term "*" factor | term "/" factor | factor
factor: NUMBER | NAME | "(" expr ")"
NUMBER: /[0-9]+/
NAME: /[a-z]+/
WS: /[ \\t\\n]+/
%ignore WS
%lexer basic
"""
KEYWORD = """start: stmt*
stmt: "if" NAME ";" | NAME ";"
NAME: /[a-z]+/
WS: / +/
%ignore WS
%lexer basic
"""
PARENS = 'start: s\ns: | s "(" s ")"\n'
MIXED = """start: "a" " " "a"
WS: / +/
%ignore WS
"""

RUNNER = r"""
import sys, json
sys.path.insert(0, sys.argv[1])
import oracle.psc_oracle as po
lib = po.build_library(force=True, defines=json.loads(sys.argv[3]), path=sys.argv[2]) if sys.argv[3] != "{}" \
    else po.build_library()
po.build_library = lambda force=False: lib
po._lib = None
from oracle import Oracle, OracleLimitError, Vocab
grammar, toks, prefix = json.loads(sys.argv[4])
toks = [t.encode() for t in toks] + [b""]
o = Oracle(grammar)
voc = Vocab.from_list(toks, len(toks) - 1)
out = {}
def run(name, fn):
    try:
        out[name] = ["ok", fn()]
    except OracleLimitError as e:
        out[name] = ["limit", e.bits]
c = o.initial()
for t in prefix:
    o.advance(c, t.encode())
run("masks", lambda: o.masks([c], voc, threads=1).tolist())
run("allowed", lambda: [o.allowed(c, t) for t in toks[:-1]])
run("advance", lambda: [o.advance(c.copy(), t) for t in toks[:-1]])
print(json.dumps(out))
"""


def _run(tmp_path, defines: dict, grammar: str, toks: list[str], prefix: list[str] = ()):
    import json
    so = tmp_path / "liboracle_variant.so"
    r = subprocess.run([sys.executable, "-c", RUNNER, ROOT, str(so), json.dumps(defines),
                        json.dumps([grammar, toks, list(prefix)])],
                       capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    return json.loads(r.stdout.strip().splitlines()[-1])


ALL = ("masks", "allowed", "advance")
CASES = [
    # (capacity, tiny value, error bit, grammar, tokens, prefix, calls that reach it)
    # two distinct pending lexemes in one mask call (each single-token call has a fresh cache)
    ("ORACLE_TP_SLOTS", 1, 16, ARITH, ["1", "ab", "+"], [], ("masks",)),
    ("ORACLE_MAX_CLASS", 1, 1, KEYWORD, ["if;", "x", ";"], [], ALL),    # "if" is a class of two terminals
    ("ORACLE_LOC_MAX", 4, 8, PARENS, ["((((((", "(", ")"], [], ALL),     # six pushes on a depth-1 stack
    ("ORACLE_MAX_EMIT", 1, 4, ARITH, ["1+2", "1", "+"], [], ALL),        # two lexemes emitted, one pending
    ("ORACLE_MAX_STEPS", 1, 32, ARITH, ["+", "*", ")"], ["1 "], ALL),    # reductions before the shift
]


@pytest.mark.parametrize("macro,value,bit,grammar,toks,prefix,calls", CASES, ids=[c[0] for c in CASES])
def test_capacity_raises_instead_of_masking(tmp_path, macro, value, bit, grammar, toks, prefix, calls):
    got = _run(tmp_path, {macro: value}, grammar, toks, prefix)
    for call in calls:
        kind, val = got[call]
        assert kind == "limit" and val & bit, (call, got)
    # the default capacities decide the same inputs
    ok = _run(tmp_path, {}, grammar, toks, prefix)
    for call in ("masks", "allowed", "advance"):
        assert ok[call][0] == "ok", (call, ok)


def test_ignored_and_kept_terminal_on_one_lexeme_raises(tmp_path):
    got = _run(tmp_path, {}, MIXED, ["a", " ", "a a"], ["a"])
    assert got["masks"][0] == "limit" and got["masks"][1] & 2, got
