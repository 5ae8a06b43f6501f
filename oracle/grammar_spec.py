"""Oracle-side reader for the grammar text format (test infrastructure only).

This package is the CPU oracle for the PSC vocabulary mask.  It is test
infrastructure: only the tests, ``__graft_entry__.smoke()`` and the CPU baseline
leg of ``bench.py`` may import it.  It shares no code with the CUDA path.

The grammar format is a small Lark-like notation (the paper builds its lexer and
LALR(1) parser from Lark grammars, Section "Experimental Setup / Implementation"):

* ``name: alt | alt ...``        a rule (lower-case name); ``start`` is the start symbol
* ``NAME: /regex/``, ``NAME: "literal"``, ``NAME.p: ...``   a named terminal with priority p
  (default 0); a quoted literal inside a rule is an anonymous terminal with priority 1
* ``%ignore NAME``                the terminal is dropped by the lexer (never reaches the parser)
* ``%lexer basic|contextual``     how a lexeme matching several terminals is resolved
* items: symbol, ``"lit"``, ``( alts )``, ``[ alts ]``, postfix ``?`` ``*`` ``+``
* a physical line whose first non-blank character is ``|`` continues the previous rule;
  ``//`` at the start of a line is a comment.

EBNF is lowered to BNF by one fixed rule set, because the LALR state a
contextual lexer consults depends on the exact BNF:

* a parenthesised group with one alternative and no postfix operator is spliced inline;
* every other group gets a fresh nonterminal whose alternatives are the group's;
* ``X?`` and ``[alts]`` become ``__oN: <empty> | X``;
* ``X*`` becomes ``__sN: <empty> | __sN X`` (left recursive);
* ``X+`` becomes ``__pN: X | __pN X``;
* fresh nonterminals are numbered in the order in which their construct is closed.
"""
from __future__ import annotations

import re
from dataclasses import dataclass, field


class GrammarError(ValueError):
    pass


@dataclass
class Terminal:
    name: str           # display name; anonymous literals are named by their quoted text
    kind: str           # "regex" or "literal"
    pattern: bytes      # regex source (as bytes) or literal bytes
    priority: int
    ignored: bool = False


@dataclass
class Grammar:
    terminals: list[Terminal]
    rules: list[tuple[str, tuple[str, ...]]]     # BNF productions (lhs, rhs symbols)
    nonterminals: list[str]
    start: str
    lexer_mode: str
    term_index: dict[str, int] = field(default_factory=dict)

    def is_terminal(self, sym: str) -> bool:
        return sym in self.term_index


def _unescape_literal(body: str) -> bytes:
    out = bytearray()
    i = 0
    while i < len(body):
        ch = body[i]
        if ch == "\\":
            i += 1
            if i >= len(body):
                raise GrammarError("dangling escape in literal")
            e = body[i]
            if e == "n":
                out.append(10)
            elif e == "t":
                out.append(9)
            elif e == "r":
                out.append(13)
            elif e == "x":
                out.append(int(body[i + 1:i + 3], 16))
                i += 2
            else:
                out.extend(e.encode("utf-8"))
        else:
            out.extend(ch.encode("utf-8"))
        i += 1
    return bytes(out)


def _unescape_slashes(body: str) -> str:
    """Inside /regex/, the pair backslash-slash stands for a slash; every other
    escape is left for the regex reader."""
    out = []
    i = 0
    while i < len(body):
        if body[i] == "\\" and i + 1 < len(body):
            out.append("/" if body[i + 1] == "/" else body[i:i + 2])
            i += 2
        else:
            out.append(body[i])
            i += 1
    return "".join(out)


_TOKEN_RE = re.compile(
    r'\s+|"(?:[^"\\]|\\.)*"|/(?:[^/\\]|\\.)+/|[A-Za-z_][A-Za-z0-9_]*|[():|?*+\[\]]')


def _tokenize(text: str):
    toks = []
    i = 0
    while i < len(text):
        m = _TOKEN_RE.match(text, i)
        if not m:
            raise GrammarError(f"cannot read grammar near {text[i:i+20]!r}")
        s = m.group(0)
        i = m.end()
        if not s.isspace():
            toks.append(s)
    return toks


def _logical_lines(text: str):
    lines = []
    for raw in text.splitlines():
        stripped = raw.strip()
        if not stripped or stripped.startswith("//"):
            continue
        if stripped.startswith("|"):
            if not lines:
                raise GrammarError("continuation line before any rule")
            lines[-1] += " " + stripped
        else:
            lines.append(stripped)
    return lines


def parse_grammar(text: str) -> Grammar:
    term_defs: list[Terminal] = []
    term_names: dict[str, int] = {}
    rule_defs: list[tuple[str, list]] = []
    ignores: list[str] = []
    lexer_mode = "basic"

    for line in _logical_lines(text):
        if line.startswith("%"):
            parts = line.split()
            if parts[0] == "%ignore" and len(parts) == 2:
                ignores.append(parts[1])
            elif parts[0] == "%lexer" and len(parts) == 2 and parts[1] in ("basic", "contextual"):
                lexer_mode = parts[1]
            else:
                raise GrammarError(f"unknown directive {line!r}")
            continue
        m = re.match(r"([A-Za-z_][A-Za-z0-9_]*)(?:\.(-?\d+))?\s*:(.*)$", line)
        if not m:
            raise GrammarError(f"cannot read line {line!r}")
        name, prio, body = m.group(1), m.group(2), m.group(3).strip()
        if name[0].isupper():
            if name in term_names:
                raise GrammarError(f"terminal {name} defined twice")
            if body.startswith('"') and body.endswith('"') and len(body) >= 2:
                kind, pat = "literal", _unescape_literal(body[1:-1])
            elif body.startswith("/") and body.endswith("/") and len(body) >= 2:
                kind, pat = "regex", _unescape_slashes(body[1:-1]).encode("utf-8")
            else:
                raise GrammarError(f"terminal {name} must be a literal or a regex")
            term_names[name] = len(term_defs)
            term_defs.append(Terminal(name, kind, pat, int(prio) if prio else 0))
        else:
            if prio is not None:
                raise GrammarError("rules take no priority")
            rule_defs.append((name, _tokenize(body)))

    nonterminals: list[str] = []
    nt_set = set()
    for lhs, _ in rule_defs:
        if lhs not in nt_set:
            nt_set.add(lhs)
            nonterminals.append(lhs)
    if "start" not in nt_set:
        raise GrammarError("grammar has no 'start' rule")

    rules: list[tuple[str, tuple[str, ...]]] = []
    counter = [0]

    def fresh(prefix: str) -> str:
        name = f"__{prefix}{counter[0]}"
        counter[0] += 1
        nonterminals.append(name)
        nt_set.add(name)
        return name

    def literal_terminal(tok: str) -> str:
        lit = _unescape_literal(tok[1:-1])
        if not lit:
            raise GrammarError("empty literal")
        disp = tok
        if disp not in term_names:
            term_names[disp] = len(term_defs)
            term_defs.append(Terminal(disp, "literal", lit, 1))
        return disp

    # recursive-descent over the token list of one rule body
    def parse_alts(toks, i, closer):
        alts = [[]]
        while i < len(toks):
            t = toks[i]
            if closer is not None and t == closer:
                return alts, i + 1
            if t == "|":
                alts.append([])
                i += 1
                continue
            item, i = parse_item(toks, i)
            alts[-1].extend(item)
        if closer is not None:
            raise GrammarError(f"missing {closer!r}")
        return alts, i

    def parse_item(toks, i):
        t = toks[i]
        if t == "(":
            alts, i = parse_alts(toks, i + 1, ")")
            group = ("group", alts)
        elif t == "[":
            alts, i = parse_alts(toks, i + 1, "]")
            group = ("opt", alts)
        elif t.startswith('"'):
            group = ("sym", literal_terminal(t))
            i += 1
        elif re.match(r"[A-Za-z_]", t):
            group = ("sym", t)
            i += 1
        else:
            raise GrammarError(f"unexpected {t!r} in rule")
        op = None
        if i < len(toks) and toks[i] in ("?", "*", "+"):
            op = toks[i]
            i += 1
        return lower(group, op), i

    def lower(group, op):
        kind, val = group
        if kind == "sym":
            inner = [[val]]
        else:
            inner = val
        if kind == "opt":
            if op is not None:
                raise GrammarError("[...] takes no postfix operator")
            op = "?"
        if op is None:
            if len(inner) == 1:
                return list(inner[0])
            nt = fresh("g")
            for alt in inner:
                rules.append((nt, tuple(alt)))
            return [nt]
        # X?, X*, X+ : X is a symbol, or the group's single alternative, or a fresh group nt
        if len(inner) == 1:
            x = list(inner[0])
        else:
            g = fresh("g")
            for alt in inner:
                rules.append((g, tuple(alt)))
            x = [g]
        if op == "?":
            nt = fresh("o")
            rules.append((nt, ()))
            rules.append((nt, tuple(x)))
        elif op == "*":
            nt = fresh("s")
            rules.append((nt, ()))
            rules.append((nt, (nt, *x)))
        else:
            nt = fresh("p")
            rules.append((nt, tuple(x)))
            rules.append((nt, (nt, *x)))
        return [nt]

    for lhs, toks in rule_defs:
        alts, _ = parse_alts(toks, 0, None)
        for alt in alts:
            rules.append((lhs, tuple(alt)))

    for ig in ignores:
        if ig not in term_names:
            raise GrammarError(f"%ignore of unknown terminal {ig}")
        term_defs[term_names[ig]].ignored = True

    for lhs, rhs in rules:
        for s in rhs:
            if s[0].isupper() or s.startswith('"'):
                if s not in term_names:
                    raise GrammarError(f"unknown terminal {s}")
                if term_defs[term_names[s]].ignored:
                    raise GrammarError(f"ignored terminal {s} used in a rule")
            elif s not in nt_set:
                raise GrammarError(f"unknown nonterminal {s}")

    g = Grammar(term_defs, rules, nonterminals, "start", lexer_mode)
    g.term_index = {t.name: i for i, t in enumerate(term_defs)}
    return g


def terminal_rank(g: Grammar) -> list[int]:
    """Resolution order of terminals that match the same lexeme: higher priority
    first, then byte-wise ascending name.  Returns rank[t] (0 = preferred)."""
    order = sorted(range(len(g.terminals)),
                   key=lambda t: (-g.terminals[t].priority, g.terminals[t].name.encode("utf-8")))
    rank = [0] * len(order)
    for r, t in enumerate(order):
        rank[t] = r
    return rank
