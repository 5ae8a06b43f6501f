"""Oracle-side regular expressions over bytes -> one Thompson NFA for all terminals.

Test infrastructure only (see ``oracle/grammar_spec.py``).  The lexer of the paper
is a finite-state transducer over the character set (Section 2.2); the oracle
takes the alphabet to be bytes and simulates the nondeterministic automaton of
the terminal regexes directly, state set by state set, with no determinisation.

Supported syntax: ``|``, concatenation, ``* + ?``, ``{m}``, ``{m,}``, ``{m,n}``,
``( )``, ``(?: )``, ``[...]`` / ``[^...]`` with ranges, ``.`` (any byte but
newline), escapes ``\\n \\t \\r \\f \\v \\xHH \\d \\D \\w \\W \\s \\S`` and an escaped
literal.  Characters outside ASCII stand for their UTF-8 bytes.
"""
from __future__ import annotations

from .grammar_spec import Grammar, GrammarError

ALL = (1 << 256) - 1


def _bit(b: int) -> int:
    return 1 << b


def _range(lo: int, hi: int) -> int:
    return ((1 << (hi + 1)) - 1) ^ ((1 << lo) - 1)


DIGIT = _range(48, 57)
WORD = DIGIT | _range(65, 90) | _range(97, 122) | _bit(95)
SPACE = _bit(32) | _bit(9) | _bit(10) | _bit(13) | _bit(12) | _bit(11)
SIMPLE_ESC = {ord("n"): 10, ord("t"): 9, ord("r"): 13, ord("f"): 12, ord("v"): 11}


class _Parser:
    """Regex source (bytes) -> AST of tuples: ('set', mask) | ('cat', [..]) |
    ('alt', [..]) | ('rep', node, lo, hi_or_None) | ('eps',)."""

    def __init__(self, src: bytes):
        self.s = src
        self.i = 0

    def peek(self):
        return self.s[self.i] if self.i < len(self.s) else None

    def take(self):
        c = self.s[self.i]
        self.i += 1
        return c

    def parse(self):
        node = self.alt()
        if self.i != len(self.s):
            raise GrammarError(f"regex: unexpected {chr(self.s[self.i])!r}")
        return node

    def alt(self):
        parts = [self.cat()]
        while self.peek() == ord("|"):
            self.take()
            parts.append(self.cat())
        return parts[0] if len(parts) == 1 else ("alt", parts)

    def cat(self):
        items = []
        while self.peek() is not None and self.peek() not in (ord("|"), ord(")")):
            items.append(self.postfix())
        if not items:
            return ("eps",)
        return items[0] if len(items) == 1 else ("cat", items)

    def postfix(self):
        node = self.atom()
        while True:
            c = self.peek()
            if c == ord("*"):
                self.take()
                node = ("rep", node, 0, None)
            elif c == ord("+"):
                self.take()
                node = ("rep", node, 1, None)
            elif c == ord("?"):
                self.take()
                node = ("rep", node, 0, 1)
            elif c == ord("{"):
                j = self.s.index(b"}", self.i)
                body = self.s[self.i + 1:j].decode()
                self.i = j + 1
                if "," in body:
                    lo, hi = body.split(",", 1)
                    node = ("rep", node, int(lo), int(hi) if hi.strip() else None)
                else:
                    node = ("rep", node, int(body), int(body))
            else:
                return node

    def escape_set(self) -> int:
        c = self.take()
        if c in SIMPLE_ESC:
            return _bit(SIMPLE_ESC[c])
        if c == ord("x"):
            v = int(self.s[self.i:self.i + 2].decode(), 16)
            self.i += 2
            return _bit(v)
        if c == ord("d"):
            return DIGIT
        if c == ord("D"):
            return ALL ^ DIGIT
        if c == ord("w"):
            return WORD
        if c == ord("W"):
            return ALL ^ WORD
        if c == ord("s"):
            return SPACE
        if c == ord("S"):
            return ALL ^ SPACE
        return _bit(c)

    def atom(self):
        c = self.take()
        if c == ord("("):
            if self.s[self.i:self.i + 2] == b"?:":
                self.i += 2
            node = self.alt()
            if self.peek() != ord(")"):
                raise GrammarError("regex: missing ')'")
            self.take()
            return node
        if c == ord("["):
            return ("set", self.char_class())
        if c == ord("."):
            return ("set", ALL ^ _bit(10))
        if c == ord("\\"):
            return ("set", self.escape_set())
        if c in (ord("*"), ord("+"), ord("?"), ord("{")):
            raise GrammarError("regex: nothing to repeat")
        return ("set", _bit(c))

    def class_atom(self):
        """One member of a character class: returns (mask, single_byte_or_None)."""
        c = self.take()
        if c == ord("\\"):
            save = self.i
            e = self.take()
            if e in SIMPLE_ESC:
                return _bit(SIMPLE_ESC[e]), SIMPLE_ESC[e]
            if e == ord("x"):
                v = int(self.s[self.i:self.i + 2].decode(), 16)
                self.i += 2
                return _bit(v), v
            if e in b"dDwWsS":
                self.i = save
                return self.escape_set(), None
            return _bit(e), e
        if c >= 128:
            raise GrammarError("regex: non-ASCII byte inside a character class")
        return _bit(c), c

    def char_class(self) -> int:
        neg = False
        if self.peek() == ord("^"):
            self.take()
            neg = True
        mask = 0
        first = True
        while True:
            c = self.peek()
            if c is None:
                raise GrammarError("regex: missing ']'")
            if c == ord("]") and not first:
                self.take()
                break
            first = False
            m, lo = self.class_atom()
            if self.peek() == ord("-") and lo is not None and self.i + 1 < len(self.s) \
                    and self.s[self.i + 1] != ord("]"):
                self.take()
                m2, hi = self.class_atom()
                if hi is None or hi < lo:
                    raise GrammarError("regex: bad range in class")
                mask |= _range(lo, hi)
            else:
                mask |= m
        return (ALL ^ mask) if neg else mask


class NFA:
    """Thompson NFA: every state has epsilon edges and at most one byte-set edge."""

    def __init__(self):
        self.eps: list[list[int]] = []
        self.edge: list[tuple[int, int] | None] = []   # (byte mask, target)
        self.accept: list[int] = []                      # terminal id or -1

    def new(self) -> int:
        self.eps.append([])
        self.edge.append(None)
        self.accept.append(-1)
        return len(self.eps) - 1

    def build(self, node) -> tuple[int, int]:
        """Fragment for an AST node: (entry, exit), exit has no edges yet."""
        kind = node[0]
        if kind == "eps":
            a = self.new()
            return a, a
        if kind == "set":
            if node[1] == 0:
                raise GrammarError("regex: empty character class")
            a, b = self.new(), self.new()
            self.edge[a] = (node[1], b)
            return a, b
        if kind == "cat":
            entry, cur = self.build(node[1][0])
            for sub in node[1][1:]:
                e2, x2 = self.build(sub)
                self.eps[cur].append(e2)
                cur = x2
            return entry, cur
        if kind == "alt":
            a, b = self.new(), self.new()
            for sub in node[1]:
                e2, x2 = self.build(sub)
                self.eps[a].append(e2)
                self.eps[x2].append(b)
            return a, b
        if kind == "rep":
            _, sub, lo, hi = node
            a = self.new()
            cur = a
            for _ in range(lo):
                e2, x2 = self.build(sub)
                self.eps[cur].append(e2)
                cur = x2
            if hi is None:
                e2, x2 = self.build(sub)
                loop_in = self.new()
                self.eps[cur].append(loop_in)
                self.eps[loop_in].append(e2)
                self.eps[x2].append(loop_in)
                out = self.new()
                self.eps[loop_in].append(out)
                return a, out
            out = self.new()
            for _ in range(hi - lo):
                self.eps[cur].append(out)
                e2, x2 = self.build(sub)
                self.eps[cur].append(e2)
                cur = x2
            self.eps[cur].append(out)
            return a, out
        raise AssertionError(kind)


def parse_regex(src: bytes):
    return _Parser(src).parse()


def literal_ast(lit: bytes):
    return ("cat", [("set", _bit(b)) for b in lit]) if len(lit) > 1 else ("set", _bit(lit[0]))


def build_lexer_nfa(g: Grammar) -> tuple[NFA, int]:
    """One NFA whose start state has an epsilon edge to every terminal's fragment;
    the exit of terminal t's fragment accepts t.  Returns (nfa, start)."""
    nfa = NFA()
    start = nfa.new()
    for t, term in enumerate(g.terminals):
        ast = literal_ast(term.pattern) if term.kind == "literal" else parse_regex(term.pattern)
        entry, exit_ = nfa.build(ast)
        nfa.accept[exit_] = t
        nfa.eps[start].append(entry)
    return nfa, start


def closure(nfa: NFA, states) -> frozenset:
    stack = list(states)
    seen = set(stack)
    while stack:
        s = stack.pop()
        for d in nfa.eps[s]:
            if d not in seen:
                seen.add(d)
                stack.append(d)
    return frozenset(seen)


def step(nfa: NFA, states: frozenset, byte: int) -> frozenset:
    nxt = []
    for s in states:
        e = nfa.edge[s]
        if e is not None and (e[0] >> byte) & 1:
            nxt.append(e[1])
    return closure(nfa, nxt)


def matches(nfa: NFA, start: int, data: bytes) -> set[int]:
    """Terminals whose language contains ``data`` (used by pins and grammar checks)."""
    cur = closure(nfa, [start])
    for b in data:
        cur = step(nfa, cur, b)
        if not cur:
            return set()
    return {nfa.accept[s] for s in cur if nfa.accept[s] >= 0}
