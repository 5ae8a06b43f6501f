"""Python restatement of the oracle's token check, used to pin ``oracle/brute.c``.

It reuses only the oracle's regex-to-NFA step (itself pinned against Python's
``re`` in ``test_oracle_pins.py``) and replaces the C lexer loop, the C T_p
exploration and the canonical LR(1) parser with plain Python and an Earley
recognizer.  Basic-lexer grammars only (class -> highest-ranked terminal).
"""
from __future__ import annotations

from oracle.grammar_spec import terminal_rank
from oracle.regex_thompson import build_lexer_nfa, closure, step

from ._earley import Earley


class PyCheck:
    def __init__(self, grammar):
        self.g = grammar
        self.nfa, self.start = build_lexer_nfa(grammar)
        self.rank = terminal_rank(grammar)
        self.start_set = closure(self.nfa, [self.start])
        names = {t.name for t in grammar.terminals}
        self.earley = Earley(grammar.rules, grammar.start, names)

    def cls(self, states):
        ts = sorted({self.nfa.accept[s] for s in states if self.nfa.accept[s] >= 0},
                    key=lambda t: self.rank[t])
        return ts

    def lex(self, data: bytes):
        """Max-munch lex from empty: (emitted terminal names, pending set, pending length) or None."""
        cur, plen, out = self.start_set, 0, []
        for c in data:
            nxt = step(self.nfa, cur, c)
            if nxt:
                cur, plen = nxt, plen + 1
                continue
            ts = self.cls(cur)
            if plen == 0 or not ts:
                return None
            if not self.g.terminals[ts[0]].ignored:
                out.append(self.g.terminals[ts[0]].name)
            cur = step(self.nfa, self.start_set, c)
            if not cur:
                return None
            plen = 1
        return out, cur, plen

    def tp(self, pend):
        """Classes (as first-ranked terminal name, or None for ignored) of every
        complete lexeme extending the pending set."""
        seen = {pend}
        work = [pend]
        res = set()
        while work:
            s = work.pop()
            ts = self.cls(s)
            if ts:
                t0 = self.g.terminals[ts[0]]
                res.add(None if t0.ignored else t0.name)
            for b in range(256):
                n = step(self.nfa, s, b)
                if n and n not in seen:
                    seen.add(n)
                    work.append(n)
        return res

    def allowed(self, prefix: bytes, token: bytes | None) -> bool:
        """Eq. (3) for the whole byte string prefix+token, parsed by Earley."""
        if token is None:
            r = self.lex(prefix)
            if r is None:
                return False
            z, pend, plen = r
            if plen == 0:
                return self.earley.accepts(z)
            ts = self.cls(pend)
            if not ts:
                return False
            t0 = self.g.terminals[ts[0]]
            return self.earley.accepts(z if t0.ignored else z + [t0.name])
        if not token:
            return False
        r = self.lex(prefix + token)
        if r is None:
            return False
        z, pend, plen = r
        if plen == 0:
            return self.earley.viable(z)
        return any(self.earley.viable(z if d is None else z + [d]) for d in self.tp(pend))

    def sentence(self, data: bytes) -> bool:
        """Membership of the whole byte string in the language (lex then parse)."""
        return self.allowed(data, None)
