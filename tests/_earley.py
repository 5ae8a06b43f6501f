"""Earley recognizer used only to pin the oracle's parser (not part of the oracle).

A general context-free recognizer (Earley 1970) with the nullable-symbol fix of
Aycock and Horspool, over the BNF the oracle's grammar reader produces.  It
answers two questions about a terminal sequence without any LR construction:
is it a prefix of some sentence (``viable``), and is it a sentence (``accepts``).
"""
from __future__ import annotations


class Earley:
    def __init__(self, rules, start: str, terminals: set[str]):
        self.rules = [(lhs, tuple(rhs)) for lhs, rhs in rules]
        self.start = start
        self.terms = terminals
        self.by_lhs: dict[str, list[int]] = {}
        for i, (lhs, _) in enumerate(self.rules):
            self.by_lhs.setdefault(lhs, []).append(i)
        self.nullable = set()
        changed = True
        while changed:
            changed = False
            for lhs, rhs in self.rules:
                if lhs not in self.nullable and all(s in self.nullable for s in rhs):
                    self.nullable.add(lhs)
                    changed = True

    def _closure(self, items: set, sets: list, k: int):
        work = list(items)
        while work:
            r, d, o = work.pop()
            rhs = self.rules[r][1]
            if d < len(rhs):
                s = rhs[d]
                if s in self.terms:
                    continue
                for r2 in self.by_lhs.get(s, []):
                    it = (r2, 0, k)
                    if it not in items:
                        items.add(it)
                        work.append(it)
                if s in self.nullable:
                    it = (r, d + 1, o)
                    if it not in items:
                        items.add(it)
                        work.append(it)
            else:
                lhs = self.rules[r][0]
                src = items if o == k else sets[o]
                for (r2, d2, o2) in list(src):
                    rhs2 = self.rules[r2][1]
                    if d2 < len(rhs2) and rhs2[d2] == lhs:
                        it = (r2, d2 + 1, o2)
                        if it not in items:
                            items.add(it)
                            work.append(it)

    def _run(self, tokens):
        sets = []
        first = {(r, 0, 0) for r in self.by_lhs[self.start]}
        self._closure(first, sets, 0)
        sets.append(first)
        for k, t in enumerate(tokens, start=1):
            nxt = set()
            for (r, d, o) in sets[k - 1]:
                rhs = self.rules[r][1]
                if d < len(rhs) and rhs[d] == t:
                    nxt.add((r, d + 1, o))
            if not nxt:
                return sets, False
            self._closure(nxt, sets, k)
            sets.append(nxt)
        return sets, True

    def viable(self, tokens) -> bool:
        """True iff ``tokens`` is a prefix of some sentence (all symbols productive)."""
        return self._run(tokens)[1]

    def accepts(self, tokens) -> bool:
        sets, ok = self._run(tokens)
        if not ok:
            return False
        return any(self.rules[r][0] == self.start and d == len(self.rules[r][1]) and o == 0
                   for (r, d, o) in sets[-1])
