"""Seeded random small grammars and vocabularies for differential tests (input
generation only: nothing here lexes, parses or masks).

Grammars mix literals with two regex terminals that collide with them (so
lexemes form classes), ignored whitespace, empty alternatives and recursion,
in both lexer modes; only productive rules are kept.
"""
from __future__ import annotations

LITS = ['"a"', '"b"', '"("', '")"', '"+"', '";"', '"ab"', '"if"']
REGEX = {"NUM": "/[0-9]+/", "ID": "/[a-z]+/"}
ALPHABET = b"ab()+;0 9zif"


def random_grammar(rng) -> str | None:
    """A random grammar text, or None when its start symbol derives no sentence."""
    nts = ["start", "x", "y", "z", "w", "v"][:int(rng.integers(2, 7))]
    terms = [str(t) for t in rng.choice(LITS, size=int(rng.integers(2, 6)), replace=False)]
    regs = [r for r in REGEX if rng.random() < 0.5]
    rules = {}
    for nt in nts:
        alts = []
        for _ in range(int(rng.integers(1, 4))):
            alts.append([str(rng.choice(nts)) if rng.random() < 0.4 else str(rng.choice(terms + regs))
                         for _ in range(int(rng.integers(0, 5)))])
        rules[nt] = alts
    productive, changed = set(), True
    while changed:
        changed = False
        for nt, alts in rules.items():
            if nt not in productive and any(all(s not in rules or s in productive for s in a) for a in alts):
                productive.add(nt)
                changed = True
    if "start" not in productive:
        return None
    lines = []
    for nt in nts:
        if nt in productive:
            alts = [a for a in rules[nt] if all(s not in rules or s in productive for s in a)]
            lines.append(f"{nt}: " + " | ".join(" ".join(a) for a in alts))
    used = {s for line in lines for s in line.split()}
    lines += [f"{r}: {REGEX[r]}" for r in regs if r in used]
    lines += ["WS: / +/", "%ignore WS", "%lexer " + ("contextual" if rng.random() < 0.5 else "basic")]
    return "\n".join(lines) + "\n"


def random_vocab(rng) -> list[bytes]:
    toks = {bytes([c]) for c in ALPHABET}
    while len(toks) < 30:
        toks.add(bytes(rng.choice(list(ALPHABET), size=int(rng.integers(2, 5)))))
    return sorted(toks) + [b""]
