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
# the larger variant: more literals (some prefixes of others), a string terminal
LITS_L = LITS + ['"{"', '"}"', '","', '"ba"', '"iff"']
REGEX_L = {**REGEX, "STR": '/"[a-z]*"/'}
ALPHABET_L = ALPHABET + b'{},"'


def random_grammar(rng, large: bool = False) -> str | None:
    """A random grammar text, or None when its start symbol derives no sentence.
    large: up to 9 nonterminals, 4 alternatives of up to 5 symbols, 8 literals."""
    lits, regex = (LITS_L, REGEX_L) if large else (LITS, REGEX)
    if large:
        nts = ["start"] + [f"n{i}" for i in range(int(rng.integers(2, 9)))]
        terms = [str(t) for t in rng.choice(lits, size=int(rng.integers(3, 9)), replace=False)]
    else:
        nts = ["start", "x", "y", "z", "w", "v"][:int(rng.integers(2, 7))]
        terms = [str(t) for t in rng.choice(lits, size=int(rng.integers(2, 6)), replace=False)]
    regs = [r for r in regex if rng.random() < 0.5]
    n_alt, n_sym, p_nt = (5, 6, 0.35) if large else (4, 5, 0.4)
    rules = {}
    for nt in nts:
        alts = []
        for _ in range(int(rng.integers(1, n_alt))):
            alts.append([str(rng.choice(nts)) if rng.random() < p_nt else str(rng.choice(terms + regs))
                         for _ in range(int(rng.integers(0, n_sym)))])
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
    lines += [f"{r}: {regex[r]}" for r in regs if r in used]
    lines += ["WS: / +/", "%ignore WS", "%lexer " + ("contextual" if rng.random() < 0.5 else "basic")]
    return "\n".join(lines) + "\n"


def random_vocab(rng, large: bool = False) -> list[bytes]:
    """Every single byte of the alphabet plus random strings; end of sequence last."""
    alphabet, size, longest = (ALPHABET_L, 60, 6) if large else (ALPHABET, 30, 5)
    toks = {bytes([c]) for c in alphabet}
    while len(toks) < size:
        toks.add(bytes(rng.choice(list(alphabet), size=int(rng.integers(2, longest)))))
    return sorted(toks) + [b""]
