"""Oracle-side canonical LR(1) parser tables (Knuth's construction), test infrastructure only.

The paper models the parser as a deterministic, terminating push-down automaton
whose stack holds parser states (Section 2.4) and builds it as Lark's LALR(1)
tables (Section "Implementation").  The oracle deliberately uses a different
construction of the same language: the canonical LR(1) collection, built item
set by item set with explicit lookahead sets.  A canonical LR(1) parser shifts a
terminal exactly when the terminal prefix read so far followed by that terminal
is a prefix of some sentence, which is the acceptance test the mask needs.

The contextual lexer consults, for the current stack top, the set of terminals
on which Lark's LALR(1) table has an action.  LALR(1) is by definition canonical
LR(1) with states of equal core merged and lookaheads united, so the oracle
obtains that set by merging its own LR(1) states by core.
"""
from __future__ import annotations

from dataclasses import dataclass

from .grammar_spec import Grammar, GrammarError

ERR, SHIFT, REDUCE, ACCEPT = 0, 1, 2, 3


@dataclass
class LR1Tables:
    n_states: int
    n_terms: int                 # grammar terminals + 1 ($END is the last id)
    n_nonterms: int
    end_term: int
    act_kind: list[list[int]]    # [state][term]
    act_val: list[list[int]]     # shift target or rule index
    goto: list[list[int]]        # [state][nonterminal] -> state or -1
    rule_lhs: list[int]          # nonterminal index; rule 0 is the augmented start rule
    rule_len: list[int]
    core_of: list[int]           # LR(1) state -> core id (LALR state)
    n_cores: int
    lalr_acceptable: list[int]   # per core: bitmask over terminals with a non-error LALR action


def build_lr1(g: Grammar) -> LR1Tables:
    n_t = len(g.terminals)
    END = n_t
    nt_index = {name: i for i, name in enumerate(g.nonterminals)}
    aug = len(g.nonterminals)              # index of the augmented start symbol S'
    n_nt = aug + 1

    # symbols: terminals are ('t', id), nonterminals ('n', id)
    def sym(s: str):
        if s in g.term_index:
            return (0, g.term_index[s])
        return (1, nt_index[s])

    prods: list[tuple[int, tuple]] = [(aug, ((1, nt_index[g.start]),))]
    for lhs, rhs in g.rules:
        prods.append((nt_index[lhs], tuple(sym(s) for s in rhs)))
    by_lhs: list[list[int]] = [[] for _ in range(n_nt)]
    for p, (lhs, _) in enumerate(prods):
        by_lhs[lhs].append(p)

    # nullable and FIRST by fixpoint
    nullable = [False] * n_nt
    first = [0] * n_nt
    changed = True
    while changed:
        changed = False
        for lhs, rhs in prods:
            f = 0
            all_null = True
            for kind, v in rhs:
                if kind == 0:
                    f |= 1 << v
                    all_null = False
                    break
                f |= first[v]
                if not nullable[v]:
                    all_null = False
                    break
            if f & ~first[lhs]:
                first[lhs] |= f
                changed = True
            if all_null and not nullable[lhs]:
                nullable[lhs] = True
                changed = True

    # FIRST of every production suffix rhs[d:]
    suffix_first: list[list[tuple[int, bool]]] = []
    for lhs, rhs in prods:
        row = [(0, True)] * (len(rhs) + 1)
        for d in range(len(rhs) - 1, -1, -1):
            kind, v = rhs[d]
            if kind == 0:
                row[d] = (1 << v, False)
            else:
                nf, nn = row[d + 1]
                row[d] = (first[v] | (nf if nullable[v] else 0), nullable[v] and nn)
        suffix_first.append(row)

    def closure(kernel: dict) -> dict:
        items = dict(kernel)
        work = list(items.keys())
        while work:
            p, d = work.pop()
            rhs = prods[p][1]
            if d >= len(rhs) or rhs[d][0] != 1:
                continue
            b = rhs[d][1]
            f, nul = suffix_first[p][d + 1]
            la = f | (items[(p, d)] if nul else 0)
            for q in by_lhs[b]:
                key = (q, 0)
                old = items.get(key)
                if old is None:
                    items[key] = la
                    work.append(key)
                elif la & ~old:
                    items[key] = old | la
                    work.append(key)
        return items

    def key_of(kernel: dict):
        return tuple(sorted(kernel.items()))

    start_kernel = {(0, 0): 1 << END}
    states_kernel = [start_kernel]
    index = {key_of(start_kernel): 0}
    transitions: list[dict] = []
    closures: list[dict] = []
    i = 0
    while i < len(states_kernel):
        items = closure(states_kernel[i])
        closures.append(items)
        moves: dict = {}
        for (p, d), la in items.items():
            rhs = prods[p][1]
            if d < len(rhs):
                moves.setdefault(rhs[d], {})[(p, d + 1)] = la
        trans = {}
        for s, kern in moves.items():
            k = key_of(kern)
            j = index.get(k)
            if j is None:
                j = len(states_kernel)
                index[k] = j
                states_kernel.append(kern)
            trans[s] = j
        transitions.append(trans)
        i += 1

    n = len(states_kernel)
    act_kind = [[ERR] * (n_t + 1) for _ in range(n)]
    act_val = [[0] * (n_t + 1) for _ in range(n)]
    goto = [[-1] * n_nt for _ in range(n)]
    for s in range(n):
        for (kind, v), j in transitions[s].items():
            if kind == 0:
                act_kind[s][v] = SHIFT
                act_val[s][v] = j
            else:
                goto[s][v] = j
        for (p, d), la in closures[s].items():
            if d != len(prods[p][1]):
                continue
            for t in range(n_t + 1):
                if not (la >> t) & 1:
                    continue
                if p == 0:
                    kind, val = ACCEPT, 0
                else:
                    kind, val = REDUCE, p
                if act_kind[s][t] != ERR and (act_kind[s][t], act_val[s][t]) != (kind, val):
                    raise GrammarError(f"grammar is not LR(1): conflict in state {s} on terminal {t}")
                act_kind[s][t] = kind
                act_val[s][t] = val

    core_ids: dict = {}
    core_of = []
    for s in range(n):
        ck = tuple(sorted(states_kernel[s].keys()))
        core_of.append(core_ids.setdefault(ck, len(core_ids)))
    acceptable = [0] * len(core_ids)
    for s in range(n):
        m = 0
        for t in range(n_t + 1):
            if act_kind[s][t] != ERR:
                m |= 1 << t
        acceptable[core_of[s]] |= m

    return LR1Tables(n, n_t + 1, n_nt, END, act_kind, act_val, goto,
                     [lhs for lhs, _ in prods], [len(rhs) for _, rhs in prods],
                     core_of, len(core_ids), acceptable)
