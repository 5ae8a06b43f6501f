"""Seeded inputs for the five workloads: sentences, vocabularies, prefixes, logits.

Shared by the library's tests and benchmark and by the oracle's tests.  Holds
none of the method's arithmetic: it draws random derivations from a grammar's
rule data, cuts strings out of them, and tokenizes by greedy longest match.

Seed scheme: every stream is ``np.random.default_rng([config_id, stream])`` with
stream 1 = grammar, 2 = vocabulary, 3 = prefixes, 4 = logits (torch CPU
generator seeded with ``1000 * config_id + 4``).
"""
from __future__ import annotations

import collections
import re
from dataclasses import dataclass

import numpy as np

from .grammars import GrammarSpec, literal_bytes


def _is_literal(sym: str) -> bool:
    return sym.startswith('"')


def min_heights(spec: GrammarSpec) -> dict[str, int]:
    """Height of the shallowest derivation tree of each nonterminal."""
    INF = 1 << 30
    h = {nt: INF for nt in spec.rules}
    changed = True
    while changed:
        changed = False
        for nt, alts in spec.rules.items():
            for alt in alts:
                m = 0
                for s in alt:
                    if s in spec.rules:
                        m = max(m, h[s])
                if m + 1 < h[nt]:
                    h[nt] = m + 1
                    changed = True
    return h


class SentenceSampler:
    """Left-to-right random derivation that yields lexemes one at a time."""

    def __init__(self, spec: GrammarSpec, max_depth: int = 40, nest_bias: float = 1.0):
        self.spec = spec
        self.h = min_heights(spec)
        self.max_depth = max_depth
        self.nest_bias = nest_bias
        self.alt_h = {nt: [max([self.h[s] for s in a if s in spec.rules] or [0]) + 1 for a in alts]
                      for nt, alts in spec.rules.items()}

    def _choose(self, rng, nt: str, depth: int) -> list[str]:
        alts = self.spec.rules[nt]
        if depth >= self.max_depth:
            best = min(self.alt_h[nt])
            cands = [i for i, hh in enumerate(self.alt_h[nt]) if hh == best]
            return alts[cands[int(rng.integers(0, len(cands)))]]
        w = np.ones(len(alts))
        for i in range(len(alts)):
            w[i] *= self.spec.weights.get((nt, i), 1.0)
            if (nt, i) in self.spec.nesting:
                w[i] *= self.nest_bias
            # stay away from alternatives that cannot finish within the depth budget
            if depth + self.alt_h[nt][i] > self.max_depth:
                w[i] = 0.0
        if w.sum() == 0:
            w[:] = 1.0
        return alts[int(rng.choice(len(alts), p=w / w.sum()))]

    def lexemes(self, rng, budget_bytes: int):
        """Yield (symbol, lexeme bytes) until about budget_bytes have been produced
        or the derivation ends."""
        stack: list[tuple[str, int]] = [("start", 0)]
        produced = 0
        while stack and produced < budget_bytes:
            sym, d = stack.pop()
            if sym in self.spec.rules:
                alt = self._choose(rng, sym, d)
                for s in reversed(alt):
                    stack.append((s, d + 1))
                continue
            lex = literal_bytes(sym) if _is_literal(sym) else self.spec.terminals[sym].sample(rng)
            produced += len(lex)
            yield sym, lex

    def text(self, rng, budget_bytes: int) -> tuple[bytes, bool]:
        """Rendered text of at least budget_bytes (if the derivation is that long);
        the flag says whether the derivation finished (a complete sentence)."""
        out = bytearray()
        prev = None
        gen = self.lexemes(rng, budget_bytes)
        finished = True
        for sym, lex in gen:
            if prev is not None and self.spec.separator is not None:
                out += self.spec.separator(rng, prev, sym)
            out += lex
            prev = sym
            if len(out) >= budget_bytes:
                finished = False
                break
        return bytes(out), finished


# ------------------------------------------------------------------ vocabularies
@dataclass
class VocabSpec:
    size: int
    max_len: int
    frac_grammar: float          # fraction of fragments cut from grammar sentences
    unicode: bool = True
    style: str = "fragments"     # "fragments" or "pretokenized"
    frac_punct: float = 0.03     # pretokenized: fraction of punctuation-run tokens


PRINTABLE = [bytes([b]) for b in range(0x20, 0x7F)] + [b"\t", b"\n", b"\r"]
_UNI = ["é", "ü", "ñ", "ß", "ø", "λ", "π", "Ω", "ж", "я", "中", "文", "日", "本", "한", "글", "€", "→",
        "✓", "😀"]


def _random_text(rng, n: int, unicode: bool) -> bytes:
    out = bytearray()
    while len(out) < n:
        if unicode and rng.random() < 0.1:
            out += _UNI[int(rng.integers(0, len(_UNI)))].encode()
        else:
            out.append(int(rng.integers(0x20, 0x7F)))
    return bytes(out[:n]) if not unicode else bytes(out)


def build_vocab(spec: GrammarSpec, vs: VocabSpec, seed_key) -> list[bytes]:
    """A BPE-like vocabulary of ``vs.size`` unique byte strings: every single
    printable byte plus tab/newline/CR, fragments of sampled sentences (cut mostly
    at lexeme starts, lengths biased short), and random printable text; the last
    id is the end-of-sequence token (empty bytes)."""
    rng = np.random.default_rng(seed_key)
    toks: list[bytes] = list(PRINTABLE)
    seen = set(toks)
    n_target = vs.size - 1
    n_gram = int((n_target - len(toks)) * vs.frac_grammar)
    sampler = SentenceSampler(spec, max_depth=30)
    # fragments of grammar sentences
    corpus = bytearray()
    starts: list[int] = []
    n_added = 0
    stall = 0
    while n_added < n_gram and stall < 200000:
        if len(starts) < 64:
            txt, _ = sampler.text(rng, 4096)
            base = len(corpus)
            corpus += txt + b" "
            starts.extend(base + i for i in range(len(txt)) if i == 0 or txt[i - 1:i] in b" \n\t")
            starts.extend(base + int(i) for i in rng.integers(0, max(len(txt), 1), len(txt) // 8))
        s = starts.pop(int(rng.integers(0, len(starts))))
        ln = 1 + int(min(rng.geometric(0.22), vs.max_len - 1))
        frag = bytes(corpus[s:s + ln])
        if frag and len(frag) <= vs.max_len and frag not in seen:
            seen.add(frag)
            toks.append(frag)
            n_added += 1
            stall = 0
        else:
            stall += 1
    # random printable text
    while len(toks) < n_target:
        ln = 1 + int(min(rng.geometric(0.18), vs.max_len - 1))
        frag = _random_text(rng, ln, vs.unicode)
        if len(frag) <= vs.max_len and frag not in seen:
            seen.add(frag)
            toks.append(frag)
    perm = rng.permutation(len(toks))
    toks = [toks[int(i)] for i in perm]
    toks.append(b"")          # end of sequence
    return toks


# The splitting rule of byte-level BPE tokenizers of the GPT / Llama 3 / Qwen2.5
# kind (ASCII form): text is cut into words with at most one leading non-letter,
# numbers of up to three digits, punctuation runs with an optional leading space
# and trailing newlines, and whitespace runs; merges never cross a cut, so no
# token mixes letters with punctuation.
PRETOKEN = re.compile(rb"[^\r\nA-Za-z0-9]?[A-Za-z]+|[0-9]{1,3}| ?[^\sA-Za-z0-9]+[\r\n]*|\s*[\r\n]+|\s+(?!\S)|\s+")
_PUNCT_RUN = re.compile(rb" ?[^\sA-Za-z0-9]+[\r\n]*")
_PUNCT_CHARS = b"(){}[];,.=<>+-*/%&|^!~?:@\"'#$\\"


def build_vocab_pretokenized(spec: GrammarSpec, vs: VocabSpec, seed_key,
                             corpus_bytes: int = 1 << 20) -> list[bytes]:
    """A vocabulary shaped like a pre-tokenized byte-level BPE vocabulary of
    ``vs.size`` unique byte strings: every single printable byte; the pre-tokens
    of sampled grammar sentences and their prefixes (the intermediate merges) by
    frequency; punctuation runs (a fraction ``vs.frac_punct`` of the vocabulary:
    the corpus's own, then random runs over code punctuation); numbers 0-999;
    indentation runs; and, for the rest, natural-language words with at most one
    leading non-letter and some non-ASCII pieces.  Every token but the single
    bytes is one pre-token (PRETOKEN matches it whole).  The last id is the
    end-of-sequence token (empty bytes)."""
    rng = np.random.default_rng(seed_key)
    sampler = SentenceSampler(spec, max_depth=30)
    cnt: collections.Counter = collections.Counter()
    n = 0
    while n < corpus_bytes:
        txt, _ = sampler.text(rng, 4096)
        n += len(txt)
        for m in PRETOKEN.finditer(txt):
            p = m.group(0)
            cnt[p] += 1.0
            for k in range(2, len(p)):
                cnt[p[:k]] += 0.2
    toks: list[bytes] = list(PRINTABLE)
    seen = set(toks)
    n_target = vs.size - 1

    def add(t: bytes) -> bool:
        if t and t not in seen and len(t) <= vs.max_len and len(toks) < n_target \
                and PRETOKEN.fullmatch(t):
            seen.add(t)
            toks.append(t)
            return True
        return False

    ranked = [p for p, _ in sorted(cnt.items(), key=lambda kv: (-kv[1], kv[0]))]
    n_punct = int(vs.size * vs.frac_punct)
    k = 0
    for p in ranked:
        if k < n_punct and _PUNCT_RUN.fullmatch(p) and add(p):
            k += 1
    stall = 0
    while k < n_punct and stall < 100000:
        ln = 1 + int(min(rng.geometric(0.35), 7))
        r = bytes(_PUNCT_CHARS[int(i)] for i in rng.integers(0, len(_PUNCT_CHARS), ln))
        if rng.random() < 0.3:
            r = b" " + r
        if rng.random() < 0.2:
            r += b"\n" * int(rng.integers(1, 3))
        if add(r):
            k += 1
            stall = 0
        else:
            stall += 1
    for p in ranked:
        if len(toks) >= n_target // 4:
            break
        if not _PUNCT_RUN.fullmatch(p):
            add(p)
    for i in range(1000):
        add(str(i).encode())
    for w in range(2, 17):
        add(b" " * w)
        add(b"\n" + b" " * w)
        add(b"\t" * (w // 2))
    lead = [b"", b" ", b" ", b" ", b".", b"(", b"_", b"@", b"\"", b"'"]
    stall = 0
    while len(toks) < n_target and stall < 100000:
        if vs.unicode and rng.random() < 0.05:
            w = b" " + "".join(_UNI[int(i)] for i in rng.integers(0, len(_UNI), int(rng.integers(1, 4)))).encode()
        else:
            ln = int(rng.integers(1, 11))
            w = bytes(int(c) for c in rng.integers(ord("a"), ord("z") + 1, ln))
            if rng.random() < 0.3:
                w = w[:1].upper() + w[1:]
            w = lead[int(rng.integers(0, len(lead)))] + w
        stall = 0 if add(w) else stall + 1
    if len(toks) < n_target:
        raise ValueError(f"pretokenized vocabulary stalled at {len(toks)} of {n_target} tokens")
    perm = rng.permutation(len(toks))
    toks = [toks[int(i)] for i in perm]
    toks.append(b"")          # end of sequence
    return toks


# ---------------------------------------------------------------- tokenization
class TrieTokenizer:
    """Greedy longest-match tokenizer over a vocabulary (the end-of-sequence id,
    whose bytes are empty, never matches)."""

    def __init__(self, toks: list[bytes]):
        self.root: dict = {}
        for i, t in enumerate(toks):
            if not t:
                continue
            node = self.root
            for b in t:
                node = node.setdefault(b, {})
            node[-1] = i

    def encode(self, data: bytes) -> list[int]:
        ids = []
        i = 0
        while i < len(data):
            node = self.root
            best, best_len = -1, 0
            j = i
            while j < len(data) and data[j] in node:
                node = node[data[j]]
                j += 1
                if -1 in node:
                    best, best_len = node[-1], j - i
            if best < 0:
                raise ValueError(f"byte {data[i]:#x} is not in the vocabulary")
            ids.append(best)
            i += best_len
        return ids


# ---------------------------------------------------------------------- prefixes
def build_prefixes(spec: GrammarSpec, n: int, min_len: int, max_len: int, seed_key,
                   max_depth: int = 40, nest_bias: float = 1.0, max_draws: int = 100000) -> list[bytes]:
    """``n`` prefixes of sampled sentences, each exactly a uniform length in
    [min_len, max_len] bytes: a sentence is drawn again until it reaches the
    drawn length, then cut there (so short sentences do not skew the lengths)."""
    rng = np.random.default_rng(seed_key)
    sampler = SentenceSampler(spec, max_depth=max_depth, nest_bias=nest_bias)
    out = []
    for _ in range(n):
        target = int(rng.integers(min_len, max_len + 1))
        for _ in range(max_draws):
            txt, _ = sampler.text(rng, target)
            if len(txt) >= target:
                break
        else:
            raise RuntimeError(f"no sentence of {spec.name} reached {target} bytes in {max_draws} draws")
        out.append(txt[:target])
    return out
