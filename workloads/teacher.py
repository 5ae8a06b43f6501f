"""Seeded teacher-forcing samples: whole sentences of a workload's grammar
(positives) and the same sentences with one foreign token spliced in
(negatives), tokenized with the workload's vocabulary.

Shared by the GPU tests and the benchmark's teacher-forcing run.  Holds none of
the method's arithmetic: it draws derivations from the grammar's rule data and
tokenizes them by greedy longest match.  Seed stream 5 of the workload's config
id (``np.random.default_rng([config_id, 5])``).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from .configs import Workload, grammar_spec
from .sample import SentenceSampler, TrieTokenizer


@dataclass
class TeacherSet:
    positives: list[list[int]]     # token ids of whole sentences (no end-of-sequence id)
    negatives: list[list[int]]     # the same with one random token inserted
    inserted_at: list[int]         # token position of the inserted token in each negative


def teacher_set(w: Workload, n: int, max_bytes: int = 600, min_tokens: int = 8,
                seed_stream: int = 5) -> TeacherSet:
    """``n`` complete sentences of at most ``max_bytes`` bytes and at least
    ``min_tokens`` tokens, and their corrupted copies."""
    spec = grammar_spec(w.spec.id)
    rng = np.random.default_rng([w.spec.id, seed_stream])
    sampler = SentenceSampler(spec, max_depth=12)
    tok = TrieTokenizer(w.vocab)
    pos: list[list[int]] = []
    tries = 0
    while len(pos) < n and tries < 200 * n:
        tries += 1
        txt, finished = sampler.text(rng, max_bytes)
        if not finished or not txt:
            continue
        ids = tok.encode(txt)
        if len(ids) >= min_tokens:
            pos.append(ids)
    neg, where = [], []
    for ids in pos:
        k = int(rng.integers(0, len(ids) + 1))
        v = int(rng.integers(0, len(w.vocab) - 1))          # any token but end-of-sequence
        neg.append(ids[:k] + [v] + ids[k:])
        where.append(k)
    return TeacherSet(pos, neg, where)
