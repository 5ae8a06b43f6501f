"""The seeded synthetic workloads (grammar, vocabulary, batch of prefixes, logits).

1. tiny arithmetic grammar, V=512, B=8, prefixes of 1-64 bytes, fp32 logits ~N(0,1)
2. JSON (RFC 8259), V=32,000, B=64, prefixes up to 512 bytes, bf16 logits ~N(0,2)
3. schema-conformant JSON, V=128,256, B=256, prefixes up to 1024 bytes, bf16 logits ~N(0,2)
4. C-like language, V=151,936, B=256, prefixes up to 2048 bytes, bf16 logits ~N(0,2)
5. C-like language, V=262,144, B=1024, prefixes of 64-4096 bytes biased to deep nesting,
   bf16 logits ~N(0,2), 32 decode steps
6. (extra) Java-sized language (1,001 LALR(1) states), V=4,096, B=64, prefixes of 64-2048 bytes
7. (extra) the same language with a pre-tokenized vocabulary of V=262,144 (the size of the
   paper's largest tokenizer), B=256, prefixes of 64-2048 bytes
8. (extra) SQL-like language (576 LALR(1) states, case-insensitive keywords), pre-tokenized
   vocabulary of V=128,256, B=256, prefixes of 64-2048 bytes

N(0,2) is read as variance 2 (sigma = sqrt 2).  The paper's datasets, JSON
schemas and tokenizers are not available; these stand in for them.
"""
from __future__ import annotations

import functools
import math
from dataclasses import dataclass

import numpy as np

from . import grammars
from .sample import TrieTokenizer, VocabSpec, build_prefixes, build_vocab, build_vocab_pretokenized


@dataclass(frozen=True)
class WorkloadSpec:
    id: int
    name: str
    B: int
    V: int
    dtype: str               # "f32" or "bf16"
    sigma: float
    prefix_min: int
    prefix_max: int
    vocab_max_len: int
    frac_grammar: float
    nest_bias: float = 1.0
    max_depth: int = 40
    decode_steps: int = 1
    vocab_style: str = "fragments"   # "fragments" or "pretokenized" (see sample.py)


SPECS = {
    1: WorkloadSpec(1, "arith_v512_b8", 8, 512, "f32", 1.0, 1, 64, 6, 400 / 413),
    2: WorkloadSpec(2, "json_v32000_b64", 64, 32000, "bf16", math.sqrt(2), 1, 512, 16, 0.4),
    3: WorkloadSpec(3, "schema_json_v128256_b256", 256, 128256, "bf16", math.sqrt(2), 1, 1024, 24,
                    0.5),
    4: WorkloadSpec(4, "c_like_v151936_b256", 256, 151936, "bf16", math.sqrt(2), 1, 2048, 32, 0.7),
    5: WorkloadSpec(5, "c_like_v262144_b1024", 1024, 262144, "bf16", math.sqrt(2), 64, 4096, 32, 0.7,
                    nest_bias=4.0, max_depth=500, decode_steps=32),
    # not one of the five benchmark configurations: a Java-sized grammar (1,001 LALR(1)
    # states, 533 productions, contextual lexer) for the construction at real-grammar
    # scale; its vocabulary is sized so that the construction fits a test run
    6: WorkloadSpec(6, "java_like_v4096_b64", 64, 4096, "bf16", math.sqrt(2), 64, 2048, 24, 0.7,
                    max_depth=60),
    # not a benchmark configuration either: the Java-sized grammar at the vocabulary size of
    # the paper's Java runs, with tokens that never mix letters and punctuation (the rule of
    # the byte-level BPE tokenizers the paper uses); 3 % of the tokens are punctuation runs
    7: WorkloadSpec(7, "java_like_pretok_v262144_b256", 256, 262144, "bf16", math.sqrt(2), 64, 2048, 24,
                    0.0, max_depth=60, vocab_style="pretokenized"),
    # not a benchmark configuration: the SQL-like grammar at the Llama 3 vocabulary size
    8: WorkloadSpec(8, "sql_like_pretok_v128256_b256", 256, 128256, "bf16", math.sqrt(2), 64, 2048, 24,
                    0.0, max_depth=40, vocab_style="pretokenized"),
}
# the Java-sized constructions build ~20 M states (6) and ~16 M states (7)
COMPILE_LIMITS = {6: {"max_states": 64_000_000}, 7: {"max_states": 64_000_000}, 8: {"max_states": 64_000_000}}


def grammar_spec(cfg: int) -> grammars.GrammarSpec:
    if cfg == 1:
        return grammars.arithmetic()
    if cfg == 2:
        return grammars.json_grammar()
    if cfg == 3:
        return grammars.schema_json(seed=int(np.random.default_rng([3, 1]).integers(0, 2**31)))
    if cfg in (6, 7):
        return grammars.java_like()
    if cfg == 8:
        return grammars.sql_like()
    return grammars.c_like()


@dataclass
class Workload:
    spec: WorkloadSpec
    grammar_text: str
    vocab: list[bytes]
    eos_id: int
    prefixes: list[bytes]
    prefix_ids: list[list[int]]

    @property
    def B(self):
        return self.spec.B

    @property
    def V(self):
        return self.spec.V

    def vocab_arrays(self):
        """(blob uint8, offsets int64[V+1]) of the vocabulary."""
        offs = np.zeros(len(self.vocab) + 1, dtype=np.int64)
        offs[1:] = np.cumsum([len(t) for t in self.vocab])
        blob = np.frombuffer(b"".join(self.vocab), dtype=np.uint8).copy()
        return blob, offs

    def token_matrix(self):
        """Prefix token ids as a [B][T] int32 matrix padded with -1 (no-op)."""
        T = max((len(p) for p in self.prefix_ids), default=0)
        m = np.full((self.B, max(T, 1)), -1, dtype=np.int32)
        for b, ids in enumerate(self.prefix_ids):
            m[b, :len(ids)] = ids
        return m

    def logits(self, step: int = 0):
        """Seeded CPU logits [B][V] (torch), fp32 or bf16."""
        import torch
        g = torch.Generator().manual_seed(1000 * self.spec.id + 4 + 7919 * step)
        x = torch.randn(self.B, self.V, generator=g) * self.spec.sigma
        return x if self.spec.dtype == "f32" else x.to(torch.bfloat16)


def vocab_spec(cfg: int, V: int | None = None) -> VocabSpec:
    s = SPECS[cfg]
    return VocabSpec(V or s.V, s.vocab_max_len, s.frac_grammar, style=s.vocab_style)


def vocab_for(cfg: int, V: int | None = None) -> list[bytes]:
    """Workload ``cfg``'s vocabulary (optionally at another size V)."""
    vs = vocab_spec(cfg, V)
    build = build_vocab_pretokenized if vs.style == "pretokenized" else build_vocab
    return build(grammar_spec(cfg), vs, [cfg, 2])


@functools.lru_cache(maxsize=8)
def load(cfg: int, batch: int | None = None) -> Workload:
    """Build workload ``cfg`` (optionally with only the first ``batch`` rows)."""
    s = SPECS[cfg]
    g = grammar_spec(cfg)
    vocab = vocab_for(cfg)
    B = s.B if batch is None else batch
    prefixes = build_prefixes(g, B, s.prefix_min, s.prefix_max, [cfg, 3],
                              max_depth=s.max_depth, nest_bias=s.nest_bias)
    tok = TrieTokenizer(vocab)
    ids = [tok.encode(p) for p in prefixes]
    spec = s if batch is None else WorkloadSpec(**{**s.__dict__, "B": B})
    return Workload(spec, g.text(), vocab, len(vocab) - 1, prefixes, ids)
