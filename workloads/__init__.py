"""Seeded synthetic inputs (grammars, vocabularies, prefixes, logits) for the PSC
mask workloads.  Holds no lexing, parsing or masking logic."""
