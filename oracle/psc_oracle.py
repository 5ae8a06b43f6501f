"""CPU oracle for the PSC per-step vocabulary mask (test infrastructure only).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this module.  It shares no code, tables or helpers with
the CUDA path; it takes the grammar text and the vocabulary bytes as its only
inputs and rebuilds everything with its own, deliberately different algorithms:

* lexer: the Thompson NFA of the terminal regexes, simulated state set by state
  set (``regex_thompson``), no determinisation or minimisation;
* parser: canonical LR(1) tables (``lr1_canonical``), not LALR(1);
* mask: for every row and every token, lex and parse (``brute.c``), which is the
  linear-in-vocabulary scheme of Fig. 1b evaluated against Eq. (3).

What it computes, per row (a prefix x with lexer state q and parser stack alpha,
Section 3.2) and token v of the vocabulary:

* an ordinary token is allowed iff lexing its bytes from the pending lexeme
  emits classes C1..Ck and leaves a pending lexeme p such that, for some D in
  T_p (Section 3.1; T_p = {empty} when p is empty, ignored classes count as
  empty), the parser consumes C1..Ck D from alpha and ends in a stable stack
  (every terminal shifted; Eq. 3 and Eq. 4);
* the end-of-sequence token is allowed iff p is empty, or p is a complete
  lexeme with class D, and consuming D (unless ignored) and then the end marker
  reaches the parser's accept action;
* a finished row allows only the end-of-sequence token, a failed row nothing.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

from .grammar_spec import Grammar, parse_grammar, terminal_rank
from .lr1_canonical import build_lr1
from .regex_thompson import build_lexer_nfa

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle_brute.so")
_lib = None

ST_OK, ST_DONE, ST_ERROR = 0, 1, 2

# bits of the checker's error word (brute.c): a capacity of the checker ran out
# (or the grammar mixes ignored and kept terminals in one lexeme); never a mask bit
ERRORS = {1: "a lexeme class has too many terminals", 2: "a lexeme matches an ignored and a kept terminal",
          4: "a token emits too many lexemes", 8: "too many stack entries pushed while checking a token",
          16: "the T_p cache is full", 32: "too many parser actions for one terminal"}


class OracleLimitError(RuntimeError):
    """The oracle could not decide: one of its checker's capacities ran out."""

    def __init__(self, bits: int):
        super().__init__("oracle capacity exceeded: " +
                         "; ".join(m for b, m in ERRORS.items() if bits & b))
        self.bits = bits


def build_library(force: bool = False, defines: dict | None = None, path: str | None = None) -> str:
    """Compile brute.c (plain C, pthreads) next to this file.  ``defines``
    overrides the checker's capacities (ORACLE_* macros) in a build at ``path``."""
    src = os.path.join(_HERE, "brute.c")
    out = path or _LIB_PATH
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    os.makedirs(os.path.dirname(out), exist_ok=True)
    tmp = out + f".{os.getpid()}.tmp"
    flags = [f"-D{k}={v}" for k, v in (defines or {}).items()]
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-pthread", *flags,
                           "-o", tmp, src])
    os.replace(tmp, out)
    return out


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build_library())
        vp = ctypes.c_void_p
        lib.oracle_config_new.restype = vp
        lib.oracle_config_new.argtypes = [vp, ctypes.c_int]
        lib.oracle_config_copy.restype = vp
        lib.oracle_config_copy.argtypes = [vp, vp]
        lib.oracle_config_free.argtypes = [vp]
        lib.oracle_config_get.argtypes = [vp, vp, vp, vp, vp, ctypes.c_int]
        lib.oracle_config_pending.argtypes = [vp, vp, vp]
        lib.oracle_advance.argtypes = [vp, vp, ctypes.c_char_p, ctypes.c_int, ctypes.c_int]
        lib.oracle_masks.argtypes = [vp, vp, ctypes.c_int, vp, vp, ctypes.c_int, ctypes.c_int,
                                     vp, ctypes.c_int]
        lib.oracle_allowed.argtypes = [vp, vp, ctypes.c_char_p, ctypes.c_int, ctypes.c_int]
        _lib = lib
    return _lib


class _OTables(ctypes.Structure):
    _fields_ = [
        ("n_nfa", ctypes.c_int), ("words", ctypes.c_int), ("nfa_start", ctypes.c_int),
        ("eps_off", ctypes.c_void_p), ("eps_dst", ctypes.c_void_p),
        ("edge_set", ctypes.c_void_p), ("edge_dst", ctypes.c_void_p), ("accept", ctypes.c_void_p),
        ("n_lex_terms", ctypes.c_int), ("term_rank", ctypes.c_void_p), ("term_ignored", ctypes.c_void_p),
        ("byte_reps", ctypes.c_void_p), ("n_byte_reps", ctypes.c_int),
        ("n_lr", ctypes.c_int), ("n_terms", ctypes.c_int), ("n_nt", ctypes.c_int),
        ("end_term", ctypes.c_int), ("contextual", ctypes.c_int),
        ("act_kind", ctypes.c_void_p), ("act_val", ctypes.c_void_p), ("go", ctypes.c_void_p),
        ("rule_lhs", ctypes.c_void_p), ("rule_len", ctypes.c_void_p), ("core_of", ctypes.c_void_p),
        ("acceptable", ctypes.c_void_p),
    ]


@dataclass
class Vocab:
    """Token byte strings packed as one blob plus offsets (token v = blob[off[v]:off[v+1]])."""
    blob: np.ndarray      # uint8
    offsets: np.ndarray   # int64, V+1
    eos_id: int

    @property
    def V(self) -> int:
        return len(self.offsets) - 1

    def token(self, v: int) -> bytes:
        return self.blob[self.offsets[v]:self.offsets[v + 1]].tobytes()

    @staticmethod
    def from_list(tokens: list[bytes], eos_id: int) -> "Vocab":
        offs = np.zeros(len(tokens) + 1, dtype=np.int64)
        offs[1:] = np.cumsum([len(t) for t in tokens])
        blob = np.frombuffer(b"".join(tokens), dtype=np.uint8).copy() if offs[-1] else np.zeros(1, np.uint8)
        return Vocab(blob, offs, eos_id)


class Config:
    """One row's lexer+parser configuration (pending lexeme NFA set, LR(1) stack, status)."""

    def __init__(self, oracle: "Oracle", ptr):
        self._o = oracle
        self._p = ptr

    def __del__(self):
        if getattr(self, "_p", None) and _lib is not None:
            _lib.oracle_config_free(self._p)
            self._p = None

    def copy(self) -> "Config":
        return Config(self._o, _load().oracle_config_copy(ctypes.byref(self._o._t), self._p))

    def info(self) -> dict:
        st, pl, d = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
        _load().oracle_config_get(self._p, ctypes.byref(st), ctypes.byref(pl), ctypes.byref(d), None, 0)
        stack = np.zeros(max(d.value, 1), dtype=np.int32)
        _load().oracle_config_get(self._p, ctypes.byref(st), ctypes.byref(pl), ctypes.byref(d),
                                  stack.ctypes.data, len(stack))
        return {"status": st.value, "pending_len": pl.value, "depth": d.value,
                "stack": stack[:d.value].tolist()}


class Oracle:
    """The oracle for one grammar: build once, then query configurations."""

    def __init__(self, grammar_text: str):
        self.grammar: Grammar = parse_grammar(grammar_text)
        g = self.grammar
        nfa, start = build_lexer_nfa(g)
        lr = build_lr1(g)
        self.lr1 = lr
        self.nfa = nfa
        n = len(nfa.eps)
        eps_off = np.zeros(n + 1, dtype=np.int32)
        eps_off[1:] = np.cumsum([len(e) for e in nfa.eps])
        eps_dst = np.array([d for e in nfa.eps for d in e] or [0], dtype=np.int32)
        edge_set = np.zeros((n, 8), dtype=np.uint32)
        edge_dst = np.full(n, -1, dtype=np.int32)
        masks = []
        for s, e in enumerate(nfa.edge):
            if e is None:
                continue
            m, d = e
            edge_dst[s] = d
            for w in range(8):
                edge_set[s, w] = (m >> (32 * w)) & 0xFFFFFFFF
            masks.append(m)
        # bytes that no edge set tells apart need only one visit while exploring T_p
        sig = {}
        for b in range(256):
            key = tuple((m >> b) & 1 for m in masks)
            sig.setdefault(key, b)
        byte_reps = np.array(sorted(sig.values()), dtype=np.int32)
        accept = np.array(nfa.accept, dtype=np.int32)
        rank = np.array(terminal_rank(g), dtype=np.int32)
        ignored = np.array([1 if t.ignored else 0 for t in g.terminals], dtype=np.uint8)
        act_kind = np.array(lr.act_kind, dtype=np.uint8)
        act_val = np.array(lr.act_val, dtype=np.int32)
        go = np.array(lr.goto, dtype=np.int32)
        acc = np.zeros((lr.n_cores, lr.n_terms), dtype=np.uint8)
        for c, m in enumerate(lr.lalr_acceptable):
            for t in range(lr.n_terms):
                acc[c, t] = (m >> t) & 1
        self._keep = [eps_off, eps_dst, edge_set, edge_dst, accept, rank, ignored, byte_reps,
                      act_kind, act_val, go, np.array(lr.rule_lhs, dtype=np.int32),
                      np.array(lr.rule_len, dtype=np.int32), np.array(lr.core_of, dtype=np.int32), acc]
        k = self._keep
        self._t = _OTables(
            n, (n + 63) // 64, start, k[0].ctypes.data, k[1].ctypes.data, k[2].ctypes.data,
            k[3].ctypes.data, k[4].ctypes.data, len(g.terminals), k[5].ctypes.data, k[6].ctypes.data,
            k[7].ctypes.data, len(byte_reps), lr.n_states, lr.n_terms, lr.n_nonterms, lr.end_term,
            1 if g.lexer_mode == "contextual" else 0, k[8].ctypes.data, k[9].ctypes.data,
            k[10].ctypes.data, k[11].ctypes.data, k[12].ctypes.data, k[13].ctypes.data,
            k[14].ctypes.data)
        _load()

    # ---------------------------------------------------------------- configs
    def initial(self) -> Config:
        """The configuration of the empty prefix: no pending lexeme, stack = [0]."""
        return Config(self, _load().oracle_config_new(ctypes.byref(self._t), 64))

    def advance(self, cfg: Config, token: bytes | None) -> int:
        """Commit one token in place (``None`` = end of sequence); returns the status."""
        if token is None:
            r = _load().oracle_advance(ctypes.byref(self._t), cfg._p, b"", 0, 1)
        else:
            r = _load().oracle_advance(ctypes.byref(self._t), cfg._p, token, len(token), 0)
        if r < 0:
            raise OracleLimitError(-r)
        return r

    def advance_tokens(self, cfg: Config, vocab: Vocab, ids) -> int:
        st = ST_OK
        for v in ids:
            v = int(v)
            st = self.advance(cfg, None if v == vocab.eos_id else vocab.token(v))
        return st

    def allowed(self, cfg: Config, token: bytes | None) -> bool:
        if token is None:
            r = _load().oracle_allowed(ctypes.byref(self._t), cfg._p, b"", 0, 1)
        else:
            r = _load().oracle_allowed(ctypes.byref(self._t), cfg._p, token, len(token), 0)
        if r < 0:
            raise OracleLimitError(-r)
        return bool(r)

    # ------------------------------------------------------------------ masks
    def masks(self, cfgs: list[Config], vocab: Vocab, threads: int | None = None) -> np.ndarray:
        """Packed masks [B][ceil(V/32)] uint32, bit v of word v>>5 at position v&31."""
        B, V = len(cfgs), vocab.V
        W = (V + 31) // 32
        out = np.zeros((B, W), dtype=np.uint32)
        arr = (ctypes.c_void_p * max(B, 1))(*[c._p for c in cfgs])
        threads = threads or os.cpu_count() or 1
        err = _load().oracle_masks(ctypes.byref(self._t), arr, B, vocab.blob.ctypes.data,
                                   vocab.offsets.ctypes.data, V, vocab.eos_id, out.ctypes.data, threads)
        if err:
            raise OracleLimitError(err)
        return out

    def mask_set(self, cfg: Config, vocab: Vocab) -> set[int]:
        m = self.masks([cfg], vocab, threads=1)[0]
        return {v for v in range(vocab.V) if (int(m[v >> 5]) >> (v & 31)) & 1}
