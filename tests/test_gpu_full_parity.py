"""Full-size GPU parity on the large workloads, through the C ABI, against
the CPU oracle.

* C-like grammar, 151,936 tokens, 256 rows: four whole decode steps
  (psc_decode_step: masking pass + greedy choice + advance) on fresh logits;
  after every step the bitmask, the masked logits and the greedy tokens of all
  rows over all tokens, and the statuses of all rows, equal the oracle's.
* C-like grammar, 262,144 tokens, 1024 rows, at the prefix states: the masks
  and masked logits of psc_fill_apply and of the decode masking pass, all rows
  over all tokens, and the greedy tokens of all rows.
* The Java-sized grammar (1,001 LALR(1) states; classifier held sparse and
  walked from the top; parser tables packed to fit shared memory), 4,096 tokens,
  64 rows: all rows over all tokens at the prefix states and through six whole
  decode steps; then three more from the prefix states with the same tables read
  from global memory.
* The same grammar with a pre-tokenized vocabulary of 262,144 tokens, 256 rows,
  default options (bottom-up classifier too): all rows over all tokens at the
  prefix states (fused masking pass with the greedy choice) and through four
  whole decode steps.
* The SQL-like grammar (576 LALR(1) states) with a pre-tokenized vocabulary of
  128,256 tokens, 256 rows: all rows over all tokens at the prefix states and
  through three whole decode steps.
* The C-like 262,144-token workload at batches of 1, 3 and 16 rows (the
  small-batch masking pass): six whole decode steps, every row over every token.
* The C-like 262,144-token workload on the benchmark's exact path: the batch restored from a
  saved copy (psc_state_copy), then 32 steps of psc_decode_step_mask +
  psc_decode_step_advance on fresh logits; the oracle is advanced by the same
  tokens.  Every step: 64 rows (a different 64 each step, so every row is
  compared in full twice) are compared over all tokens (bitmask and masked
  logits); on every row, the chosen token is the greedy choice over the
  oracle's mask, checked exactly: the oracle allows the token and rejects every
  token whose logit is larger (or equal at a lower index); the bitmask of every
  row equals the oracle's on those tokens and on 512 random ones; the statuses
  of every row equal the oracle's.
"""
from __future__ import annotations

import os

import numpy as np
import pytest

from oracle import ST_DONE, ST_ERROR, ST_OK, Oracle, Vocab
from workloads import configs

from .test_gpu_parity import bits_of, cpu_greedy, raw_bits, reference_masked

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

THREADS = os.cpu_count() or 1
CAP = 256      # the benchmark's stack capacity


@pytest.fixture(scope="module")
def psc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_03065_gb300 import build, psc as mod
    build.build()
    mod.load()
    return mod


class Big:
    """A large workload compiled on the device: the prefix states saved in a
    states object, and the oracle's configurations of the same prefixes."""

    def __init__(self, psc, cfg_id, **opts):
        self.w = w = configs.load(cfg_id)
        self._prefix_states(psc, psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, **opts))
        self.o = Oracle(w.grammar_text)
        self.voc = Vocab.from_list(w.vocab, w.eos_id)
        self.ocs0 = []
        for ids in w.prefix_ids:
            oc = self.o.initial()
            self.o.advance_tokens(oc, self.voc, ids)
            self.ocs0.append(oc)

    def _prefix_states(self, psc, h):
        self.h = h
        self.snap = psc.psc_state_init(h, self.w.B, CAP)
        tm = torch.from_numpy(self.w.token_matrix()).cuda()
        for j in range(tm.shape[1]):
            psc.psc_advance(h, self.snap, tm[:, j].contiguous())
        torch.cuda.synchronize()

    def reloaded(self, psc, path, **opts):
        """The same workload on the tables saved and loaded back with other
        placement options (prefix states rebuilt on the new handle)."""
        psc.psc_save(self.h, path)
        other = object.__new__(Big)
        other.w, other.o, other.voc, other.ocs0 = self.w, self.o, self.voc, self.ocs0
        other._prefix_states(psc, psc.psc_load(path, **opts))
        return other

    def restored(self, psc):
        """A fresh states object restored from the saved prefix states, and
        copies of the oracle's configurations."""
        st = psc.psc_state_init(self.h, self.w.B, CAP)
        psc.psc_state_copy(st, self.snap)
        return st, [oc.copy() for oc in self.ocs0]


_big = {}


def big(psc, cfg_id, **opts):
    if cfg_id not in _big:
        _big[cfg_id] = Big(psc, cfg_id, **opts)
    return _big[cfg_id]


def device_logits(B, V, seed, sigma):
    """Seeded N(0, sigma^2) bf16 logits made on the device (as the benchmark
    makes them), and their host copy for the reference side."""
    g = torch.Generator(device="cuda").manual_seed(seed)
    x = (torch.randn(B, V, generator=g, device="cuda") * sigma).to(torch.bfloat16)
    return x, x.cpu()


STATUS = {ST_OK: 0, ST_DONE: 1, ST_ERROR: 2}


def whole_decode_all_rows_all_tokens(psc, b, steps, seed):
    """``steps`` whole decode steps (psc_decode_step) on fresh logits from the
    restored prefix states; after every step the bitmask, the masked logits and
    the greedy tokens of all rows over all tokens, and the statuses of all rows,
    equal the oracle's."""
    w = b.w
    B, V = w.B, w.V
    st, ocs = b.restored(psc)
    tok = torch.empty(B, dtype=torch.int32, device="cuda")
    stat = torch.empty(B, dtype=torch.int32, device="cuda")
    for step in range(steps):
        x, logits = device_logits(B, V, seed + step, w.spec.sigma)
        bm = torch.zeros(B, b.h.W, dtype=torch.int32, device="cuda")
        psc.psc_decode_step(b.h, st, x, tok, bm, stat)
        torch.cuda.synchronize()
        ref = b.o.masks(ocs, b.voc, threads=THREADS)
        np.testing.assert_array_equal(bm.cpu().numpy().view(np.uint32), ref, err_msg=f"step {step}")
        allowed = bits_of(ref, V)
        np.testing.assert_array_equal(raw_bits(x), reference_masked(logits, allowed), err_msg=f"step {step}")
        t = tok.cpu().numpy()
        np.testing.assert_array_equal(t, cpu_greedy(logits, allowed), err_msg=f"step {step}")
        s = stat.cpu().numpy()
        for r in range(B):
            if t[r] >= 0:
                ost = b.o.advance(ocs[r], None if t[r] == w.eos_id else w.vocab[t[r]])
                assert s[r] == STATUS[ost], (step, r, s[r], ost)


def test_c_like_151936_whole_decode_all_rows_all_tokens(psc):
    whole_decode_all_rows_all_tokens(psc, big(psc, 4), 4, 4000)


def test_java_sized_grammar_whole_decode_all_rows_all_tokens(psc, tmp_path):
    """Packed parser tables staged in shared memory (the default for this
    grammar), then the same tables read from global memory (k_advance +
    k_classify); the classifier sparse and walked from the top."""
    b = big(psc, 6, bottom_up=False, **configs.COMPILE_LIMITS[6])
    info = b.h.info()
    assert info.n_parser_states >= 1000 and info.classifier_sparse == 1
    assert info.advance_tables_packed == 1 and info.advance_table_bytes > 0
    whole_decode_all_rows_all_tokens(psc, b, 6, 7000)
    bg = b.reloaded(psc, str(tmp_path / "java.psc"), global_tables=True, bottom_up=False)
    assert bg.h.info().advance_table_bytes == 0
    whole_decode_all_rows_all_tokens(psc, bg, 3, 7100)


def test_java_sized_grammar_262144_pretokenized_all_rows_all_tokens(psc):
    """The Java-sized grammar at the paper's largest vocabulary size, with a
    pre-tokenized vocabulary, compiled with the default options (sparse
    classifier, bottom-up classifier, packed parser tables staged in shared
    memory): the fused masking pass at the prefix states, then four whole decode
    steps, every row over every token."""
    b = big(psc, 7, **configs.COMPILE_LIMITS[7])
    w = b.w
    info = b.h.info()
    assert info.n_parser_states >= 1000 and info.classifier_sparse == 1 and info.bottom_up_states > 0
    assert info.advance_tables_packed == 1
    assert w.V == 262144 and w.B == 256
    ref = b.o.masks(b.ocs0, b.voc, threads=THREADS)
    st, _ = b.restored(psc)
    x, logits = device_logits(w.B, w.V, 7500, w.spec.sigma)
    bm = torch.zeros(w.B, b.h.W, dtype=torch.int32, device="cuda")
    tok = torch.empty(w.B, dtype=torch.int32, device="cuda")
    psc.psc_fill_apply_argmax(b.h, st, x, tok, bm)
    torch.cuda.synchronize()
    allowed = bits_of(ref, w.V)
    np.testing.assert_array_equal(bm.cpu().numpy().view(np.uint32), ref)
    np.testing.assert_array_equal(raw_bits(x), reference_masked(logits, allowed))
    np.testing.assert_array_equal(tok.cpu().numpy(), cpu_greedy(logits, allowed))
    whole_decode_all_rows_all_tokens(psc, b, 4, 7600)


def test_c_like_262144_prefix_states_all_rows_all_tokens(psc):
    b = big(psc, 5)
    w = b.w
    B, V = w.B, w.V
    ref = b.o.masks(b.ocs0, b.voc, threads=THREADS)
    allowed = bits_of(ref, V)
    # fill + apply (classification from the kept state, masks from the device table)
    st, _ = b.restored(psc)
    x, logits = device_logits(B, V, 5000, w.spec.sigma)
    bm = torch.zeros(B, b.h.W, dtype=torch.int32, device="cuda")
    psc.psc_fill_apply(b.h, st, x, bm)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(bm.cpu().numpy().view(np.uint32), ref)
    np.testing.assert_array_equal(raw_bits(x), reference_masked(logits, allowed))
    # the decode masking pass (TMA-pipelined, greedy choice) on fresh logits
    x, logits = device_logits(B, V, 5001, w.spec.sigma)
    bm.zero_()
    tok = torch.empty(B, dtype=torch.int32, device="cuda")
    psc.psc_fill_apply_argmax(b.h, st, x, tok, bm)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(bm.cpu().numpy().view(np.uint32), ref)
    np.testing.assert_array_equal(raw_bits(x), reference_masked(logits, allowed))
    np.testing.assert_array_equal(tok.cpu().numpy(), cpu_greedy(logits, allowed))


def test_sql_like_128256_pretokenized_all_rows_all_tokens(psc):
    """The SQL-like grammar (576 LALR(1) states, case-insensitive keywords ranked
    above names, contextual lexer) with a pre-tokenized vocabulary of 128,256
    tokens, 256 rows (parser tables packed to fit shared memory, stacks walked from
    the top): the fused masking pass at the prefix states, then three whole decode
    steps, every row over every token."""
    b = big(psc, 8, bottom_up=False, **configs.COMPILE_LIMITS[8])
    w = b.w
    info = b.h.info()
    assert info.n_parser_states >= 500 and info.advance_tables_packed == 1
    assert w.V == 128256 and w.B == 256
    ref = b.o.masks(b.ocs0, b.voc, threads=THREADS)
    st, _ = b.restored(psc)
    x, logits = device_logits(w.B, w.V, 8500, w.spec.sigma)
    bm = torch.zeros(w.B, b.h.W, dtype=torch.int32, device="cuda")
    tok = torch.empty(w.B, dtype=torch.int32, device="cuda")
    psc.psc_fill_apply_argmax(b.h, st, x, tok, bm)
    torch.cuda.synchronize()
    allowed = bits_of(ref, w.V)
    np.testing.assert_array_equal(bm.cpu().numpy().view(np.uint32), ref)
    np.testing.assert_array_equal(raw_bits(x), reference_masked(logits, allowed))
    np.testing.assert_array_equal(tok.cpu().numpy(), cpu_greedy(logits, allowed))
    whole_decode_all_rows_all_tokens(psc, b, 3, 8600)


@pytest.mark.parametrize("B", [1, 3, 16])
def test_c_like_262144_small_batches_whole_decode(psc, B):
    """Batches of 1, 3 and 16 rows of the 262,144-token workload (the small-batch
    masking pass, a warp per 1024-column chunk, when the mask ids are current):
    six whole decode steps; after every step the bitmask (left out on odd steps),
    the masked logits and the greedy tokens of every row over every token, and
    the statuses, equal the oracle's."""
    b = big(psc, 5)
    w = b.w
    V = w.V
    st = psc.psc_state_init(b.h, B, CAP)
    tm = torch.from_numpy(w.token_matrix()[:B]).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(b.h, st, tm[:, j].contiguous())
    ocs = [oc.copy() for oc in b.ocs0[:B]]
    tok = torch.empty(B, dtype=torch.int32, device="cuda")
    stat = torch.empty(B, dtype=torch.int32, device="cuda")
    for step in range(6):
        x, logits = device_logits(B, V, 8000 + 10 * B + step, w.spec.sigma)
        bm = torch.zeros(B, b.h.W, dtype=torch.int32, device="cuda") if step % 2 == 0 else None
        psc.psc_decode_step(b.h, st, x, tok, bm, stat)
        torch.cuda.synchronize()
        ref = b.o.masks(ocs, b.voc, threads=THREADS)
        if bm is not None:
            np.testing.assert_array_equal(bm.cpu().numpy().view(np.uint32), ref, err_msg=f"step {step}")
        allowed = bits_of(ref, V)
        np.testing.assert_array_equal(raw_bits(x), reference_masked(logits, allowed), err_msg=f"step {step}")
        t = tok.cpu().numpy()
        np.testing.assert_array_equal(t, cpu_greedy(logits, allowed), err_msg=f"step {step}")
        s = stat.cpu().numpy()
        for r in range(B):
            if t[r] >= 0:
                ost = b.o.advance(ocs[r], None if t[r] == w.eos_id else w.vocab[t[r]])
                assert s[r] == STATUS[ost], (step, r, s[r], ost)


def greedy_rivals(xf, t):
    """Columns that would beat column t in the greedy choice over row xf (a
    larger value, or an equal value at a lower index; NaN never wins)."""
    xt = xf[t]
    idx = np.arange(len(xf))
    return np.nonzero((xf > xt) | ((xf == xt) & (idx < t)))[0]


def test_c_like_262144_benchmark_decode_path_32_steps(psc):
    b = big(psc, 5)
    w = b.w
    B, V, steps = w.B, w.V, w.spec.decode_steps
    assert steps == 32
    st, ocs = b.restored(psc)
    dead = np.zeros(B, dtype=bool)       # rows whose device stack overflowed (the oracle has no capacity)
    tok = torch.empty(B, dtype=torch.int32, device="cuda")
    stat = torch.empty(B, dtype=torch.int32, device="cuda")
    rng = np.random.default_rng(32)
    for step in range(steps):
        x, logits = device_logits(B, V, 6000 + step, w.spec.sigma)
        bm = torch.zeros(B, b.h.W, dtype=torch.int32, device="cuda")
        psc.psc_decode_step_mask(b.h, st, x, bm)
        psc.psc_decode_step_advance(b.h, st, tok, stat)
        torch.cuda.synchronize()
        dev_mask = bm.cpu().numpy().view(np.uint32)
        dev_bits = bits_of(dev_mask, V)
        t = tok.cpu().numpy()
        s = stat.cpu().numpy()
        live = [r for r in range(B) if not dead[r]]
        # 64 rows in full: bitmask and masked logits
        full = [r for r in range(step % 16, B, 16) if not dead[r]]
        ref_full = b.o.masks([ocs[r] for r in full], b.voc, threads=THREADS)
        np.testing.assert_array_equal(dev_mask[full], ref_full, err_msg=f"step {step}")
        rows_t = torch.tensor(full, device="cuda")
        np.testing.assert_array_equal(raw_bits(x.index_select(0, rows_t)),
                                      reference_masked(logits[full], bits_of(ref_full, V)), err_msg=f"step {step}")
        # every row: the token is the greedy choice over the oracle's mask
        xf = logits.float().numpy()
        rivals = {r: greedy_rivals(xf[r], int(t[r])) for r in live if t[r] >= 0}
        cols = set(rng.choice(V, size=512, replace=False).tolist()) | {w.eos_id}
        for r in live:
            if t[r] >= 0:
                cols.add(int(t[r]))
                cols.update(rivals[r].tolist())
        cols = sorted(cols)
        pos = {c: i for i, c in enumerate(cols)}
        eos_pos = pos[w.eos_id]
        sub = Vocab.from_list([w.vocab[c] for c in cols], eos_pos)
        ob = bits_of(b.o.masks([ocs[r] for r in live], sub, threads=THREADS), len(cols))
        np.testing.assert_array_equal(dev_bits[live][:, cols], ob, err_msg=f"step {step}")
        for i, r in enumerate(live):
            if t[r] >= 0:
                assert ob[i, pos[int(t[r])]], (step, r)
                assert not ob[i, [pos[c] for c in rivals[r].tolist()]].any(), (step, r)
            else:   # nothing allowed: the oracle's whole row is empty
                assert not b.o.masks([ocs[r]], b.voc, threads=THREADS).any(), (step, r)
        # statuses of every row after the advance
        for r in live:
            if t[r] < 0:
                continue
            if s[r] == psc.ROW_OVERFLOW:
                dead[r] = True
                continue
            ost = b.o.advance(ocs[r], None if t[r] == w.eos_id else w.vocab[t[r]])
            assert s[r] == STATUS[ost], (step, r, s[r], ost)
    # an overflow is the capacity, never a parse difference: those rows are deep
    for r in np.nonzero(dead)[0]:
        assert ocs[r].info()["depth"] > CAP - 64, r
    assert dead.sum() <= B // 100
