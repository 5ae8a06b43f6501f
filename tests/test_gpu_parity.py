"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Masks, masked logits and advanced parser states must be bit-exact.  Configs 1-3
are compared on every row and every token here; the two large workloads (configs
4 and 5) at full size in test_gpu_full_parity.py.
"""
from __future__ import annotations

import os

import numpy as np
import pytest

from oracle import ST_DONE, ST_ERROR, ST_OK, Oracle, Vocab
from workloads import configs, grammars

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

THREADS = os.cpu_count() or 1


@pytest.fixture(scope="module")
def psc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_03065_gb300 import build, psc as mod
    build.build()
    mod.load()
    return mod


class Case:
    """A workload compiled on the device, with device states and oracle configs
    advanced over the same prefix tokens."""

    def __init__(self, psc, cfg_id, cap=256, global_tables=False, packed_tables=False):
        self.w = configs.load(cfg_id)
        w = self.w
        self.h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, global_tables=global_tables,
                                 packed_tables=packed_tables)
        self.st = psc.psc_state_init(self.h, w.B, cap)
        tm = torch.from_numpy(w.token_matrix()).cuda()
        for j in range(tm.shape[1]):
            psc.psc_advance(self.h, self.st, tm[:, j].contiguous())
        torch.cuda.synchronize()
        self.o = Oracle(w.grammar_text)
        self.voc = Vocab.from_list(w.vocab, w.eos_id)
        self.ocs = []
        for ids in w.prefix_ids:
            oc = self.o.initial()
            self.o.advance_tokens(oc, self.voc, ids)
            self.ocs.append(oc)


_cases = {}


def case(psc, cfg_id):
    if cfg_id not in _cases:
        _cases[cfg_id] = Case(psc, cfg_id)
    return _cases[cfg_id]


def bits_of(mask_np, V):
    return np.unpackbits(mask_np.view(np.uint8), axis=-1, bitorder="little")[..., :V].astype(bool)


def sampled_oracle(c: Case, rows, tokens):
    """Oracle mask bits [len(rows)][len(tokens)] on a sub-vocabulary."""
    toks = [c.w.vocab[t] for t in tokens]
    eos_pos = [i for i, t in enumerate(tokens) if t == c.w.eos_id]
    sub = Vocab.from_list(toks, eos_pos[0] if eos_pos else -1)
    m = c.o.masks([c.ocs[r] for r in rows], sub, threads=THREADS)
    return bits_of(m, len(tokens))


def fill(psc, c):
    out = torch.empty(c.w.B, c.h.W, dtype=torch.int32, device="cuda")
    psc.psc_fill_mask(c.h, c.st, out)
    torch.cuda.synchronize()
    return out.cpu().numpy().view(np.uint32)


def reference_masked(logits_cpu, allowed):
    """where(allowed, logits, -inf) on raw bits."""
    if logits_cpu.dtype == torch.bfloat16:
        raw = logits_cpu.view(torch.int16).numpy().copy()
        raw[~allowed] = np.int16(-128)        # 0xFF80
    else:
        raw = logits_cpu.view(torch.int32).numpy().copy()
        raw[~allowed] = np.int32(-8388608)    # 0xFF800000
    return raw


def raw_bits(t):
    t = t.cpu()
    return t.view(torch.int16 if t.dtype == torch.bfloat16 else torch.int32).numpy()


# --------------------------------------------------------------- full parity
@pytest.mark.parametrize("cfg_id", [1, 2, 3])
def test_fill_mask_bit_exact(psc, cfg_id):
    c = case(psc, cfg_id)
    dev = fill(psc, c)
    ref = c.o.masks(c.ocs, c.voc, threads=THREADS)
    assert dev.shape == ref.shape
    bad = np.nonzero((dev != ref).any(axis=1))[0]
    assert len(bad) == 0, f"rows {bad[:10]} differ"


@pytest.mark.parametrize("cfg_id", [1, 2, 3])
def test_apply_and_fused_bit_exact(psc, cfg_id):
    c = case(psc, cfg_id)
    ref_mask = c.o.masks(c.ocs, c.voc, threads=THREADS)
    allowed = bits_of(ref_mask, c.w.V)
    logits = c.w.logits()
    want = reference_masked(logits, allowed)
    # unfused: fill_mask then apply_mask
    bm = torch.empty(c.w.B, c.h.W, dtype=torch.int32, device="cuda")
    psc.psc_fill_mask(c.h, c.st, bm)
    x = logits.cuda()
    psc.psc_apply_mask(x, bm, c.w.B, c.w.V)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(raw_bits(x), want)
    # fused, with the bitmask copy
    x2 = logits.cuda()
    bm2 = torch.zeros_like(bm)
    psc.psc_fill_apply(c.h, c.st, x2, bm2)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(raw_bits(x2), want)
    np.testing.assert_array_equal(bm2.cpu().numpy().view(np.uint32), ref_mask)


@pytest.mark.parametrize("cfg_id", [1, 2, 3])
def test_argmax_masked(psc, cfg_id):
    c = case(psc, cfg_id)
    allowed = bits_of(c.o.masks(c.ocs, c.voc, threads=THREADS), c.w.V)
    logits = c.w.logits()
    x = logits.cuda()
    tok = torch.empty(c.w.B, dtype=torch.int32, device="cuda")
    psc.psc_fill_apply(c.h, c.st, x)
    psc.psc_argmax_masked(c.h, c.st, x, tok)
    torch.cuda.synchronize()
    lf = logits.float().numpy()
    for b in range(c.w.B):
        idx = np.nonzero(allowed[b])[0]
        want = -1 if len(idx) == 0 else int(idx[np.argmax(lf[b, idx])])
        assert int(tok[b]) == want, b


def cpu_greedy(logits_cpu, allowed):
    """Lowest index of the largest allowed logit (NaN never wins), -1 if none."""
    lf = logits_cpu.float().numpy()
    out = np.full(lf.shape[0], -1, dtype=np.int64)
    for b in range(lf.shape[0]):
        idx = np.nonzero(allowed[b] & ~np.isnan(lf[b]))[0]
        if len(idx):
            out[b] = idx[np.argmax(lf[b, idx])]
    return out


@pytest.mark.parametrize("cfg_id", [1, 2, 3])
def test_fused_apply_argmax_bit_exact(psc, cfg_id):
    c = case(psc, cfg_id)
    ref_mask = c.o.masks(c.ocs, c.voc, threads=THREADS)
    allowed = bits_of(ref_mask, c.w.V)
    logits = c.w.logits(7)
    x = logits.cuda()
    bm = torch.zeros(c.w.B, c.h.W, dtype=torch.int32, device="cuda")
    tok = torch.empty(c.w.B, dtype=torch.int32, device="cuda")
    psc.psc_fill_apply_argmax(c.h, c.st, x, tok, bm)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(raw_bits(x), reference_masked(logits, allowed))
    np.testing.assert_array_equal(bm.cpu().numpy().view(np.uint32), ref_mask)
    np.testing.assert_array_equal(tok.cpu().numpy(), cpu_greedy(logits, allowed))


def test_fused_argmax_ties_nan_and_empty_rows(psc):
    """Ties go to the lowest index (+0 and -0 tie), NaN never wins, a row whose
    allowed logits are all NaN gets -1; vector (f32, bf16) and element paths."""
    g = grammars.json_grammar().text()
    singles = [bytes([b]) for b in range(0x20, 0x7F)]
    toks = singles + [a + b for a in singles[:40] for b in singles[:40]][:2000] + [b"true", b"false", b""]
    V = len(toks)
    h = psc.psc_compile(g, toks, V - 1)
    st = psc.psc_state_init(h, 3, 32)
    psc.psc_advance(h, st, torch.tensor([toks.index(b"["), -1, toks.index(b"{")], dtype=torch.int32,
                                        device="cuda"))
    bm = torch.empty(3, h.W, dtype=torch.int32, device="cuda")
    psc.psc_fill_mask(h, st, bm)
    allowed = bits_of(bm.cpu().numpy().view(np.uint32), V)
    for dt in (torch.float32, torch.bfloat16):
        for stride in (2048 + 16, V + 1):
            x = torch.zeros(3, stride, dtype=torch.float32)
            for b in range(3):
                idx = np.nonzero(allowed[b])[0]
                x[b, idx[0]] = float("nan")                     # the lowest allowed is NaN
                x[b, idx[1::2]] = -0.0                           # the rest tie at zero
            x[2, np.nonzero(allowed[2])[0]] = float("nan")       # row 2: nothing but NaN
            xd = x.to(dt).cuda()
            tok = torch.empty(3, dtype=torch.int32, device="cuda")
            psc.psc_fill_apply_argmax(h, st, xd, tok)
            t = tok.cpu().numpy()
            assert t[0] == np.nonzero(allowed[0])[0][1], (dt, stride)
            assert t[1] == np.nonzero(allowed[1])[0][1], (dt, stride)
            assert t[2] == -1, (dt, stride)


# ------------------------------------------------------------- decode loop
@pytest.mark.parametrize("cfg_id,steps,mode", [(2, 6, "separate"), (3, 3, "fused"), (2, 4, "step"),
                                                (3, 3, "split")])
def test_decode_loop_advance(psc, cfg_id, steps, mode):
    _decode_loop(psc, case(psc, cfg_id), steps, mode)


@pytest.mark.parametrize("tables", ["global", "packed"])
def test_decode_loop_table_paths(psc, tables):
    """The advance kernel with its tables read from global memory, or staged in
    the packed layout, decodes as the oracle says (JSON, whole decode steps)."""
    c = Case(psc, 2, global_tables=tables == "global", packed_tables=tables == "packed")
    assert (c.h.info().advance_table_bytes > 0) == (tables == "packed")
    assert c.h.info().advance_tables_packed == (tables == "packed")
    _decode_loop(psc, c, 5, "step")


def test_decode_step_advance_without_mask(psc):
    """The advance half with no masking pass before it finds no greedy choices:
    every token -1 and the rows unchanged."""
    w = configs.load(2, batch=8)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    st = psc.psc_state_init(h, w.B, 64)
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(min(tm.shape[1], 6)):
        psc.psc_advance(h, st, tm[:, j].contiguous())
    before = psc.psc_states_download(st)
    tok = torch.full((w.B,), 7, dtype=torch.int32, device="cuda")
    stat = torch.empty(w.B, dtype=torch.int32, device="cuda")
    psc.psc_decode_step_advance(h, st, tok, stat)
    after = psc.psc_states_download(st)
    assert (tok.cpu().numpy() == -1).all()
    np.testing.assert_array_equal(stat.cpu().numpy(), before["status"])
    for k in ("q", "depth", "stack", "status"):
        np.testing.assert_array_equal(after[k], before[k])


def test_state_copy_forks_a_batch(psc):
    """A copied batch decodes exactly like its source (same tokens, statuses and
    states after several steps); copies between mismatched batches are refused."""
    w = configs.load(2)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    a = psc.psc_state_init(h, w.B, 128)
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(h, a, tm[:, j].contiguous())
    b = psc.psc_state_init(h, w.B, 128)
    psc.psc_state_copy(b, a)
    ta = torch.empty(w.B, dtype=torch.int32, device="cuda")
    tb = torch.empty_like(ta)
    for step in range(4):
        logits = w.logits(50 + step)
        xa, xb = logits.cuda(), logits.cuda()
        psc.psc_decode_step(h, a, xa, ta)
        psc.psc_decode_step(h, b, xb, tb)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(ta.cpu().numpy(), tb.cpu().numpy())
        np.testing.assert_array_equal(raw_bits(xa), raw_bits(xb))
    da, db = psc.psc_states_download(a), psc.psc_states_download(b)
    for k in ("q", "depth", "status"):
        np.testing.assert_array_equal(da[k], db[k])
    for r in range(w.B):
        np.testing.assert_array_equal(da["stack"][r, :da["depth"][r]], db["stack"][r, :db["depth"][r]])
    small = psc.psc_state_init(h, w.B, 64)
    with pytest.raises(psc.PscError) as e:
        psc.psc_state_copy(small, a)
    assert e.value.code == 1


def test_decode_sequence_in_a_cuda_graph(psc):
    """A decode sequence (restore the batch from a saved copy, then 4 steps of
    psc_decode_step on fresh logits) captured once in a CUDA graph and replayed
    gives the same tokens, masked logits and states as running it eagerly."""
    w = configs.load(3, batch=32)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id)
    snap = psc.psc_state_init(h, w.B, 256)
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(h, snap, tm[:, j].contiguous())
    steps = 4
    pristine = [w.logits(70 + i).cuda() for i in range(steps)]
    # eager
    st_e = psc.psc_state_init(h, w.B, 256)
    psc.psc_state_copy(st_e, snap)
    tok_e, x_e = [], []
    for i in range(steps):
        x = pristine[i].clone()
        t = torch.empty(w.B, dtype=torch.int32, device="cuda")
        psc.psc_decode_step(h, st_e, x, t)
        tok_e.append(t)
        x_e.append(x)
    torch.cuda.synchronize()
    # captured
    st_g = psc.psc_state_init(h, w.B, 256)
    xs = [torch.empty_like(p) for p in pristine]
    toks = [torch.empty(w.B, dtype=torch.int32, device="cuda") for _ in range(steps)]
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        psc.psc_state_copy(st_g, snap)
        for i in range(steps):
            xs[i].copy_(pristine[i])
            psc.psc_decode_step(h, st_g, xs[i], toks[i])
    for rep in range(2):
        g.replay()
        torch.cuda.synchronize()
        for i in range(steps):
            np.testing.assert_array_equal(toks[i].cpu().numpy(), tok_e[i].cpu().numpy(), err_msg=f"step {i}")
            np.testing.assert_array_equal(raw_bits(xs[i]), raw_bits(x_e[i]))
        a, b = psc.psc_states_download(st_e), psc.psc_states_download(st_g)
        for k in ("q", "depth", "status"):
            np.testing.assert_array_equal(a[k], b[k])


def _decode_loop(psc, c, steps, mode):
    """fill_apply -> argmax -> advance for several steps; after every step the
    device masks equal the oracle's after advancing it by the same tokens
    (runs after the other tests of the same workload: it advances its states)."""
    B, V = c.w.B, c.w.V
    rng = np.random.default_rng(10 + B)
    rows = list(range(B)) if B <= 64 else sorted(rng.choice(B, size=16, replace=False).tolist())
    tok = torch.empty(B, dtype=torch.int32, device="cuda")
    stat = torch.empty(B, dtype=torch.int32, device="cuda")
    for step in range(steps):
        logits = c.w.logits(step + 1)
        x = logits.cuda()
        bm = torch.zeros(B, c.h.W, dtype=torch.int32, device="cuda")
        if mode == "step":
            psc.psc_decode_step(c.h, c.st, x, tok, bm, stat)
        elif mode == "split":
            psc.psc_decode_step_mask(c.h, c.st, x, bm)
            psc.psc_decode_step_advance(c.h, c.st, tok, stat)
        elif mode == "fused":
            psc.psc_fill_apply_argmax(c.h, c.st, x, tok, bm)
        else:
            psc.psc_fill_apply(c.h, c.st, x, bm)
            psc.psc_argmax_masked(c.h, c.st, x, tok)
        torch.cuda.synchronize()
        dev_mask = bm.cpu().numpy().view(np.uint32)
        ref = c.o.masks([c.ocs[r] for r in rows], c.voc, threads=THREADS)
        np.testing.assert_array_equal(dev_mask[rows], ref)
        allowed = bits_of(dev_mask, V)
        np.testing.assert_array_equal(tok.cpu().numpy(), cpu_greedy(logits, allowed))
        np.testing.assert_array_equal(raw_bits(x)[rows], reference_masked(logits[rows], allowed[rows]))
        if mode not in ("step", "split"):
            psc.psc_advance(c.h, c.st, tok, stat)
        torch.cuda.synchronize()
        t = tok.cpu().numpy()
        s = stat.cpu().numpy()
        for r in rows:
            if t[r] < 0:
                continue
            ost = c.o.advance(c.ocs[r], None if t[r] == c.w.eos_id else c.w.vocab[t[r]])
            want = {ST_OK: psc.ROW_OK, ST_DONE: psc.ROW_DONE, ST_ERROR: psc.ROW_REJECTED}[ost]
            assert s[r] == want, (step, r)


# ---------------------------------------------------------------- edge cases
def _small_vocab(n=1000, seed=0):
    rng = np.random.default_rng(seed)
    toks = {bytes([b]) for b in range(0x20, 0x7F)}
    alphabet = b"0123456789abcxyz+-*/() "
    while len(toks) < n - 1:
        k = int(rng.integers(2, 6))
        toks.add(bytes(alphabet[int(i)] for i in rng.integers(0, len(alphabet), k)))
    return sorted(toks) + [b""]


def test_ragged_vocab_unaligned_rows_and_statuses(psc):
    """V = 1000 (not a multiple of 32 or 1024), odd row strides (element path),
    rejected / finished / overflowed rows."""
    g = grammars.arithmetic().text()
    toks = _small_vocab()
    V, eos = len(toks), len(toks) - 1
    h = psc.psc_compile(g, toks, eos)
    o = Oracle(g)
    voc = Vocab.from_list(toks, eos)
    idx = {t: i for i, t in enumerate(toks)}
    prefixes = [b"", b"(1+", b"((((((((a", b"12*x", b"1", b"(", b")", b"((((((((((((((((((((((((1"]
    B, cap = len(prefixes), 16
    st = psc.psc_state_init(h, B, cap)
    ocs = []
    for b, p in enumerate(prefixes):
        oc = o.initial()
        for ch in p:
            o.advance(oc, bytes([ch]))
        ocs.append(oc)
    T = max(len(p) for p in prefixes)
    tm = np.full((B, T), -1, dtype=np.int32)
    for b, p in enumerate(prefixes):
        for j, ch in enumerate(p):
            tm[b, j] = idx[bytes([ch])]
    stat = torch.empty(B, dtype=torch.int32, device="cuda")
    tmd = torch.from_numpy(tm).cuda()
    for j in range(T):
        psc.psc_advance(h, st, tmd[:, j].contiguous(), stat)
    # row 4 finishes with EOS; row 7 overflows the 16-entry stack
    psc.psc_advance(h, st, torch.tensor([-1, -1, -1, -1, eos, -1, -1, -1], dtype=torch.int32, device="cuda"), stat)
    o.advance(ocs[4], None)
    info = psc.psc_states_download(st)
    assert info["status"][6] == psc.ROW_REJECTED           # ")" at the start
    assert info["status"][4] == psc.ROW_DONE
    assert info["status"][7] == psc.ROW_OVERFLOW
    ref = o.masks(ocs, voc)
    ref[7] = 0                                              # the oracle has no capacity limit
    bm = torch.empty(B, h.W, dtype=torch.int32, device="cuda")
    psc.psc_fill_mask(h, st, bm)
    np.testing.assert_array_equal(bm.cpu().numpy().view(np.uint32), ref)
    allowed = bits_of(ref, V)
    for dt in (torch.float32, torch.bfloat16):
        for stride in (V, V + 3, 1024):
            base = torch.randn(B, stride, generator=torch.Generator().manual_seed(stride)).to(dt)
            x = base.cuda()
            psc.psc_fill_apply(h, st, x[:, :V] if stride == V else x, None, V=V)
            torch.cuda.synchronize()
            want = reference_masked(base[:, :V].contiguous(), allowed)
            got = raw_bits(x)
            np.testing.assert_array_equal(got[:, :V], want)
            np.testing.assert_array_equal(got[:, V:], raw_bits(base)[:, V:])   # columns >= V untouched
    tok = torch.empty(B, dtype=torch.int32, device="cuda")
    x = torch.randn(B, V).cuda()
    psc.psc_argmax_masked(h, st, x, tok)
    t = tok.cpu().numpy()
    assert t[6] == -1 and t[7] == -1 and t[4] == eos


def test_nan_payloads_and_infinities_kept(psc):
    """Allowed logits keep their exact bits (NaN payloads, infinities, denormals),
    on the 16-byte vector path and on the element path."""
    g = grammars.json_grammar().text()
    singles = [bytes([b]) for b in range(0x20, 0x7F)]
    toks = singles + [a + b for a in singles[:40] for b in singles[:40]][:2000] + [b"true", b"false", b""]
    V = len(toks)
    h = psc.psc_compile(g, toks, V - 1)
    st = psc.psc_state_init(h, 2, 32)
    psc.psc_advance(h, st, torch.tensor([toks.index(b"["), -1], dtype=torch.int32, device="cuda"))
    bm = torch.empty(2, h.W, dtype=torch.int32, device="cuda")
    psc.psc_fill_mask(h, st, bm)
    allowed = bits_of(bm.cpu().numpy().view(np.uint32), V)
    pattern = np.array([0x7FC00001, 0x7F800000, -8388608, 0x00000001, 0x7FBFFFFF], dtype=np.int64)
    for stride in (2048 + 8, V + 1):
        raw = np.resize(pattern, (2, stride)).astype(np.int32)
        x = torch.from_numpy(raw.copy()).cuda().view(torch.float32)
        psc.psc_fill_apply(h, st, x, None, V=V)
        got = x.cpu().view(torch.int32).numpy()
        want = raw.copy()
        want[:, :V][~allowed] = np.int32(-8388608)
        np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("tables", ["staged", "global", "packed"])
def test_deep_stacks_and_long_pushes(psc, tables):
    """Balanced parentheses with tokens of up to 32 brackets: stacks grow to
    thousands of entries, past the advance kernel's shared-memory window (192
    entries copied in, 256 held), pushes of one token run beyond the window into
    global memory, and closing tokens pop below it; masks and statuses after every
    step equal the oracle's."""
    g = 'start: s\ns: | s "(" s ")"\n'
    toks = [b"(" * n for n in (1, 2, 7, 16, 31, 32)] + [b")" * n for n in (1, 3, 16, 32)] + [b"()", b")(", b""]
    eos = len(toks) - 1
    h = psc.psc_compile(g, toks, eos, global_tables=tables == "global", packed_tables=tables == "packed")
    o = Oracle(g)
    voc = Vocab.from_list(toks, eos)
    B, cap = 6, 8192
    st = psc.psc_state_init(h, B, cap)
    ocs = [o.initial() for _ in range(B)]
    rng = np.random.default_rng(77)
    bm = torch.empty(B, h.W, dtype=torch.int32, device="cuda")
    stat = torch.empty(B, dtype=torch.int32, device="cuda")
    for step in range(70):
        psc.psc_fill_mask(h, st, bm)
        m = bm.cpu().numpy().view(np.uint32)
        np.testing.assert_array_equal(m, o.masks(ocs, voc), err_msg=f"step {step}")
        allowed = bits_of(m, len(toks))
        tok = np.full(B, -1, dtype=np.int32)
        for r in range(B):
            opts = [t for t in np.nonzero(allowed[r])[0] if t != eos]
            # rows 0-2 mostly open (deep stacks), rows 3-5 open and close at random
            opens = [t for t in opts if toks[t].startswith(b"((")] if r < 3 else []
            tok[r] = int(rng.choice(opens)) if opens and rng.random() < 0.8 else int(rng.choice(opts))
        psc.psc_advance(h, st, torch.from_numpy(tok).cuda(), stat)
        s_dev = stat.cpu().numpy()
        for r in range(B):
            ost = o.advance(ocs[r], toks[tok[r]])
            want = {ST_OK: psc.ROW_OK, ST_DONE: psc.ROW_DONE, ST_ERROR: psc.ROW_REJECTED}[ost]
            assert s_dev[r] == want, (step, r, s_dev[r], want)
    d = psc.psc_states_download(st)
    assert d["depth"].max() > 1024     # the deep rows went far past the window
    for r in range(B):
        assert d["depth"][r] == ocs[r].info()["depth"]


@pytest.mark.parametrize("cfg_id,global_tables", [(4, False), (2, True)])
def test_bottom_up_and_top_down_classification_agree(psc, cfg_id, global_tables):
    """Decoding with the bottom-up classifier (each advance re-reads only the
    stack entries it pushed, from the blocks kept per stack prefix) and with
    top-down walks of the whole stack gives the same tokens, masked logits,
    statuses and stacks, also after a batch is forked (psc_state_copy) and some
    of its rows are reset."""
    w = configs.load(cfg_id, batch=64)
    hb = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, global_tables=global_tables)
    ht = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, global_tables=global_tables, bottom_up=False)
    assert hb.info().bottom_up_states > 0 and ht.info().bottom_up_states == 0
    B, cap = w.B, 512
    sb0, st = psc.psc_state_init(hb, B, cap), psc.psc_state_init(ht, B, cap)
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(hb, sb0, tm[:, j].contiguous())
        psc.psc_advance(ht, st, tm[:, j].contiguous())
    sb = psc.psc_state_init(hb, B, cap)
    psc.psc_state_copy(sb, sb0)
    rows = torch.tensor([1, 5, B - 1], dtype=torch.int32, device="cuda")
    psc.psc_state_reset(sb, rows)
    psc.psc_state_reset(st, rows)
    tb, tt = (torch.empty(B, dtype=torch.int32, device="cuda") for _ in range(2))
    sbs, sts = (torch.empty(B, dtype=torch.int32, device="cuda") for _ in range(2))
    mb, mt = (torch.zeros(B, hb.W, dtype=torch.int32, device="cuda") for _ in range(2))
    for step in range(8):
        logits = w.logits(90 + step)
        xb, xt = logits.cuda(), logits.cuda()
        psc.psc_decode_step(hb, sb, xb, tb, mb, sbs)
        psc.psc_decode_step(ht, st, xt, tt, mt, sts)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(mb.cpu().numpy(), mt.cpu().numpy(), err_msg=f"step {step}")
        np.testing.assert_array_equal(tb.cpu().numpy(), tt.cpu().numpy(), err_msg=f"step {step}")
        np.testing.assert_array_equal(sbs.cpu().numpy(), sts.cpu().numpy(), err_msg=f"step {step}")
        np.testing.assert_array_equal(raw_bits(xb), raw_bits(xt))
    psc.psc_fill_mask(hb, sb, mb)
    psc.psc_fill_mask(ht, st, mt)
    np.testing.assert_array_equal(mb.cpu().numpy(), mt.cpu().numpy())
    db, dt = psc.psc_states_download(sb), psc.psc_states_download(st)
    for k in ("q", "depth", "status"):
        np.testing.assert_array_equal(db[k], dt[k])
    for r in range(B):
        np.testing.assert_array_equal(db["stack"][r, :db["depth"][r]], dt["stack"][r, :dt["depth"][r]])
        if db["status"][r] == psc.ROW_OK:   # the host's bottom-up tables agree on the final stacks
            stack = db["stack"][r, :db["depth"][r]]
            assert hb.host_classify_bottom_up(int(db["q"][r]), stack) == ht.host_classify(int(db["q"][r]), stack)


def test_state_reset_rows(psc):
    c = case(psc, 2)
    rows = torch.tensor([0, 3, 5], dtype=torch.int32, device="cuda")
    h, w = c.h, c.w
    st = psc.psc_state_init(h, w.B, 256)
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(h, st, tm[:, j].contiguous())
    psc.psc_state_reset(st, rows)
    info = psc.psc_states_download(st)
    for r in (0, 3, 5):
        assert info["depth"][r] == 1 and info["q"][r] == 0 and info["status"][r] == psc.ROW_OK
    dev = torch.empty(w.B, h.W, dtype=torch.int32, device="cuda")
    psc.psc_fill_mask(h, st, dev)
    m0 = c.o.masks([c.o.initial()], c.voc)[0]
    for r in (0, 3, 5):
        np.testing.assert_array_equal(dev[r].cpu().numpy().view(np.uint32), m0)


def test_saved_tables_load_onto_the_device(psc, tmp_path):
    """psc_save then psc_load: the loaded handle's device path gives the same
    masks, masked logits and advanced states."""
    c = case(psc, 2)
    path = str(tmp_path / "json.psc")
    psc.psc_save(c.h, path)
    h2 = psc.psc_load(path)
    w = c.w
    st2 = psc.psc_state_init(h2, w.B, 256)
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(h2, st2, tm[:, j].contiguous())
    ocs = []
    for ids in w.prefix_ids:           # fresh configurations: other tests advance c.ocs
        oc = c.o.initial()
        c.o.advance_tokens(oc, c.voc, ids)
        ocs.append(oc)
    ref = c.o.masks(ocs, c.voc, threads=THREADS)
    bm = torch.empty(w.B, h2.W, dtype=torch.int32, device="cuda")
    psc.psc_fill_mask(h2, st2, bm)
    np.testing.assert_array_equal(bm.cpu().numpy().view(np.uint32), ref)


def test_bad_arguments_are_reported(psc):
    c = case(psc, 1)
    lib = psc.load()
    x = torch.zeros(c.w.B, c.w.V, device="cuda")
    bm = torch.zeros(c.w.B, c.h.W, dtype=torch.int32, device="cuda")
    assert lib.psc_fill_apply(c.h.ptr, c.st.ptr, c.w.B + 1, x.data_ptr(), 0, c.w.V, c.w.V, None, None) == 1
    assert lib.psc_apply_mask(x.data_ptr(), 0, c.w.V - 1, bm.data_ptr(), c.w.B, c.w.V, None) == 1
    assert lib.psc_apply_mask(x.data_ptr(), 7, c.w.V, bm.data_ptr(), c.w.B, c.w.V, None) == 1
    assert lib.psc_fill_mask(c.h.ptr, c.st.ptr, c.w.B, None, None) == 1
    assert b"bad arguments" in lib.psc_last_error()


def test_no_device_wait_gave_up(psc):
    """Every bounded wait inside the kernels (TMA pipeline, table staging) of all
    the tests above completed: the process-wide timeout counter is still zero."""
    c = case(psc, 1)
    assert c.h.info().device_timeouts == 0


@pytest.mark.parametrize("cfg_id", [1, 2, 3])
def test_sparse_classifier_layout_on_the_device(psc, cfg_id):
    """The classifier in the sparse layout (a default target and the exceptions
    to it per state; a warp reads one row per step) and no bottom-up classifier,
    so the device walks the sparse rows from the stack top: the masks of every
    row over every token equal the oracle's; four decode steps give the same
    masks, tokens, masked logits and statuses as the dense handle; the no-alloc
    entry point (its own classifier walk) agrees with psc_fill_apply."""
    w = configs.load(cfg_id)
    hs = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, bottom_up=False, max_dense_classifier_bytes=-1)
    hd = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, bottom_up=False)
    assert hs.info().classifier_sparse == 1 and hd.info().classifier_sparse == 0
    ss, sd = psc.psc_state_init(hs, w.B, 256), psc.psc_state_init(hd, w.B, 256)
    tm = torch.from_numpy(w.token_matrix()).cuda()
    for j in range(tm.shape[1]):
        psc.psc_advance(hs, ss, tm[:, j].contiguous())
        psc.psc_advance(hd, sd, tm[:, j].contiguous())
    o = Oracle(w.grammar_text)
    voc = Vocab.from_list(w.vocab, w.eos_id)
    ocs = []
    for ids in w.prefix_ids:
        oc = o.initial()
        o.advance_tokens(oc, voc, ids)
        ocs.append(oc)
    bm = torch.empty(w.B, hs.W, dtype=torch.int32, device="cuda")
    psc.psc_fill_mask(hs, ss, bm)
    np.testing.assert_array_equal(bm.cpu().numpy().view(np.uint32), o.masks(ocs, voc, threads=THREADS))
    # the no-alloc call classifies with its own walk over the sparse rows
    d = psc.psc_states_download(ss)
    logits = w.logits(60).cuda()
    a, b = logits.clone(), logits.clone()
    psc.psc_fill_apply(hs, ss, a)
    psc.psc_fill_apply_noalloc(hs, torch.from_numpy(d["q"]).cuda(), torch.from_numpy(d["depth"]).cuda(),
                               torch.from_numpy(d["status"]).cuda(), torch.from_numpy(d["stack"].view(np.int16)).cuda(), b)
    np.testing.assert_array_equal(raw_bits(a), raw_bits(b))
    ts, td = (torch.empty(w.B, dtype=torch.int32, device="cuda") for _ in range(2))
    xs_, xd_ = (torch.empty(w.B, dtype=torch.int32, device="cuda") for _ in range(2))
    for step in range(4):
        logits = w.logits(61 + step)
        x1, x2 = logits.cuda(), logits.cuda()
        b1, b2 = (torch.zeros(w.B, hs.W, dtype=torch.int32, device="cuda") for _ in range(2))
        psc.psc_decode_step(hs, ss, x1, ts, b1, xs_)
        psc.psc_decode_step(hd, sd, x2, td, b2, xd_)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(b1.cpu().numpy(), b2.cpu().numpy(), err_msg=f"step {step}")
        np.testing.assert_array_equal(ts.cpu().numpy(), td.cpu().numpy(), err_msg=f"step {step}")
        np.testing.assert_array_equal(xs_.cpu().numpy(), xd_.cpu().numpy(), err_msg=f"step {step}")
        np.testing.assert_array_equal(raw_bits(x1), raw_bits(x2))
