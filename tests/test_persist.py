"""psc_save / psc_load: compiled tables round-trip through a file, and a
corrupt or truncated file is refused (host tables, no GPU needed)."""
from __future__ import annotations

import os

import numpy as np
import pytest

from workloads import configs


@pytest.fixture(scope="module")
def psc():
    from paper_2608_03065_gb300 import build, psc as mod
    build.build()
    mod.load()
    return mod


def test_round_trip_gives_identical_masks(psc, tmp_path):
    w = configs.load(2, batch=12)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True)
    path = str(tmp_path / "json.psc")
    psc.psc_save(h, path)
    h2 = psc.psc_load(path, host_only=True)
    i1, i2 = h.info(), h2.info()
    for f in ("V", "W", "n_lexer_states", "n_parser_states", "n_classifier_states", "n_masks", "eos_id",
              "classifier_bytes", "mask_bytes", "bottom_up_states", "bottom_up_bytes"):
        assert getattr(i1, f) == getattr(i2, f), f
    assert i2.bottom_up_states > 0
    h3 = psc.psc_load(path, host_only=True, bottom_up=False)   # loaded without the bottom-up classifier
    assert h3.info().bottom_up_states == 0
    for ids in w.prefix_ids:
        c1, c2 = h.host_initial(), h2.host_initial()
        for v in ids:
            c1, c2 = h.host_advance(c1, v), h2.host_advance(c2, v)
        assert c1 == c2
        m1 = h.host_mask_row(h.host_classify(c1["q"], c1["stack"], c1["status"]))
        m2 = h2.host_mask_row(h2.host_classify(c2["q"], c2["stack"], c2["status"]))
        np.testing.assert_array_equal(m1, m2)
        assert h2.host_classify_bottom_up(c2["q"], c2["stack"]) == h.host_classify(c1["q"], c1["stack"])
        assert h3.host_classify_bottom_up(c2["q"], c2["stack"]) == -2


def test_corrupt_and_truncated_files_are_refused(psc, tmp_path):
    w = configs.load(1, batch=2)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True)
    path = str(tmp_path / "a.psc")
    psc.psc_save(h, path)
    data = bytearray(open(path, "rb").read())
    bad = bytearray(data)
    bad[len(bad) // 2] ^= 0x40
    open(path + ".flip", "wb").write(bytes(bad))
    open(path + ".cut", "wb").write(bytes(data[:len(data) // 3]))
    open(path + ".junk", "wb").write(b"not a table file at all")
    for suffix in (".flip", ".cut", ".junk", ".missing"):
        with pytest.raises(psc.PscError) as e:
            psc.psc_load(path + suffix, host_only=True)
        assert e.value.code == 8, suffix


def test_tables_without_bottom_up_round_trip(psc, tmp_path):
    """A handle compiled without the bottom-up classifier saves and loads (the
    loaded handle has none either) and classifies as before."""
    w = configs.load(1, batch=4)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True, bottom_up=False)
    path = str(tmp_path / "plain.psc")
    psc.psc_save(h, path)
    h2 = psc.psc_load(path, host_only=True)
    assert h2.info().bottom_up_states == 0
    for ids in w.prefix_ids:
        c = h.host_initial()
        for v in ids:
            c = h.host_advance(c, v)
        assert h2.host_classify(c["q"], c["stack"]) == h.host_classify(c["q"], c["stack"])
        assert h2.host_classify_bottom_up(c["q"], c["stack"]) == -2


@pytest.fixture()
def uncompressed(monkeypatch):
    monkeypatch.setenv("PSC_SAVE_CODEC", "none")


def _payload_start(data: bytes) -> int:
    """Offset of the table payload in an uncompressed format-04 file: magic,
    codec and reserved words, payload size and block count, then the sizes of
    every block."""
    assert data[:8] == b"PSCTAB04" and int.from_bytes(data[8:12], "little") == 0
    nb = int.from_bytes(data[24:32], "little")
    return 32 + 16 * nb


@pytest.mark.parametrize("cfg_id,V", [(2, None), (8, 2048)])
def test_compiled_tables_do_not_depend_on_the_thread_count(psc, tmp_path, uncompressed, cfg_id, V):
    """Files compiled with 1 and with 8 host threads are byte-identical except
    for the recorded compile time (and so the checksum): table ids are numbered
    in an order that does not depend on which thread finishes first.  The
    SQL-like grammar at 2,048 tokens builds a million classifier states, so the
    minimisation's rounds run on many chunks in parallel."""
    text = configs.grammar_spec(cfg_id).text()
    toks = configs.vocab_for(cfg_id, V)
    data = []
    for th in (1, 8):
        h = psc.psc_compile(text, toks, len(toks) - 1, host_only=True, threads=th, bottom_up=V is None)
        path = str(tmp_path / f"t{th}.psc")
        psc.psc_save(h, path)
        data.append(open(path, "rb").read())
    a, b = data
    t0 = _payload_start(a) + 15 * 4 + 3 * 8   # 15 int32 and 3 int64 scalars, then the compile time (double)
    assert len(a) == len(b)
    assert a[:t0] == b[:t0] and a[t0 + 8:-8] == b[t0 + 8:-8]


def test_saved_files_are_compressed(psc, tmp_path, monkeypatch):
    """By default the tables are compressed (zstd when the system library loads,
    else zlib); every codec round-trips to the same tables."""
    w = configs.load(2, batch=4)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True)
    sizes = {}
    for codec in ("default", "none", "zlib", "zstd"):
        if codec == "default":
            monkeypatch.delenv("PSC_SAVE_CODEC", raising=False)
        else:
            monkeypatch.setenv("PSC_SAVE_CODEC", codec)
        path = str(tmp_path / f"{codec}.psc")
        psc.psc_save(h, path)
        data = open(path, "rb").read()
        sizes[codec] = (len(data), int.from_bytes(data[8:12], "little"))
        h2 = psc.psc_load(path, host_only=True)
        assert h2.info().n_classifier_states == h.info().n_classifier_states
        for ids in w.prefix_ids:
            c = h.host_initial()
            for v in ids:
                c = h.host_advance(c, v)
            assert h2.host_classify(c["q"], c["stack"]) == h.host_classify(c["q"], c["stack"])
    assert sizes["none"][1] == 0
    assert sizes["default"][1] in (1, 2) and sizes["default"][0] * 4 < sizes["none"][0]


def _fnv1a64(data: bytes) -> int:
    h = 1469598103934665603
    for b in data:
        h = ((h ^ b) * 1099511628211) & 0xFFFFFFFFFFFFFFFF
    return h


def test_inconsistent_bottom_up_tables_are_refused(psc, tmp_path, uncompressed):
    """A file whose checksum is right but whose bottom-up classifier names an LR
    state out of range (the last table of the file) fails validation."""
    w = configs.load(1, batch=2)
    h = psc.psc_compile(w.grammar_text, w.vocab, w.eos_id, host_only=True)
    path = str(tmp_path / "a.psc")
    psc.psc_save(h, path)
    data = bytearray(open(path, "rb").read())
    p0 = _payload_start(bytes(data))
    body = data[p0:-8]
    body[-4:] = (0x7FFF0000).to_bytes(4, "little")      # LR state of the last bottom-up block
    bad = bytes(data[:p0]) + bytes(body) + _fnv1a64(bytes(body)).to_bytes(8, "little")
    open(path + ".bad", "wb").write(bad)
    with pytest.raises(psc.PscError) as e:
        psc.psc_load(path + ".bad", host_only=True)
    assert e.value.code == 8 and "bottom-up" in str(e.value)
