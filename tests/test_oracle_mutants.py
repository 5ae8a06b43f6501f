"""The oracle's pins catch planted mistakes: each case below copies the oracle's
C checker, plants one plausible mistake in the copy, builds it, and runs a
battery of the pins of test_oracle_pins.py against it in a child process.  The
unmodified source passes the battery; every mutant must fail at least one pin
(a crash counts as caught too, but none is expected).  Mistakes are planted in
the oracle only, on the CPU.  (Allowing the end of sequence on any non-error
result of the end marker instead of on accept is no mistake: the end marker is
never shifted, so that variant is equivalent and is not listed.)"""
from __future__ import annotations

import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "brute.c")

BATTERY = [
    "test_golden_hand_enumerated_masks", "test_golden_json_micro_masks",
    "test_closed_form_balanced_parentheses_deep", "test_closed_form_single_literal",
    "test_closed_form_any_bytes", "test_eq1_completion_search_arithmetic",
    "test_contextual_keyword_resolution", "test_contextual_uses_lalr_action_set",
    "test_terminal_rank_priority_then_name",
    "test_eos_only_after_complete_sentence", "test_sampled_sentences_are_sentences",
    ("test_earley_cross_check_workload", 1), ("test_invariants_on_workloads", 1),
    ("test_tokenwise_equals_bytewise", 1), ("test_tokenwise_equals_bytewise", 2),
    ("test_earley_cross_check_random_grammars", 40),
]

# name: (text in brute.c, replacement)
MUTANTS = {
    "pending lexeme's T_p ignored": (
        "if (plen == 0) return 1; /* T_p = {empty} */", "return 1;"),
    "basic lexer takes the lowest-ranked terminal": (
        "if (!T->contextual) return c->t[0];", "if (!T->contextual) return c->t[c->n - 1];"),
    "contextual lexer resolved like the basic one": (
        "if (!T->contextual) return c->t[0];", "return c->t[0];"),
    "end of sequence skips the pending lexeme's class": (
        "if (!T->term_ignored[cl.t[0]] && !feed_class(T, &W->ov, &cl)) return 0;", ";"),
    "end of sequence allowed without parsing to accept": (
        "return feed_terminal(T, &W->ov, T->end_term) == 2;", "return 1;"),
    "accept taken as a shift": (
        "if (k == K_ACCEPT) return 2;", "if (k == K_ACCEPT) return 1;"),
    "reductions pop one symbol too few": (
        "if (ov_pop(o, T->rule_len[v]) < 0) return 0;",
        "if (ov_pop(o, T->rule_len[v] > 1 ? T->rule_len[v] - 1 : T->rule_len[v]) < 0) return 0;"),
    "ignored lexemes fed to the parser": (
        "if (!cl.ignored) {", "if (1) {"),
    "byte after an emitted lexeme dropped": (
        """        set_start(L, pend);
        *plen = 0;
        set_step(L, pend, c, tmp);
        if (set_empty(tmp, T->words)) return -1;
        memcpy(pend, tmp, sizeof(uint64_t) * T->words);
        *plen = 1;""",
        """        set_start(L, pend);
        *plen = 0;"""),
}

RUNNER = r"""
import sys
sys.path.insert(0, sys.argv[1])
import oracle.psc_oracle as po
lib = sys.argv[2]
po.build_library = lambda force=False: lib
po._lib = None
import tests.test_oracle_pins as P
battery = %r
failed = []
for item in battery:
    name, args = (item, ()) if isinstance(item, str) else (item[0], item[1:])
    try:
        getattr(P, name)(*args)
    except AssertionError:
        failed.append(name)
print("failed pins:", failed)
sys.exit(3 if failed else 0)
""" % (BATTERY,)


def _build_and_run(tmp_path, source: str, tag: str):
    c = tmp_path / f"{tag}.c"
    so = tmp_path / f"lib{tag}.so"
    c.write_text(source)
    subprocess.check_call(["gcc", "-O1", "-std=c11", "-shared", "-fPIC", "-pthread", "-o", str(so), str(c)])
    return subprocess.run([sys.executable, "-c", RUNNER, ROOT, str(so)], capture_output=True, text=True,
                          timeout=300)


@pytest.fixture(scope="module")
def source():
    if shutil.which("gcc") is None:
        pytest.skip("gcc not available")
    return open(SRC).read()


def test_unmodified_oracle_passes_the_battery(source, tmp_path):
    r = _build_and_run(tmp_path, source, "control")
    assert r.returncode == 0, r.stdout + r.stderr


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(source, tmp_path, name):
    old, new = MUTANTS[name]
    assert source.count(old) == 1, "mutation site not found once: " + old
    r = _build_and_run(tmp_path, source.replace(old, new), "mutant")
    assert r.returncode != 0, f"mutant '{name}' passed every pin\n{r.stdout}{r.stderr}"
    assert r.returncode == 3 or r.returncode < 0, r.stdout + r.stderr
