"""Seeded synthetic grammars for the five benchmark workloads.

Each grammar is held as plain data (BNF rules, terminal patterns and a lexeme
sampler per terminal) so that this module can render the grammar text that the
library and the oracle both read, and can also sample sentences from the same
data to build vocabularies and prefixes.  Nothing here lexes, parses or masks:
it only writes grammar text and draws random strings.

The grammars stand in for the paper's workloads (Section "Datasets"), which are
not available: JSON, schema-conformant JSON generated from a JSON schema, and
programming-language grammars (Java, Go, SQL there; a synthetic C-like language
here).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Callable

import numpy as np

Sampler = Callable[[np.random.Generator], bytes]


@dataclass
class TermSpec:
    pattern: str                    # grammar-text form: /regex/ or "literal"
    sample: Sampler
    priority: int | None = None
    ignored: bool = False


@dataclass
class GrammarSpec:
    name: str
    rules: dict[str, list[list[str]]]        # BNF; a symbol in double quotes is a literal
    terminals: dict[str, TermSpec]
    lexer: str = "basic"
    # separator(rng, prev_sym, next_sym) -> bytes placed between two lexemes
    separator: Callable[[np.random.Generator, str, str], bytes] | None = None
    # extra weight per (nonterminal, alternative index) while sampling
    weights: dict[tuple[str, int], float] = field(default_factory=dict)
    # alternatives that nest (used to grow deep prefixes)
    nesting: set[tuple[str, int]] = field(default_factory=set)

    def text(self) -> str:
        lines = [f"// synthetic grammar: {self.name}"]
        for lhs, alts in self.rules.items():
            body = " | ".join(" ".join(a) for a in alts)
            lines.append(f"{lhs}: {body}")
        for name, t in self.terminals.items():
            pr = f".{t.priority}" if t.priority is not None else ""
            lines.append(f"{name}{pr}: {t.pattern}")
        for name, t in self.terminals.items():
            if t.ignored:
                lines.append(f"%ignore {name}")
        lines.append(f"%lexer {self.lexer}")
        return "\n".join(lines) + "\n"


def literal_bytes(sym: str) -> bytes:
    """Bytes of a quoted literal symbol as written in the grammar text."""
    body = sym[1:-1]
    out = bytearray()
    i = 0
    while i < len(body):
        c = body[i]
        if c == "\\":
            e = body[i + 1]
            out.extend({"n": b"\n", "t": b"\t", "r": b"\r"}.get(e, e.encode()))
            i += 2
        else:
            out.extend(c.encode())
            i += 1
    return bytes(out)


def _lit(s: str) -> str:
    """Grammar-text literal for the byte string s."""
    return '"' + s.replace("\\", "\\\\").replace('"', '\\"') + '"'


# ----------------------------------------------------------------- samplers
_LOWER = "abcdefghijklmnopqrstuvwxyz"
_ALNUM = _LOWER + "ABCDEFGHIJKLMNOPQRSTUVWXYZ0123456789_"


def _word(rng, lo=1, hi=8, alphabet=_LOWER) -> str:
    n = int(rng.integers(lo, hi + 1))
    return "".join(alphabet[int(i)] for i in rng.integers(0, len(alphabet), n))


def _digits(rng, lo=1, hi=6) -> str:
    n = int(rng.integers(lo, hi + 1))
    s = str(int(rng.integers(1, 10)))
    return s + "".join(str(int(d)) for d in rng.integers(0, 10, n - 1))


def _json_string(rng, hi=12) -> bytes:
    parts = []
    for _ in range(int(rng.integers(0, hi + 1))):
        r = rng.random()
        if r < 0.85:
            parts.append(chr(int(rng.integers(0x20, 0x7F))).replace('"', "'").replace("\\", "/"))
        elif r < 0.95:
            parts.append("\\" + "\"\\/bfnrt"[int(rng.integers(0, 8))])
        else:
            parts.append("\\u%04x" % int(rng.integers(0, 0x10000)))
    return ('"' + "".join(parts) + '"').encode()


def _json_number(rng) -> bytes:
    s = "-" if rng.random() < 0.2 else ""
    s += "0" if rng.random() < 0.1 else _digits(rng, 1, 5)
    if rng.random() < 0.3:
        s += "." + _digits(rng, 1, 3)
    if rng.random() < 0.1:
        s += "e" + "+-"[int(rng.integers(0, 2))] + _digits(rng, 1, 2)
    return s.encode()


def _json_integer(rng) -> bytes:
    s = "-" if rng.random() < 0.2 else ""
    return (s + ("0" if rng.random() < 0.1 else _digits(rng, 1, 6))).encode()


# ------------------------------------------------------------ 1: arithmetic
def arithmetic() -> GrammarSpec:
    """Tiny arithmetic-expression grammar: digits, [a-z]+ identifiers, + - * /,
    parentheses, optional whitespace (8 productions, LALR(1), basic lexer)."""
    rules = {
        "start": [["expr"]],
        "expr": [["expr", '"+"', "term"], ["expr", '"-"', "term"], ["term"]],
        "term": [["term", '"*"', "factor"], ["term", '"/"', "factor"], ["factor"]],
        "factor": [["NUMBER"], ["NAME"], ['"("', "expr", '")"']],
    }
    terms = {
        "NUMBER": TermSpec("/[0-9]+/", lambda r: _digits(r, 1, 4).encode()),
        "NAME": TermSpec("/[a-z]+/", lambda r: _word(r, 1, 5).encode()),
        "WS": TermSpec("/[ \\t\\n]+/", lambda r: b" ", ignored=True),
    }

    def sep(rng, a, b):
        return b" " if rng.random() < 0.4 else b""

    return GrammarSpec("arithmetic", rules, terms, "basic", sep,
                       weights={("factor", 2): 2.0, ("expr", 0): 1.5, ("term", 0): 1.5},
                       nesting={("factor", 2)})


# ------------------------------------------------------------------ 2: JSON
_JSON_STRING_RE = r'/"([^"\\\x00-\x1f]|\\(["\\\/bfnrt]|u[0-9a-fA-F]{4}))*"/'
_JSON_NUMBER_RE = r"/-?(0|[1-9][0-9]*)(\.[0-9]+)?([eE][+-]?[0-9]+)?/"


def _json_sep(rng, a, b):
    r = rng.random()
    if r < 0.55:
        return b""
    if r < 0.85:
        return b" "
    return b"\n" + b"  " * int(rng.integers(0, 4))


def json_grammar() -> GrammarSpec:
    """RFC 8259 JSON: objects, arrays, strings with escapes, numbers, true/false/null."""
    rules = {
        "start": [["value"]],
        "value": [["object"], ["array"], ["STRING"], ["NUMBER"], ['"true"'], ['"false"'], ['"null"']],
        "object": [['"{"', '"}"'], ['"{"', "members", '"}"']],
        "members": [["pair"], ["members", '","', "pair"]],
        "pair": [["STRING", '":"', "value"]],
        "array": [['"["', '"]"'], ['"["', "elements", '"]"']],
        "elements": [["value"], ["elements", '","', "value"]],
    }
    terms = {
        "STRING": TermSpec(_JSON_STRING_RE, _json_string),
        "NUMBER": TermSpec(_JSON_NUMBER_RE, _json_number),
        "WS": TermSpec("/[ \\t\\n\\r]+/", lambda r: b" ", ignored=True),
    }
    return GrammarSpec("json", rules, terms, "basic", _json_sep,
                       weights={("value", 0): 2.0, ("value", 1): 1.5, ("members", 1): 2.0,
                                ("elements", 1): 2.0},
                       nesting={("value", 0), ("value", 1)})


# ------------------------------------------------------- 3: schema JSON
def schema_json(seed: int = 1, n_props: int = 20, max_depth: int = 3) -> GrammarSpec:
    """Grammar of the instances of a seeded synthetic JSON schema: one object with
    ``n_props`` required properties in fixed order, nested objects to depth
    ``max_depth``, string enums of 4-12 values, integer/number/boolean fields and
    arrays of objects.  Contextual lexer (keys and enum values are literals that
    also match STRING; integers also match NUMBER)."""
    rng = np.random.default_rng(seed)
    rules: dict[str, list[list[str]]] = {}
    words = set()

    def fresh_word():
        while True:
            w = _word(rng, 3, 9)
            if w not in words:
                words.add(w)
                return w

    counter = [0]

    def obj(depth: int, n: int) -> str:
        name = f"obj{counter[0]}"
        counter[0] += 1
        seq = ['"{"']
        for k in range(n):
            key = _lit('"' + fresh_word() + '"')
            if k:
                seq.append('","')
            seq += [key, '":"', field_type(depth)]
        seq.append('"}"')
        rules[name] = [seq]
        return name

    def field_type(depth: int) -> str:
        r = rng.random()
        if depth < max_depth and r < 0.12:
            return obj(depth + 1, int(rng.integers(3, 7)))
        if depth < max_depth and r < 0.20:
            arr = f"arr{counter[0]}"
            counter[0] += 1
            item = obj(depth + 1, int(rng.integers(2, 5)))
            rules[arr] = [['"["', '"]"'], ['"["', arr + "_items", '"]"']]
            rules[arr + "_items"] = [[item], [arr + "_items", '","', item]]
            return arr
        if r < 0.40:
            en = f"enum{counter[0]}"
            counter[0] += 1
            rules[en] = [[_lit('"' + fresh_word() + '"')] for _ in range(int(rng.integers(4, 13)))]
            return en
        if r < 0.60:
            return "STRING"
        if r < 0.75:
            return "INTEGER"
        if r < 0.88:
            return "NUMBER"
        return "boolean"

    rules["start"] = []
    rules["boolean"] = [['"true"'], ['"false"']]
    root = obj(0, n_props)
    rules["start"] = [[root]]
    # keep "start" first in the text
    rules = {"start": rules.pop("start"), **rules}
    terms = {
        "STRING": TermSpec(_JSON_STRING_RE, _json_string),
        "INTEGER": TermSpec("/-?(0|[1-9][0-9]*)/", _json_integer),
        "NUMBER": TermSpec(_JSON_NUMBER_RE, _json_number),
        "WS": TermSpec("/[ \\t\\n\\r]+/", lambda r: b" ", ignored=True),
    }
    weights = {}
    for lhs, alts in rules.items():
        if lhs.endswith("_items"):
            weights[(lhs, 1)] = 2.0
    return GrammarSpec("schema_json", rules, terms, "contextual", _json_sep, weights=weights)


# --------------------------------------------------------------- 4/5: C-like
C_KEYWORDS = ["int", "char", "void", "float", "double", "long", "short", "unsigned", "signed",
              "bool", "const", "struct", "typedef", "if", "else", "while", "for", "do", "return",
              "break", "continue", "switch", "case", "default", "sizeof"]


def _c_name(rng) -> bytes:
    while True:
        r = rng.random()
        if r < 0.5:
            w = _word(rng, 1, 8)
        elif r < 0.8:
            w = _word(rng, 1, 5) + "_" + _word(rng, 1, 5)
        else:
            w = _word(rng, 1, 1) + _word(rng, 0, 6, _ALNUM)
        if w not in C_KEYWORDS:
            return w.encode()


def _c_number(rng) -> bytes:
    r = rng.random()
    if r < 0.6:
        return _digits(rng, 1, 4).encode()
    if r < 0.75:
        return b"0"
    if r < 0.9:
        return (_digits(rng, 1, 3) + "." + _digits(rng, 1, 3)).encode()
    return ("0x" + "".join("0123456789abcdef"[int(i)] for i in rng.integers(0, 16, 4))).encode()


def _c_string(rng) -> bytes:
    s = []
    for _ in range(int(rng.integers(0, 12))):
        if rng.random() < 0.9:
            s.append(chr(int(rng.integers(0x20, 0x7F))).replace('"', "'").replace("\\", "/"))
        else:
            s.append("\\" + "ntr0\\\""[int(rng.integers(0, 6))])
    return ('"' + "".join(s) + '"').encode()


def _c_char(rng) -> bytes:
    if rng.random() < 0.8:
        c = chr(int(rng.integers(0x20, 0x7F)))
        if c in "'\\":
            c = "x"
        return ("'" + c + "'").encode()
    return ("'\\" + "ntr0"[int(rng.integers(0, 4))] + "'").encode()


def _c_sep(rng, a, b):
    r = rng.random()
    if r < 0.80:
        return b" "
    if r < 0.95:
        return b"\n" + b"    " * int(rng.integers(0, 4))
    if r < 0.98:
        return b" /* " + _word(rng, 1, 8).encode() + b" */ "
    return b" // " + _word(rng, 1, 8).encode() + b"\n"


def c_like() -> GrammarSpec:
    """Synthetic C-like language: declarations, typed functions, structs, if/else,
    while, do, for, switch, return/break/continue, expressions over 15 binary and
    unary precedence levels, string/char/number/identifier terminals, line and
    block comments.  Keywords are literals that also match NAME (contextual lexer)."""
    L = lambda s: _lit(s)  # noqa: E731
    rules = {
        "start": [["unit"]],
        "unit": [["item"], ["unit", "item"]],
        "item": [["func_def"], ["decl_stmt"], ["struct_def"], ["typedef_decl"]],
        "struct_def": [[L("struct"), "NAME", L("{"), "field_list", L("}"), L(";")]],
        "field_list": [["field"], ["field_list", "field"]],
        "field": [["type", "NAME", L(";")], ["type", "NAME", L("["), "NUMBER", L("]"), L(";")]],
        "typedef_decl": [[L("typedef"), "type", "NAME", L(";")]],
        "type": [["base_type"], ["base_type", "stars"], [L("const"), "base_type"],
                 [L("const"), "base_type", "stars"], [L("struct"), "NAME"],
                 [L("struct"), "NAME", "stars"]],
        "stars": [[L("*")], ["stars", L("*")]],
        "base_type": [[L(k)] for k in ["int", "char", "void", "float", "double", "long", "short",
                                       "unsigned", "signed", "bool"]],
        "func_def": [["type", "NAME", L("("), L(")"), "block"],
                     ["type", "NAME", L("("), "params", L(")"), "block"]],
        "params": [["param"], ["params", L(","), "param"]],
        "param": [["type", "NAME"], ["type", "NAME", L("["), L("]")]],
        "block": [[L("{"), L("}")], [L("{"), "stmts", L("}")]],
        "stmts": [["stmt"], ["stmts", "stmt"]],
        "stmt": [["block"], ["decl_stmt"], ["expr", L(";")], [L(";")], ["if_stmt"],
                 [L("while"), L("("), "expr", L(")"), "stmt"], ["for_stmt"],
                 [L("do"), "stmt", L("while"), L("("), "expr", L(")"), L(";")],
                 [L("return"), L(";")], [L("return"), "expr", L(";")],
                 [L("break"), L(";")], [L("continue"), L(";")], ["switch_stmt"]],
        "if_stmt": [[L("if"), L("("), "expr", L(")"), "block"],
                    [L("if"), L("("), "expr", L(")"), "block", L("else"), "block"],
                    [L("if"), L("("), "expr", L(")"), "block", L("else"), "if_stmt"]],
        "decl_stmt": [["type", "init_list", L(";")]],
        "init_list": [["init_decl"], ["init_list", L(","), "init_decl"]],
        "init_decl": [["NAME"], ["NAME", L("="), "assign"], ["NAME", L("["), "NUMBER", L("]")],
                      ["NAME", L("["), "NUMBER", L("]"), L("="), L("{"), "args", L("}")]],
        "for_stmt": [[L("for"), L("("), "for_init", L(";"), "opt_expr", L(";"), "opt_expr", L(")"),
                      "stmt"]],
        "for_init": [[], ["expr"], ["type", "init_list"]],
        "opt_expr": [[], ["expr"]],
        "switch_stmt": [[L("switch"), L("("), "expr", L(")"), L("{"), "case_list", L("}")]],
        "case_list": [["case_item"], ["case_list", "case_item"]],
        "case_item": [[L("case"), "cond", L(":"), "stmts"], [L("default"), L(":"), "stmts"],
                      [L("case"), "cond", L(":")], [L("default"), L(":")]],
        "expr": [["assign"], ["expr", L(","), "assign"]],
        "assign": [["cond"], ["unary", "assign_op", "assign"]],
        "assign_op": [[L(o)] for o in ["=", "+=", "-=", "*=", "/=", "%=", "<<=", ">>=", "&=", "^=",
                                       "|="]],
        "cond": [["lor"], ["lor", L("?"), "expr", L(":"), "cond"]],
        "lor": [["land"], ["lor", L("||"), "land"]],
        "land": [["bor"], ["land", L("&&"), "bor"]],
        "bor": [["bxor"], ["bor", L("|"), "bxor"]],
        "bxor": [["band"], ["bxor", L("^"), "band"]],
        "band": [["eq"], ["band", L("&"), "eq"]],
        "eq": [["rel"], ["eq", L("=="), "rel"], ["eq", L("!="), "rel"]],
        "rel": [["shift"], ["rel", L("<"), "shift"], ["rel", L(">"), "shift"],
                ["rel", L("<="), "shift"], ["rel", L(">="), "shift"]],
        "shift": [["add"], ["shift", L("<<"), "add"], ["shift", L(">>"), "add"]],
        "add": [["mul"], ["add", L("+"), "mul"], ["add", L("-"), "mul"]],
        "mul": [["cast"], ["mul", L("*"), "cast"], ["mul", L("/"), "cast"], ["mul", L("%"), "cast"]],
        "cast": [["unary"], [L("("), "type", L(")"), "cast"]],
        "unary": [["postfix"], [L("++"), "unary"], [L("--"), "unary"], ["unary_op", "cast"],
                  [L("sizeof"), L("("), "type", L(")")]],
        "unary_op": [[L(o)] for o in ["&", "*", "+", "-", "~", "!"]],
        "postfix": [["primary"], ["postfix", L("["), "expr", L("]")], ["postfix", L("("), L(")")],
                    ["postfix", L("("), "args", L(")")], ["postfix", L("."), "NAME"],
                    ["postfix", L("->"), "NAME"], ["postfix", L("++")], ["postfix", L("--")]],
        "args": [["assign"], ["args", L(","), "assign"]],
        "primary": [["NAME"], ["NUMBER"], ["STRING"], ["CHARLIT"], [L("("), "expr", L(")")]],
    }
    terms = {
        "NAME": TermSpec("/[A-Za-z_][A-Za-z0-9_]*/", _c_name),
        "NUMBER": TermSpec("/(0|[1-9][0-9]*)(\\.[0-9]+)?([eE][+-]?[0-9]+)?|0[xX][0-9a-fA-F]+/",
                           _c_number),
        "STRING": TermSpec('/"([^"\\\\\\n]|\\\\.)*"/', _c_string),
        "CHARLIT": TermSpec("/'([^'\\\\\\n]|\\\\.)'/", _c_char),
        "LINE_COMMENT": TermSpec("/\\/\\/[^\\n]*/", lambda r: b"// x", ignored=True),
        "BLOCK_COMMENT": TermSpec("/\\/\\*([^*]|\\*+[^*\\/])*\\*+\\//", lambda r: b"/* x */",
                                  ignored=True),
        "WS": TermSpec("/[ \\t\\r\\n]+/", lambda r: b" ", ignored=True),
    }
    weights = {("stmts", 1): 3.0, ("unit", 1): 2.0, ("stmt", 2): 2.0, ("stmt", 1): 1.5,
               ("stmt", 4): 1.2, ("stmt", 5): 1.0, ("args", 1): 1.5, ("postfix", 3): 1.5,
               ("item", 0): 3.0}
    nesting = {("stmt", 0), ("stmt", 4), ("stmt", 5), ("stmt", 6), ("primary", 4),
               ("if_stmt", 0), ("if_stmt", 1), ("if_stmt", 2)}
    return GrammarSpec("c_like", rules, terms, "contextual", _c_sep, weights=weights,
                       nesting=nesting)
