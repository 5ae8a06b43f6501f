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


# ------------------------------------------------------------ Java-sized
JAVA_KEYWORDS = [
    "abstract", "assert", "boolean", "break", "byte", "case", "catch", "char", "class", "const", "continue",
    "default", "do", "double", "else", "enum", "exports", "extends", "final", "finally", "float", "for", "goto",
    "if", "implements", "import", "instanceof", "int", "interface", "long", "module", "native", "new", "null",
    "open", "opens", "package", "private", "protected", "provides", "public", "record", "requires", "return",
    "short", "static", "strictfp", "super", "switch", "synchronized", "this", "throw", "throws", "to",
    "transient", "transitive", "true", "false", "try", "uses", "var", "void", "volatile", "while", "with",
    "yield"]


def _java_name(rng) -> bytes:
    while True:
        r = rng.random()
        if r < 0.45:
            w = _word(rng, 1, 8)
        elif r < 0.75:
            w = _word(rng, 1, 6) + _word(rng, 1, 1, "ABCDEFGHIJKLMNOPQRSTUVWXYZ") + _word(rng, 1, 5)
        elif r < 0.9:
            w = _word(rng, 1, 1, "ABCDEFGHIJKLMNOPQRSTUVWXYZ") + _word(rng, 2, 8)
        else:
            w = _word(rng, 1, 4) + "_" + _word(rng, 1, 4, _ALNUM)
        if w not in JAVA_KEYWORDS:
            return w.encode()


def _java_int(rng) -> bytes:
    r = rng.random()
    if r < 0.6:
        s = _digits(rng, 1, 4)
    elif r < 0.72:
        s = "0"
    elif r < 0.84:
        s = "0x" + _word(rng, 1, 6, "0123456789abcdefABCDEF")
    elif r < 0.9:
        s = "0b" + _word(rng, 1, 8, "01")
    else:
        s = _digits(rng, 1, 3) + "_" + _digits(rng, 3, 3)
    return (s + ("L" if rng.random() < 0.1 else "")).encode()


def _java_float(rng) -> bytes:
    r = rng.random()
    if r < 0.6:
        s = _digits(rng, 1, 3) + "." + _digits(rng, 1, 3)
    elif r < 0.8:
        s = _digits(rng, 1, 2) + "e" + "+-"[int(rng.integers(0, 2))] + _digits(rng, 1, 2)
    else:
        s = _digits(rng, 1, 3)
    return (s + ("fFdD"[int(rng.integers(0, 4))] if r >= 0.8 or rng.random() < 0.3 else "")).encode()


def _java_text_block(rng) -> bytes:
    lines = [_word(rng, 0, 10, _LOWER + " .,") for _ in range(int(rng.integers(1, 4)))]
    return ('"""\n' + "\n".join(lines) + '"""').encode()


def java_like() -> GrammarSpec:
    """Synthetic Java-sized language (stands in for the paper's Java grammar): package
    and import declarations, a module declaration, classes, interfaces, enums,
    records and annotation types with generics, modifiers and annotations; fields,
    methods, constructors, initializers; every Java statement form (if/else in the
    no-short-if form, loops, enhanced for, labelled statements, switch with groups and
    arrow rules, try/catch/finally with resources, synchronized, assert, throw);
    expressions over 15 precedence levels with casts, instanceof patterns, class
    literals, array creation and access, method invocation and object creation.
    Written LALR(1): generic type arguments only where no expression can start,
    casts as in Java's own LALR grammar (a parenthesized expression followed by a
    unary expression), declarations and expressions sharing the qualified-name
    prefix.  Keywords are literals that also match NAME (contextual lexer); nested
    generic closers need a space (the lexer reads ">>" as one lexeme)."""
    L = lambda s: _lit(s)  # noqa: E731
    prim = ["byte", "short", "char", "int", "long", "float", "double", "boolean"]
    mods = ["public", "protected", "private", "static", "abstract", "final", "native", "synchronized",
            "transient", "volatile", "strictfp", "default", "sealed", "non-sealed"]
    assign_ops = ["=", "+=", "-=", "*=", "/=", "%=", "&=", "|=", "^=", "<<=", ">>=", ">>>="]

    def if_forms(s, body):   # if statements whose last sub-statement is `body`
        return [[L("if"), L("("), "expr", L(")"), "stmt_nsi", L("else"), body]]

    rules = {
        "start": [["compilation_unit"]],
        "compilation_unit": [["type_decls"], ["package_decl", "type_decls"], ["import_decls", "type_decls"],
                             ["package_decl", "import_decls", "type_decls"], ["module_decl"],
                             ["import_decls", "module_decl"]],
        "package_decl": [[L("package"), "qualified_name", L(";")]],
        "import_decls": [["import_decl"], ["import_decls", "import_decl"]],
        "import_decl": [[L("import"), "qualified_name", L(";")],
                        [L("import"), "qualified_name", L("."), L("*"), L(";")],
                        [L("import"), L("static"), "qualified_name", L(";")],
                        [L("import"), L("static"), "qualified_name", L("."), L("*"), L(";")]],
        "qualified_name": [["NAME"], ["qualified_name", L("."), "NAME"]],
        # modules
        "module_decl": [[L("module"), "qualified_name", L("{"), L("}")],
                        [L("module"), "qualified_name", L("{"), "module_directives", L("}")],
                        [L("open"), L("module"), "qualified_name", L("{"), "module_directives", L("}")]],
        "module_directives": [["module_directive"], ["module_directives", "module_directive"]],
        "module_directive": [[L("requires"), "qualified_name", L(";")],
                             [L("requires"), L("transitive"), "qualified_name", L(";")],
                             [L("requires"), L("static"), "qualified_name", L(";")],
                             [L("exports"), "qualified_name", L(";")],
                             [L("exports"), "qualified_name", L("to"), "name_list", L(";")],
                             [L("opens"), "qualified_name", L(";")],
                             [L("opens"), "qualified_name", L("to"), "name_list", L(";")],
                             [L("uses"), "qualified_name", L(";")],
                             [L("provides"), "qualified_name", L("with"), "name_list", L(";")]],
        "name_list": [["qualified_name"], ["name_list", L(","), "qualified_name"]],
        # type declarations
        "type_decls": [["type_decl"], ["type_decls", "type_decl"]],
        "type_decl": [["class_decl"], ["interface_decl"], ["enum_decl"], ["record_decl"],
                      ["annotation_type_decl"], [L(";")]],
        "modifiers": [["modifier"], ["modifiers", "modifier"]],
        "modifier": [[L(m)] for m in mods] + [["annotation"]],
        "annotation": [[L("@"), "qualified_name"], [L("@"), "qualified_name", L("("), L(")")],
                       [L("@"), "qualified_name", L("("), "element_value", L(")")],
                       [L("@"), "qualified_name", L("("), "element_value_pairs", L(")")]],
        "element_value_pairs": [["element_value_pair"], ["element_value_pairs", L(","), "element_value_pair"]],
        "element_value_pair": [["NAME", L("="), "element_value"]],
        "element_value": [["cond_expr"], ["annotation"], [L("{"), L("}")], [L("{"), "element_values", L("}")],
                          [L("{"), "element_values", L(","), L("}")]],
        "element_values": [["element_value"], ["element_values", L(","), "element_value"]],
        "class_decl": [["class_head", "class_body"]],
        "class_head": [["class_name"], ["class_name", "superclass"], ["class_name", "interfaces"],
                       ["class_name", "superclass", "interfaces"], ["class_name", "permits"],
                       ["class_name", "superclass", "permits"], ["class_name", "superclass", "interfaces", "permits"]],
        "permits": [[L("permits"), "class_type_list"]],
        "class_name": [[L("class"), "NAME"], ["modifiers", L("class"), "NAME"],
                       [L("class"), "NAME", "type_params"], ["modifiers", L("class"), "NAME", "type_params"]],
        "superclass": [[L("extends"), "class_type"]],
        "interfaces": [[L("implements"), "class_type_list"]],
        "class_type_list": [["class_type"], ["class_type_list", L(","), "class_type"]],
        "type_params": [[L("<"), "type_param_list", L(">")]],
        "type_param_list": [["type_param"], ["type_param_list", L(","), "type_param"]],
        "type_param": [["NAME"], ["NAME", L("extends"), "type_bound"]],
        "type_bound": [["class_type"], ["type_bound", L("&"), "class_type"]],
        "class_type": [["NAME"], ["NAME", "type_args"], ["class_type", L("."), "NAME"],
                       ["class_type", L("."), "NAME", "type_args"]],
        "type_args": [[L("<"), "type_arg_list", L(">")], [L("<"), L(">")]],
        "type_arg_list": [["type_arg"], ["type_arg_list", L(","), "type_arg"]],
        "type_arg": [["ref_type"], [L("?")], [L("?"), L("extends"), "ref_type"], [L("?"), L("super"), "ref_type"]],
        "ref_type": [["class_type"], ["class_type", "dims"], ["prim_type", "dims"]],
        "type": [["prim_type"], ["prim_type", "dims"], ["class_type"], ["class_type", "dims"]],
        "prim_type": [[L(p)] for p in prim],
        "dims": [[L("["), L("]")], ["dims", L("["), L("]")]],
        "class_body": [[L("{"), L("}")], [L("{"), "class_body_decls", L("}")]],
        "class_body_decls": [["class_body_decl"], ["class_body_decls", "class_body_decl"]],
        "class_body_decl": [["field_decl"], ["method_decl"], ["constructor_decl"], ["block"],
                            [L("static"), "block"], ["class_decl"], ["interface_decl"], ["enum_decl"],
                            ["record_decl"], ["annotation_type_decl"], ["compact_constructor"], [L(";")]],
        "field_decl": [["type", "var_declarators", L(";")], ["modifiers", "type", "var_declarators", L(";")]],
        "var_declarators": [["var_declarator"], ["var_declarators", L(","), "var_declarator"]],
        "var_declarator": [["NAME"], ["NAME", L("="), "var_init"], ["NAME", "dims"],
                           ["NAME", "dims", L("="), "var_init"]],
        "var_init": [["expr"], ["array_init"], ["switch_expr"]],
        "array_init": [[L("{"), L("}")], [L("{"), "var_inits", L("}")], [L("{"), "var_inits", L(","), L("}")]],
        "var_inits": [["var_init"], ["var_inits", L(","), "var_init"]],
        "method_decl": [["method_header", "method_body"]],
        "method_header": [["method_sig"], ["method_sig", "throws"]],
        "method_sig": [["type", "method_declarator"], [L("void"), "method_declarator"],
                       ["modifiers", "type", "method_declarator"], ["modifiers", L("void"), "method_declarator"],
                       ["type_params", "type", "method_declarator"],
                       ["type_params", L("void"), "method_declarator"],
                       ["modifiers", "type_params", "type", "method_declarator"],
                       ["modifiers", "type_params", L("void"), "method_declarator"]],
        "method_declarator": [["NAME", L("("), L(")")], ["NAME", L("("), "formal_params", L(")")]],
        "formal_params": [["formal_param"], ["formal_params", L(","), "formal_param"]],
        "formal_param": [["type", "NAME"], ["var_modifiers", "type", "NAME"], ["type", L("..."), "NAME"],
                         ["var_modifiers", "type", L("..."), "NAME"]],
        "var_modifiers": [["var_modifier"], ["var_modifiers", "var_modifier"]],
        "var_modifier": [[L("final")], ["annotation"]],
        "throws": [[L("throws"), "class_type_list"]],
        "method_body": [["block"], [L(";")]],
        "constructor_decl": [["constructor_sig", "block"], ["constructor_sig", "throws", "block"]],
        "constructor_sig": [["NAME", L("("), L(")")], ["NAME", L("("), "formal_params", L(")")],
                            ["modifiers", "NAME", L("("), L(")")],
                            ["modifiers", "NAME", L("("), "formal_params", L(")")],
                            ["type_params", "NAME", L("("), L(")")],
                            ["type_params", "NAME", L("("), "formal_params", L(")")],
                            ["modifiers", "type_params", "NAME", L("("), "formal_params", L(")")]],
        # compact constructor of a record
        "compact_constructor": [["NAME", "block"], ["modifiers", "NAME", "block"]],
        "interface_decl": [["interface_name", "interface_body"],
                           ["interface_name", L("extends"), "class_type_list", "interface_body"]],
        "interface_name": [[L("interface"), "NAME"], ["modifiers", L("interface"), "NAME"],
                           [L("interface"), "NAME", "type_params"],
                           ["modifiers", L("interface"), "NAME", "type_params"]],
        "interface_body": [[L("{"), L("}")], [L("{"), "interface_members", L("}")]],
        "interface_members": [["interface_member"], ["interface_members", "interface_member"]],
        "interface_member": [["field_decl"], ["method_decl"], ["class_decl"], ["interface_decl"],
                             ["enum_decl"], ["record_decl"], ["annotation_type_decl"], [L(";")]],
        "enum_decl": [["enum_name", "enum_body"], ["enum_name", "interfaces", "enum_body"]],
        "enum_name": [[L("enum"), "NAME"], ["modifiers", L("enum"), "NAME"]],
        "enum_body": [[L("{"), L("}")], [L("{"), "enum_constants", L("}")],
                      [L("{"), "enum_constants", L(","), L("}")],
                      [L("{"), "enum_constants", L(";"), "class_body_decls", L("}")],
                      [L("{"), "enum_constants", L(","), L(";"), "class_body_decls", L("}")],
                      [L("{"), L(";"), "class_body_decls", L("}")]],
        "enum_constants": [["enum_constant"], ["enum_constants", L(","), "enum_constant"]],
        "enum_constant": [["NAME"], ["NAME", "arguments"], ["NAME", "class_body"], ["NAME", "arguments", "class_body"]],
        "record_decl": [["record_head", "class_body"], ["record_head", "interfaces", "class_body"]],
        "record_head": [["record_name", L("("), L(")")], ["record_name", L("("), "record_components", L(")")]],
        "record_name": [[L("record"), "NAME"], ["modifiers", L("record"), "NAME"],
                        [L("record"), "NAME", "type_params"]],
        "record_components": [["record_component"], ["record_components", L(","), "record_component"]],
        "record_component": [["type", "NAME"], ["annotation", "type", "NAME"]],
        "annotation_type_decl": [[L("@"), L("interface"), "NAME", "annotation_type_body"],
                                 ["modifiers", L("@"), L("interface"), "NAME", "annotation_type_body"]],
        "annotation_type_body": [[L("{"), L("}")], [L("{"), "annotation_type_elements", L("}")]],
        "annotation_type_elements": [["annotation_type_element"],
                                     ["annotation_type_elements", "annotation_type_element"]],
        "annotation_type_element": [["type", "NAME", L("("), L(")"), L(";")],
                                    ["type", "NAME", L("("), L(")"), L("default"), "element_value", L(";")],
                                    ["modifiers", "type", "NAME", L("("), L(")"), L(";")],
                                    ["modifiers", "type", "NAME", L("("), L(")"), L("default"), "element_value",
                                     L(";")],
                                    ["field_decl_const"], ["class_decl"], ["enum_decl"], [L(";")]],
        "field_decl_const": [["type", "NAME", L("="), "var_init", L(";")],
                             ["modifiers", "type", "NAME", L("="), "var_init", L(";")]],
        # blocks and statements
        "block": [[L("{"), L("}")], [L("{"), "block_stmts", L("}")]],
        "block_stmts": [["block_stmt"], ["block_stmts", "block_stmt"]],
        "block_stmt": [["local_var_decl", L(";")], ["stmt"], ["local_type_decl"],
                       [L("this"), "arguments", L(";")], [L("super"), "arguments", L(";")]],
        # local classes, records, interfaces and enums (modifiers: final, abstract, annotations)
        "local_type_decl": [["local_class_name", "class_body"], ["local_class_name", "superclass", "class_body"],
                            ["local_class_name", "interfaces", "class_body"],
                            ["local_class_name", "superclass", "interfaces", "class_body"],
                            [L("record"), "NAME", L("("), "record_components", L(")"), "class_body"],
                            [L("record"), "NAME", L("("), L(")"), "class_body"],
                            [L("interface"), "NAME", "interface_body"],
                            [L("enum"), "NAME", "enum_body"]],
        "local_class_name": [[L("class"), "NAME"], ["local_class_mods", L("class"), "NAME"],
                             [L("class"), "NAME", "type_params"]],
        "local_class_mods": [["var_modifiers"], [L("abstract")], ["var_modifiers", L("abstract")]],
        "local_var_decl": [["local_type", "var_declarators"], ["var_modifiers", "local_type", "var_declarators"],
                           [L("var"), "NAME", L("="), "expr"], ["var_modifiers", L("var"), "NAME", L("="), "expr"]],
        "local_type": [["prim_type"], ["prim_type", "dims"], ["name"], ["name", "dims"]],
        "name": [["NAME"], ["name", L("."), "NAME"]],
        "stmt": [["stmt_wts"], ["labeled_stmt"], [L("if"), L("("), "expr", L(")"), "stmt"],
                 ["if_else_stmt"], ["while_stmt"], ["for_stmt"], ["foreach_stmt"]],
        "stmt_nsi": [["stmt_wts"], ["labeled_stmt_nsi"], ["if_else_stmt_nsi"], ["while_stmt_nsi"],
                     ["for_stmt_nsi"], ["foreach_stmt_nsi"]],
        "if_else_stmt": if_forms("stmt", "stmt"),
        "if_else_stmt_nsi": if_forms("stmt_nsi", "stmt_nsi"),
        "labeled_stmt": [["NAME", L(":"), "stmt"]],
        "labeled_stmt_nsi": [["NAME", L(":"), "stmt_nsi"]],
        "while_stmt": [[L("while"), L("("), "expr", L(")"), "stmt"]],
        "while_stmt_nsi": [[L("while"), L("("), "expr", L(")"), "stmt_nsi"]],
        "for_stmt": [["for_head", "stmt"]],
        "for_stmt_nsi": [["for_head", "stmt_nsi"]],
        "for_head": [[L("for"), L("("), "for_init", L(";"), "opt_expr", L(";"), "for_update", L(")")]],
        "for_init": [[], ["stmt_expr_list"], ["local_var_decl"]],
        "for_update": [[], ["stmt_expr_list"]],
        "opt_expr": [[], ["expr"]],
        "stmt_expr_list": [["expr"], ["stmt_expr_list", L(","), "expr"]],
        "foreach_stmt": [["foreach_head", "stmt"]],
        "foreach_stmt_nsi": [["foreach_head", "stmt_nsi"]],
        "foreach_head": [[L("for"), L("("), "local_type", "NAME", L(":"), "expr", L(")")],
                         [L("for"), L("("), "var_modifiers", "local_type", "NAME", L(":"), "expr", L(")")],
                         [L("for"), L("("), L("var"), "NAME", L(":"), "expr", L(")")]],
        "stmt_wts": [["block"], [L(";")], ["expr", L(";")], ["switch_stmt"],
                     [L("return"), "switch_expr", L(";")], [L("yield"), "switch_expr", L(";")],
                     [L("do"), "stmt", L("while"), L("("), "expr", L(")"), L(";")],
                     [L("break"), L(";")], [L("break"), "NAME", L(";")], [L("continue"), L(";")],
                     [L("continue"), "NAME", L(";")], [L("return"), L(";")], [L("return"), "expr", L(";")],
                     [L("throw"), "expr", L(";")], [L("yield"), "expr", L(";")],
                     [L("synchronized"), L("("), "expr", L(")"), "block"], ["try_stmt"],
                     [L("assert"), "expr", L(";")], [L("assert"), "expr", L(":"), "expr", L(";")]],
        "switch_stmt": [[L("switch"), L("("), "expr", L(")"), "switch_block"]],
        "switch_block": [[L("{"), L("}")], [L("{"), "switch_groups", L("}")],
                         [L("{"), "switch_groups", "switch_labels", L("}")], [L("{"), "switch_labels", L("}")],
                         [L("{"), "switch_rules", L("}")]],
        "switch_groups": [["switch_group"], ["switch_groups", "switch_group"]],
        "switch_group": [["switch_labels", "block_stmts"]],
        "switch_labels": [["switch_label"], ["switch_labels", "switch_label"]],
        "switch_label": [[L("case"), "case_consts", L(":")], [L("default"), L(":")],
                         [L("case"), "pattern", L(":")], [L("case"), "pattern", L("when"), "cond_expr", L(":")]],
        "pattern": [["local_type", "NAME"], [L("final"), "local_type", "NAME"]],
        "case_consts": [["cond_expr"], ["case_consts", L(","), "cond_expr"]],
        "switch_rules": [["switch_rule"], ["switch_rules", "switch_rule"]],
        "switch_rule": [["rule_label", "expr", L(";")], ["rule_label", "block"],
                        ["rule_label", L("throw"), "expr", L(";")]],
        "rule_label": [[L("case"), "case_consts", L("->")], [L("default"), L("->")],
                       [L("case"), "pattern", L("->")], [L("case"), "pattern", L("when"), "cond_expr", L("->")]],
        "try_stmt": [[L("try"), "block", "catches"], [L("try"), "block", "finally"],
                     [L("try"), "block", "catches", "finally"], [L("try"), "resource_spec", "block"],
                     [L("try"), "resource_spec", "block", "catches"], [L("try"), "resource_spec", "block", "finally"],
                     [L("try"), "resource_spec", "block", "catches", "finally"]],
        "catches": [["catch_clause"], ["catches", "catch_clause"]],
        "catch_clause": [[L("catch"), L("("), "catch_type", "NAME", L(")"), "block"],
                         [L("catch"), L("("), L("final"), "catch_type", "NAME", L(")"), "block"]],
        "catch_type": [["name"], ["catch_type", L("|"), "name"]],
        "finally": [[L("finally"), "block"]],
        "resource_spec": [[L("("), "resources", L(")")], [L("("), "resources", L(";"), L(")")]],
        "resources": [["resource"], ["resources", L(";"), "resource"]],
        "resource": [["local_type", "NAME", L("="), "expr"], [L("var"), "NAME", L("="), "expr"], ["name"],
                     ["var_modifiers", "local_type", "NAME", L("="), "expr"]],
        # expressions
        "expr": [["assign_expr"], ["lambda"]],
        "assign_expr": [["cond_expr"], ["lhs", "assign_op", "assign_expr"], ["lhs", "assign_op", "switch_expr"],
                        ["lhs", "assign_op", "lambda"]],
        # lambdas: one untyped parameter, or typed parameters in parentheses (an untyped
        # parenthesized list would need more than one token of lookahead after ")")
        "lambda": [["NAME", L("->"), "lambda_body"], [L("("), L(")"), L("->"), "lambda_body"],
                   [L("("), "lambda_params", L(")"), L("->"), "lambda_body"]],
        "lambda_params": [["lambda_param"], ["lambda_params", L(","), "lambda_param"]],
        "lambda_param": [["local_type", "NAME"], [L("final"), "local_type", "NAME"], [L("var"), "NAME"]],
        "lambda_body": [["expr"], ["block"]],
        # switch expressions where no statement can start (initializers, right-hand sides,
        # arguments, return and yield)
        "switch_expr": [[L("switch"), L("("), "expr", L(")"), L("{"), "switch_rules", L("}")]],
        "lhs": [["name"], ["field_access"], ["array_access"]],
        "assign_op": [[L(o)] for o in assign_ops],
        "cond_expr": [["cond_or"], ["cond_or", L("?"), "expr", L(":"), "cond_expr"]],
        "cond_or": [["cond_and"], ["cond_or", L("||"), "cond_and"]],
        "cond_and": [["incl_or"], ["cond_and", L("&&"), "incl_or"]],
        "incl_or": [["excl_or"], ["incl_or", L("|"), "excl_or"]],
        "excl_or": [["and_expr"], ["excl_or", L("^"), "and_expr"]],
        "and_expr": [["eq_expr"], ["and_expr", L("&"), "eq_expr"]],
        "eq_expr": [["rel_expr"], ["eq_expr", L("=="), "rel_expr"], ["eq_expr", L("!="), "rel_expr"]],
        "rel_expr": [["shift_expr"], ["rel_expr", L("<"), "shift_expr"], ["rel_expr", L(">"), "shift_expr"],
                     ["rel_expr", L("<="), "shift_expr"], ["rel_expr", L(">="), "shift_expr"],
                     ["rel_expr", L("instanceof"), "local_type"],
                     ["rel_expr", L("instanceof"), "local_type", "NAME"]],
        "shift_expr": [["add_expr"], ["shift_expr", L("<<"), "add_expr"], ["shift_expr", L(">>"), "add_expr"],
                       ["shift_expr", L(">>>"), "add_expr"]],
        "add_expr": [["mul_expr"], ["add_expr", L("+"), "mul_expr"], ["add_expr", L("-"), "mul_expr"]],
        "mul_expr": [["unary"], ["mul_expr", L("*"), "unary"], ["mul_expr", L("/"), "unary"],
                     ["mul_expr", L("%"), "unary"]],
        "unary": [[L("++"), "unary"], [L("--"), "unary"], [L("+"), "unary"], [L("-"), "unary"], ["unary_nnpm"]],
        "unary_nnpm": [["postfix"], [L("~"), "unary"], [L("!"), "unary"], ["cast"]],
        "cast": [[L("("), "prim_type", L(")"), "unary"], [L("("), "prim_type", "dims", L(")"), "unary"],
                 [L("("), "expr", L(")"), "unary_nnpm"], [L("("), "name", "dims", L(")"), "unary_nnpm"]],
        "postfix": [["primary"], ["name"], ["postfix", L("++")], ["postfix", L("--")]],
        "primary": [["primary_nna"], ["array_creation"]],
        "primary_nna": [["literal"], [L("this")], ["name", L("."), L("this")], [L("("), "expr", L(")")],
                        ["instance_creation"], ["field_access"], ["method_call"], ["array_access"],
                        ["name", L("."), L("class")], ["prim_type", L("."), L("class")],
                        [L("void"), L("."), L("class")], ["name", "dims", L("."), L("class")],
                        ["prim_type", "dims", L("."), L("class")], ["method_ref"]],
        "literal": [["INT"], ["FLOAT"], ["STRING"], ["TEXT_BLOCK"], ["CHARLIT"], [L("true")], [L("false")],
                    [L("null")]],
        "field_access": [["primary", L("."), "NAME"], [L("super"), L("."), "NAME"],
                         ["name", L("."), L("super"), L("."), "NAME"]],
        "method_call": [["name", "arguments"], ["primary", L("."), "NAME", "arguments"],
                        [L("super"), L("."), "NAME", "arguments"],
                        ["name", L("."), "type_args", "NAME", "arguments"],
                        ["primary", L("."), "type_args", "NAME", "arguments"],
                        [L("super"), L("."), "type_args", "NAME", "arguments"]],
        "method_ref": [["name", L("::"), "NAME"], ["primary", L("::"), "NAME"], [L("super"), L("::"), "NAME"],
                       ["name", L("::"), L("new")], ["prim_type", "dims", L("::"), L("new")]],
        "arguments": [[L("("), L(")")], [L("("), "arg_list", L(")")]],
        "arg_list": [["arg"], ["arg_list", L(","), "arg"]],
        "arg": [["expr"], ["switch_expr"]],
        "array_access": [["name", L("["), "expr", L("]")], ["primary_nna", L("["), "expr", L("]")]],
        "instance_creation": [[L("new"), "class_type", "arguments"],
                              [L("new"), "class_type", "arguments", "class_body"],
                              ["primary", L("."), L("new"), "NAME", "arguments"],
                              ["primary", L("."), L("new"), "NAME", "type_args", "arguments"],
                              ["primary", L("."), L("new"), "NAME", "arguments", "class_body"],
                              ["name", L("."), L("new"), "NAME", "arguments"]],
        "array_creation": [[L("new"), "prim_type", "dim_exprs"], [L("new"), "prim_type", "dim_exprs", "dims"],
                           [L("new"), "class_type", "dim_exprs"], [L("new"), "class_type", "dim_exprs", "dims"],
                           [L("new"), "prim_type", "dims", "array_init"],
                           [L("new"), "class_type", "dims", "array_init"]],
        "dim_exprs": [["dim_expr"], ["dim_exprs", "dim_expr"]],
        "dim_expr": [[L("["), "expr", L("]")]],
    }
    terms = {
        "NAME": TermSpec("/[A-Za-z_$][A-Za-z0-9_$]*/", _java_name),
        "INT": TermSpec("/(0|[1-9][0-9_]*)[lL]?|0[xX][0-9a-fA-F_]+[lL]?|0[bB][01_]+[lL]?/", _java_int),
        "FLOAT": TermSpec("/[0-9]+\\.[0-9]+([eE][+-]?[0-9]+)?[fFdD]?|[0-9]+[eE][+-]?[0-9]+[fFdD]?|[0-9]+[fFdD]/",
                          _java_float),
        "STRING": TermSpec('/"([^"\\\\\\n]|\\\\.)*"/', _c_string),
        # a text block: three quotes, a line break, then text without three quotes in a row
        "TEXT_BLOCK": TermSpec('/"""[ \\t]*\\n([^"\\\\]|\\\\.|"[^"\\\\]|""[^"\\\\])*"""/', _java_text_block),
        "CHARLIT": TermSpec("/'([^'\\\\\\n]|\\\\.)'/", _c_char),
        "LINE_COMMENT": TermSpec("/\\/\\/[^\\n]*/", lambda r: b"// x", ignored=True),
        "BLOCK_COMMENT": TermSpec("/\\/\\*([^*]|\\*+[^*\\/])*\\*+\\//", lambda r: b"/* x */", ignored=True),
        "WS": TermSpec("/[ \\t\\r\\n]+/", lambda r: b" ", ignored=True),
    }
    weights = {("type_decls", 1): 1.5, ("class_body_decls", 1): 4.0, ("class_body_decl", 1): 3.0,
               ("class_body_decl", 0): 2.0, ("block_stmts", 1): 3.0, ("block_stmt", 1): 1.5,
               ("stmt_wts", 2): 3.0, ("arg_list", 1): 1.2, ("type_decl", 0): 4.0}
    nesting = {("stmt", 2), ("if_else_stmt", 0), ("stmt_wts", 0), ("while_stmt", 0), ("for_stmt", 0),
               ("primary_nna", 3), ("class_body_decl", 1)}
    return GrammarSpec("java_like", rules, terms, "contextual", _c_sep, weights=weights, nesting=nesting)


# ------------------------------------------------------------------- SQL-like
SQL_KEYWORDS = [
    "select", "distinct", "all", "from", "where", "group", "by", "having", "order", "asc", "desc", "nulls",
    "first", "last", "limit", "offset", "union", "except", "intersect", "with", "recursive", "as", "join",
    "inner", "left", "right", "full", "outer", "cross", "natural", "on", "using", "and", "or", "not", "is",
    "null", "true", "false", "between", "in", "like", "exists", "case", "when", "then", "else", "end", "cast",
    "over", "partition", "insert", "into", "values", "update", "set", "delete", "create", "table", "if",
    "index", "unique", "view", "drop", "alter", "add", "column", "rename", "to", "primary", "key", "foreign",
    "references", "check", "constraint", "default", "begin", "commit", "rollback", "integer", "int",
    "bigint", "smallint", "real", "double", "precision", "float", "boolean", "text", "date", "timestamp",
    "varchar", "char", "decimal", "numeric", "any", "some", "escape", "returning", "conflict", "do",
    "nothing", "rows", "range", "unbounded", "preceding", "following", "current", "row", "filter", "extract",
    "coalesce", "nullif", "interval", "temporary", "cascade", "restrict",
]


def _sql_keyword(word: str):
    def sample(rng) -> bytes:
        r = rng.random()
        if r < 0.5:
            return word.upper().encode()
        if r < 0.9:
            return word.encode()
        return "".join(c.upper() if rng.random() < 0.5 else c for c in word).encode()
    return sample


def _sql_name(rng) -> bytes:
    while True:
        r = rng.random()
        if r < 0.6:
            w = _word(rng, 1, 10)
        elif r < 0.9:
            w = _word(rng, 1, 6) + "_" + _word(rng, 1, 6)
        else:
            w = _word(rng, 1, 1) + _digits(rng, 1, 2)
        if w not in SQL_KEYWORDS:
            return w.encode()


def _sql_string(rng) -> bytes:
    s = "".join("''" if rng.random() < 0.05 else _word(rng, 1, 1, _LOWER + " %_-.")
                for _ in range(int(rng.integers(0, 10))))
    return ("'" + s + "'").encode()


def _sql_number(rng) -> bytes:
    r = rng.random()
    if r < 0.6:
        return (_digits(rng, 1, 3) + "." + _digits(rng, 1, 3)).encode()
    if r < 0.8:
        return ("." + _digits(rng, 1, 3)).encode()
    return (_digits(rng, 1, 2) + "e" + _digits(rng, 1, 2)).encode()


def _sql_param(rng) -> bytes:
    r = rng.random()
    if r < 0.4:
        return b"?"
    if r < 0.7:
        return (":" + _word(rng, 1, 6)).encode()
    return ("$" + _digits(rng, 1, 2)).encode()


def _sql_sep(rng, a, b):
    r = rng.random()
    if r < 0.85:
        return b" "
    if r < 0.97:
        return b"\n" + b"  " * int(rng.integers(0, 4))
    return b" -- " + _word(rng, 1, 8).encode() + b"\n"


def sql_like() -> GrammarSpec:
    """Synthetic SQL-like language (stands in for the paper's SQL grammar): statement
    lists of queries (WITH [RECURSIVE] common table expressions, set operations,
    SELECT with DISTINCT, joins of every kind with ON / USING, WHERE, GROUP BY,
    HAVING, ORDER BY with NULLS FIRST/LAST, LIMIT / OFFSET), expressions over
    OR / AND / NOT, comparisons with quantified subqueries, IS [NOT] NULL,
    [NOT] BETWEEN / IN / LIKE [ESCAPE], EXISTS, CASE, CAST, EXTRACT, COALESCE,
    function calls with DISTINCT, FILTER and window clauses (PARTITION BY, ORDER BY,
    ROWS / RANGE frames), INSERT (VALUES or a query, ON CONFLICT, RETURNING),
    UPDATE, DELETE, CREATE TABLE / INDEX / VIEW, DROP, ALTER TABLE and transaction
    statements.  Keywords are case-insensitive regex terminals ranked above NAME
    (contextual lexer: a keyword spelling is a name wherever the keyword cannot
    follow).  Written LALR(1): a parenthesized query appears only where an
    expression or a table reference is expected, and INSERT takes a bare SELECT."""
    K = {w: w.upper() for w in SQL_KEYWORDS}   # keyword terminal names
    L = lambda s: _lit(s)  # noqa: E731
    k = lambda w: K[w]  # noqa: E731
    rules = {
        "start": [["stmts"]],
        "stmts": [["stmt", L(";")], ["stmts", "stmt", L(";")]],
        "stmt": [["query"], ["insert"], ["update"], ["delete"], ["create_table"], ["create_index"],
                 ["create_view"], ["drop"], ["alter"], [k("begin")], [k("commit")], [k("rollback")]],
        # queries
        "query": [["query_body"], ["with_clause", "query_body"]],
        "with_clause": [[k("with"), "ctes"], [k("with"), k("recursive"), "ctes"]],
        "ctes": [["cte"], ["ctes", L(","), "cte"]],
        "cte": [["NAME", k("as"), L("("), "query", L(")")],
                ["NAME", L("("), "name_list", L(")"), k("as"), L("("), "query", L(")")]],
        "query_body": [["set_expr"], ["set_expr", "order_by"], ["set_expr", "limit_clause"],
                       ["set_expr", "order_by", "limit_clause"]],
        "set_expr": [["set_term"], ["set_expr", k("union"), "set_term"], ["set_expr", k("union"), k("all"), "set_term"],
                     ["set_expr", k("except"), "set_term"]],
        "set_term": [["select_core"], ["set_term", k("intersect"), "select_core"]],
        "select_core": [[k("select"), "set_quant", "select_list", "opt_from", "opt_where", "opt_group",
                         "opt_having"]],
        "set_quant": [[], [k("distinct")], [k("all")]],
        "select_list": [["select_item"], ["select_list", L(","), "select_item"]],
        "select_item": [["expr"], ["expr", "NAME"], ["expr", k("as"), "NAME"], [L("*")], ["qname", L("."), L("*")]],
        "opt_from": [[], [k("from"), "table_refs"]],
        "table_refs": [["table_ref"], ["table_refs", L(","), "table_ref"]],
        "table_ref": [["table_primary"], ["joined"]],
        "joined": [["table_ref", "join_type", k("join"), "table_primary", "join_cond"],
                   ["table_ref", k("cross"), k("join"), "table_primary"],
                   ["table_ref", k("natural"), "join_type", k("join"), "table_primary"]],
        "join_type": [[], [k("inner")], [k("left")], [k("left"), k("outer")], [k("right")],
                      [k("right"), k("outer")], [k("full")], [k("full"), k("outer")]],
        "join_cond": [[k("on"), "expr"], [k("using"), L("("), "name_list", L(")")]],
        "table_primary": [["qname"], ["qname", "alias"], [L("("), "query", L(")"), "alias"],
                          [L("("), "joined", L(")")]],
        "alias": [["NAME"], [k("as"), "NAME"], [k("as"), "NAME", L("("), "name_list", L(")")]],
        "opt_where": [[], [k("where"), "expr"]],
        "opt_group": [[], [k("group"), k("by"), "expr_list"]],
        "opt_having": [[], [k("having"), "expr"]],
        "order_by": [[k("order"), k("by"), "order_items"]],
        "order_items": [["order_item"], ["order_items", L(","), "order_item"]],
        "order_item": [["expr", "opt_dir", "opt_nulls"]],
        "opt_dir": [[], [k("asc")], [k("desc")]],
        "opt_nulls": [[], [k("nulls"), k("first")], [k("nulls"), k("last")]],
        "limit_clause": [[k("limit"), "expr"], [k("limit"), "expr", k("offset"), "expr"], [k("offset"), "expr"]],
        # expressions
        "expr": [["or_expr"]],
        "or_expr": [["and_expr"], ["or_expr", k("or"), "and_expr"]],
        "and_expr": [["not_expr"], ["and_expr", k("and"), "not_expr"]],
        "not_expr": [["pred"], [k("not"), "not_expr"]],
        "pred": [["add_expr"], ["add_expr", "comp_op", "add_expr"],
                 ["add_expr", "comp_op", "quantifier", L("("), "query", L(")")],
                 ["add_expr", k("is"), k("null")], ["add_expr", k("is"), k("not"), k("null")],
                 ["add_expr", k("is"), k("true")], ["add_expr", k("is"), k("false")],
                 ["add_expr", k("between"), "add_expr", k("and"), "add_expr"],
                 ["add_expr", k("not"), k("between"), "add_expr", k("and"), "add_expr"],
                 ["add_expr", k("in"), L("("), "expr_list", L(")")],
                 ["add_expr", k("not"), k("in"), L("("), "expr_list", L(")")],
                 ["add_expr", k("in"), L("("), "query", L(")")],
                 ["add_expr", k("not"), k("in"), L("("), "query", L(")")],
                 ["add_expr", k("like"), "add_expr"], ["add_expr", k("not"), k("like"), "add_expr"],
                 ["add_expr", k("like"), "add_expr", k("escape"), "STRING"],
                 [k("exists"), L("("), "query", L(")")]],
        "quantifier": [[k("any")], [k("some")], [k("all")]],
        "comp_op": [[L(o)] for o in ["=", "<>", "!=", "<", "<=", ">", ">="]],
        "add_expr": [["mul_expr"], ["add_expr", L("+"), "mul_expr"], ["add_expr", L("-"), "mul_expr"],
                     ["add_expr", L("||"), "mul_expr"]],
        "mul_expr": [["unary"], ["mul_expr", L("*"), "unary"], ["mul_expr", L("/"), "unary"],
                     ["mul_expr", L("%"), "unary"]],
        "unary": [["primary"], [L("-"), "unary"], [L("+"), "unary"]],
        "primary": [["literal"], ["qname"], ["PARAM"], [L("("), "expr", L(")")], [L("("), "query", L(")")],
                    ["func_call"], ["case_expr"], [k("cast"), L("("), "expr", k("as"), "type_name", L(")")],
                    [k("extract"), L("("), "NAME", k("from"), "expr", L(")")],
                    [k("coalesce"), L("("), "expr_list", L(")")],
                    [k("nullif"), L("("), "expr", L(","), "expr", L(")")],
                    [k("interval"), "STRING"]],
        "literal": [["INT"], ["NUMBER"], ["STRING"], [k("null")], [k("true")], [k("false")],
                    [k("date"), "STRING"], [k("timestamp"), "STRING"]],
        "func_call": [["qname", L("("), "func_args", L(")"), "opt_filter", "opt_over"]],
        "func_args": [[], ["expr_list"], [k("distinct"), "expr_list"], [L("*")]],
        "opt_filter": [[], [k("filter"), L("("), k("where"), "expr", L(")")]],
        "opt_over": [[], [k("over"), L("("), "window_spec", L(")")], [k("over"), "NAME"]],
        "window_spec": [["opt_partition", "opt_window_order", "opt_frame"]],
        "opt_partition": [[], [k("partition"), k("by"), "expr_list"]],
        "opt_window_order": [[], ["order_by"]],
        "opt_frame": [[], ["frame_unit", "frame_bound"],
                      ["frame_unit", k("between"), "frame_bound", k("and"), "frame_bound"]],
        "frame_unit": [[k("rows")], [k("range")]],
        "frame_bound": [[k("unbounded"), k("preceding")], [k("unbounded"), k("following")],
                        [k("current"), k("row")], ["INT", k("preceding")], ["INT", k("following")]],
        "case_expr": [[k("case"), "when_list", "opt_else", k("end")],
                      [k("case"), "expr", "when_list", "opt_else", k("end")]],
        "when_list": [[k("when"), "expr", k("then"), "expr"], ["when_list", k("when"), "expr", k("then"), "expr"]],
        "opt_else": [[], [k("else"), "expr"]],
        "expr_list": [["expr"], ["expr_list", L(","), "expr"]],
        "name_list": [["NAME"], ["name_list", L(","), "NAME"]],
        "qname": [["NAME"], ["qname", L("."), "NAME"]],
        "type_name": [[k("integer")], [k("int")], [k("bigint")], [k("smallint")], [k("real")],
                      [k("double"), k("precision")], [k("float")], [k("boolean")], [k("text")], [k("date")],
                      [k("timestamp")], [k("varchar"), L("("), "INT", L(")")], [k("char"), L("("), "INT", L(")")],
                      [k("decimal"), L("("), "INT", L(","), "INT", L(")")],
                      [k("numeric"), L("("), "INT", L(","), "INT", L(")")]],
        # data manipulation
        "insert": [[k("insert"), k("into"), "qname", "insert_src", "opt_conflict", "opt_returning"],
                   [k("insert"), k("into"), "qname", L("("), "name_list", L(")"), "insert_src", "opt_conflict",
                    "opt_returning"]],
        "insert_src": [[k("values"), "value_rows"], ["select_core"], ["select_core", "order_by"],
                       [k("default"), k("values")]],
        "value_rows": [[L("("), "expr_list", L(")")], ["value_rows", L(","), L("("), "expr_list", L(")")]],
        "opt_conflict": [[], [k("on"), k("conflict"), k("do"), k("nothing")],
                         [k("on"), k("conflict"), L("("), "name_list", L(")"), k("do"), k("nothing")],
                         [k("on"), k("conflict"), L("("), "name_list", L(")"), k("do"), k("update"), k("set"),
                          "assignments"]],
        "opt_returning": [[], [k("returning"), "select_list"]],
        "update": [[k("update"), "qname", k("set"), "assignments", "opt_from", "opt_where", "opt_returning"]],
        "assignments": [["assignment"], ["assignments", L(","), "assignment"]],
        "assignment": [["NAME", L("="), "expr"], ["NAME", L("="), k("default")]],
        "delete": [[k("delete"), k("from"), "qname", "opt_where", "opt_returning"]],
        # definitions
        "create_table": [[k("create"), "opt_temp", k("table"), "opt_if_not_exists", "qname", L("("), "table_elems",
                          L(")")],
                         [k("create"), "opt_temp", k("table"), "opt_if_not_exists", "qname", k("as"), "query"]],
        "opt_temp": [[], [k("temporary")]],
        "opt_if_not_exists": [[], [k("if"), k("not"), k("exists")]],
        "table_elems": [["table_elem"], ["table_elems", L(","), "table_elem"]],
        "table_elem": [["NAME", "type_name", "col_constraints"], ["table_constraint"],
                       [k("constraint"), "NAME", "table_constraint"]],
        "col_constraints": [[], ["col_constraints", "col_constraint"]],
        "col_constraint": [[k("not"), k("null")], [k("null")], [k("primary"), k("key")], [k("unique")],
                           [k("default"), "default_value"], [k("references"), "qname"],
                           [k("references"), "qname", L("("), "name_list", L(")")],
                           [k("check"), L("("), "expr", L(")")]],
        "default_value": [["literal"], [L("-"), "INT"], [L("("), "expr", L(")")]],
        "table_constraint": [[k("primary"), k("key"), L("("), "name_list", L(")")],
                             [k("unique"), L("("), "name_list", L(")")],
                             [k("foreign"), k("key"), L("("), "name_list", L(")"), k("references"), "qname",
                              L("("), "name_list", L(")")],
                             [k("check"), L("("), "expr", L(")")]],
        "create_index": [[k("create"), k("index"), "NAME", k("on"), "qname", L("("), "index_items", L(")")],
                         [k("create"), k("unique"), k("index"), "NAME", k("on"), "qname", L("("), "index_items",
                          L(")")]],
        "index_items": [["index_item"], ["index_items", L(","), "index_item"]],
        "index_item": [["NAME", "opt_dir"]],
        "create_view": [[k("create"), k("view"), "qname", k("as"), "query"],
                        [k("create"), k("view"), "qname", L("("), "name_list", L(")"), k("as"), "query"]],
        "drop": [[k("drop"), "drop_kind", "qname", "opt_drop_mode"],
                 [k("drop"), "drop_kind", k("if"), k("exists"), "qname", "opt_drop_mode"]],
        "drop_kind": [[k("table")], [k("view")], [k("index")]],
        "opt_drop_mode": [[], [k("cascade")], [k("restrict")]],
        "alter": [[k("alter"), k("table"), "qname", "alter_action"]],
        "alter_action": [[k("add"), k("column"), "NAME", "type_name", "col_constraints"],
                         [k("add"), "table_constraint"],
                         [k("drop"), k("column"), "NAME"], [k("rename"), k("to"), "NAME"],
                         [k("rename"), k("column"), "NAME", k("to"), "NAME"],
                         [k("alter"), k("column"), "NAME", k("set"), k("default"), "default_value"],
                         [k("alter"), k("column"), "NAME", k("drop"), k("default")]],
    }
    terms = {K[w]: TermSpec("/" + "".join(f"[{c.lower()}{c.upper()}]" if c.isalpha() else c for c in w) + "/",
                            _sql_keyword(w), priority=2) for w in SQL_KEYWORDS}
    terms.update({
        "NAME": TermSpec("/[A-Za-z_][A-Za-z0-9_]*|\"([^\"]|\"\")+\"/", _sql_name),
        "INT": TermSpec("/[0-9]+/", lambda r: _digits(r, 1, 4).encode()),
        "NUMBER": TermSpec("/[0-9]+\\.[0-9]*([eE][+-]?[0-9]+)?|\\.[0-9]+([eE][+-]?[0-9]+)?|[0-9]+[eE][+-]?[0-9]+/",
                           _sql_number),
        "STRING": TermSpec("/'([^']|'')*'/", _sql_string),
        "PARAM": TermSpec("/\\?|:[A-Za-z_][A-Za-z0-9_]*|\\$[0-9]+/", _sql_param),
        "LINE_COMMENT": TermSpec("/--[^\\n]*/", lambda r: b"-- x", ignored=True),
        "BLOCK_COMMENT": TermSpec("/\\/\\*([^*]|\\*+[^*\\/])*\\*+\\//", lambda r: b"/* x */", ignored=True),
        "WS": TermSpec("/[ \\t\\r\\n]+/", lambda r: b" ", ignored=True),
    })
    weights = {("stmts", 1): 2.0, ("stmt", 0): 4.0, ("select_list", 1): 1.5, ("and_expr", 1): 1.2}
    nesting = {("primary", 3), ("primary", 4), ("table_primary", 2), ("pred", 11)}
    return GrammarSpec("sql_like", rules, terms, "contextual", _sql_sep, weights=weights, nesting=nesting)
