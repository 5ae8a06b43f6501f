// Grammar text reader and EBNF lowering.
//
// The paper builds its lexer and LALR(1) parser from Lark grammars (Section
// "Experimental Setup", Implementation).  The accepted notation is a small
// Lark-like subset:
//   name: alt | alt ...            rule; the start symbol is `start`
//   NAME(.p)?: /regex/ | "literal"  named terminal, priority p (default 0)
//   "literal" inside a rule         anonymous terminal with priority 1
//   %ignore NAME, %lexer basic|contextual
//   items: symbol, "lit", ( alts ), [ alts ], postfix ? * +
//   a line starting with | continues the previous rule; // starts a comment line
// EBNF lowering (fixed, because a contextual lexer consults LALR states, which
// depend on the exact BNF): a one-alternative group without postfix is spliced
// inline; other groups get a fresh nonterminal; X? and [..] -> N: <empty> | X;
// X* -> N: <empty> | N X; X+ -> N: X | N X.
#include <algorithm>
#include <cctype>
#include <map>
#include <set>

#include "psc_internal.h"

namespace psc {
namespace {

std::string trim(const std::string& s) {
    size_t a = 0, b = s.size();
    while (a < b && std::isspace((unsigned char)s[a])) a++;
    while (b > a && std::isspace((unsigned char)s[b - 1])) b--;
    return s.substr(a, b - a);
}

[[noreturn]] void fail(const std::string& m) { throw Error(ST_ERR_GRAMMAR, m); }

int hexval(char c) {
    if (c >= '0' && c <= '9') return c - '0';
    if (c >= 'a' && c <= 'f') return c - 'a' + 10;
    if (c >= 'A' && c <= 'F') return c - 'A' + 10;
    fail("bad hex digit in literal");
}

std::string unescape_literal(const std::string& body) {
    std::string out;
    for (size_t i = 0; i < body.size(); i++) {
        char c = body[i];
        if (c != '\\') {
            out.push_back(c);
            continue;
        }
        if (++i >= body.size()) fail("dangling escape in literal");
        char e = body[i];
        if (e == 'n') out.push_back('\n');
        else if (e == 't') out.push_back('\t');
        else if (e == 'r') out.push_back('\r');
        else if (e == 'x') {
            if (i + 2 >= body.size()) fail("short \\x escape");
            out.push_back((char)(hexval(body[i + 1]) * 16 + hexval(body[i + 2])));
            i += 2;
        } else out.push_back(e);
    }
    return out;
}

std::string unescape_slashes(const std::string& body) {
    std::string out;
    for (size_t i = 0; i < body.size(); i++) {
        if (body[i] == '\\' && i + 1 < body.size()) {
            if (body[i + 1] == '/') out.push_back('/');
            else {
                out.push_back(body[i]);
                out.push_back(body[i + 1]);
            }
            i++;
        } else {
            out.push_back(body[i]);
        }
    }
    return out;
}

bool is_ident_start(char c) { return std::isalpha((unsigned char)c) || c == '_'; }
bool is_ident(char c) { return std::isalnum((unsigned char)c) || c == '_'; }

std::vector<std::string> tokenize(const std::string& s) {
    std::vector<std::string> out;
    size_t i = 0;
    while (i < s.size()) {
        char c = s[i];
        if (std::isspace((unsigned char)c)) {
            i++;
        } else if (c == '"') {
            size_t j = i + 1;
            while (j < s.size() && s[j] != '"') j += (s[j] == '\\') ? 2 : 1;
            if (j >= s.size()) fail("unterminated literal in rule");
            out.push_back(s.substr(i, j - i + 1));
            i = j + 1;
        } else if (is_ident_start(c)) {
            size_t j = i;
            while (j < s.size() && is_ident(s[j])) j++;
            out.push_back(s.substr(i, j - i));
            i = j;
        } else if (std::string("():|?*+[]").find(c) != std::string::npos) {
            out.push_back(std::string(1, c));
            i++;
        } else {
            fail("cannot read rule text near '" + s.substr(i, 20) + "'");
        }
    }
    return out;
}

struct Lowering {
    Grammar& g;
    std::map<std::string, int> term_id;
    std::map<std::string, int> nt_id;
    int counter = 0;
    std::vector<std::pair<int, std::vector<std::string>>> pending_rules;  // lhs nt, symbol names

    explicit Lowering(Grammar& gr) : g(gr) {}

    int fresh(const char* prefix) {
        std::string name = std::string("__") + prefix + std::to_string(counter++);
        int id = (int)g.nts.size();
        g.nts.push_back(name);
        nt_id[name] = id;
        return id;
    }

    std::string literal_terminal(const std::string& tok) {
        std::string lit = unescape_literal(tok.substr(1, tok.size() - 2));
        if (lit.empty()) fail("empty literal");
        if (!term_id.count(tok)) {
            Terminal t;
            t.name = tok;
            t.literal = true;
            t.pattern = lit;
            t.priority = 1;
            term_id[tok] = (int)g.terms.size();
            g.terms.push_back(t);
        }
        return tok;
    }

    using Alts = std::vector<std::vector<std::string>>;

    void add_rule(int lhs, const std::vector<std::string>& rhs) { pending_rules.push_back({lhs, rhs}); }

    std::string ntname(int id) { return g.nts[id]; }

    // returns the symbols an item expands to
    std::vector<std::string> lower(const std::string& kind, const Alts& inner_in, const std::string& sym,
                                   char op) {
        Alts inner = inner_in;
        if (kind == "sym") inner = {{sym}};
        if (kind == "opt") {
            if (op) fail("[...] takes no postfix operator");
            op = '?';
        }
        if (!op) {
            if (inner.size() == 1) return inner[0];
            int nt = fresh("g");
            for (auto& a : inner) add_rule(nt, a);
            return {ntname(nt)};
        }
        std::vector<std::string> x;
        if (inner.size() == 1) {
            x = inner[0];
        } else {
            int gnt = fresh("g");
            for (auto& a : inner) add_rule(gnt, a);
            x = {ntname(gnt)};
        }
        int nt;
        if (op == '?') {
            nt = fresh("o");
            add_rule(nt, {});
            add_rule(nt, x);
        } else if (op == '*') {
            nt = fresh("s");
            add_rule(nt, {});
            std::vector<std::string> r = {ntname(nt)};
            r.insert(r.end(), x.begin(), x.end());
            add_rule(nt, r);
        } else {
            nt = fresh("p");
            add_rule(nt, x);
            std::vector<std::string> r = {ntname(nt)};
            r.insert(r.end(), x.begin(), x.end());
            add_rule(nt, r);
        }
        return {ntname(nt)};
    }

    Alts parse_alts(const std::vector<std::string>& t, size_t& i, const std::string& closer) {
        Alts alts(1);
        while (i < t.size()) {
            if (!closer.empty() && t[i] == closer) {
                i++;
                return alts;
            }
            if (t[i] == "|") {
                alts.emplace_back();
                i++;
                continue;
            }
            auto item = parse_item(t, i);
            alts.back().insert(alts.back().end(), item.begin(), item.end());
        }
        if (!closer.empty()) fail("missing '" + closer + "'");
        return alts;
    }

    std::vector<std::string> parse_item(const std::vector<std::string>& t, size_t& i) {
        std::string kind, sym;
        Alts inner;
        const std::string& tok = t[i];
        if (tok == "(") {
            i++;
            inner = parse_alts(t, i, ")");
            kind = "group";
        } else if (tok == "[") {
            i++;
            inner = parse_alts(t, i, "]");
            kind = "opt";
        } else if (tok[0] == '"') {
            sym = literal_terminal(tok);
            kind = "sym";
            i++;
        } else if (is_ident_start(tok[0])) {
            sym = tok;
            kind = "sym";
            i++;
        } else {
            fail("unexpected '" + tok + "' in rule");
        }
        char op = 0;
        if (i < t.size() && (t[i] == "?" || t[i] == "*" || t[i] == "+")) {
            op = t[i][0];
            i++;
        }
        return lower(kind, inner, sym, op);
    }
};

}  // namespace

Grammar parse_grammar(const std::string& text) {
    Grammar g;
    // logical lines
    std::vector<std::string> lines;
    size_t pos = 0;
    while (pos <= text.size()) {
        size_t nl = text.find('\n', pos);
        if (nl == std::string::npos) nl = text.size();
        std::string s = trim(text.substr(pos, nl - pos));
        pos = nl + 1;
        if (s.empty() || s.rfind("//", 0) == 0) continue;
        if (s[0] == '|') {
            if (lines.empty()) fail("continuation line before any rule");
            lines.back() += " " + s;
        } else {
            lines.push_back(s);
        }
    }
    Lowering L(g);
    std::vector<std::string> ignores;
    std::vector<std::pair<std::string, std::vector<std::string>>> rule_defs;
    for (auto& line : lines) {
        if (line[0] == '%') {
            std::vector<std::string> parts;
            size_t a = 0;
            while (a < line.size()) {
                while (a < line.size() && std::isspace((unsigned char)line[a])) a++;
                size_t b = a;
                while (b < line.size() && !std::isspace((unsigned char)line[b])) b++;
                if (b > a) parts.push_back(line.substr(a, b - a));
                a = b;
            }
            if (parts.size() == 2 && parts[0] == "%ignore") ignores.push_back(parts[1]);
            else if (parts.size() == 2 && parts[0] == "%lexer" && (parts[1] == "basic" || parts[1] == "contextual"))
                g.contextual = parts[1] == "contextual";
            else fail("unknown directive '" + line + "'");
            continue;
        }
        size_t i = 0;
        if (!is_ident_start(line[0])) fail("cannot read line '" + line + "'");
        while (i < line.size() && is_ident(line[i])) i++;
        std::string name = line.substr(0, i);
        bool has_prio = false;
        int prio = 0;
        if (i < line.size() && line[i] == '.') {
            size_t j = i + 1;
            if (j < line.size() && line[j] == '-') j++;
            size_t k = j;
            while (k < line.size() && std::isdigit((unsigned char)line[k])) k++;
            if (k == j) fail("bad priority in '" + line + "'");
            prio = std::stoi(line.substr(i + 1, k - i - 1));
            has_prio = true;
            i = k;
        }
        while (i < line.size() && std::isspace((unsigned char)line[i])) i++;
        if (i >= line.size() || line[i] != ':') fail("cannot read line '" + line + "'");
        std::string body = trim(line.substr(i + 1));
        if (std::isupper((unsigned char)name[0])) {
            if (L.term_id.count(name)) fail("terminal " + name + " defined twice");
            Terminal t;
            t.name = name;
            t.priority = has_prio ? prio : 0;
            if (body.size() >= 2 && body.front() == '"' && body.back() == '"') {
                t.literal = true;
                t.pattern = unescape_literal(body.substr(1, body.size() - 2));
            } else if (body.size() >= 2 && body.front() == '/' && body.back() == '/') {
                t.literal = false;
                t.pattern = unescape_slashes(body.substr(1, body.size() - 2));
            } else {
                fail("terminal " + name + " must be a literal or a regex");
            }
            if (t.pattern.empty()) fail("terminal " + name + " is empty");
            L.term_id[name] = (int)g.terms.size();
            g.terms.push_back(t);
        } else {
            if (has_prio) fail("rules take no priority");
            rule_defs.push_back({name, tokenize(body)});
        }
    }
    for (auto& rd : rule_defs) {
        if (!L.nt_id.count(rd.first)) {
            L.nt_id[rd.first] = (int)g.nts.size();
            g.nts.push_back(rd.first);
        }
    }
    if (!L.nt_id.count("start")) fail("grammar has no 'start' rule");
    g.start_nt = L.nt_id["start"];
    std::vector<std::pair<int, std::vector<std::string>>> ordered;
    for (auto& rd : rule_defs) {
        size_t i = 0;
        L.pending_rules.clear();
        auto alts = L.parse_alts(rd.second, i, "");
        for (auto& pr : L.pending_rules) ordered.push_back(pr);
        for (auto& a : alts) ordered.push_back({L.nt_id[rd.first], a});
    }
    for (auto& ig : ignores) {
        if (!L.term_id.count(ig)) fail("%ignore of unknown terminal " + ig);
        g.terms[L.term_id[ig]].ignored = true;
    }
    for (auto& pr : ordered) {
        Rule r;
        r.lhs = pr.first;
        for (auto& s : pr.second) {
            bool term = std::isupper((unsigned char)s[0]) || s[0] == '"';
            if (term) {
                auto it = L.term_id.find(s);
                if (it == L.term_id.end()) fail("unknown terminal " + s);
                if (g.terms[it->second].ignored) fail("ignored terminal " + s + " used in a rule");
                r.rhs.push_back(it->second);
            } else {
                auto it = L.nt_id.find(s);
                if (it == L.nt_id.end()) fail("unknown nonterminal " + s);
                r.rhs.push_back(~it->second);
            }
        }
        g.rules.push_back(r);
    }
    if (g.terms.size() > 30000) fail("too many terminals");
    return g;
}

std::vector<int> terminal_rank(const Grammar& g) {
    std::vector<int> order(g.terms.size());
    for (size_t i = 0; i < order.size(); i++) order[i] = (int)i;
    std::sort(order.begin(), order.end(), [&](int a, int b) {
        if (g.terms[a].priority != g.terms[b].priority) return g.terms[a].priority > g.terms[b].priority;
        return g.terms[a].name < g.terms[b].name;  // byte-wise
    });
    std::vector<int> rank(order.size());
    for (size_t r = 0; r < order.size(); r++) rank[order[r]] = (int)r;
    return rank;
}

}  // namespace psc
