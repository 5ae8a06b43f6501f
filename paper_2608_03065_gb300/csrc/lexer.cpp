// Byte-level lexer: terminal regexes -> one NFA -> DFA (subset construction) ->
// minimal DFA.  The lexing transducer of Section 2.2 is read as maximal munch
// with one byte of lookahead: a pending lexeme grows while the DFA has a move
// on the next byte; when it has none, the complete pending lexeme is emitted as
// the class of all terminals it matches and the byte starts a new lexeme.
// State q0 is the empty pending lexeme and is never merged with another state,
// so "pending lexeme is empty" is a property of the state alone.
//
// For every state p the finite set T_p of Section 3.1 (the terminal classes the
// pending lexeme can still become) is precomputed; a class of ignored terminals
// stands for the empty sequence, and T_q0 = {empty}.
#include <algorithm>
#include <bitset>
#include <map>
#include <queue>
#include <unordered_map>

#include "psc_internal.h"

namespace psc {
namespace {

using ByteSet = std::bitset<256>;

[[noreturn]] void fail(const std::string& m) { throw Error(ST_ERR_GRAMMAR, m); }

// ---- regex AST
struct Node {
    enum Kind { SET, CAT, ALT, REP, EPS } kind;
    ByteSet set;
    std::vector<int> kids;
    int lo = 0, hi = -1;  // REP: hi = -1 means unbounded
};

struct RegexParser {
    const std::string& s;
    size_t i = 0;
    std::vector<Node>& pool;
    RegexParser(const std::string& src, std::vector<Node>& p) : s(src), pool(p) {}

    int mk(Node n) {
        pool.push_back(n);
        return (int)pool.size() - 1;
    }
    int peek() const { return i < s.size() ? (unsigned char)s[i] : -1; }
    int take() { return (unsigned char)s[i++]; }

    static ByteSet range(int lo, int hi) {
        ByteSet b;
        for (int c = lo; c <= hi; c++) b.set(c);
        return b;
    }
    static ByteSet digit() { return range('0', '9'); }
    static ByteSet word() { return range('0', '9') | range('a', 'z') | range('A', 'Z') | range('_', '_'); }
    static ByteSet space() {
        ByteSet b;
        for (int c : {' ', '\t', '\n', '\r', '\f', '\v'}) b.set(c);
        return b;
    }

    int hex2() {
        if (i + 2 > s.size()) fail("regex: short \\x escape");
        auto hv = [](int c) -> int {
            if (c >= '0' && c <= '9') return c - '0';
            if (c >= 'a' && c <= 'f') return c - 'a' + 10;
            if (c >= 'A' && c <= 'F') return c - 'A' + 10;
            fail("regex: bad hex digit");
        };
        int v = hv((unsigned char)s[i]) * 16 + hv((unsigned char)s[i + 1]);
        i += 2;
        return v;
    }

    // escape after a backslash: returns the set; single = the byte if it is one byte
    ByteSet escape(int& single) {
        int c = take();
        single = -1;
        switch (c) {
            case 'n': single = '\n'; break;
            case 't': single = '\t'; break;
            case 'r': single = '\r'; break;
            case 'f': single = '\f'; break;
            case 'v': single = '\v'; break;
            case 'x': single = hex2(); break;
            case 'd': return digit();
            case 'D': return ~digit();
            case 'w': return word();
            case 'W': return ~word();
            case 's': return space();
            case 'S': return ~space();
            default: single = c;
        }
        ByteSet b;
        b.set(single);
        return b;
    }

    int parse() {
        int n = alt();
        if (i != s.size()) fail("regex: unexpected character");
        return n;
    }
    int alt() {
        std::vector<int> parts{cat()};
        while (peek() == '|') {
            take();
            parts.push_back(cat());
        }
        if (parts.size() == 1) return parts[0];
        Node n{Node::ALT, {}, parts};
        return mk(n);
    }
    int cat() {
        std::vector<int> items;
        while (peek() != -1 && peek() != '|' && peek() != ')') items.push_back(postfix());
        if (items.empty()) return mk(Node{Node::EPS, {}, {}});
        if (items.size() == 1) return items[0];
        return mk(Node{Node::CAT, {}, items});
    }
    int postfix() {
        int n = atom();
        for (;;) {
            int c = peek();
            Node r{Node::REP, {}, {n}};
            if (c == '*') { take(); r.lo = 0; r.hi = -1; }
            else if (c == '+') { take(); r.lo = 1; r.hi = -1; }
            else if (c == '?') { take(); r.lo = 0; r.hi = 1; }
            else if (c == '{') {
                size_t j = s.find('}', i);
                if (j == std::string::npos) fail("regex: missing '}'");
                std::string body = s.substr(i + 1, j - i - 1);
                i = j + 1;
                size_t comma = body.find(',');
                if (comma == std::string::npos) {
                    r.lo = r.hi = std::stoi(body);
                } else {
                    r.lo = std::stoi(body.substr(0, comma));
                    std::string h = body.substr(comma + 1);
                    r.hi = h.find_first_not_of(' ') == std::string::npos ? -1 : std::stoi(h);
                }
                if (r.hi >= 0 && r.hi < r.lo) fail("regex: bad repeat bounds");
            } else {
                return n;
            }
            n = mk(r);
        }
    }
    int atom() {
        int c = take();
        if (c == '(') {
            if (s.compare(i, 2, "?:") == 0) i += 2;
            int n = alt();
            if (peek() != ')') fail("regex: missing ')'");
            take();
            return n;
        }
        Node n{Node::SET, {}, {}};
        if (c == '[') n.set = char_class();
        else if (c == '.') { n.set.set(); n.set.reset('\n'); }
        else if (c == '\\') { int single; n.set = escape(single); }
        else if (c == '*' || c == '+' || c == '?' || c == '{') fail("regex: nothing to repeat");
        else n.set.set(c);
        return mk(n);
    }
    // one class member: set, and the byte if it is a single byte
    ByteSet class_atom(int& single) {
        int c = take();
        if (c == '\\') return escape(single);
        if (c >= 128) fail("regex: non-ASCII byte inside a character class");
        single = c;
        ByteSet b;
        b.set(c);
        return b;
    }
    ByteSet char_class() {
        bool neg = false;
        if (peek() == '^') { take(); neg = true; }
        ByteSet m;
        bool first = true;
        for (;;) {
            int c = peek();
            if (c == -1) fail("regex: missing ']'");
            if (c == ']' && !first) { take(); break; }
            first = false;
            int lo;
            ByteSet a = class_atom(lo);
            if (peek() == '-' && lo >= 0 && i + 1 < s.size() && s[i + 1] != ']') {
                take();
                int hi;
                class_atom(hi);
                if (hi < 0 || hi < lo) fail("regex: bad range in class");
                m |= range(lo, hi);
            } else {
                m |= a;
            }
        }
        return neg ? ~m : m;
    }
};

// ---- Thompson-style NFA
struct NFA {
    std::vector<std::vector<int>> eps;
    std::vector<int> edge_to;
    std::vector<ByteSet> edge_set;
    std::vector<int> accept;
    int add() {
        eps.emplace_back();
        edge_to.push_back(-1);
        edge_set.emplace_back();
        accept.push_back(-1);
        return (int)eps.size() - 1;
    }
    std::pair<int, int> build(const std::vector<Node>& pool, int id) {
        const Node& n = pool[id];
        switch (n.kind) {
            case Node::EPS: { int a = add(); return {a, a}; }
            case Node::SET: {
                if (n.set.none()) fail("regex: empty character class");
                int a = add(), b = add();
                edge_to[a] = b;
                edge_set[a] = n.set;
                return {a, b};
            }
            case Node::CAT: {
                auto f = build(pool, n.kids[0]);
                int cur = f.second;
                for (size_t k = 1; k < n.kids.size(); k++) {
                    auto g = build(pool, n.kids[k]);
                    eps[cur].push_back(g.first);
                    cur = g.second;
                }
                return {f.first, cur};
            }
            case Node::ALT: {
                int a = add(), b = add();
                for (int k : n.kids) {
                    auto g = build(pool, k);
                    eps[a].push_back(g.first);
                    eps[g.second].push_back(b);
                }
                return {a, b};
            }
            case Node::REP: {
                int a = add();
                int cur = a;
                for (int k = 0; k < n.lo; k++) {
                    auto g = build(pool, n.kids[0]);
                    eps[cur].push_back(g.first);
                    cur = g.second;
                }
                int out = add();
                if (n.hi < 0) {
                    auto g = build(pool, n.kids[0]);
                    eps[cur].push_back(g.first);
                    eps[g.second].push_back(cur);
                    eps[cur].push_back(out);
                } else {
                    for (int k = n.lo; k < n.hi; k++) {
                        eps[cur].push_back(out);
                        auto g = build(pool, n.kids[0]);
                        eps[cur].push_back(g.first);
                        cur = g.second;
                    }
                    eps[cur].push_back(out);
                }
                return {a, out};
            }
        }
        return {-1, -1};
    }
    void closure(std::vector<int>& set) const {
        std::vector<char> in(eps.size(), 0);
        for (int s : set) in[s] = 1;
        std::vector<int> stack = set;
        while (!stack.empty()) {
            int s = stack.back();
            stack.pop_back();
            for (int d : eps[s])
                if (!in[d]) {
                    in[d] = 1;
                    set.push_back(d);
                    stack.push_back(d);
                }
        }
        std::sort(set.begin(), set.end());
    }
};

struct VecHash {
    size_t operator()(const std::vector<int>& v) const {
        uint64_t h = 1469598103934665603ull;
        for (int x : v) h = (h ^ (uint64_t)(uint32_t)x) * 1099511628211ull;
        return (size_t)h;
    }
};

}  // namespace

Lexer build_lexer(const Grammar& g, const std::vector<int>& rank) {
    NFA nfa;
    int start = nfa.add();
    for (size_t t = 0; t < g.terms.size(); t++) {
        std::vector<Node> pool;
        int root;
        const Terminal& term = g.terms[t];
        if (term.literal) {
            std::vector<int> kids;
            for (unsigned char c : term.pattern) {
                Node n{Node::SET, {}, {}};
                n.set.set(c);
                pool.push_back(n);
                kids.push_back((int)pool.size() - 1);
            }
            if (kids.size() == 1) root = kids[0];
            else { pool.push_back(Node{Node::CAT, {}, kids}); root = (int)pool.size() - 1; }
        } else {
            RegexParser rp(term.pattern, pool);
            root = rp.parse();
        }
        auto fr = nfa.build(pool, root);
        nfa.accept[fr.second] = (int)t;
        nfa.eps[start].push_back(fr.first);
    }
    // byte classes: bytes that every edge set treats alike
    std::vector<int> byte_class(256, -1), reps;
    {
        std::map<std::vector<bool>, int> sig;
        for (int b = 0; b < 256; b++) {
            std::vector<bool> k;
            for (size_t s = 0; s < nfa.eps.size(); s++)
                if (nfa.edge_to[s] >= 0) k.push_back(nfa.edge_set[s].test(b));
            auto it = sig.find(k);
            if (it == sig.end()) {
                int id = (int)reps.size();
                sig[k] = id;
                reps.push_back(b);
                byte_class[b] = id;
            } else {
                byte_class[b] = it->second;
            }
        }
    }
    int nbc = (int)reps.size();
    // subset construction
    std::vector<std::vector<int>> dstates;
    std::unordered_map<std::vector<int>, int, VecHash> index;
    std::vector<int> init{start};
    nfa.closure(init);
    dstates.push_back(init);
    index[init] = 0;
    std::vector<int> dtrans;  // [n][nbc]
    for (size_t i = 0; i < dstates.size(); i++) {
        if (dstates.size() > 200000) throw Error(ST_ERR_LIMIT, "lexer DFA too large");
        dtrans.resize((i + 1) * nbc, -1);
        for (int bc = 0; bc < nbc; bc++) {
            int b = reps[bc];
            std::vector<int> nxt;
            for (int s : dstates[i])
                if (nfa.edge_to[s] >= 0 && nfa.edge_set[s].test(b)) nxt.push_back(nfa.edge_to[s]);
            if (nxt.empty()) continue;
            std::sort(nxt.begin(), nxt.end());
            nxt.erase(std::unique(nxt.begin(), nxt.end()), nxt.end());
            nfa.closure(nxt);
            auto it = index.find(nxt);
            int j;
            if (it == index.end()) {
                j = (int)dstates.size();
                index[nxt] = j;
                dstates.push_back(nxt);
            } else {
                j = it->second;
            }
            dtrans[i * nbc + bc] = j;
        }
    }
    int n = (int)dstates.size();
    // classes of complete lexemes
    Lexer L;
    std::map<std::vector<int>, int> class_index;
    std::vector<int> dclass(n, -1);
    for (int i = 0; i < n; i++) {
        std::vector<int> ts;
        for (int s : dstates[i])
            if (nfa.accept[s] >= 0) ts.push_back(nfa.accept[s]);
        if (ts.empty()) continue;
        std::sort(ts.begin(), ts.end(), [&](int a, int b) { return rank[a] < rank[b]; });
        ts.erase(std::unique(ts.begin(), ts.end()), ts.end());
        int ign = 0;
        for (int t : ts) ign += g.terms[t].ignored;
        if (ign && ign != (int)ts.size())
            throw Error(ST_ERR_LEXER_AMBIGUOUS, "a lexeme matches both an ignored terminal (" +
                        g.terms[ts[0]].name + ") and a kept one");
        if (i == 0) throw Error(ST_ERR_GRAMMAR, "a terminal matches the empty string");
        auto it = class_index.find(ts);
        if (it == class_index.end()) {
            int id = (int)L.classes.size();
            class_index[ts] = id;
            L.classes.push_back(ts);
            L.class_ignored.push_back(ign ? 1 : 0);
            dclass[i] = id;
        } else {
            dclass[i] = it->second;
        }
    }
    // Moore refinement; the initial state stays alone
    std::vector<int> cls(n);
    for (int i = 0; i < n; i++) cls[i] = i == 0 ? 0 : dclass[i] + 2;
    int ncls = -1;
    for (;;) {
        std::map<std::vector<int>, int> sig;
        std::vector<int> nc(n);
        for (int i = 0; i < n; i++) {
            std::vector<int> k;
            k.reserve(nbc + 1);
            k.push_back(cls[i]);
            for (int bc = 0; bc < nbc; bc++) {
                int d = dtrans[i * nbc + bc];
                k.push_back(d < 0 ? -1 : cls[d]);
            }
            auto it = sig.find(k);
            if (it == sig.end()) {
                int id = (int)sig.size();
                sig[k] = id;
                nc[i] = id;
            } else {
                nc[i] = it->second;
            }
        }
        int m = (int)sig.size();
        cls.swap(nc);
        if (m == ncls) break;
        ncls = m;
    }
    // renumber so that q0 = 0 in BFS order
    std::vector<int> rep(ncls, -1), order, newid(ncls, -1);
    for (int i = 0; i < n; i++)
        if (rep[cls[i]] < 0) rep[cls[i]] = i;
    std::queue<int> bfs;
    bfs.push(cls[0]);
    newid[cls[0]] = 0;
    order.push_back(cls[0]);
    while (!bfs.empty()) {
        int c = bfs.front();
        bfs.pop();
        for (int bc = 0; bc < nbc; bc++) {
            int d = dtrans[rep[c] * nbc + bc];
            if (d < 0) continue;
            int dc = cls[d];
            if (newid[dc] < 0) {
                newid[dc] = (int)order.size();
                order.push_back(dc);
                bfs.push(dc);
            }
        }
    }
    int nq = (int)order.size();
    if (nq > 32000) throw Error(ST_ERR_LIMIT, "lexer DFA has more than 32000 states");
    L.nq = nq;
    L.q0 = 0;
    L.trans.assign((size_t)nq * 256, -1);
    L.accept_cls.assign(nq, -1);
    for (int q = 0; q < nq; q++) {
        int r = rep[order[q]];
        L.accept_cls[q] = dclass[r];
        for (int b = 0; b < 256; b++) {
            int d = dtrans[r * nbc + byte_class[b]];
            L.trans[(size_t)q * 256 + b] = (int16_t)(d < 0 ? -1 : newid[cls[d]]);
        }
    }
    // T_p by reachability over the minimal DFA
    L.tp.assign(nq, {});
    L.tp[0] = {-1};
    for (int p = 1; p < nq; p++) {
        std::vector<char> seen(nq, 0);
        std::vector<int> stack{p};
        seen[p] = 1;
        std::vector<int> out;
        bool empty_seq = false;
        while (!stack.empty()) {
            int s = stack.back();
            stack.pop_back();
            int c = L.accept_cls[s];
            if (c >= 0) {
                if (L.class_ignored[c]) empty_seq = true;
                else out.push_back(c);
            }
            for (int b = 0; b < 256; b++) {
                int d = L.trans[(size_t)s * 256 + b];
                if (d >= 0 && !seen[d]) {
                    seen[d] = 1;
                    stack.push_back(d);
                }
            }
        }
        std::sort(out.begin(), out.end());
        out.erase(std::unique(out.begin(), out.end()), out.end());
        if (empty_seq) out.insert(out.begin(), -1);
        L.tp[p] = out;
    }
    return L;
}

}  // namespace psc
