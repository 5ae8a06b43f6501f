// LALR(1) parser tables: LR(0) automaton plus DeRemer-Pennello lookaheads.
//
// The paper's parser is a deterministic terminating PDA whose stack holds
// parser states (Section 2.4); it builds it with Lark's LALR(1) generator.
// The grammar is augmented with S' -> start END; the state reached by `start`
// from state 0 accepts on END.  LALR(1) lookaheads are the relations of
// DeRemer and Pennello (1982): DR, reads, includes, lookback, solved with the
// SCC digraph traversal.  Any shift/reduce or reduce/reduce conflict is an error
// (the method requires a deterministic parser, Section 2.4 and "Threats").
#include <algorithm>
#include <map>
#include <unordered_map>

#include "psc_internal.h"

namespace psc {
namespace {

struct Bits {
    std::vector<uint64_t> w;
    explicit Bits(int n = 0) : w((n + 63) / 64, 0) {}
    void set(int i) { w[i >> 6] |= 1ull << (i & 63); }
    bool test(int i) const { return (w[i >> 6] >> (i & 63)) & 1; }
    void merge(const Bits& o) {
        for (size_t i = 0; i < w.size(); i++) w[i] |= o.w[i];
    }
};

// DeRemer-Pennello digraph: F(x) = F'(x) U union{F(y) : x R y}
void digraph(int n, const std::vector<std::vector<int>>& R, std::vector<Bits>& F) {
    std::vector<int> N(n, 0), stack;
    const int INF = 1 << 30;
    // iterative Tarjan-style traversal
    for (int x0 = 0; x0 < n; x0++) {
        if (N[x0] != 0) continue;
        struct Frame { int x, i, d; };
        std::vector<Frame> call{{x0, 0, 0}};
        stack.push_back(x0);
        N[x0] = (int)stack.size();
        call.back().d = N[x0];
        while (!call.empty()) {
            Frame& f = call.back();
            if (f.i < (int)R[f.x].size()) {
                int y = R[f.x][f.i++];
                if (N[y] == 0) {
                    stack.push_back(y);
                    N[y] = (int)stack.size();
                    call.push_back({y, 0, N[y]});
                } else {
                    N[f.x] = std::min(N[f.x], N[y]);
                    F[f.x].merge(F[y]);
                }
                continue;
            }
            int x = f.x, d = f.d;
            call.pop_back();
            if (N[x] == d) {
                for (;;) {
                    int top = stack.back();
                    stack.pop_back();
                    N[top] = INF;
                    if (top == x) break;
                    F[top] = F[x];
                }
            }
            if (!call.empty()) {
                Frame& p = call.back();
                N[p.x] = std::min(N[p.x], N[x]);
                F[p.x].merge(F[x]);
            }
        }
    }
}

}  // namespace

Parser build_lalr(const Grammar& g) {
    const int nT = (int)g.terms.size();
    const int END = nT;
    const int nTerms = nT + 1;
    const int nN = (int)g.nts.size();
    const int AUG = nN;
    const int nNts = nN + 1;
    // productions: 0 = S' -> start END
    struct Prod { int lhs; std::vector<int> rhs; };   // rhs symbol: >= 0 terminal (END included), < 0 ~nt
    std::vector<Prod> P;
    P.push_back({AUG, {~g.start_nt, END}});
    for (auto& r : g.rules) P.push_back({r.lhs, r.rhs});
    std::vector<std::vector<int>> by_lhs(nNts);
    for (size_t p = 0; p < P.size(); p++) by_lhs[P[p].lhs].push_back((int)p);
    for (int a = 0; a < nN; a++)
        if (by_lhs[a].empty()) throw Error(ST_ERR_GRAMMAR, "nonterminal " + g.nts[a] + " has no rule");
    std::vector<char> nullable(nNts, 0);
    for (bool ch = true; ch;) {
        ch = false;
        for (auto& p : P) {
            if (nullable[p.lhs]) continue;
            bool all = true;
            for (int s : p.rhs)
                if (s >= 0 || !nullable[~s]) { all = false; break; }
            if (all) { nullable[p.lhs] = 1; ch = true; }
        }
    }
    // LR(0) automaton
    using Item = std::pair<int, int>;
    std::vector<std::vector<Item>> kernels;
    std::map<std::vector<Item>, int> index;
    std::vector<std::map<int, int>> trans;   // symbol -> state (terminal >= 0, nonterminal ~n)
    std::vector<std::vector<Item>> closures;
    kernels.push_back({{0, 0}});
    index[kernels[0]] = 0;
    for (size_t i = 0; i < kernels.size(); i++) {
        if (kernels.size() > 60000) throw Error(ST_ERR_LIMIT, "more than 60000 LR(0) states");
        std::vector<Item> items = kernels[i];
        std::vector<char> added(nNts, 0);
        for (size_t k = 0; k < items.size(); k++) {
            auto [p, d] = items[k];
            if (d < (int)P[p].rhs.size() && P[p].rhs[d] < 0) {
                int b = ~P[p].rhs[d];
                if (!added[b]) {
                    added[b] = 1;
                    for (int q : by_lhs[b]) items.push_back({q, 0});
                }
            }
        }
        closures.push_back(items);
        std::map<int, std::vector<Item>> moves;
        for (auto& [p, d] : items)
            if (d < (int)P[p].rhs.size()) moves[P[p].rhs[d]].push_back({p, d + 1});
        std::map<int, int> tr;
        for (auto& [sym, kern] : moves) {
            std::sort(kern.begin(), kern.end());
            auto it = index.find(kern);
            int j;
            if (it == index.end()) {
                j = (int)kernels.size();
                index[kern] = j;
                kernels.push_back(kern);
            } else {
                j = it->second;
            }
            tr[sym] = j;
        }
        trans.push_back(tr);
    }
    const int nS = (int)kernels.size();
    auto go_state = [&](int s, int sym) -> int {
        auto it = trans[s].find(sym);
        return it == trans[s].end() ? -1 : it->second;
    };
    // nonterminal transitions
    std::vector<std::pair<int, int>> ntt;   // (state, nonterminal)
    std::map<std::pair<int, int>, int> ntt_id;
    for (int s = 0; s < nS; s++)
        for (auto& [sym, d] : trans[s])
            if (sym < 0) {
                ntt_id[{s, ~sym}] = (int)ntt.size();
                ntt.push_back({s, ~sym});
            }
    const int nX = (int)ntt.size();
    std::vector<Bits> F(nX, Bits(nTerms));
    std::vector<std::vector<int>> reads(nX), includes(nX);
    for (int x = 0; x < nX; x++) {
        int r = go_state(ntt[x].first, ~ntt[x].second);
        for (auto& [sym, d] : trans[r]) {
            if (sym >= 0) F[x].set(sym);
            else if (nullable[~sym]) reads[x].push_back(ntt_id[{r, ~sym}]);
        }
    }
    digraph(nX, reads, F);   // F = Read
    // includes and lookback
    std::map<std::pair<int, int>, std::vector<int>> lookback;   // (state, prod) -> ntt ids
    for (int x = 0; x < nX; x++) {
        int p0 = ntt[x].first, B = ntt[x].second;
        for (int pr : by_lhs[B]) {
            const auto& rhs = P[pr].rhs;
            int s = p0;
            for (size_t i = 0; i < rhs.size(); i++) {
                if (rhs[i] < 0) {
                    bool rest_null = true;
                    for (size_t j = i + 1; j < rhs.size(); j++)
                        if (rhs[j] >= 0 || !nullable[~rhs[j]]) { rest_null = false; break; }
                    if (rest_null) includes[ntt_id[{s, ~rhs[i]}]].push_back(x);
                }
                s = go_state(s, rhs[i]);
                if (s < 0) break;
            }
            if (s >= 0) lookback[{s, pr}].push_back(x);
        }
    }
    digraph(nX, includes, F);   // F = Follow
    // tables
    Parser out;
    out.n_states = nS;
    out.n_terms = nTerms;
    out.n_nts = nNts;
    out.end_term = END;
    out.action.assign((size_t)nS * nTerms, act_make(ACT_ERR, 0));
    out.go.assign((size_t)nS * nNts, -1);
    out.term_entered.assign(nS, 0);
    out.term_entered[0] = 1;
    for (auto& p : P) {
        out.rule_len.push_back((int)p.rhs.size());
        out.rule_lhs.push_back(p.lhs);
    }
    auto sym_name = [&](int t) { return t == END ? std::string("$END") : g.terms[t].name; };
    for (int s = 0; s < nS; s++) {
        for (auto& [sym, d] : trans[s]) {
            if (sym >= 0) {
                out.term_entered[d] = 1;
                if (sym == END) out.action[(size_t)s * nTerms + END] = act_make(ACT_ACCEPT, 0);
                else out.action[(size_t)s * nTerms + sym] = act_make(ACT_SHIFT, d);
            } else {
                out.go[(size_t)s * nNts + ~sym] = d;
            }
        }
        for (auto& [p, d] : closures[s]) {
            if (p == 0 || d != (int)P[p].rhs.size()) continue;
            Bits la(nTerms);
            auto it = lookback.find({s, p});
            if (it != lookback.end())
                for (int x : it->second) la.merge(F[x]);
            for (int t = 0; t < nTerms; t++) {
                if (!la.test(t)) continue;
                int32_t& a = out.action[(size_t)s * nTerms + t];
                int32_t want = act_make(ACT_REDUCE, p);
                if (act_kind(a) != ACT_ERR && a != want) {
                    std::string what = act_kind(a) == ACT_SHIFT ? "shift/reduce" : "reduce/reduce";
                    throw Error(ST_ERR_CONFLICT, what + " conflict in LALR(1) state " + std::to_string(s) +
                                " on " + sym_name(t) + " (rule for " +
                                (P[p].lhs == AUG ? std::string("start'") : g.nts[P[p].lhs]) + ")");
                }
                a = want;
            }
        }
    }
    if (nS > 65535) throw Error(ST_ERR_LIMIT, "more than 65535 parser states");
    return out;
}

}  // namespace psc
