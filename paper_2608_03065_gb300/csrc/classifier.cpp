// PSC offline construction: the one-pass stack classifier (Section 3, Algorithm 1).
//
// For every lexer state q and token v the realizable terminal sequences
// R_q(v) = x T_p are obtained by lexing v from q (Section 3.1).  Per q they are
// pooled into a trie whose edges are lexeme classes (the END marker for the
// end-of-sequence token) and whose nodes carry the tokens whose sequence ends
// there.  The classifier A of Eq. (9) reads q and then the parser stack from the
// top down.  Instead of building the transducers P_eps, P~_a and P_w of Eq.
// (5)-(8) and unioning their acceptors, it runs the same simulation directly:
// a "thread" is one walk of the trie together with the part of the stack the
// parser has built or read so far (the known top); it performs the parser's
// epsilon moves (reductions, Eq. 5) and single-terminal moves (shifts, Eq. 6-7)
// on the known top, and parks when a reduction pops below it, waiting for the
// next stack symbol (the read-up move of Eq. 5a).  A thread that consumes the
// whole sequence of a trie node with tokens has reached a stable stack
// (Eq. 5b), so those tokens are accepted (Eq. 3).  Subset construction over
// sets of parked threads (plus the set of tokens accepted so far) gives a DFA
// over stack symbols; it is minimised with the initial partition by mask
// (Algorithm 1, Minimize), and the mask A_s of every state is its accepted set.
//
// Terminals: a class consumed with the stack top s stands for resolve[class][s]:
// its highest-ranked terminal (basic lexer), or the highest-ranked one on which
// the LALR(1) state s has an action (contextual lexer).
#include <algorithm>
#include <atomic>
#include <chrono>
#include <cstring>
#include <mutex>
#include <climits>
#include <memory>
#include <map>
#include <thread>
#include <cstdio>
#include <cstdlib>
#include <unordered_map>

#include "psc_internal.h"

namespace psc {
namespace {

double now() {
    return std::chrono::duration<double>(std::chrono::steady_clock::now().time_since_epoch()).count();
}

uint64_t mix64(uint64_t h) {
    h ^= h >> 33;
    h *= 0xff51afd7ed558ccdull;
    h ^= h >> 33;
    h *= 0xc4ceb9fe1a85ec53ull;
    h ^= h >> 33;
    return h;
}

uint64_t hash_span(const int32_t* p, size_t n, uint64_t seed) {
    uint64_t h = seed ^ (n * 0x9e3779b97f4a7c15ull);
    for (size_t i = 0; i < n; i++) h = mix64(h ^ (uint32_t)p[i]) + i;
    return h;
}

// Hash of a mask row: the XOR of one mixed value per non-zero word (mix64 is a
// bijection, so distinct (index, word) pairs give distinct values).  Setting
// bits in a few words updates it in O(words changed) instead of O(W).
uint64_t word_hash(size_t i, uint32_t w) { return w ? mix64(((uint64_t)i << 32) ^ w ^ 0x5bd1e995u) : 0; }

uint64_t row_hash(const uint32_t* r, int W) {
    uint64_t h = 0;
    for (int i = 0; i < W; i++) h ^= word_hash((size_t)i, r[i]);
    return h;
}

// ----------------------------------------------------------------- tries
struct Trie {
    std::vector<int32_t> child_off{0}, child_cls, child_node;
    std::vector<int32_t> tok_off{0}, toks;
    std::vector<int32_t> root;   // per lexer state
    int n() const { return (int)tok_off.size() - 1; }
};

bool lex_token(const Lexer& L, int q, const uint8_t* b, int64_t len, std::vector<int>& out, int& p) {
    out.clear();
    int cur = q;
    for (int64_t i = 0; i < len; i++) {
        int c = b[i];
        int nx = L.trans[(size_t)cur * 256 + c];
        if (nx >= 0) {
            cur = nx;
            continue;
        }
        if (cur == L.q0) return false;
        int cls = L.accept_cls[cur];
        if (cls < 0) return false;
        if (!L.class_ignored[cls]) out.push_back(cls);
        nx = L.trans[(size_t)L.q0 * 256 + c];
        if (nx < 0) return false;
        cur = nx;
    }
    p = cur;
    return true;
}

struct LocalTrie {
    // edges (node, class) -> child in an open-addressing table (keys ~0 = empty)
    std::vector<uint64_t> keys = std::vector<uint64_t>(1024, ~0ull);
    std::vector<int32_t> vals = std::vector<int32_t>(1024, 0);
    size_t used = 0;
    std::vector<std::pair<int32_t, int32_t>> toks;  // (node, token)
    int32_t n = 1;
    static uint64_t key_of(int32_t node, int cls) { return ((uint64_t)(uint32_t)node << 24) | (uint32_t)(cls + 1); }
    int32_t child(int32_t node, int cls) {
        uint64_t key = key_of(node, cls);
        size_t m = keys.size() - 1, i = mix64(key) & m;
        for (; keys[i] != ~0ull; i = (i + 1) & m)
            if (keys[i] == key) return vals[i];
        keys[i] = key;
        vals[i] = n;
        if (++used * 2 > keys.size()) grow();
        return n++;
    }
    void grow() {
        std::vector<uint64_t> k2(keys.size() * 2, ~0ull);
        std::vector<int32_t> v2(keys.size() * 2, 0);
        size_t m = k2.size() - 1;
        for (size_t j = 0; j < keys.size(); j++) {
            if (keys[j] == ~0ull) continue;
            size_t i = mix64(keys[j]) & m;
            while (k2[i] != ~0ull) i = (i + 1) & m;
            k2[i] = keys[j];
            v2[i] = vals[j];
        }
        keys.swap(k2);
        vals.swap(v2);
    }
};

Trie build_tries(const Lexer& L, const uint8_t* vb, const int64_t* vo, int V, int eos_id, int end_cls,
                 int threads) {
    int nq = L.nq;
    std::vector<LocalTrie> local(nq);
    std::atomic<int> next{0};
    auto work = [&]() {
        std::vector<int> x;
        for (;;) {
            int q = next.fetch_add(1);
            if (q >= nq) break;
            LocalTrie& T = local[q];
            for (int v = 0; v < V; v++) {
                if (v == eos_id) continue;
                int64_t len = vo[v + 1] - vo[v];
                if (len <= 0) continue;
                int p;
                if (!lex_token(L, q, vb + vo[v], len, x, p)) continue;
                int32_t node = 0;
                for (int c : x) node = T.child(node, c);
                for (int d : L.tp[p]) {
                    if (d < 0) T.toks.push_back({node, v});
                    else T.toks.push_back({T.child(node, d), v});
                }
            }
            if (eos_id >= 0 && eos_id < V) {
                if (q == L.q0) {
                    T.toks.push_back({T.child(0, end_cls), eos_id});
                } else if (L.accept_cls[q] >= 0) {
                    int c = L.accept_cls[q];
                    int32_t node = L.class_ignored[c] ? 0 : T.child(0, c);
                    T.toks.push_back({T.child(node, end_cls), eos_id});
                }
            }
        }
    };
    double t0 = now();
    std::vector<std::thread> pool;
    for (int i = 0; i < threads; i++) pool.emplace_back(work);
    for (auto& t : pool) t.join();
    double t1 = now();
    // each lexer state's part laid out on its own (in parallel), then concatenated
    struct Part {
        std::vector<int32_t> child_cls, child_node, child_cnt, toks, tok_cnt;
    };
    std::vector<Part> parts(nq);
    std::vector<int32_t> base(nq + 1, 0);
    for (int q = 0; q < nq; q++) base[q + 1] = base[q] + local[q].n;
    {
        std::atomic<int> next_q{0};
        auto lay_out = [&]() {
            for (int q; (q = next_q.fetch_add(1)) < nq;) {
                LocalTrie& T = local[q];
                Part& P = parts[q];
                std::vector<std::tuple<int32_t, int32_t, int32_t>> edges;  // parent, cls, child
                edges.reserve(T.used);
                for (size_t j = 0; j < T.keys.size(); j++)
                    if (T.keys[j] != ~0ull)
                        edges.emplace_back((int32_t)(T.keys[j] >> 24), (int32_t)(T.keys[j] & 0xFFFFFF) - 1, T.vals[j]);
                std::sort(edges.begin(), edges.end());
                std::sort(T.toks.begin(), T.toks.end());
                T.toks.erase(std::unique(T.toks.begin(), T.toks.end()), T.toks.end());
                P.child_cnt.assign(T.n, 0);
                P.tok_cnt.assign(T.n, 0);
                for (auto& [parent, cls, ch] : edges) {
                    P.child_cls.push_back(cls);
                    P.child_node.push_back(base[q] + ch);
                    P.child_cnt[parent]++;
                }
                for (auto& [node, tok] : T.toks) {
                    P.toks.push_back(tok);
                    P.tok_cnt[node]++;
                }
                std::vector<uint64_t>().swap(T.keys);
                std::vector<int32_t>().swap(T.vals);
                std::vector<std::pair<int32_t, int32_t>>().swap(T.toks);
            }
        };
        std::vector<std::thread> workers;
        for (int i = 0; i < threads; i++) workers.emplace_back(lay_out);
        for (auto& t : workers) t.join();
    }
    Trie tr;
    for (int q = 0; q < nq; q++) {
        Part& P = parts[q];
        tr.root.push_back(base[q]);
        tr.child_cls.insert(tr.child_cls.end(), P.child_cls.begin(), P.child_cls.end());
        tr.child_node.insert(tr.child_node.end(), P.child_node.begin(), P.child_node.end());
        tr.toks.insert(tr.toks.end(), P.toks.begin(), P.toks.end());
        int32_t co = tr.child_off.back(), to = tr.tok_off.back();
        for (int32_t nd = 0; nd < (int32_t)P.child_cnt.size(); nd++) {
            co += P.child_cnt[nd];
            to += P.tok_cnt[nd];
            tr.child_off.push_back(co);
            tr.tok_off.push_back(to);
        }
        Part().child_cls.swap(P.child_cls);
        P = Part();
    }
    if (getenv("PSC_LOG"))
        fprintf(stderr, "psc: token tries: %d nodes, lexing %.2f s, merging %.2f s\n", tr.n(), t1 - t0, now() - t1);
    return tr;
}

// --------------------------------------------------------- interning pools
struct ListPool {   // interned int32 lists
    std::vector<int32_t> data;
    std::vector<int64_t> off{0};
    std::unordered_multimap<uint64_t, int32_t> index;
    int32_t intern(const std::vector<int32_t>& v, uint64_t seed = 7) {
        uint64_t h = hash_span(v.data(), v.size(), seed);
        auto range = index.equal_range(h);
        for (auto it = range.first; it != range.second; ++it) {
            int32_t id = it->second;
            int64_t a = off[id], b = off[id + 1];
            if ((size_t)(b - a) == v.size() && std::equal(v.begin(), v.end(), data.begin() + a)) return id;
        }
        int32_t id = (int32_t)(off.size() - 1);
        data.insert(data.end(), v.begin(), v.end());
        off.push_back((int64_t)data.size());
        index.emplace(h, id);
        return id;
    }
    size_t size() const { return off.size() - 1; }
    const int32_t* ptr(int32_t id) const { return data.data() + off[id]; }
    int64_t len(int32_t id) const { return off[id + 1] - off[id]; }
};

struct Thread {
    int32_t node, t, r, A;   // START: t = -1
    bool operator==(const Thread& o) const { return node == o.node && t == o.t && r == o.r && A == o.A; }
};
struct ThreadHash {
    size_t operator()(const Thread& x) const {
        return (size_t)mix64(((uint64_t)(uint32_t)x.node << 32) ^ ((uint64_t)(uint32_t)x.t << 20) ^
                             ((uint64_t)(uint32_t)x.r << 12) ^ (uint64_t)(uint32_t)x.A * 0x9e37ull);
    }
};

struct Builder {
    const Lexer& L;
    const Parser& P;
    const Trie& tr;
    const std::vector<int16_t>& resolve;   // [n_classes][n_lr]
    int end_cls, n_lr, V, W;
    const Options& opt;

    // threads
    std::vector<Thread> threads;
    std::unordered_map<Thread, int32_t, ThreadHash> thread_id;
    // per-(thread, top) successor results
    std::unordered_map<uint64_t, int32_t> memo;
    std::vector<int64_t> res_th_off{0}, res_acc_off{0};
    std::vector<int32_t> res_th, res_acc;
    // masks
    std::vector<uint32_t> rows;                    // [n_masks][W]
    std::vector<uint64_t> row_hashes;              // row_hash of each row
    std::unordered_multimap<uint64_t, int32_t> row_index;
    std::unordered_map<uint64_t, int32_t> mask_memo;   // (mask, acc list id) -> mask
    ListPool acc_lists;
    // DFA states: (mask, thread list id)
    std::vector<int32_t> st_mask, st_list;
    std::unordered_map<uint64_t, int32_t> st_index;
    ListPool th_lists;
    std::vector<int32_t> st_def;
    std::vector<int64_t> exc_off{0};
    std::vector<int32_t> exc_y, exc_t;
    std::vector<std::vector<int32_t>> goto_src;     // nonterminal -> states with a goto on it
    // scratch for expansion: one frame of GCAP stack entries per trie level
    static constexpr int GCAP = 1024;
    std::vector<int32_t> out_th, out_acc;
    std::vector<int32_t> arena = std::vector<int32_t>(GCAP * 256);
    int arena_top = 0;

    int32_t* frame_push() {
        if (arena_top + GCAP > (int)arena.size()) throw Error(ST_ERR_LIMIT, "classifier simulation too deep");
        int32_t* f = arena.data() + arena_top;
        arena_top += GCAP;
        return f;
    }
    void frame_pop() { arena_top -= GCAP; }

    Builder(const Lexer& l, const Parser& p, const Trie& t, const std::vector<int16_t>& res, int endc, int v,
            const Options& o)
        : L(l), P(p), tr(t), resolve(res), end_cls(endc), n_lr(p.n_states), V(v), W((v + 31) / 32), opt(o) {
        goto_src.assign(P.n_nts, {});
        for (int s = 0; s < n_lr; s++)
            for (int a = 0; a < P.n_nts; a++)
                if (P.go[(size_t)s * P.n_nts + a] >= 0) goto_src[a].push_back(s);
        // rows 0 (nothing allowed) and 1 (end of sequence only, filled by the caller)
        rows.assign(2 * (size_t)W, 0);
    }

    int32_t add_row(const uint32_t* r, uint64_t h) {   // h = row_hash(r)
        auto range = row_index.equal_range(h);
        for (auto it = range.first; it != range.second; ++it)
            if (!memcmp(rows.data() + (size_t)it->second * W, r, sizeof(uint32_t) * W)) return it->second;
        int32_t id = (int32_t)(rows.size() / W);
        if ((int64_t)(rows.size() + W) * 4 > opt.max_mask_bytes)
            throw Error(ST_ERR_LIMIT, "mask rows exceed the memory limit");
        rows.insert(rows.end(), r, r + W);
        row_hashes.push_back(h);
        row_index.emplace(h, id);
        return id;
    }

    int32_t thread(const Thread& t) {
        auto it = thread_id.find(t);
        if (it != thread_id.end()) return it->second;
        int32_t id = (int32_t)threads.size();
        threads.push_back(t);
        thread_id.emplace(t, id);
        return id;
    }

    void park(int32_t c, int t, int r, int A) { out_th.push_back(thread({c, t, r, A})); }

    void expand(int32_t n, const int32_t* g, int glen);

    void consume(int32_t c, int t, int32_t* g, int glen) {
        for (int guard = 0; guard < 1000000; guard++) {
            int s = g[glen - 1];
            int32_t a = P.action[(size_t)s * P.n_terms + t];
            int kind = act_kind(a), val = act_val(a);
            if (glen + 1 >= GCAP) throw Error(ST_ERR_LIMIT, "classifier simulation stack overflow");
            if (kind == ACT_SHIFT) {
                g[glen++] = val;
                expand(c, g, glen);
                return;
            }
            if (kind == ACT_ACCEPT) {
                if (tr.tok_off[c + 1] > tr.tok_off[c]) out_acc.push_back(c);
                return;
            }
            if (kind != ACT_REDUCE) return;
            int k = P.rule_len[val], A = P.rule_lhs[val];
            if (glen > k) {
                glen -= k;
                int go = P.go[(size_t)g[glen - 1] * P.n_nts + A];
                if (go < 0) return;
                g[glen++] = go;
                continue;
            }
            park(c, t, k - glen, A);
            return;
        }
        throw Error(ST_ERR_LIMIT, "reduction loop did not end");
    }

    // successors of thread th when the next stack symbol read is Y
    int32_t step(int32_t th, int Y) {
        uint64_t key = ((uint64_t)(uint32_t)th << 16) | (uint32_t)Y;
        auto it = memo.find(key);
        if (it != memo.end()) return it->second;
        out_th.clear();
        out_acc.clear();
        const Thread t = threads[th];
        int32_t* g = frame_push();
        if (t.t < 0) {
            g[0] = Y;
            expand(t.node, g, 1);
        } else {
            int go = P.go[(size_t)Y * P.n_nts + t.A];
            if (go >= 0) {
                g[0] = Y;
                g[1] = go;
                consume(t.node, t.t, g, 2);
            }
        }
        frame_pop();
        std::sort(out_th.begin(), out_th.end());
        out_th.erase(std::unique(out_th.begin(), out_th.end()), out_th.end());
        std::sort(out_acc.begin(), out_acc.end());
        out_acc.erase(std::unique(out_acc.begin(), out_acc.end()), out_acc.end());
        int32_t rid = (int32_t)(res_th_off.size() - 1);
        res_th.insert(res_th.end(), out_th.begin(), out_th.end());
        res_th_off.push_back((int64_t)res_th.size());
        res_acc.insert(res_acc.end(), out_acc.begin(), out_acc.end());
        res_acc_off.push_back((int64_t)res_acc.size());
        memo.emplace(key, rid);
        return rid;
    }

    int32_t mask_add(int32_t m, const std::vector<int32_t>& acc) {
        if (acc.empty()) return m;
        int32_t aid = acc_lists.intern(acc);
        uint64_t key = ((uint64_t)(uint32_t)m << 32) | (uint32_t)aid;
        auto it = mask_memo.find(key);
        if (it != mask_memo.end()) return it->second;
        const uint32_t* base = rows.data() + (size_t)m * W;
        bool fresh = false;
        for (int32_t n : acc)
            for (int32_t k = tr.tok_off[n]; k < tr.tok_off[n + 1] && !fresh; k++) {
                int v = tr.toks[k];
                fresh = !((base[v >> 5] >> (v & 31)) & 1);
            }
        int32_t out = m;
        if (fresh) {
            std::vector<uint32_t> row(base, base + W);
            uint64_t h = row_hashes[m];
            for (int32_t n : acc)
                for (int32_t k = tr.tok_off[n]; k < tr.tok_off[n + 1]; k++) {
                    int v = tr.toks[k];
                    uint32_t old = row[v >> 5], now = old | (1u << (v & 31));
                    if (now != old) {
                        h ^= word_hash((size_t)(v >> 5), old) ^ word_hash((size_t)(v >> 5), now);
                        row[v >> 5] = now;
                    }
                }
            out = add_row(row.data(), h);
        }
        mask_memo.emplace(key, out);
        return out;
    }

    int32_t state(int32_t mask, const std::vector<int32_t>& th) {
        int32_t lid = th_lists.intern(th, 13);
        uint64_t key = ((uint64_t)(uint32_t)mask << 32) | (uint32_t)lid;
        auto it = st_index.find(key);
        if (it != st_index.end()) return it->second;
        int32_t id = (int32_t)st_mask.size();
        if (id >= opt.max_states) throw Error(ST_ERR_LIMIT, "classifier exceeds the state limit");
        st_mask.push_back(mask);
        st_list.push_back(lid);
        st_index.emplace(key, id);
        return id;
    }

    void build_transitions(int32_t s) {
        int32_t lid = st_list[s], m = st_mask[s];
        std::vector<int32_t> ths(th_lists.ptr(lid), th_lists.ptr(lid) + th_lists.len(lid));
        if (ths.empty()) {   // absorbing
            st_def.push_back(s);
            exc_off.push_back((int64_t)exc_y.size());
            return;
        }
        bool has_start = false;
        std::vector<int32_t> base;
        std::vector<int32_t> ys;
        std::vector<char> seen(n_lr, 0);
        for (int32_t th : ths) {
            const Thread t = threads[th];
            if (t.t < 0) {
                has_start = true;
            } else if (t.r > 0) {
                base.push_back(thread({t.node, t.t, t.r - 1, t.A}));
            } else {
                for (int32_t y : goto_src[t.A])
                    if (!seen[y]) { seen[y] = 1; ys.push_back(y); }
            }
        }
        if (has_start)
            for (int y = 0; y < n_lr; y++)
                if (P.term_entered[y] && !seen[y]) { seen[y] = 1; ys.push_back(y); }
        std::sort(base.begin(), base.end());
        base.erase(std::unique(base.begin(), base.end()), base.end());
        std::sort(ys.begin(), ys.end());
        // stable tops are entered by a terminal: any other top under the start
        // state cannot occur and leads to the dead state
        int32_t def = has_start ? state(0, {}) : state(m, base);
        st_def.push_back(def);
        std::vector<int32_t> cur, acc;
        for (int32_t y : ys) {
            cur = base;
            acc.clear();
            for (int32_t th : ths) {
                const Thread& t = threads[th];
                if (t.t >= 0 && (t.r > 0 || P.go[(size_t)y * P.n_nts + t.A] < 0)) continue;
                int32_t rid = step(th, y);
                cur.insert(cur.end(), res_th.begin() + res_th_off[rid], res_th.begin() + res_th_off[rid + 1]);
                acc.insert(acc.end(), res_acc.begin() + res_acc_off[rid], res_acc.begin() + res_acc_off[rid + 1]);
            }
            std::sort(cur.begin(), cur.end());
            cur.erase(std::unique(cur.begin(), cur.end()), cur.end());
            std::sort(acc.begin(), acc.end());
            acc.erase(std::unique(acc.begin(), acc.end()), acc.end());
            int32_t m2 = mask_add(m, acc);
            int32_t tgt = state(m2, cur);
            if (tgt != def) {
                exc_y.push_back(y);
                exc_t.push_back(tgt);
            }
        }
        exc_off.push_back((int64_t)exc_y.size());
    }
};

void Builder::expand(int32_t n, const int32_t* g, int glen) {
    if (tr.tok_off[n + 1] > tr.tok_off[n]) out_acc.push_back(n);
    if (tr.child_off[n + 1] == tr.child_off[n]) return;
    int top = g[glen - 1];
    int32_t* g2 = frame_push();
    for (int32_t e = tr.child_off[n]; e < tr.child_off[n + 1]; e++) {
        int cls = tr.child_cls[e];
        int t = cls == end_cls ? P.end_term : resolve[(size_t)cls * n_lr + top];
        if (t < 0) continue;
        std::copy(g, g + glen, g2);
        consume(tr.child_node[e], t, g2, glen);
    }
    frame_pop();
}

}  // namespace

namespace {

// The chunk table of mask rows given by pointer (row m = rows[m], W words):
// chunk hashes are computed in parallel, then chunk ids are given serially in
// the order chunks are first met (row by row), so the result does not depend on
// the thread count.
void set_mask_rows_from(Tables& t, const std::vector<const uint32_t*>& rows, int W, int threads) {
    int n = (int)rows.size();
    int nch = (W + 31) / 32;
    t.W = W;
    t.n_masks = n;
    t.nch = nch;
    t.mask_rows.assign((size_t)n * nch, 0);
    t.mask_chunks.clear();
    auto load_chunk = [&](int m, int c, uint32_t* chunk) {
        int w0 = c * 32, nw = std::min(32, W - w0);
        std::memcpy(chunk, rows[m] + w0, sizeof(uint32_t) * nw);
        for (int k = nw; k < 32; k++) chunk[k] = 0;
    };
    auto fnv = [](const uint32_t* chunk) {
        uint64_t h = 1469598103934665603ull;
        for (int k = 0; k < 32; k++) h = (h ^ chunk[k]) * 1099511628211ull;
        return h;
    };
    std::vector<uint64_t> hs((size_t)n * nch);
    {
        std::atomic<int> next{0};
        auto work = [&]() {
            uint32_t chunk[32];
            for (int m; (m = next.fetch_add(1)) < n;)
                for (int c = 0; c < nch; c++) {
                    load_chunk(m, c, chunk);
                    hs[(size_t)m * nch + c] = fnv(chunk);
                }
        };
        std::vector<std::thread> pool;
        for (int i = 0; i < std::max(1, threads); i++) pool.emplace_back(work);
        for (auto& th : pool) th.join();
    }
    // open addressing over chunk contents (load factor below 1/2)
    size_t cap = 1024;
    while (cap < (size_t)n * nch / 4 + 1024) cap <<= 1;
    std::vector<int64_t> slot(cap, -1);
    std::vector<uint64_t> slot_hash(cap, 0);
    uint32_t chunk[32];
    for (int m = 0; m < n; m++) {
        for (int c = 0; c < nch; c++) {
            uint64_t h = hs[(size_t)m * nch + c];
            load_chunk(m, c, chunk);
            if ((size_t)t.mask_chunks.size() / 32 * 2 >= cap) {
                size_t ncap = cap << 1;
                std::vector<int64_t> ns(ncap, -1);
                std::vector<uint64_t> nh(ncap, 0);
                for (size_t i = 0; i < cap; i++) {
                    if (slot[i] < 0) continue;
                    size_t j = slot_hash[i] & (ncap - 1);
                    while (ns[j] >= 0) j = (j + 1) & (ncap - 1);
                    ns[j] = slot[i];
                    nh[j] = slot_hash[i];
                }
                slot.swap(ns);
                slot_hash.swap(nh);
                cap = ncap;
            }
            size_t j = h & (cap - 1);
            int64_t id = -1;
            while (slot[j] >= 0) {
                if (slot_hash[j] == h &&
                    std::memcmp(t.mask_chunks.data() + (size_t)slot[j] * 32, chunk, sizeof(chunk)) == 0) {
                    id = slot[j];
                    break;
                }
                j = (j + 1) & (cap - 1);
            }
            if (id < 0) {
                id = (int64_t)(t.mask_chunks.size() / 32);
                t.mask_chunks.insert(t.mask_chunks.end(), chunk, chunk + 32);
                slot[j] = id;
                slot_hash[j] = h;
            }
            t.mask_rows[(size_t)m * nch + c] = (uint32_t)id;
        }
    }
    t.n_chunks = (int)(t.mask_chunks.size() / 32);
}

}  // namespace

void set_mask_rows(Tables& t, const uint32_t* rows, int n, int W) {
    std::vector<const uint32_t*> ptr(n);
    for (int m = 0; m < n; m++) ptr[m] = rows + (size_t)m * W;
    set_mask_rows_from(t, ptr, W, (int)std::max(1u, std::thread::hardware_concurrency()));
}

Tables compile_tables(const std::string& text, const uint8_t* vb, const int64_t* vo, int V, int eos_id,
                      const Options& opt) {
    double t0 = now();
    Tables T;
    Grammar g = parse_grammar(text);
    std::vector<int> rank = terminal_rank(g);
    Lexer L = build_lexer(g, rank);
    Parser P = build_lalr(g);
    if (getenv("PSC_LOG")) {
        size_t na = 0, ng = 0, nr = 0;
        for (int32_t x : P.action) na += act_kind(x) != ACT_ERR, nr += act_kind(x) == ACT_REDUCE;
        for (int32_t x : P.go) ng += x >= 0;
        fprintf(stderr, "psc: LALR(1): %d states, %d terminals, %d nonterminals, %zu actions (%zu reduce), %zu gotos, "
                        "%zu lexeme classes\n", P.n_states, P.n_terms, P.n_nts, na, nr, ng, L.classes.size());
    }
    int threads = opt.threads > 0 ? opt.threads : (int)std::max(1u, std::thread::hardware_concurrency());
    int ncls = (int)L.classes.size();
    int end_cls = ncls;   // pseudo class of the end marker

    // class -> terminal, per stack top
    std::vector<int16_t> resolve((size_t)ncls * P.n_states, -1);
    for (int c = 0; c < ncls; c++)
        for (int s = 0; s < P.n_states; s++) {
            int pick = -1;
            if (!g.contextual) {
                pick = L.classes[c][0];
            } else {
                for (int t : L.classes[c])
                    if (act_kind(P.action[(size_t)s * P.n_terms + t]) != ACT_ERR) { pick = t; break; }
            }
            resolve[(size_t)c * P.n_states + s] = (int16_t)pick;
        }

    double t1 = now();
    Trie tr = build_tries(L, vb, vo, V, eos_id, end_cls, threads);
    double t2 = now();

    // ---- one builder per lexer state, in parallel (their states are disjoint)
    int W = (V + 31) / 32;
    std::vector<uint32_t> eos_row(W, 0);
    if (eos_id >= 0 && eos_id < V) eos_row[eos_id >> 5] |= 1u << (eos_id & 31);
    // global mask pool: row 0 = nothing, row 1 = end-of-sequence only
    std::vector<uint32_t> grows(2 * (size_t)W, 0);
    std::copy(eos_row.begin(), eos_row.end(), grows.begin() + W);
    std::unordered_multimap<uint64_t, int32_t> gindex;
    gindex.emplace(row_hash(grows.data(), W), 0);
    gindex.emplace(row_hash(grows.data() + W, W), 1);
    struct Part {
        std::vector<int32_t> st_mask, st_def, exc_y, exc_t;
        std::vector<int64_t> exc_off;
        int32_t start = 0;
        int64_t n_threads = 0;
        double seconds = 0;
    };
    std::vector<Part> parts(L.nq);
    std::vector<int> qorder(L.nq);
    for (int q = 0; q < L.nq; q++) qorder[q] = q;
    std::sort(qorder.begin(), qorder.end(), [&](int a, int b) {
        int32_t ea = (a + 1 < L.nq ? tr.root[a + 1] : tr.n()) - tr.root[a];
        int32_t eb = (b + 1 < L.nq ? tr.root[b + 1] : tr.n()) - tr.root[b];
        return ea > eb;
    });
    std::atomic<int> next_q{0};
    std::atomic<int64_t> total_states{0};
    std::mutex pool_mu;
    std::string first_error;
    int first_code = 0;
    auto worker = [&]() {
        for (;;) {
            int k = next_q.fetch_add(1);
            if (k >= L.nq) break;
            int q = qorder[k];
            double tq = now();
            try {
                Builder B(L, P, tr, resolve, end_cls, V, opt);
                std::copy(eos_row.begin(), eos_row.end(), B.rows.begin() + W);
                B.row_index.clear();
                B.row_hashes = {row_hash(B.rows.data(), W), row_hash(B.rows.data() + W, W)};
                B.row_index.emplace(B.row_hashes[0], 0);
                B.row_index.emplace(B.row_hashes[1], 1);
                B.state(0, {});
                int32_t th = B.thread({tr.root[q], -1, 0, -1});
                Part& pt = parts[q];
                pt.start = B.state(0, {th});
                for (int32_t s = 0; s < (int32_t)B.st_mask.size(); s++) {
                    B.build_transitions(s);
                    if ((s & 1023) == 0 && total_states.load() + (int64_t)B.st_mask.size() > opt.max_states)
                        throw Error(ST_ERR_LIMIT, "classifier exceeds the state limit");
                }
                total_states += (int64_t)B.st_mask.size();
                // move this part's masks into the global pool
                int nm = (int)(B.rows.size() / W);
                std::vector<int32_t> gid(nm);
                {
                    std::lock_guard<std::mutex> lk(pool_mu);
                    for (int m = 0; m < nm; m++) {
                        const uint32_t* r = B.rows.data() + (size_t)m * W;
                        uint64_t h = B.row_hashes[m];
                        int32_t found = -1;
                        auto range = gindex.equal_range(h);
                        for (auto it = range.first; it != range.second; ++it)
                            if (!memcmp(grows.data() + (size_t)it->second * W, r, sizeof(uint32_t) * W)) {
                                found = it->second;
                                break;
                            }
                        if (found < 0) {
                            if ((int64_t)(grows.size() + W) * 4 > opt.max_mask_bytes)
                                throw Error(ST_ERR_LIMIT, "mask rows exceed the memory limit");
                            found = (int32_t)(grows.size() / W);
                            grows.insert(grows.end(), r, r + W);
                            gindex.emplace(h, found);
                        }
                        gid[m] = found;
                    }
                }
                pt.st_mask.resize(B.st_mask.size());
                for (size_t i = 0; i < B.st_mask.size(); i++) pt.st_mask[i] = gid[B.st_mask[i]];
                pt.st_def = std::move(B.st_def);
                pt.exc_off = std::move(B.exc_off);
                pt.exc_y = std::move(B.exc_y);
                pt.exc_t = std::move(B.exc_t);
                pt.n_threads = (int64_t)B.threads.size();
            } catch (const Error& e) {
                std::lock_guard<std::mutex> lk(pool_mu);
                if (!first_code) {
                    first_code = e.code;
                    first_error = e.what();
                }
                next_q = L.nq;
            } catch (const std::bad_alloc&) {
                std::lock_guard<std::mutex> lk(pool_mu);
                if (!first_code) {
                    first_code = ST_ERR_OOM;
                    first_error = "out of host memory while building the classifier";
                }
                next_q = L.nq;
            }
            parts[q].seconds = now() - tq;
        }
    };
    {
        std::vector<std::thread> pool;
        for (int i = 0; i < threads; i++) pool.emplace_back(worker);
        for (auto& t : pool) t.join();
    }
    if (first_code) throw Error(first_code, first_error);
    if (getenv("PSC_LOG")) {
        double busy = 0, longest = 0;
        for (int q = 0; q < L.nq; q++) {
            busy += parts[q].seconds;
            longest = std::max(longest, parts[q].seconds);
        }
        fprintf(stderr, "psc: %d lexer states on %d threads: %.2f s of builder time, longest %.2f s\n", L.nq,
                threads, busy, longest);
        for (int k = 0; k < std::min(L.nq, 12); k++) {
            int q = qorder[k];
            fprintf(stderr, "psc: lexer state %d: %zu classifier states, %lld threads, %.2f s\n", q,
                    parts[q].st_mask.size(), (long long)parts[q].n_threads, parts[q].seconds);
        }
    }
    // concatenate the parts
    struct Concat {
        std::vector<int32_t> st_mask, st_def, exc_y, exc_t;
        std::vector<int64_t> exc_off{0};
    } B;
    std::vector<int32_t> start_state(L.nq);
    int64_t n_threads_total = 0;
    for (int q = 0; q < L.nq; q++) {
        Part& pt = parts[q];
        int32_t base = (int32_t)B.st_mask.size();
        start_state[q] = base + pt.start;
        for (size_t i = 0; i < pt.st_mask.size(); i++) {
            B.st_mask.push_back(pt.st_mask[i]);
            B.st_def.push_back(base + pt.st_def[i]);
            for (int64_t e = pt.exc_off[i]; e < pt.exc_off[i + 1]; e++) {
                B.exc_y.push_back(pt.exc_y[e]);
                B.exc_t.push_back(base + pt.exc_t[e]);
            }
            B.exc_off.push_back((int64_t)B.exc_y.size());
        }
        n_threads_total += pt.n_threads;
        Part().st_mask.swap(pt.st_mask);
        pt = Part();
    }
    double t3 = now();

    // ---- Moore minimisation, initial partition by mask.  Each round gives every
    // state the signature (its class, the class of its default target, then the
    // (symbol, class) of each exception whose target class differs from the
    // default's) and numbers the distinct signatures in the order of their first
    // state, which is what a serial scan gives.  The signatures are hashed in
    // parallel; a shared open-addressing table keeps the first state of every hash,
    // every state is compared with that state's full signature, and a state whose
    // hash is shared by a different signature is grouped through a serial map.
    const int N = (int)B.st_mask.size();
    std::vector<int32_t> cls(N);
    {
        std::unordered_map<int32_t, int32_t> m2c;
        for (int s = 0; s < N; s++) {
            auto it = m2c.find(B.st_mask[s]);
            if (it == m2c.end()) it = m2c.emplace(B.st_mask[s], (int32_t)m2c.size()).first;
            cls[s] = it->second;
        }
    }
    auto sig_of = [&](int s, std::vector<int64_t>& sig) {
        sig.clear();
        int32_t dc = cls[B.st_def[s]];
        sig.push_back(cls[s]);
        sig.push_back(dc);
        for (int64_t e = B.exc_off[s]; e < B.exc_off[s + 1]; e++) {
            int32_t tc = cls[B.exc_t[e]];
            if (tc != dc) sig.push_back(((int64_t)B.exc_y[e] << 32) | (uint32_t)tc);
        }
    };
    auto hash_of = [](const std::vector<int64_t>& sig) {
        uint64_t h = 1469598103934665603ull;
        for (int64_t x : sig) h = mix64(h ^ (uint64_t)x);
        return h ? h : 1ull;   // 0 marks an empty slot
    };
    // contiguous chunks of [0, n), one worker per thread
    auto chunks_of = [&](int64_t n, auto&& body) {
        const int64_t step = 1 << 16;
        std::atomic<int64_t> next{0};
        auto run = [&]() {
            std::vector<int64_t> a, b;
            for (;;) {
                int64_t lo = next.fetch_add(step);
                if (lo >= n) break;
                body(lo, std::min<int64_t>(n, lo + step), a, b);
            }
        };
        int nt = (int)std::max<int64_t>(1, std::min<int64_t>(threads, (n + step - 1) / step));
        if (nt <= 1) {
            run();
            return;
        }
        std::vector<std::thread> pool;
        for (int k = 0; k < nt; k++) pool.emplace_back(run);
        for (auto& th : pool) th.join();
    };
    auto chunks = [&](auto&& body) { chunks_of(N, body); };
    size_t cap = 1024;
    while (cap < 2 * (size_t)N) cap <<= 1;
    std::unique_ptr<std::atomic<uint64_t>[]> tkey(new std::atomic<uint64_t>[cap]);
    std::unique_ptr<std::atomic<int32_t>[]> tval(new std::atomic<int32_t>[cap]);
    auto clear_table = [&]() {
        chunks_of((int64_t)cap, [&](int64_t lo, int64_t hi, std::vector<int64_t>&, std::vector<int64_t>&) {
            for (int64_t i = lo; i < hi; i++) {
                tkey[i].store(0, std::memory_order_relaxed);
                tval[i].store(INT32_MAX, std::memory_order_relaxed);
            }
        });
    };
    clear_table();
    auto slot_of = [&](uint64_t h, bool insert) -> size_t {
        size_t i = (size_t)h & (cap - 1);
        for (;;) {
            uint64_t k = tkey[i].load(std::memory_order_relaxed);
            if (k == h) return i;
            if (k == 0 && insert) {
                uint64_t z = 0;
                if (tkey[i].compare_exchange_strong(z, h) || z == h) return i;
            }
            i = (i + 1) & (cap - 1);
        }
    };
    std::vector<uint64_t> hs(N);
    std::vector<int32_t> first(N), nc(N);
    std::vector<char> odd(N);
    int ncl = -1;
    for (int iter = 0; iter < 100000; iter++) {
        // hashes, and the first state of every hash
        chunks([&](int64_t lo, int64_t hi, std::vector<int64_t>& sig, std::vector<int64_t>&) {
            for (int s = (int)lo; s < (int)hi; s++) {
                sig_of(s, sig);
                uint64_t h = hash_of(sig);
                hs[s] = h;
                std::atomic<int32_t>& v = tval[slot_of(h, true)];
                int32_t cur = v.load(std::memory_order_relaxed);
                while (s < cur && !v.compare_exchange_weak(cur, s)) {
                }
            }
        });
        // every state against the first state of its hash
        chunks([&](int64_t lo, int64_t hi, std::vector<int64_t>& a, std::vector<int64_t>& b) {
            for (int s = (int)lo; s < (int)hi; s++) {
                int32_t r = tval[slot_of(hs[s], false)].load(std::memory_order_relaxed);
                first[s] = r;
                odd[s] = 0;
                if (r != s) {
                    sig_of(s, a);
                    sig_of(r, b);
                    odd[s] = a != b;
                }
            }
        });
        // states whose hash is shared by another signature: grouped by full signature
        {
            std::map<std::vector<int64_t>, int32_t> groups;
            std::vector<int64_t> sig;
            for (int s = 0; s < N; s++)
                if (odd[s]) {
                    sig_of(s, sig);
                    auto it = groups.emplace(sig, s).first;
                    first[s] = it->second;
                }
        }
        // the distinct signatures numbered in the order of their first state
        int count = 0;
        for (int s = 0; s < N; s++)
            if (first[s] == s) nc[s] = count++;
        chunks([&](int64_t lo, int64_t hi, std::vector<int64_t>&, std::vector<int64_t>&) {
            for (int s = (int)lo; s < (int)hi; s++)
                if (first[s] != s) nc[s] = nc[first[s]];   // a first state is numbered above and not written here
        });
        cls.swap(nc);
        clear_table();
        if (count == ncl) break;
        ncl = count;
    }
    if (getenv("PSC_LOG")) fprintf(stderr, "psc: minimisation: %d states -> %d classes\n", N, ncl);
    double t4 = now();

    // ---- flatten
    std::vector<int32_t> rep(ncl, -1);
    for (int s = 0; s < N; s++)
        if (rep[cls[s]] < 0) rep[cls[s]] = s;
    std::vector<char> absorbing(ncl, 0);
    for (int c = 0; c < ncl; c++) {
        int r = rep[c];
        bool ab = cls[B.st_def[r]] == c;
        for (int64_t e = B.exc_off[r]; e < B.exc_off[r + 1] && ab; e++) ab = cls[B.exc_t[e]] == c;
        absorbing[c] = ab;
    }
    // masks actually used (0 and 1 always kept)
    std::vector<int32_t> mask_new(grows.size() / W, -1);
    mask_new[0] = 0;
    mask_new[1] = 1;
    int n_masks = 2;
    for (int c = 0; c < ncl; c++) {
        int32_t m = B.st_mask[rep[c]];
        if (mask_new[m] < 0) mask_new[m] = n_masks++;
    }
    std::vector<int32_t> dense(ncl, -1);
    int S = 0;
    for (int c = 0; c < ncl; c++)
        if (!absorbing[c]) dense[c] = S++;
    auto enc = [&](int32_t c) -> int32_t {
        return absorbing[c] ? -(mask_new[B.st_mask[rep[c]]] + 1) : dense[c];
    };
    T.S = S;
    T.n_lr = P.n_states;
    T.dfa_mask.assign(S, 0);
    // dense [S][n_lr] table, or (above the size budget) a default target and the
    // exceptions to it per state, as the construction produced them
    int64_t dense_budget = opt.max_dense_classifier_bytes == 0 ? (int64_t(512) << 20) : opt.max_dense_classifier_bytes;
    T.dfa_sparse = dense_budget < 0 || (int64_t)S * P.n_states * 4 > dense_budget;
    if (!T.dfa_sparse) T.dfa.assign((size_t)S * P.n_states, 0);
    else {
        T.dfa_def.assign(S, 0);
        T.dfa_exc_off.assign(1, 0);
    }
    for (int c = 0; c < ncl; c++) {   // dense ids increase with c
        if (absorbing[c]) continue;
        int r = rep[c];
        int32_t d = enc(cls[B.st_def[r]]);
        if (!T.dfa_sparse) {
            int32_t* row = T.dfa.data() + (size_t)dense[c] * P.n_states;
            for (int y = 0; y < P.n_states; y++) row[y] = d;
            for (int64_t e = B.exc_off[r]; e < B.exc_off[r + 1]; e++) row[B.exc_y[e]] = enc(cls[B.exc_t[e]]);
        } else {
            T.dfa_def[dense[c]] = d;
            for (int64_t e = B.exc_off[r]; e < B.exc_off[r + 1]; e++) {   // symbols ascending
                int32_t x = enc(cls[B.exc_t[e]]);
                if (x == d) continue;
                T.dfa_exc_y.push_back((uint16_t)B.exc_y[e]);
                T.dfa_exc_t.push_back(x);
            }
            T.dfa_exc_off.push_back((int64_t)T.dfa_exc_y.size());
        }
        T.dfa_mask[dense[c]] = mask_new[B.st_mask[r]];
    }
    T.dfa_start.resize(L.nq);
    for (int q = 0; q < L.nq; q++) T.dfa_start[q] = enc(cls[start_state[q]]);
    T.V = V;
    double t5 = now();
    {
        std::vector<const uint32_t*> rows_by_id(n_masks, nullptr);   // final mask id -> its pool row
        for (size_t m = 0; m < mask_new.size(); m++)
            if (mask_new[m] >= 0) rows_by_id[mask_new[m]] = grows.data() + m * W;
        set_mask_rows_from(T, rows_by_id, W, threads);
    }
    double t6 = now();

    // lexer and parser tables for the device
    T.nq = L.nq;
    T.q0 = L.q0;
    T.lex_trans = L.trans;
    T.lex_accept = L.accept_cls;
    T.cls_ignored = L.class_ignored;
    T.n_classes = ncls;
    T.n_terms = P.n_terms;
    T.n_nts = P.n_nts;
    T.end_term = P.end_term;
    T.action = P.action;
    T.go = P.go;
    T.rule_len = P.rule_len;
    T.rule_lhs = P.rule_lhs;
    T.resolve = resolve;
    T.contextual = g.contextual;
    T.vocab_bytes.assign(vb, vb + vo[V]);
    T.vocab_off.assign(vo, vo + V + 1);
    T.eos_id = eos_id;
    T.n_dfa_states_built = N;
    T.n_threads = n_threads_total;
    T.n_trie_nodes = tr.n();
    T.seconds_lex = t2 - t1;
    T.seconds_dfa = t3 - t2;
    T.seconds_min = t4 - t3;
    double t7 = now();
    // optional: empty tables when a size limit or the host's memory stops it (the device
    // then walks stacks from the top)
    bool built = false;
    try {
        built = build_bottom_up(T, opt);
    } catch (const std::bad_alloc&) {
        Options off = opt;
        off.max_bottom_up_bytes = -1;
        build_bottom_up(T, off);   // clears the partial tables
    }
    if (!built && getenv("PSC_LOG"))
        fprintf(stderr, "psc: no bottom-up classifier (switched off, or over max_bottom_up_bytes or "
                        "max_states): stacks are walked from the top\n");
    T.seconds_total = now() - t0;
    if (getenv("PSC_LOG"))
        fprintf(stderr, "psc: compile %.2f s: grammar+lexer+LALR %.2f s, token tries %.2f s, classifier %.2f s, "
                        "minimisation %.2f s, flatten %.2f s (mask rows %.2f s), bottom-up %.2f s\n",
                T.seconds_total, t1 - t0, t2 - t1, t3 - t2, t4 - t3, t7 - t4, t6 - t5, now() - t7);
    return T;
}

int classify_host(const Tables& t, int q, const uint16_t* stack, int depth, int status) {
    if (status == 1) return 1;
    if (status != 0) return 0;
    if (q < 0 || q >= t.nq) return 0;
    int32_t s = t.dfa_start[q];
    if (s < 0) return -s - 1;
    for (int i = depth - 1; i >= 0; i--) {
        int32_t nx = dfa_next(t, s, stack[i]);
        if (nx < 0) return -nx - 1;
        s = nx;
    }
    return t.dfa_mask[s];
}

}  // namespace psc
