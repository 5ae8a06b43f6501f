// Bottom-up stack classifier: the classifier of Eq. (9) turned around so that
// it reads the parser stack from the bottom, with its state after every stack
// prefix kept per row.  A decode step that pops the stack to depth d and then
// pushes k states re-reads only those k states (plus one lookup by the lexer
// state), instead of walking the stack from the top (Algorithm 2 step 3,
// O(|stack|) per step).
//
// Why it exists: the set of (lexer state, stack) pairs that select a given mask
// is regular (the regularity theorem of Section 3.5), and regular languages are
// closed under reversal, so a deterministic automaton reading q·α_top…α_bottom
// backwards exists.  It is built here from the forward classifier DFA `dfa`:
//
//   g_α(s) = mask id the forward walk reaches when it starts in forward state s
//            and reads α from the top down (the stack's bottom is always LR
//            state 0; a walk that reads the whole stack ends with dfa_mask[s]).
//
// g_α·u (u pushed on top of α) is g_α composed with one forward step on u:
// g_α·u(s) = mask of the absorbing step when dfa[s][u] absorbs, else
// g_α(dfa[s][u]).  The mask of a configuration (q, α) is g_α(dfa_start[q]).  A
// bottom-up state is a distinct pair (top LR state t, g restricted to D(t)),
// where D(t) is the set of forward states that can be about to read an entry t
// (found by propagating from the start states down the LR automaton's edges);
// only stacks that are paths of the LR automaton (every entry a shift or goto
// successor of the one below it, which every parser stack is) are explored.
//
// Device layout: one int32 array of blocks, a block per bottom-up state:
//   [F row id, next block for successor slot 0, slot 1, ...]
// slot[t][u] = index of u among t's successors (-1: not an LR edge); the final
// table F[row][q] holds the mask id of every lexer state.
#include <algorithm>
#include <atomic>
#include <chrono>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <thread>
#include <unordered_map>

#include <unistd.h>

#include "psc_internal.h"

namespace psc {
namespace {

uint64_t mix(uint64_t h) {
    h ^= h >> 33;
    h *= 0xff51afd7ed558ccdull;
    h ^= h >> 33;
    h *= 0xc4ceb9fe1a85ec53ull;
    h ^= h >> 33;
    return h;
}

template <typename G>
uint64_t hash_state(int t, const G* g, size_t n) {
    uint64_t h = mix(0x9e3779b97f4a7c15ull ^ (uint64_t)t);
    for (size_t i = 0; i < n; i++) h = mix(h ^ ((uint64_t)(uint32_t)g[i] << 1) ^ i);
    return h;
}

template <typename F>
void parallel_for(int threads, size_t n, F&& f) {
    if (threads <= 1 || n < 2) {
        for (size_t i = 0; i < n; i++) f(i);
        return;
    }
    std::atomic<size_t> next{0};
    std::vector<std::thread> pool;
    int nt = (int)std::min<size_t>((size_t)threads, n);
    for (int k = 0; k < nt; k++)
        pool.emplace_back([&]() {
            for (;;) {
                size_t i = next.fetch_add(1);
                if (i >= n) break;
                f(i);
            }
        });
    for (auto& th : pool) th.join();
}

double seconds() {
    return std::chrono::duration<double>(std::chrono::steady_clock::now().time_since_epoch()).count();
}

// G: the element type of the g vectors (mask ids): uint16_t when every mask id
// fits, which halves the construction's memory, else int32_t.
template <typename G>
bool build_bottom_up_g(Tables& T, const Options& opt) {
    T.bu.clear();
    T.bu_slot.clear();
    T.bu_F.clear();
    T.bu_t.clear();
    T.bu_root = -1;
    T.n_bu = 0;
    T.n_frow = 0;
    if (opt.max_bottom_up_bytes < 0) return false;
    // default budget: 16 GiB, at most half of the machine's memory
    int64_t dflt = int64_t(16) << 30;
    long pages = sysconf(_SC_PHYS_PAGES), psize = sysconf(_SC_PAGESIZE);
    if (pages > 0 && psize > 0) dflt = std::min<int64_t>(dflt, (int64_t)pages * psize / 2);
    const int64_t budget = opt.max_bottom_up_bytes > 0 ? opt.max_bottom_up_bytes : dflt;
    const int n = T.n_lr, S = T.S, nq = T.nq;
    if (n <= 0 || n > 32767 || (int64_t)n * n * 2 > (int64_t(64) << 20)) return false;
    int threads = opt.threads > 0 ? opt.threads : (int)std::max(1u, std::thread::hardware_concurrency());
    const bool log = getenv("PSC_LOG") != nullptr;
    double t0 = seconds();

    // LR automaton edges: t -> u when u is entered from t by a shift or a goto
    std::vector<std::vector<int32_t>> succ(n), pred(n);
    for (int t = 0; t < n; t++) {
        for (int a = 0; a < T.n_terms; a++) {
            int32_t x = T.action[(size_t)t * T.n_terms + a];
            if (act_kind(x) == ACT_SHIFT) succ[t].push_back(act_val(x));
        }
        for (int nt = 0; nt < T.n_nts; nt++) {
            int32_t g = T.go[(size_t)t * T.n_nts + nt];
            if (g >= 0) succ[t].push_back(g);
        }
        std::sort(succ[t].begin(), succ[t].end());
        succ[t].erase(std::unique(succ[t].begin(), succ[t].end()), succ[t].end());
        for (int32_t u : succ[t]) pred[u].push_back(t);   // pred[u] ends up sorted by t
    }
    std::vector<int16_t> slot((size_t)n * n, -1);
    for (int t = 0; t < n; t++)
        for (size_t k = 0; k < succ[t].size(); k++) slot[(size_t)t * n + succ[t][k]] = (int16_t)k;

    // D(t) as bitsets over forward states, with per-word prefix counts for ranks
    const size_t words = ((size_t)S + 63) / 64;
    if ((int64_t)(n * words * 12) > budget) return false;
    std::vector<uint64_t> bits((size_t)n * words, 0);
    auto has = [&](int t, int32_t s) { return (bits[(size_t)t * words + (s >> 6)] >> (s & 63)) & 1; };
    auto add = [&](int t, int32_t s) { bits[(size_t)t * words + (s >> 6)] |= 1ull << (s & 63); };
    std::vector<int32_t> starts;
    for (int q = 0; q < nq; q++)
        if (T.dfa_start[q] >= 0) starts.push_back(T.dfa_start[q]);
    std::sort(starts.begin(), starts.end());
    starts.erase(std::unique(starts.begin(), starts.end()), starts.end());
    std::vector<std::pair<int32_t, int32_t>> work;   // (forward state, LR entry it is about to read)
    for (int t = 0; t < n; t++)
        for (int32_t s : starts) {
            add(t, s);
            work.push_back({s, t});
        }
    while (!work.empty()) {
        auto [s, t] = work.back();
        work.pop_back();
        int32_t nx = dfa_next(T, s, t);
        if (nx < 0) continue;
        for (int32_t u : pred[t])
            if (!has(u, nx)) {
                add(u, nx);
                work.push_back({nx, u});
            }
    }
    std::vector<uint32_t> prefix((size_t)n * words + 1, 0);
    std::vector<std::vector<int32_t>> D(n);
    for (int t = 0; t < n; t++) {
        uint32_t c = 0;
        for (size_t w = 0; w < words; w++) {
            prefix[(size_t)t * words + w] = c;
            uint64_t x = bits[(size_t)t * words + w];
            c += (uint32_t)__builtin_popcountll(x);
            while (x) {
                int b = __builtin_ctzll(x);
                D[t].push_back((int32_t)(w * 64 + b));
                x &= x - 1;
            }
        }
    }
    auto rank = [&](int t, int32_t s) -> int32_t {
        size_t w = (size_t)t * words + (s >> 6);
        uint64_t below = bits[w] & ((1ull << (s & 63)) - 1);
        return (int32_t)(prefix[w] + (uint32_t)__builtin_popcountll(below));
    };

    double t1 = seconds();
    // one forward step per LR edge t -> u, as a map from D(u) to D(t) (or a final mask)
    std::vector<std::vector<int32_t>> step(n);   // step[u] holds the edges into u, one after the other
    std::vector<std::vector<int64_t>> step_off(n);
    int64_t step_bytes = 0;
    for (int u = 0; u < n; u++) {
        step_off[u].push_back(0);
        for (int32_t t : pred[u]) {
            for (int32_t s : D[u]) {
                int32_t nx = dfa_next(T, s, u);
                step[u].push_back(nx < 0 ? nx : rank(t, nx));   // nx < 0: -(mask + 1)
            }
            step_off[u].push_back((int64_t)step[u].size());
        }
        step_bytes += (int64_t)step[u].size() * 4;
        if (step_bytes > budget) return false;
    }
    auto pred_index = [&](int u, int t) {
        return (int)(std::lower_bound(pred[u].begin(), pred[u].end(), t) - pred[u].begin());
    };

    double t2 = seconds();
    // breadth-first construction of the distinct (t, g) pairs.  The g vectors live
    // in one growing block (realloc moves large blocks by remapping, not copying);
    // new states of a batch are numbered serially and copied in parallel.
    struct Arena {
        G* p = nullptr;
        size_t n = 0, cap = 0;
        ~Arena() { free(p); }
        bool grow(size_t need) {
            if (need <= cap) return true;
            size_t c = std::max(need, std::max<size_t>(cap * 2, (size_t)1 << 24));
            void* q = realloc(p, c * sizeof(G));
            if (!q) return false;
            p = static_cast<G*>(q);
            cap = c;
            return true;
        }
    } arena;
    std::vector<int64_t> g_off;           // per state
    std::vector<int32_t> st_t;            // per state: top LR state
    std::vector<int64_t> tr_off;          // per state: first successor id in tr
    std::vector<int32_t> tr;              // successor state ids, |succ(t)| per state
    std::unordered_multimap<uint64_t, int32_t> index;
    auto new_state = [&](int t, uint64_t h) -> int32_t {
        int32_t r = (int32_t)st_t.size();
        g_off.push_back((int64_t)arena.n);
        arena.n += D[t].size();
        st_t.push_back(t);
        tr_off.push_back((int64_t)tr.size());
        tr.insert(tr.end(), succ[t].size(), -1);
        index.emplace(h, r);
        return r;
    };
    {
        std::vector<G> g0(D[0].size());
        for (size_t i = 0; i < D[0].size(); i++) {
            int32_t nx = dfa_next(T, D[0][i], 0);
            g0[i] = (G)(nx < 0 ? -nx - 1 : T.dfa_mask[nx]);
        }
        new_state(0, hash_state(0, g0.data(), g0.size()));
        if (!arena.grow(arena.n)) return false;
        std::memcpy(arena.p, g0.data(), g0.size() * sizeof(G));
    }
    double t_par = 0, t_ser = 0;
    int n_batches = 0;
    std::vector<int32_t> frontier{0}, next;
    struct Cand {
        int32_t from, k, u;
        int64_t off;
        uint64_t h;
        int32_t found;
    };
    std::vector<Cand> cands;
    std::vector<G> buf;
    std::vector<std::pair<int32_t, int64_t>> fresh;   // (new state, its vector's offset in buf)
    const int64_t batch_bytes = std::min<int64_t>(budget / 8, int64_t(256) << 20);
    while (!frontier.empty()) {
        next.clear();
        size_t i0 = 0;
        while (i0 < frontier.size()) {
            // a batch of frontier states whose candidate vectors fit the batch budget
            cands.clear();
            int64_t total = 0;
            size_t i1 = i0;
            while (i1 < frontier.size() && (i1 == i0 || total * 4 < batch_bytes)) {
                int32_t r = frontier[i1++];
                int t = st_t[r];
                for (size_t k = 0; k < succ[t].size(); k++) {
                    int u = succ[t][k];
                    cands.push_back({r, (int32_t)k, u, total, 0, -1});
                    total += (int64_t)D[u].size();
                }
            }
            buf.resize((size_t)total);
            double tp = seconds();
            parallel_for(threads, cands.size(), [&](size_t ci) {
                Cand& c = cands[ci];
                int t = st_t[c.from];
                const G* g = arena.p + g_off[c.from];
                int pi = pred_index(c.u, t);
                const int32_t* sp = step[c.u].data() + step_off[c.u][pi];
                G* out = buf.data() + c.off;
                size_t m = D[c.u].size();
                for (size_t j = 0; j < m; j++) {
                    int32_t x = sp[j];
                    out[j] = x < 0 ? (G)(-x - 1) : g[x];
                }
                c.h = hash_state(c.u, out, m);
                auto range = index.equal_range(c.h);   // read-only while the batch runs
                for (auto it = range.first; it != range.second; ++it) {
                    int32_t r = it->second;
                    if (st_t[r] == c.u && !memcmp(arena.p + g_off[r], out, m * sizeof(G))) {
                        c.found = r;
                        break;
                    }
                }
            });
            t_par += seconds() - tp;
            tp = seconds();
            // number the batch's new states (equal candidates of one batch compared in buf)
            fresh.clear();
            int32_t first_new = (int32_t)st_t.size();
            for (Cand& c : cands) {
                int32_t r = c.found;
                if (r < 0) {
                    size_t m = D[c.u].size();
                    auto range = index.equal_range(c.h);
                    for (auto it = range.first; it != range.second && r < 0; ++it) {
                        int32_t x = it->second;
                        if (x < first_new || st_t[x] != c.u) continue;   // older states were checked above
                        if (!memcmp(buf.data() + fresh[x - first_new].second, buf.data() + c.off, m * sizeof(G)))
                            r = x;
                    }
                    if (r < 0) {
                        r = new_state(c.u, c.h);
                        fresh.push_back({r, c.off});
                        next.push_back(r);
                    }
                }
                tr[tr_off[c.from] + c.k] = r;
            }
            if ((int64_t)(arena.n * sizeof(G)) + (int64_t)tr.size() * 4 + step_bytes > budget ||
                (int64_t)st_t.size() > opt.max_states || !arena.grow(arena.n)) {
                if (log)
                    fprintf(stderr, "psc: bottom-up classifier given up at %zu states, %.2f GiB of %.2f GiB\n",
                            st_t.size(),
                            ((double)arena.n * sizeof(G) + (double)tr.size() * 4 + (double)step_bytes) / (1 << 30),
                            (double)budget / (1 << 30));
                return false;
            }
            parallel_for(threads, fresh.size(), [&](size_t i) {
                int32_t r = fresh[i].first;
                std::memcpy(arena.p + g_off[r], buf.data() + fresh[i].second, D[st_t[r]].size() * sizeof(G));
            });
            t_ser += seconds() - tp;
            n_batches++;
            i0 = i1;
        }
        frontier.swap(next);
    }

    double t3 = seconds();
    // final table: the mask id of every lexer state, per state; equal rows stored once
    int32_t R = (int32_t)st_t.size();
    std::vector<int32_t> frow(R);
    std::vector<int32_t> F;
    {
        std::unordered_multimap<uint64_t, int32_t> fidx;
        std::vector<int32_t> row(nq);
        for (int32_t r = 0; r < R; r++) {
            int t = st_t[r];
            const G* g = arena.p + g_off[r];
            for (int q = 0; q < nq; q++) {
                int32_t s = T.dfa_start[q];
                row[q] = s < 0 ? -s - 1 : g[rank(t, s)];
            }
            uint64_t h = hash_state(-1, row.data(), nq);
            int32_t found = -1;
            auto range = fidx.equal_range(h);
            for (auto it = range.first; it != range.second; ++it)
                if (!memcmp(F.data() + (size_t)it->second * nq, row.data(), (size_t)nq * 4)) {
                    found = it->second;
                    break;
                }
            if (found < 0) {
                found = (int32_t)(F.size() / nq);
                F.insert(F.end(), row.begin(), row.end());
                fidx.emplace(h, found);
            }
            frow[r] = found;
        }
    }
    // blocks
    std::vector<int64_t> base(R);
    int64_t len = 0;
    for (int32_t r = 0; r < R; r++) {
        base[r] = len;
        len += 1 + (int64_t)succ[st_t[r]].size();
    }
    if (len >= (int64_t(1) << 31)) return false;
    T.bu.assign((size_t)len, 0);
    for (int32_t r = 0; r < R; r++) {
        int32_t* blk = T.bu.data() + base[r];
        blk[0] = frow[r];
        for (size_t k = 0; k < succ[st_t[r]].size(); k++) blk[1 + k] = (int32_t)base[tr[tr_off[r] + k]];
    }
    T.bu_slot = std::move(slot);
    T.bu_F = std::move(F);
    T.bu_t = std::move(st_t);
    T.bu_root = 0;
    T.n_bu = R;
    T.n_frow = (int)(T.bu_F.size() / nq);
    if (log)
        fprintf(stderr, "psc: bottom-up classifier: %d states, %d final rows, %.2f GiB of construction vectors; "
                        "domains %.2f s, steps %.2f s, states %.2f s (%d batches: parallel %.2f s, serial %.2f s), "
                        "final %.2f s\n",
                R, T.n_frow, ((double)arena.n * sizeof(G) + (double)tr.size() * 4 + (double)step_bytes) / (1 << 30),
                t1 - t0, t2 - t1, t3 - t2, n_batches, t_par, t_ser, seconds() - t3);
    return true;
}

}  // namespace

int classify_host_bottom_up(const Tables& t, int q, const uint16_t* stack, int depth, int status) {
    if (status == 1) return 1;
    if (status != 0) return 0;
    if (t.bu_root < 0) return -2;
    if (q < 0 || q >= t.nq || depth < 1 || stack[0] != 0) return -2;
    int64_t e = t.bu_root;
    for (int i = 1; i < depth; i++) {
        if (stack[i - 1] >= t.n_lr || stack[i] >= t.n_lr) return -2;
        int k = t.bu_slot[(size_t)stack[i - 1] * t.n_lr + stack[i]];
        if (k < 0) return -2;   // not an edge of the LR automaton: no parser builds this stack
        e = t.bu[(size_t)e + 1 + k];
    }
    return t.bu_F[(size_t)t.bu[(size_t)e] * t.nq + q];
}

bool build_bottom_up(Tables& T, const Options& opt) {
    return T.n_masks < 65536 ? build_bottom_up_g<uint16_t>(T, opt) : build_bottom_up_g<int32_t>(T, opt);
}

}  // namespace psc
