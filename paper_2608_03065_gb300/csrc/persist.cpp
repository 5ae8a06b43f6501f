// Persistence of compiled tables.  The paper stores its preprocessing results
// on disk so that providers can ship them to decoding users (Section 5,
// preprocessing overhead); here the flat tables of a compiled handle are
// written as one binary file: a magic/version header, every table as
// (element count, raw little-endian bytes), and a 64-bit FNV-1a checksum of
// everything before it (format 03: with the bottom-up classifier's tables).
// The mask rows are stored as they are held in memory:
// chunk ids plus the distinct 1024-token chunks (no general-purpose compression;
// the paper uses zstd).
#include <cstdio>
#include <cstring>
#include <type_traits>

#include "psc_internal.h"

namespace psc {
namespace {

const char MAGIC[8] = {'P', 'S', 'C', 'T', 'A', 'B', '0', '3'};

struct Writer {
    FILE* f;
    uint64_t h = 1469598103934665603ull;
    void raw(const void* p, size_t n) {
        const uint8_t* b = static_cast<const uint8_t*>(p);
        for (size_t i = 0; i < n; i++) h = (h ^ b[i]) * 1099511628211ull;
        if (n && fwrite(p, 1, n, f) != n) throw Error(ST_ERR_IO, "write failed");
    }
    template <typename T>
    void scalar(T v) { raw(&v, sizeof(T)); }
    template <typename T>
    void vec(const std::vector<T>& v) {
        scalar<uint64_t>(v.size());
        raw(v.data(), v.size() * sizeof(T));
    }
};

struct Reader {
    FILE* f;
    uint64_t h = 1469598103934665603ull;
    void raw(void* p, size_t n) {
        if (n && fread(p, 1, n, f) != n) throw Error(ST_ERR_IO, "table file is truncated");
        const uint8_t* b = static_cast<const uint8_t*>(p);
        for (size_t i = 0; i < n; i++) h = (h ^ b[i]) * 1099511628211ull;
    }
    template <typename T>
    T scalar() {
        T v;
        raw(&v, sizeof(T));
        return v;
    }
    template <typename T>
    void vec(std::vector<T>& v, uint64_t limit = (uint64_t)1 << 36) {
        uint64_t n = scalar<uint64_t>();
        if (n > limit / sizeof(T)) throw Error(ST_ERR_IO, "table file has an implausible size field");
        v.resize(n);
        raw(v.data(), n * sizeof(T));
    }
};

template <typename S>
void fields(S& s, Tables& t) {
    // scalars
    auto sc = [&](auto& x) {
        using X = std::remove_reference_t<decltype(x)>;
        if constexpr (std::is_same_v<S, Writer>) s.template scalar<X>(x);
        else x = s.template scalar<X>();
    };
    auto vc = [&](auto& v) {
        if constexpr (std::is_same_v<S, Writer>) s.vec(v);
        else s.vec(v);
    };
    int32_t contextual = t.contextual ? 1 : 0;
    sc(t.nq); sc(t.q0); sc(t.n_classes); sc(t.n_lr); sc(t.n_terms); sc(t.n_nts); sc(t.end_term);
    sc(contextual); sc(t.S); sc(t.V); sc(t.W); sc(t.n_masks); sc(t.nch); sc(t.n_chunks); sc(t.eos_id);
    sc(t.n_dfa_states_built); sc(t.n_threads); sc(t.n_trie_nodes); sc(t.seconds_total);
    t.contextual = contextual != 0;
    vc(t.lex_trans); vc(t.lex_accept); vc(t.cls_ignored);
    vc(t.action); vc(t.go); vc(t.rule_len); vc(t.rule_lhs); vc(t.resolve);
    vc(t.dfa); vc(t.dfa_start); vc(t.dfa_mask); vc(t.mask_rows); vc(t.mask_chunks);
    vc(t.vocab_bytes); vc(t.vocab_off);
    sc(t.bu_root); sc(t.n_bu); sc(t.n_frow);
    vc(t.bu); vc(t.bu_slot); vc(t.bu_F); vc(t.bu_t);
}

void validate(const Tables& t) {
    auto bad = [](const char* what) { throw Error(ST_ERR_IO, std::string("table file is inconsistent: ") + what); };
    if (t.nq <= 0 || t.lex_trans.size() != (size_t)t.nq * 256 || t.lex_accept.size() != (size_t)t.nq) bad("lexer");
    if (t.q0 < 0 || t.q0 >= t.nq) bad("lexer start");
    if (t.n_lr <= 0 || t.action.size() != (size_t)t.n_lr * t.n_terms || t.go.size() != (size_t)t.n_lr * t.n_nts)
        bad("parser");
    if (t.resolve.size() != (size_t)t.n_classes * t.n_lr || t.cls_ignored.size() != (size_t)t.n_classes) bad("classes");
    if (t.dfa.size() != (size_t)t.S * t.n_lr || t.dfa_mask.size() != (size_t)t.S || t.dfa_start.size() != (size_t)t.nq)
        bad("classifier");
    if (t.W != (t.V + 31) / 32 || t.nch != (t.W + 31) / 32 || t.n_masks < 2 || t.n_chunks < 1 ||
        t.mask_rows.size() != (size_t)t.n_masks * t.nch || t.mask_chunks.size() != (size_t)t.n_chunks * 32)
        bad("masks");
    for (uint32_t c : t.mask_rows) if (c >= (uint32_t)t.n_chunks) bad("mask chunk id");
    if (t.vocab_off.size() != (size_t)t.V + 1 || (uint64_t)t.vocab_off[t.V] != t.vocab_bytes.size()) bad("vocabulary");
    for (int32_t x : t.lex_trans) if (x < -1 || x >= t.nq) bad("lexer transition");
    for (int32_t c : t.lex_accept) if (c < -1 || c >= t.n_classes) bad("lexer class");
    for (int32_t a : t.action) {
        int k = act_kind(a), v = act_val(a);
        if ((k == ACT_SHIFT && (v < 0 || v >= t.n_lr)) || (k == ACT_REDUCE && (v < 0 || v >= (int)t.rule_len.size())))
            bad("action");
    }
    for (int32_t g : t.go) if (g < -1 || g >= t.n_lr) bad("goto");
    for (size_t r = 0; r < t.rule_lhs.size(); r++)
        if (t.rule_lhs[r] < 0 || t.rule_lhs[r] >= t.n_nts || t.rule_len[r] < 0) bad("rule");
    for (int16_t x : t.resolve) if (x < -1 || x >= t.n_terms) bad("class resolution");
    auto state_ok = [&](int32_t s) { return s >= 0 ? s < t.S : (-s - 1) < t.n_masks; };
    for (int32_t s : t.dfa) if (!state_ok(s)) bad("classifier transition");
    for (int32_t s : t.dfa_start) if (!state_ok(s)) bad("classifier start");
    for (int32_t m : t.dfa_mask) if (m < 0 || m >= t.n_masks) bad("classifier mask id");
    if (t.eos_id < -1 || t.eos_id >= t.V) bad("end-of-sequence id");
    // bottom-up classifier: absent, or every block's successors are block starts
    if (t.bu_root < 0) {
        if (!t.bu.empty() || !t.bu_slot.empty() || !t.bu_F.empty() || !t.bu_t.empty() || t.n_bu || t.n_frow)
            bad("bottom-up classifier");
        return;
    }
    if (t.bu_slot.size() != (size_t)t.n_lr * t.n_lr || t.n_bu < 1 || t.bu_t.size() != (size_t)t.n_bu ||
        t.n_frow < 1 || t.bu_F.size() != (size_t)t.n_frow * t.nq)
        bad("bottom-up classifier");
    std::vector<int> deg(t.n_lr, 0);
    for (int a = 0; a < t.n_lr; a++)
        for (int u = 0; u < t.n_lr; u++) {
            int k = t.bu_slot[(size_t)a * t.n_lr + u];
            if (k < -1 || k >= t.n_lr) bad("bottom-up slot");
            if (k >= 0) deg[a]++;
        }
    for (int a = 0; a < t.n_lr; a++)   // slots of a state are 0 .. deg-1, each once
        for (int u = 0; u < t.n_lr; u++) {
            int k = t.bu_slot[(size_t)a * t.n_lr + u];
            if (k >= deg[a]) bad("bottom-up slot");
        }
    std::vector<uint8_t> is_base(t.bu.size() + 1, 0);
    size_t len = 0;
    for (int32_t r = 0; r < t.n_bu; r++) {
        if (t.bu_t[r] < 0 || t.bu_t[r] >= t.n_lr) bad("bottom-up state");
        if (len >= t.bu.size()) bad("bottom-up blocks");
        is_base[len] = 1;
        len += 1 + (size_t)deg[t.bu_t[r]];
    }
    if (len != t.bu.size() || t.bu_root != 0 || t.bu_t[0] != 0) bad("bottom-up blocks");
    len = 0;
    for (int32_t r = 0; r < t.n_bu; r++) {
        const int32_t* blk = t.bu.data() + len;
        if (blk[0] < 0 || blk[0] >= t.n_frow) bad("bottom-up row id");
        for (int k = 0; k < deg[t.bu_t[r]]; k++)
            if (blk[1 + k] < 0 || (size_t)blk[1 + k] >= t.bu.size() || !is_base[blk[1 + k]]) bad("bottom-up successor");
        len += 1 + (size_t)deg[t.bu_t[r]];
    }
    for (int32_t m : t.bu_F) if (m < 0 || m >= t.n_masks) bad("bottom-up mask id");
}

}  // namespace

void save_tables(const Tables& t, const std::string& path) {
    std::string tmp = path + ".tmp";
    FILE* f = fopen(tmp.c_str(), "wb");
    if (!f) throw Error(ST_ERR_IO, "cannot open " + tmp + " for writing");
    try {
        Writer w{f};
        w.raw(MAGIC, 8);
        Tables copy = t;   // fields() takes a mutable reference
        fields(w, copy);
        uint64_t h = w.h;
        if (fwrite(&h, 8, 1, f) != 1) throw Error(ST_ERR_IO, "write failed");
        if (fclose(f) != 0) throw Error(ST_ERR_IO, "close failed");
    } catch (...) {
        fclose(f);
        remove(tmp.c_str());
        throw;
    }
    if (rename(tmp.c_str(), path.c_str()) != 0) throw Error(ST_ERR_IO, "cannot rename " + tmp + " to " + path);
}

Tables load_tables(const std::string& path) {
    FILE* f = fopen(path.c_str(), "rb");
    if (!f) throw Error(ST_ERR_IO, "cannot open " + path);
    Tables t;
    try {
        Reader r{f};
        char magic[8];
        r.raw(magic, 8);
        if (memcmp(magic, MAGIC, 8) != 0) throw Error(ST_ERR_IO, path + " is not a PSC table file");
        fields(r, t);
        uint64_t want = r.h, got = 0;
        if (fread(&got, 8, 1, f) != 1 || got != want) throw Error(ST_ERR_IO, path + ": checksum mismatch");
        fclose(f);
    } catch (...) {
        fclose(f);
        throw;
    }
    validate(t);
    return t;
}

}  // namespace psc
