// Persistence of compiled tables.  The paper stores its preprocessing results
// on disk, zstd-compressed, so that providers can ship them to decoding users
// (Section 5, preprocessing overhead); here the flat tables of a compiled handle
// are written as one file (format 04):
//   "PSCTAB04", codec (u32: 0 none, 1 zstd, 2 zlib), reserved (u32),
//   size of the table payload (u64), number of blocks (u64),
//   per block: payload bytes and stored bytes (u64 each), then the blocks,
//   then a 64-bit FNV-1a checksum of the payload.
// The payload lists every table as (element count, raw little-endian bytes).
// Blocks of 16 MiB of payload are compressed and decompressed in parallel.  The
// compressor is the system's zstd library (libzstd.so.1) when it can be loaded,
// else zlib (libz.so.1), else none: both are loaded at run time through their
// stable C interfaces, so the library does not depend on them to link or run; a
// file needs the codec it was written with to be read.  The environment variable
// PSC_SAVE_CODEC (none, zstd or zlib) overrides the choice.
#include <dlfcn.h>

#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <thread>
#include <type_traits>

#include "psc_internal.h"

namespace psc {
namespace {

const char MAGIC[8] = {'P', 'S', 'C', 'T', 'A', 'B', '0', '4'};
constexpr size_t BLOCK = size_t(16) << 20;
enum { CODEC_NONE = 0, CODEC_ZSTD = 1, CODEC_ZLIB = 2 };

// ------------------------------------------------------------------ codecs
struct Codecs {
    // zstd
    size_t (*zstd_bound)(size_t) = nullptr;
    size_t (*zstd_compress)(void*, size_t, const void*, size_t, int) = nullptr;
    size_t (*zstd_decompress)(void*, size_t, const void*, size_t) = nullptr;
    unsigned (*zstd_is_error)(size_t) = nullptr;
    // zlib (uLong = unsigned long, Bytef = unsigned char)
    unsigned long (*z_bound)(unsigned long) = nullptr;
    int (*z_compress2)(unsigned char*, unsigned long*, const unsigned char*, unsigned long, int) = nullptr;
    int (*z_uncompress)(unsigned char*, unsigned long*, const unsigned char*, unsigned long) = nullptr;
    bool zstd() const { return zstd_bound && zstd_compress && zstd_decompress && zstd_is_error; }
    bool zlib() const { return z_bound && z_compress2 && z_uncompress; }
};

const Codecs& codecs() {
    static Codecs c;
    static std::once_flag once;
    std::call_once(once, [] {
        if (void* z = dlopen("libzstd.so.1", RTLD_NOW | RTLD_LOCAL)) {
            c.zstd_bound = reinterpret_cast<size_t (*)(size_t)>(dlsym(z, "ZSTD_compressBound"));
            c.zstd_compress = reinterpret_cast<size_t (*)(void*, size_t, const void*, size_t, int)>(dlsym(z, "ZSTD_compress"));
            c.zstd_decompress = reinterpret_cast<size_t (*)(void*, size_t, const void*, size_t)>(dlsym(z, "ZSTD_decompress"));
            c.zstd_is_error = reinterpret_cast<unsigned (*)(size_t)>(dlsym(z, "ZSTD_isError"));
        }
        if (void* z = dlopen("libz.so.1", RTLD_NOW | RTLD_LOCAL)) {
            c.z_bound = reinterpret_cast<unsigned long (*)(unsigned long)>(dlsym(z, "compressBound"));
            c.z_compress2 = reinterpret_cast<int (*)(unsigned char*, unsigned long*, const unsigned char*,
                                                     unsigned long, int)>(dlsym(z, "compress2"));
            c.z_uncompress = reinterpret_cast<int (*)(unsigned char*, unsigned long*, const unsigned char*,
                                                      unsigned long)>(dlsym(z, "uncompress"));
        }
    });
    return c;
}

// compresses src into dst (resized); false when the codec fails
bool encode(int codec, const uint8_t* src, size_t n, std::vector<uint8_t>& dst) {
    const Codecs& c = codecs();
    if (codec == CODEC_ZSTD) {
        dst.resize(c.zstd_bound(n));
        size_t r = c.zstd_compress(dst.data(), dst.size(), src, n, 9);
        if (c.zstd_is_error(r)) return false;
        dst.resize(r);
        return true;
    }
    unsigned long cap = c.z_bound((unsigned long)n);
    dst.resize(cap);
    if (c.z_compress2(dst.data(), &cap, src, (unsigned long)n, 6) != 0) return false;
    dst.resize(cap);
    return true;
}

bool decode(int codec, const uint8_t* src, size_t n, uint8_t* dst, size_t want) {
    const Codecs& c = codecs();
    if (codec == CODEC_ZSTD) {
        size_t r = c.zstd_decompress(dst, want, src, n);
        return !c.zstd_is_error(r) && r == want;
    }
    unsigned long got = (unsigned long)want;
    return c.z_uncompress(dst, &got, src, (unsigned long)n) == 0 && got == want;
}

// runs f(i) for i in [0, n) on up to hardware-concurrency threads
template <typename F>
void parallel_for(size_t n, F f) {
    size_t nt = std::min<size_t>(n, std::max(1u, std::thread::hardware_concurrency()));
    std::vector<std::thread> pool;
    std::mutex mu;
    size_t next = 0;
    for (size_t t = 0; t < nt; t++)
        pool.emplace_back([&] {
            for (;;) {
                size_t i;
                {
                    std::lock_guard<std::mutex> lk(mu);
                    if (next >= n) return;
                    i = next++;
                }
                f(i);
            }
        });
    for (auto& th : pool) th.join();
}

uint64_t fnv1a(const uint8_t* b, size_t n) {
    uint64_t h = 1469598103934665603ull;
    for (size_t i = 0; i < n; i++) h = (h ^ b[i]) * 1099511628211ull;
    return h;
}

// ------------------------------------------------------- payload (de)coding
struct Writer {
    std::vector<uint8_t> out;
    void raw(const void* p, size_t n) {
        const uint8_t* b = static_cast<const uint8_t*>(p);
        out.insert(out.end(), b, b + n);
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
    const uint8_t* p;
    size_t n, pos = 0;
    void raw(void* dst, size_t k) {
        if (k > n - pos) throw Error(ST_ERR_IO, "table file is truncated");
        std::memcpy(dst, p + pos, k);
        pos += k;
    }
    template <typename T>
    T scalar() {
        T v;
        raw(&v, sizeof(T));
        return v;
    }
    template <typename T>
    void vec(std::vector<T>& v) {
        uint64_t k = scalar<uint64_t>();
        if (k > (n - pos) / sizeof(T)) throw Error(ST_ERR_IO, "table file has an implausible size field");
        v.resize(k);
        raw(v.data(), k * sizeof(T));
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
    sc(t.dfa_sparse); vc(t.dfa_def); vc(t.dfa_exc_off); vc(t.dfa_exc_y); vc(t.dfa_exc_t);
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
    if (t.dfa_mask.size() != (size_t)t.S || t.dfa_start.size() != (size_t)t.nq) bad("classifier");
    if (t.dfa_sparse == 0) {
        if (t.dfa.size() != (size_t)t.S * t.n_lr || !t.dfa_def.empty() || !t.dfa_exc_off.empty() ||
            !t.dfa_exc_y.empty() || !t.dfa_exc_t.empty())
            bad("classifier");
    } else {
        if (t.dfa_sparse != 1 || !t.dfa.empty() || t.dfa_def.size() != (size_t)t.S ||
            t.dfa_exc_off.size() != (size_t)t.S + 1 || t.dfa_exc_off[0] != 0 ||
            (uint64_t)t.dfa_exc_off[t.S] != t.dfa_exc_y.size() || t.dfa_exc_t.size() != t.dfa_exc_y.size())
            bad("sparse classifier");
        for (int s = 0; s < t.S; s++) {
            if (t.dfa_exc_off[s + 1] < t.dfa_exc_off[s]) bad("sparse classifier");
            for (int64_t e = t.dfa_exc_off[s]; e < t.dfa_exc_off[s + 1]; e++)
                if (t.dfa_exc_y[e] >= t.n_lr || (e > t.dfa_exc_off[s] && t.dfa_exc_y[e] <= t.dfa_exc_y[e - 1]))
                    bad("sparse classifier symbols");
        }
    }
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
    for (int32_t s : t.dfa_def) if (!state_ok(s)) bad("classifier transition");
    for (int32_t s : t.dfa_exc_t) if (!state_ok(s)) bad("classifier transition");
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
    Writer w;
    Tables copy = t;   // fields() takes a mutable reference
    fields(w, copy);
    const std::vector<uint8_t>& payload = w.out;
    const Codecs& c = codecs();
    int codec = c.zstd() ? CODEC_ZSTD : c.zlib() ? CODEC_ZLIB : CODEC_NONE;
    if (const char* want = getenv("PSC_SAVE_CODEC")) {   // none | zstd | zlib (if it can be loaded)
        if (!strcmp(want, "none")) codec = CODEC_NONE;
        else if (!strcmp(want, "zlib") && c.zlib()) codec = CODEC_ZLIB;
        else if (!strcmp(want, "zstd") && c.zstd()) codec = CODEC_ZSTD;
    }
    size_t nb = (payload.size() + BLOCK - 1) / BLOCK;
    std::vector<std::vector<uint8_t>> blocks(nb);
    if (codec != CODEC_NONE) {
        std::vector<char> ok(nb, 1);
        parallel_for(nb, [&](size_t i) {
            size_t lo = i * BLOCK, n = std::min(BLOCK, payload.size() - lo);
            ok[i] = encode(codec, payload.data() + lo, n, blocks[i]);
        });
        for (char k : ok)
            if (!k) throw Error(ST_ERR_IO, "compressing the tables failed");
    }
    std::string tmp = path + ".tmp";
    FILE* f = fopen(tmp.c_str(), "wb");
    if (!f) throw Error(ST_ERR_IO, "cannot open " + tmp + " for writing");
    auto put = [&](const void* p, size_t n) {
        if (n && fwrite(p, 1, n, f) != n) throw Error(ST_ERR_IO, "write failed");
    };
    try {
        uint32_t hdr[2] = {(uint32_t)codec, 0};
        uint64_t sizes[2] = {payload.size(), nb};
        put(MAGIC, 8);
        put(hdr, sizeof(hdr));
        put(sizes, sizeof(sizes));
        for (size_t i = 0; i < nb; i++) {
            uint64_t raw = std::min(BLOCK, payload.size() - i * BLOCK);
            uint64_t stored = codec == CODEC_NONE ? raw : blocks[i].size();
            put(&raw, 8);
            put(&stored, 8);
        }
        for (size_t i = 0; i < nb; i++) {
            if (codec == CODEC_NONE) put(payload.data() + i * BLOCK, std::min(BLOCK, payload.size() - i * BLOCK));
            else put(blocks[i].data(), blocks[i].size());
        }
        uint64_t h = fnv1a(payload.data(), payload.size());
        put(&h, 8);
        if (fclose(f) != 0) {
            f = nullptr;
            throw Error(ST_ERR_IO, "close failed");
        }
        f = nullptr;
    } catch (...) {
        if (f) fclose(f);
        remove(tmp.c_str());
        throw;
    }
    if (rename(tmp.c_str(), path.c_str()) != 0) throw Error(ST_ERR_IO, "cannot rename " + tmp + " to " + path);
}

Tables load_tables(const std::string& path) {
    FILE* f = fopen(path.c_str(), "rb");
    if (!f) throw Error(ST_ERR_IO, "cannot open " + path);
    std::vector<uint8_t> payload;
    try {
        auto get = [&](void* p, size_t n) {
            if (n && fread(p, 1, n, f) != n) throw Error(ST_ERR_IO, path + ": table file is truncated");
        };
        char magic[8];
        get(magic, 8);
        if (memcmp(magic, MAGIC, 8) != 0) throw Error(ST_ERR_IO, path + " is not a PSC table file (format 04)");
        uint32_t hdr[2];
        uint64_t sizes[2];
        get(hdr, sizeof(hdr));
        get(sizes, sizeof(sizes));
        int codec = (int)hdr[0];
        uint64_t total = sizes[0], nb = sizes[1];
        if (codec > CODEC_ZLIB || total > (uint64_t(1) << 40) || nb != (total + BLOCK - 1) / BLOCK)
            throw Error(ST_ERR_IO, path + ": bad table file header");
        if ((codec == CODEC_ZSTD && !codecs().zstd()) || (codec == CODEC_ZLIB && !codecs().zlib()))
            throw Error(ST_ERR_IO, path + std::string(": written with ") + (codec == CODEC_ZSTD ? "zstd" : "zlib") +
                                       ", which cannot be loaded on this host");
        std::vector<uint64_t> raw(nb), stored(nb);
        for (uint64_t i = 0; i < nb; i++) {
            get(&raw[i], 8);
            get(&stored[i], 8);
            if (raw[i] != std::min<uint64_t>(BLOCK, total - i * BLOCK) || stored[i] > (uint64_t(1) << 32))
                throw Error(ST_ERR_IO, path + ": bad block size");
        }
        std::vector<std::vector<uint8_t>> blocks(nb);
        for (uint64_t i = 0; i < nb; i++) {
            blocks[i].resize(stored[i]);
            get(blocks[i].data(), stored[i]);
        }
        uint64_t want = 0;
        get(&want, 8);
        payload.resize(total);
        std::vector<char> ok(nb, 1);
        parallel_for(nb, [&](size_t i) {
            uint8_t* dst = payload.data() + i * BLOCK;
            if (codec == CODEC_NONE) {
                if (stored[i] != raw[i]) ok[i] = 0;
                else std::memcpy(dst, blocks[i].data(), raw[i]);
            } else {
                ok[i] = decode(codec, blocks[i].data(), blocks[i].size(), dst, raw[i]);
            }
            std::vector<uint8_t>().swap(blocks[i]);
        });
        for (char k : ok)
            if (!k) throw Error(ST_ERR_IO, path + ": a block does not decompress");
        if (fnv1a(payload.data(), payload.size()) != want) throw Error(ST_ERR_IO, path + ": checksum mismatch");
        fclose(f);
    } catch (...) {
        fclose(f);
        throw;
    }
    Tables t;
    Reader r{payload.data(), payload.size()};
    fields(r, t);
    if (r.pos != r.n) throw Error(ST_ERR_IO, path + ": trailing bytes in the table payload");
    validate(t);
    return t;
}

}  // namespace psc
