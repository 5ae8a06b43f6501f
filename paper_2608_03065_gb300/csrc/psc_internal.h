// Internal data structures of the PSC library (host side).
//
// The compile step (psc_compile) turns a grammar and a vocabulary into flat
// tables: a byte-level lexer DFA (the lexing transducer of Section 2.2), LALR(1)
// ACTION/GOTO tables (the deterministic push-down automaton of Section 2.4), the
// stack classifier DFA built from every token's acceptance condition (Section
// 3.5, Eq. 9, Algorithm 1), and the deduplicated vocabulary mask of every
// classifier state (Section 3.5, the sets A_s).
#pragma once

#include <cstdint>
#include <stdexcept>
#include <string>
#include <vector>

namespace psc {

// status codes shared with include/psc.h
enum {
    ST_OK = 0, ST_ERR_ARG = 1, ST_ERR_GRAMMAR = 2, ST_ERR_CONFLICT = 3, ST_ERR_LEXER_AMBIGUOUS = 4,
    ST_ERR_LIMIT = 5, ST_ERR_OOM = 6, ST_ERR_CUDA = 7, ST_ERR_IO = 8
};

struct Error : std::runtime_error {
    int code;
    Error(int c, const std::string& m) : std::runtime_error(m), code(c) {}
};

// ---------------------------------------------------------------- grammar
struct Terminal {
    std::string name;      // display name; an anonymous literal is named by its quoted text
    bool literal = false;
    std::string pattern;   // literal bytes, or regex source
    int priority = 0;
    bool ignored = false;
};

struct Rule {
    int lhs;                // nonterminal index
    std::vector<int> rhs;   // symbol >= 0: terminal id; < 0: nonterminal ~index
};

struct Grammar {
    std::vector<Terminal> terms;
    std::vector<std::string> nts;
    std::vector<Rule> rules;
    int start_nt = -1;
    bool contextual = false;
};

Grammar parse_grammar(const std::string& text);
// rank[t]: order in which a lexeme matching several terminals prefers them
// (higher priority first, then byte-wise ascending display name)
std::vector<int> terminal_rank(const Grammar& g);

// ------------------------------------------------------------------ lexer
struct Lexer {
    int nq = 0, q0 = 0;                       // q0: the empty pending lexeme
    std::vector<int16_t> trans;               // [nq][256], -1: the byte ends the lexeme
    std::vector<int32_t> accept_cls;          // [nq], class of a complete lexeme or -1
    std::vector<std::vector<int>> classes;    // class id -> terminal ids in rank order
    std::vector<uint8_t> class_ignored;
    std::vector<std::vector<int>> tp;         // per state: T_p as class ids, -1 = empty sequence
};

Lexer build_lexer(const Grammar& g, const std::vector<int>& rank);

// ----------------------------------------------------------------- parser
enum { ACT_ERR = 0, ACT_SHIFT = 1, ACT_REDUCE = 2, ACT_ACCEPT = 3 };
inline int32_t act_make(int kind, int v) { return (int32_t)((v << 2) | kind); }
inline int act_kind(int32_t a) { return a & 3; }
inline int act_val(int32_t a) { return a >> 2; }

struct Parser {
    int n_states = 0, n_terms = 0, n_nts = 0, end_term = 0;   // n_terms includes the end marker
    std::vector<int32_t> action;      // [n_states][n_terms]
    std::vector<int32_t> go;          // [n_states][n_nts], -1 = none
    std::vector<int32_t> rule_len, rule_lhs;
    std::vector<uint8_t> term_entered;  // state is entered by shifting a terminal (or is state 0)
};

Parser build_lalr(const Grammar& g);

// ---------------------------------------------------------- compiled tables
struct Options {
    int64_t max_states = 4000000;     // classifier states before PSC_ERR_LIMIT
    int64_t max_mask_bytes = int64_t(24) << 30;
    int threads = 0;                  // 0 = hardware concurrency
    int64_t max_bottom_up_bytes = 0;  // construction memory of the bottom-up classifier
                                      // (0 = 16 GiB, at most half the memory; < 0 = not built;
                                      // over the limit: not built)
    int64_t max_dense_classifier_bytes = 0;  // dense classifier table above this: sparse layout
                                             // (0 = 512 MiB; < 0 = always sparse)
};

struct Tables {
    // lexer
    int nq = 0, q0 = 0;
    std::vector<int16_t> lex_trans;      // [nq][256]
    std::vector<int32_t> lex_accept;     // [nq]
    std::vector<uint8_t> cls_ignored;    // [n_classes]
    int n_classes = 0;
    // parser
    int n_lr = 0, n_terms = 0, n_nts = 0, end_term = 0;
    std::vector<int32_t> action, go, rule_len, rule_lhs;
    std::vector<int16_t> resolve;        // [n_classes][n_lr]: terminal a class stands for, -1 none
    bool contextual = false;
    // classifier DFA over (lexer state, stack read from the top), dense or sparse
    int S = 0;
    std::vector<int32_t> dfa;            // dense: [S][n_lr]: next state, or -(mask+1) when absorbing
    std::vector<int32_t> dfa_start;      // [nq]: first state after reading q (same encoding)
    std::vector<int32_t> dfa_mask;       // [S]: mask id when the stack ends in this state
    int dfa_sparse = 0;                  // 1: held as a default target and exceptions per state
    std::vector<int32_t> dfa_def;        // sparse: [S] default target (same encoding)
    std::vector<int64_t> dfa_exc_off;    // sparse: [S+1] range of the state's exceptions
    std::vector<uint16_t> dfa_exc_y;     // sparse: stack symbols whose target is not the default, ascending
    std::vector<int32_t> dfa_exc_t;      // sparse: their targets
    // masks: row 0 = nothing allowed, row 1 = only the end-of-sequence token.
    // A row is stored as nch = ceil(W/32) ids of 32-word chunks (1024 tokens each);
    // equal chunks are stored once (the table shrinks about tenfold on the C-like
    // workloads).  Words past W in a row's last chunk are zero.
    int V = 0, W = 0, n_masks = 0, nch = 0, n_chunks = 0;
    std::vector<uint32_t> mask_rows;     // [n_masks][nch] chunk ids
    std::vector<uint32_t> mask_chunks;   // [n_chunks][32]
    // bottom-up classifier (the same classification, reading the stack from the
    // bottom; empty when not built): blocks [F row, next block per successor slot],
    // slot of an LR edge t -> u, final mask ids [F row][nq], LR state of each block
    int bu_root = -1, n_bu = 0, n_frow = 0;
    std::vector<int32_t> bu;
    std::vector<int16_t> bu_slot;        // [n_lr][n_lr], -1: no edge
    std::vector<int32_t> bu_F;           // [n_frow][nq]
    std::vector<int32_t> bu_t;           // [n_bu] (host only: validation)
    // vocabulary
    std::vector<uint8_t> vocab_bytes;
    std::vector<int64_t> vocab_off;      // [V+1]
    int eos_id = -1;
    // statistics
    int64_t n_dfa_states_built = 0, n_threads = 0, n_trie_nodes = 0;
    double seconds_lex = 0, seconds_dfa = 0, seconds_min = 0, seconds_total = 0;
};

// Classifier transition from state s on stack symbol y (either layout).
inline int32_t dfa_next(const Tables& t, int32_t s, int y) {
    if (!t.dfa_sparse) return t.dfa[(size_t)s * t.n_lr + y];
    int64_t lo = t.dfa_exc_off[s], end = t.dfa_exc_off[s + 1], hi = end;
    while (lo < hi) {
        int64_t m = (lo + hi) >> 1;
        if (t.dfa_exc_y[m] < y) lo = m + 1;
        else hi = m;
    }
    return lo < end && t.dfa_exc_y[lo] == y ? t.dfa_exc_t[lo] : t.dfa_def[s];
}

// Word w of mask row m.
inline uint32_t mask_word(const Tables& t, int m, int w) {
    return t.mask_chunks[(size_t)t.mask_rows[(size_t)m * t.nch + (w >> 5)] * 32 + (w & 31)];
}

// Stores n dense mask rows of W words each (row m at rows + m * W) as chunk ids
// and distinct chunks (ids numbered in the order chunks are first met).
void set_mask_rows(Tables& t, const uint32_t* rows, int n, int W);

Tables compile_tables(const std::string& grammar, const uint8_t* vocab_bytes, const int64_t* offsets,
                      int V, int eos_id, const Options& opt);

// binary persistence of the flat tables (throws Error(ST_ERR_IO) on failure)
void save_tables(const Tables& t, const std::string& path);
Tables load_tables(const std::string& path);

// host-side walk of the flattened classifier (inspection / tests): mask id of (q, stack)
int classify_host(const Tables& t, int q, const uint16_t* stack, int depth, int status);

// Builds the bottom-up classifier tables from the forward classifier (false, and
// empty tables, when a size limit stops it).
bool build_bottom_up(Tables& t, const Options& opt);
// The same classification through the bottom-up tables; -2 when they are not
// built or the stack is not a path of the LR automaton.
int classify_host_bottom_up(const Tables& t, int q, const uint16_t* stack, int depth, int status);

}  // namespace psc
