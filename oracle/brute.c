/*
 * Oracle brute force for the PSC vocabulary mask (test infrastructure only).
 *
 * This file is part of the CPU oracle.  Only the tests, __graft_entry__.smoke()
 * and the CPU-baseline leg of bench.py may load it.  It shares no code with the
 * CUDA path: it reads the oracle's own Thompson NFA (oracle/regex_thompson.py)
 * and canonical LR(1) tables (oracle/lr1_canonical.py).
 *
 * What it computes is the mask of Eq. (1) rewritten as Eq. (3): token v is
 * allowed after prefix x iff some realizable terminal sequence w in R_q(v)
 * (Section 3.1: the terminals emitted while lexing v from the lexer state q,
 * followed by one element of T_p, the finite set of terminal prefixes the
 * pending lexeme p can still become) takes the parser from the current stack to
 * a stable stack.  It does this the slow way: for every row and every token it
 * lexes the token's bytes and simulates the LR(1) parser on a copy-on-write view
 * of the row's stack: the scheme that runs the parser once per token, which the
 * paper sets against PSC (Fig. 1b).
 *
 * Lexer reading (the paper defers its lexer to prior work): bytes, maximal munch
 * with one byte of lookahead and no backtracking.  A pending lexeme is extended
 * while the extension is a prefix of some terminal's language; otherwise a
 * complete pending lexeme is emitted as the class of all terminals it matches
 * and the byte is read again from an empty lexeme; otherwise the token fails.
 * Classes made only of %ignore terminals reach no parser.  The parser resolves a
 * class to one terminal: the first in rank order (basic lexer), or the first in
 * rank order on which the LALR(1) state of the current stack top has an action
 * (contextual lexer).
 */
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum { K_ERR = 0, K_SHIFT = 1, K_REDUCE = 2, K_ACCEPT = 3 };
enum { ST_OK = 0, ST_DONE = 1, ST_ERROR = 2 };

/* Capacities of the checker.  None of them is part of the method: reaching one
 * is a failure of the checker, never a "token not allowed".  Each sets a bit of
 * the worker's error word, the call that hit it returns that word (negated or
 * as its result) and the Python wrapper raises.  They can be set at build time
 * so that a test can reach each of them on a small grammar. */
#ifndef ORACLE_MAX_CLASS
#define ORACLE_MAX_CLASS 32      /* terminals in one lexeme class */
#endif
#ifndef ORACLE_MAX_EMIT
#define ORACLE_MAX_EMIT 256      /* classes emitted while lexing one token */
#endif
#ifndef ORACLE_LOC_MAX
#define ORACLE_LOC_MAX 8192      /* entries pushed above the row's stack while checking one token */
#endif
#ifndef ORACLE_TP_SLOTS
#define ORACLE_TP_SLOTS 1024     /* pending lexemes whose T_p a worker keeps */
#endif
#ifndef ORACLE_MAX_STEPS
#define ORACLE_MAX_STEPS 10000000L  /* parser actions while feeding one terminal */
#endif
enum { MAX_CLASS = ORACLE_MAX_CLASS, MAX_EMIT = ORACLE_MAX_EMIT, LOC_MAX = ORACLE_LOC_MAX };
enum {
    ERR_CLASS = 1,     /* a class with more than MAX_CLASS terminals */
    ERR_MIXED = 2,     /* a lexeme matched by an ignored and a kept terminal (a grammar error) */
    ERR_EMIT = 4,      /* more than MAX_EMIT classes from one token */
    ERR_LOC = 8,       /* more than LOC_MAX pushed entries */
    ERR_TP_CACHE = 16, /* the T_p cache is full */
    ERR_STEPS = 32     /* more than ORACLE_MAX_STEPS parser actions for one terminal */
};

typedef struct {
    int n_nfa, words, nfa_start;
    const int32_t *eps_off, *eps_dst;
    const uint32_t *edge_set; /* [n_nfa][8] */
    const int32_t *edge_dst, *accept;
    int n_lex_terms;
    const int32_t *term_rank;
    const uint8_t *term_ignored;
    const int32_t *byte_reps; /* one representative byte per byte equivalence class */
    int n_byte_reps;
    int n_lr, n_terms, n_nt, end_term, contextual;
    const uint8_t *act_kind;
    const int32_t *act_val, *go, *rule_lhs, *rule_len, *core_of;
    const uint8_t *acceptable; /* [n_cores][n_terms] */
} OTables;

typedef struct {
    uint64_t *pend;
    int pend_len;
    int32_t *stack;
    int depth, cap;
    int status;
} OConfig;

/* ---------------------------------------------------------------- NFA sets */

typedef struct {
    const OTables *T;
    int32_t *dfs;
    int *err;   /* the worker's error word */
} Lex;

static int set_empty(const uint64_t *a, int w) {
    for (int i = 0; i < w; i++)
        if (a[i]) return 0;
    return 1;
}

static void set_closure(Lex *L, uint64_t *set) {
    const OTables *T = L->T;
    int top = 0;
    for (int i = 0; i < T->words; i++) {
        uint64_t m = set[i];
        while (m) {
            int b = __builtin_ctzll(m);
            m &= m - 1;
            L->dfs[top++] = i * 64 + b;
        }
    }
    while (top) {
        int s = L->dfs[--top];
        for (int e = T->eps_off[s]; e < T->eps_off[s + 1]; e++) {
            int d = T->eps_dst[e];
            if (!((set[d >> 6] >> (d & 63)) & 1)) {
                set[d >> 6] |= 1ull << (d & 63);
                L->dfs[top++] = d;
            }
        }
    }
}

static void set_start(Lex *L, uint64_t *set) {
    memset(set, 0, sizeof(uint64_t) * L->T->words);
    set[L->T->nfa_start >> 6] |= 1ull << (L->T->nfa_start & 63);
    set_closure(L, set);
}

static void set_step(Lex *L, const uint64_t *cur, int byte, uint64_t *out) {
    const OTables *T = L->T;
    memset(out, 0, sizeof(uint64_t) * T->words);
    for (int i = 0; i < T->words; i++) {
        uint64_t m = cur[i];
        while (m) {
            int s = i * 64 + __builtin_ctzll(m);
            m &= m - 1;
            int d = T->edge_dst[s];
            if (d >= 0 && ((T->edge_set[s * 8 + (byte >> 5)] >> (byte & 31)) & 1))
                out[d >> 6] |= 1ull << (d & 63);
        }
    }
    set_closure(L, out);
}

/* The class of a set: all terminals accepted in it, sorted by rank.  Returns
 * the count (0 = not complete), or -1 (with a bit of *err set) if the class
 * overflows or ignored and kept terminals mix. */
static int set_class(const OTables *T, const uint64_t *set, int32_t *cls, int *err) {
    int n = 0;
    for (int i = 0; i < T->words; i++) {
        uint64_t m = set[i];
        while (m) {
            int s = i * 64 + __builtin_ctzll(m);
            m &= m - 1;
            int t = T->accept[s];
            if (t < 0) continue;
            int dup = 0;
            for (int k = 0; k < n; k++) dup |= cls[k] == t;
            if (!dup) {
                if (n == MAX_CLASS) {
                    *err |= ERR_CLASS;
                    return -1;
                }
                cls[n++] = t;
            }
        }
    }
    for (int i = 1; i < n; i++) { /* insertion sort by rank */
        int32_t t = cls[i];
        int j = i - 1;
        while (j >= 0 && T->term_rank[cls[j]] > T->term_rank[t]) {
            cls[j + 1] = cls[j];
            j--;
        }
        cls[j + 1] = t;
    }
    int ign = 0;
    for (int k = 0; k < n; k++) ign += T->term_ignored[cls[k]];
    if (ign && ign != n) {
        *err |= ERR_MIXED;
        return -1;
    }
    return n;
}

typedef struct {
    int n;
    int32_t t[MAX_CLASS];
    int ignored;
} Class;

/* Lex `len` bytes from the pending lexeme (pend, *plen).  Emitted non-ignored
 * classes go to out[]; returns their count, or -1 if the bytes do not lex. */
static int lex_bytes(Lex *L, uint64_t *pend, int *plen, const uint8_t *bytes, int len,
                     Class *out, uint64_t *tmp) {
    const OTables *T = L->T;
    int n_out = 0;
    for (int i = 0; i < len; i++) {
        int c = bytes[i];
        set_step(L, pend, c, tmp);
        if (!set_empty(tmp, T->words)) {
            memcpy(pend, tmp, sizeof(uint64_t) * T->words);
            (*plen)++;
            continue;
        }
        if (*plen == 0) return -1;
        Class cl;
        cl.n = set_class(T, pend, cl.t, L->err);
        if (cl.n <= 0) return -1;
        cl.ignored = T->term_ignored[cl.t[0]];
        if (!cl.ignored) {
            if (n_out == MAX_EMIT) {
                *L->err |= ERR_EMIT;
                return -1;
            }
            out[n_out++] = cl;
        }
        set_start(L, pend);
        *plen = 0;
        set_step(L, pend, c, tmp);
        if (set_empty(tmp, T->words)) return -1;
        memcpy(pend, tmp, sizeof(uint64_t) * T->words);
        *plen = 1;
    }
    return n_out;
}

/* ----------------------------------------------------- T_p by exploration */

/* T_p for a non-empty pending lexeme: every class of a complete lexeme that
 * extends it, found by visiting every NFA state set reachable from it.  An
 * ignored class stands for the empty terminal sequence (ignored = 1). */
typedef struct {
    int n, cap;
    Class *c;
} TpSet;

typedef struct {
    uint64_t *keys; /* [slots][words] */
    int *used;
    TpSet *vals;
    int slots;
} TpCache;

static uint64_t set_hash(const uint64_t *s, int w) {
    uint64_t h = 1469598103934665603ull;
    for (int i = 0; i < w; i++) h = (h ^ s[i]) * 1099511628211ull;
    return h ^ (h >> 29);
}

static int tp_explore(Lex *L, const uint64_t *p, TpSet *res) {
    const OTables *T = L->T;
    int w = T->words;
    int cap = 256, n = 0;
    uint64_t *seen = malloc(sizeof(uint64_t) * w * cap);
    uint64_t *tmp = malloc(sizeof(uint64_t) * w);
    memcpy(seen, p, sizeof(uint64_t) * w);
    n = 1;
    res->n = 0;
    res->cap = 0;
    res->c = NULL;
    int rc = 0;
    for (int i = 0; i < n; i++) {
        Class cl;
        cl.n = set_class(T, seen + (size_t)i * w, cl.t, L->err);
        if (cl.n < 0) { rc = -1; break; }
        if (cl.n > 0) {
            cl.ignored = T->term_ignored[cl.t[0]];
            int dup = 0;
            for (int k = 0; k < res->n && !dup; k++) {
                if (res->c[k].ignored && cl.ignored) dup = 1;
                else if (!res->c[k].ignored && !cl.ignored && res->c[k].n == cl.n &&
                         !memcmp(res->c[k].t, cl.t, sizeof(int32_t) * cl.n)) dup = 1;
            }
            if (!dup) {
                if (res->n == res->cap) {
                    res->cap = res->cap ? 2 * res->cap : 8;
                    res->c = realloc(res->c, sizeof(Class) * res->cap);
                }
                res->c[res->n++] = cl;
            }
        }
        for (int r = 0; r < T->n_byte_reps; r++) {
            set_step(L, seen + (size_t)i * w, T->byte_reps[r], tmp);
            if (set_empty(tmp, w)) continue;
            int found = 0;
            for (int j = 0; j < n && !found; j++)
                found = !memcmp(seen + (size_t)j * w, tmp, sizeof(uint64_t) * w);
            if (found) continue;
            if (n == cap) {
                cap *= 2;
                seen = realloc(seen, sizeof(uint64_t) * w * cap);
            }
            memcpy(seen + (size_t)n * w, tmp, sizeof(uint64_t) * w);
            n++;
        }
    }
    free(seen);
    free(tmp);
    return rc;
}

static const TpSet *tp_lookup(Lex *L, TpCache *C, const uint64_t *p) {
    int w = L->T->words;
    uint64_t h = set_hash(p, w);
    int slot = (int)(h % (uint64_t)C->slots);
    for (int probe = 0; probe < C->slots; probe++) {
        int s = (slot + probe) % C->slots;
        if (!C->used[s]) {
            if (tp_explore(L, p, &C->vals[s]) < 0) return NULL;
            memcpy(C->keys + (size_t)s * w, p, sizeof(uint64_t) * w);
            C->used[s] = 1;
            return &C->vals[s];
        }
        if (!memcmp(C->keys + (size_t)s * w, p, sizeof(uint64_t) * w)) return &C->vals[s];
    }
    *L->err |= ERR_TP_CACHE;
    return NULL;
}

/* ------------------------------------------------------- parser simulation */

typedef struct {
    const int32_t *base;
    int base_top;           /* entries base[0..base_top) are still on the stack */
    int nloc;
    int *err;               /* the worker's error word */
    int32_t loc[LOC_MAX];   /* pushed on top of base[0..base_top) */
} Ov;

static int ov_top(const Ov *o) { return o->nloc ? o->loc[o->nloc - 1] : o->base[o->base_top - 1]; }

static int ov_pop(Ov *o, int k) {
    while (k > 0) {
        if (o->nloc) o->nloc--;
        else if (o->base_top > 1) o->base_top--;
        else return -1; /* would pop the bottom state */
        k--;
    }
    return 0;
}

static int ov_push(Ov *o, int s) {
    if (o->nloc == LOC_MAX) {
        *o->err |= ERR_LOC;
        return -1;
    }
    o->loc[o->nloc++] = s;
    return 0;
}

/* Feed terminal t: reductions until t is shifted (1), accepted (2) or rejected (0). */
static int feed_terminal(const OTables *T, Ov *o, int t) {
    for (long guard = 0; guard < ORACLE_MAX_STEPS; guard++) {
        int s = ov_top(o);
        int k = T->act_kind[(size_t)s * T->n_terms + t];
        int v = T->act_val[(size_t)s * T->n_terms + t];
        if (k == K_SHIFT) return ov_push(o, v) == 0 ? 1 : 0;
        if (k == K_ACCEPT) return 2;
        if (k != K_REDUCE) return 0;
        if (ov_pop(o, T->rule_len[v]) < 0) return 0;
        int g = T->go[(size_t)ov_top(o) * T->n_nt + T->rule_lhs[v]];
        if (g < 0 || ov_push(o, g) < 0) return 0;
    }
    *o->err |= ERR_STEPS;
    return 0;
}

static int resolve(const OTables *T, const Ov *o, const Class *c) {
    if (!T->contextual) return c->t[0];
    const uint8_t *acc = T->acceptable + (size_t)T->core_of[ov_top(o)] * T->n_terms;
    for (int k = 0; k < c->n; k++)
        if (acc[c->t[k]]) return c->t[k];
    return -1;
}

static int feed_class(const OTables *T, Ov *o, const Class *c) {
    int t = resolve(T, o, c);
    if (t < 0) return 0;
    return feed_terminal(T, o, t) == 1;
}

/* ----------------------------------------------------------- token checks */

typedef struct {
    Lex L;
    TpCache cache;
    uint64_t *pend, *tmp;
    Class *emit;
    Ov ov, ov2;
    int err;   /* capacity failures (ERR_* bits) since the worker was made */
} Worker;

static void worker_init(Worker *W, const OTables *T) {
    memset(W, 0, sizeof(*W));
    W->L.T = T;
    W->L.err = &W->err;
    W->ov.err = &W->err;
    W->ov2.err = &W->err;
    W->L.dfs = malloc(sizeof(int32_t) * (T->n_nfa + 1) * 2);
    W->cache.slots = ORACLE_TP_SLOTS;
    W->cache.keys = malloc(sizeof(uint64_t) * T->words * W->cache.slots);
    W->cache.used = calloc(W->cache.slots, sizeof(int));
    W->cache.vals = malloc(sizeof(TpSet) * W->cache.slots);
    W->pend = malloc(sizeof(uint64_t) * T->words);
    W->tmp = malloc(sizeof(uint64_t) * T->words);
    W->emit = malloc(sizeof(Class) * MAX_EMIT);
}

static void worker_free(Worker *W) {
    for (int s = 0; s < W->cache.slots; s++)
        if (W->cache.used[s]) free(W->cache.vals[s].c);
    free(W->L.dfs);
    free(W->cache.keys);
    free(W->cache.used);
    free(W->cache.vals);
    free(W->pend);
    free(W->tmp);
    free(W->emit);
}

static void ov_init(Ov *o, const OConfig *c) {
    o->base = c->stack;
    o->base_top = c->depth;
    o->nloc = 0;
}

static void ov_copy(Ov *dst, const Ov *src) {
    dst->err = src->err;
    dst->base = src->base;
    dst->base_top = src->base_top;
    dst->nloc = src->nloc;
    memcpy(dst->loc, src->loc, sizeof(int32_t) * src->nloc);
}

/* Is the end-of-sequence token allowed in configuration c? */
static int check_eos(Worker *W, const OConfig *c) {
    const OTables *T = W->L.T;
    if (c->status == ST_DONE) return 1;
    if (c->status != ST_OK) return 0;
    ov_init(&W->ov, c);
    if (c->pend_len > 0) {
        Class cl;
        cl.n = set_class(T, c->pend, cl.t, &W->err);
        if (cl.n <= 0) return 0;
        if (!T->term_ignored[cl.t[0]] && !feed_class(T, &W->ov, &cl)) return 0;
    }
    return feed_terminal(T, &W->ov, T->end_term) == 2;
}

/* Is the ordinary token with these bytes allowed in configuration c? */
static int check_token(Worker *W, const OConfig *c, const uint8_t *bytes, int len) {
    const OTables *T = W->L.T;
    if (c->status != ST_OK || len <= 0) return 0;
    memcpy(W->pend, c->pend, sizeof(uint64_t) * T->words);
    int plen = c->pend_len;
    int n = lex_bytes(&W->L, W->pend, &plen, bytes, len, W->emit, W->tmp);
    if (n < 0) return 0;
    ov_init(&W->ov, c);
    for (int i = 0; i < n; i++)
        if (!feed_class(T, &W->ov, &W->emit[i])) return 0;
    if (plen == 0) return 1; /* T_p = {empty} */
    const TpSet *tp = tp_lookup(&W->L, &W->cache, W->pend);
    if (!tp) return 0;
    for (int k = 0; k < tp->n; k++) {
        if (tp->c[k].ignored) return 1;
        ov_copy(&W->ov2, &W->ov);
        if (feed_class(T, &W->ov2, &tp->c[k])) return 1;
    }
    return 0;
}

/* ------------------------------------------------------------- public API */

OConfig *oracle_config_new(const OTables *T, int cap) {
    OConfig *c = calloc(1, sizeof(OConfig));
    int err = 0;
    Lex L = {T, malloc(sizeof(int32_t) * (T->n_nfa + 1) * 2), &err};
    c->pend = malloc(sizeof(uint64_t) * T->words);
    set_start(&L, c->pend);
    free(L.dfs);
    c->cap = cap < 16 ? 16 : cap;
    c->stack = malloc(sizeof(int32_t) * c->cap);
    c->stack[0] = 0;
    c->depth = 1;
    return c;
}

OConfig *oracle_config_copy(const OTables *T, const OConfig *src) {
    OConfig *c = calloc(1, sizeof(OConfig));
    *c = *src;
    c->pend = malloc(sizeof(uint64_t) * T->words);
    memcpy(c->pend, src->pend, sizeof(uint64_t) * T->words);
    c->stack = malloc(sizeof(int32_t) * c->cap);
    memcpy(c->stack, src->stack, sizeof(int32_t) * c->depth);
    return c;
}

void oracle_config_free(OConfig *c) {
    if (!c) return;
    free(c->pend);
    free(c->stack);
    free(c);
}

int oracle_config_get(const OConfig *c, int32_t *status, int32_t *pend_len, int32_t *depth,
                      int32_t *stack_out, int stack_cap) {
    *status = c->status;
    *pend_len = c->pend_len;
    *depth = c->depth;
    for (int i = 0; i < c->depth && i < stack_cap; i++) stack_out[i] = c->stack[i];
    return 0;
}

int oracle_config_pending(const OTables *T, const OConfig *c, uint64_t *out_words) {
    memcpy(out_words, c->pend, sizeof(uint64_t) * T->words);
    return T->words;
}

/* Commit one token (is_eos: the end-of-sequence token).  A token the mask does
 * not allow moves the row to the error status.  Returns the new status, or
 * -(ERR_* bits) with the row unchanged if a capacity of the checker ran out. */
int oracle_advance(const OTables *T, OConfig *c, const uint8_t *bytes, int len, int is_eos) {
    if (c->status == ST_ERROR) return c->status;
    Worker *W = malloc(sizeof(Worker));
    worker_init(W, T);
    int allowed = is_eos ? check_eos(W, c) : check_token(W, c, bytes, len);
    if (W->err) {
        int e = W->err;
        worker_free(W);
        free(W);
        return -e;
    }
    if (!allowed) {
        c->status = ST_ERROR;
    } else if (is_eos) {
        c->status = ST_DONE;
    } else {
        int plen = c->pend_len;
        int n = lex_bytes(&W->L, c->pend, &plen, bytes, len, W->emit, W->tmp);
        c->pend_len = plen;
        ov_init(&W->ov, c);
        for (int i = 0; i < n; i++) feed_class(T, &W->ov, &W->emit[i]);
        /* write the view back into the row's stack */
        int d = W->ov.base_top + W->ov.nloc;
        if (d > c->cap) {
            int nc = c->cap;
            while (nc < d) nc *= 2;
            c->stack = realloc(c->stack, sizeof(int32_t) * nc);
            c->cap = nc;
        }
        memcpy(c->stack + W->ov.base_top, W->ov.loc, sizeof(int32_t) * W->ov.nloc);
        c->depth = d;
    }
    worker_free(W);
    free(W);
    return c->status;
}

typedef struct {
    const OTables *T;
    OConfig *const *rows;
    int B, V, W, eos_id;
    const uint8_t *vb;
    const int64_t *vo;
    uint32_t *out;
    int tid, nthreads;
    int err;   /* the worker's error word when it finished */
} Job;

static void *mask_worker(void *arg) {
    Job *J = arg;
    Worker *W = malloc(sizeof(Worker));
    worker_init(W, J->T);
    long total = (long)J->B * J->V;
    long chunk = (total + J->nthreads - 1) / J->nthreads;
    long lo = chunk * J->tid, hi = lo + chunk < total ? lo + chunk : total;
    for (long i = lo; i < hi; i++) {
        int b = (int)(i / J->V), v = (int)(i % J->V);
        const OConfig *c = J->rows[b];
        int ok;
        if (c->status == ST_DONE) ok = v == J->eos_id;
        else if (v == J->eos_id) ok = check_eos(W, c);
        else ok = check_token(W, c, J->vb + J->vo[v], (int)(J->vo[v + 1] - J->vo[v]));
        if (W->err) break;
        if (ok) __atomic_fetch_or(&J->out[(size_t)b * J->W + (v >> 5)], 1u << (v & 31), __ATOMIC_RELAXED);
    }
    J->err = W->err;
    worker_free(W);
    free(W);
    return NULL;
}

/* Masks of B rows over a vocabulary of V tokens (token v = vb[vo[v]..vo[v+1])),
 * packed LSB-first into out[B][ceil(V/32)] (bits v >= V stay zero).  Returns 0,
 * or the ERR_* bits of the capacities that ran out (the masks are then void). */
int oracle_masks(const OTables *T, OConfig *const *rows, int B, const uint8_t *vb,
                 const int64_t *vo, int V, int eos_id, uint32_t *out, int nthreads) {
    int W = (V + 31) / 32;
    memset(out, 0, sizeof(uint32_t) * (size_t)B * W);
    if (nthreads < 1) nthreads = 1;
    pthread_t *th = malloc(sizeof(pthread_t) * nthreads);
    Job *jobs = malloc(sizeof(Job) * nthreads);
    for (int t = 0; t < nthreads; t++) {
        jobs[t] = (Job){T, rows, B, V, W, eos_id, vb, vo, out, t, nthreads, 0};
        pthread_create(&th[t], NULL, mask_worker, &jobs[t]);
    }
    int err = 0;
    for (int t = 0; t < nthreads; t++) {
        pthread_join(th[t], NULL);
        err |= jobs[t].err;
    }
    free(th);
    free(jobs);
    return err;
}

/* One (row, token) decision; used to sample outputs of large workloads.
 * Returns 1 / 0, or -(ERR_* bits) if a capacity of the checker ran out. */
int oracle_allowed(const OTables *T, const OConfig *c, const uint8_t *bytes, int len,
                   int is_eos) {
    Worker *W = malloc(sizeof(Worker));
    worker_init(W, T);
    int ok;
    if (c->status == ST_DONE) ok = is_eos;
    else if (is_eos) ok = check_eos(W, c);
    else ok = check_token(W, c, bytes, len);
    if (W->err) ok = -W->err;
    worker_free(W);
    free(W);
    return ok;
}
