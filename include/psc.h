/*
 * psc.h - C ABI of the GB300 PSC library: grammar-constrained decoding masks by
 * Parser Stack Classification (Li, Dong, Li, Li, "Efficient Grammar-Constrained
 * Decoding via Parser Stack Classification").
 *
 * The library computes, once per decoding step and for a whole batch of
 * sequences, the vocabulary mask of Eq. (1): the tokens v such that the prefix
 * followed by v can still be completed to a string of the grammar's language.
 * Following the paper, the offline step (psc_compile, Algorithm 1) folds every
 * token's acceptance condition on the parser stack into one classifier DFA over
 * (lexer state, parser stack read from the top) and precomputes the mask of
 * every classifier state; the online step (Algorithm 2) walks each sequence's
 * stack once through that DFA and returns the precomputed mask.  Here the
 * online step runs in CUDA kernels on the GPU that also applies the mask to
 * the logits, and the classification is kept incremental: the same classifier
 * is also built reading the stack from the bottom, its state is kept for every
 * stack prefix, and a step re-reads only the stack entries it changed.
 *
 * Conventions for every call:
 *  - Pointers named d_* are device memory owned by the caller (for example the
 *    data_ptr() of a torch tensor); h_* are host memory owned by the caller.
 *  - A psc_handle owns its device tables and a psc_states owns its device
 *    arrays; both are freed only by their *_destroy call.
 *  - Calls that take a cudaStream_t (passed as void*, NULL = the legacy default
 *    stream) only enqueue work on that stream and return; they never
 *    synchronise.  Their return value reports argument and launch errors only.
 *  - Errors in the data (a token the mask does not allow, a stack that
 *    overflows its capacity) are per-row statuses written by the kernels;
 *    kernels never trap and never spin.  Every in-kernel wait is bounded; one
 *    that gives up is counted on the states object (psc_state_faults).
 *  - psc_last_error() returns a thread-local message for the last failing call.
 *  - Bit v of a packed mask row is bit (v & 31) of 32-bit word (v >> 5)
 *    (least significant bit first); bits v >= V are zero.
 */
#ifndef PSC_H
#define PSC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    PSC_OK = 0,
    PSC_ERR_ARG = 1,              /* bad argument (NULL, size, dtype, stride, host-only handle) */
    PSC_ERR_GRAMMAR = 2,          /* grammar text cannot be read */
    PSC_ERR_CONFLICT = 3,         /* grammar is not LALR(1) */
    PSC_ERR_LEXER_AMBIGUOUS = 4,  /* a lexeme matches an ignored and a kept terminal */
    PSC_ERR_LIMIT = 5,            /* a size limit of psc_options was exceeded */
    PSC_ERR_OOM = 6,              /* host or device allocation failed */
    PSC_ERR_CUDA = 7,             /* a CUDA runtime call failed */
    PSC_ERR_IO = 8
} psc_status;

typedef enum { PSC_F32 = 0, PSC_BF16 = 1 } psc_dtype;

/* per-row status words of a psc_states batch */
enum {
    PSC_ROW_OK = 0,        /* the row is inside the language's prefixes */
    PSC_ROW_DONE = 1,      /* the end-of-sequence token was accepted; only it stays allowed */
    PSC_ROW_REJECTED = 2,  /* a token outside the mask was advanced; nothing is allowed */
    PSC_ROW_OVERFLOW = 3,  /* the parser stack exceeded the batch capacity; nothing is allowed */
    PSC_ROW_LIMIT = 4      /* a bounded loop in the advance kernel ran out; nothing is allowed */
};

typedef struct psc_handle psc_handle;
typedef struct psc_states psc_states;

typedef struct {
    int64_t max_states;      /* classifier states before PSC_ERR_LIMIT (0 = 4,000,000) */
    int64_t max_mask_bytes;  /* host bytes of distinct mask rows before PSC_ERR_LIMIT (0 = 24 GiB) */
    int32_t threads;         /* host threads for compilation (0 = all cores) */
    int32_t host_only;       /* 1: build host tables only (no GPU needed; device calls fail) */
    int32_t global_tables;   /* where the advance kernel reads the lexer and parser tables:
                                0 = staged in shared memory, dense when they fit in 200 KiB, else
                                packed (ACTION and GOTO row-displaced into one table of owner-
                                checked entries, lexeme classes resolved through candidate lists)
                                when those fit, else global memory; 1 = global memory;
                                2 = staged packed tables whenever they fit.  Other values:
                                PSC_ERR_ARG. */
    int64_t max_bottom_up_bytes;  /* host memory for building the bottom-up classifier (0 = 16 GiB,
                                     at most half of the machine's memory);
                                     negative: not built (psc_load: dropped), and the device walks
                                     every stack from the top.  Over the limit it is not built
                                     (no error). */
    int64_t max_dense_classifier_bytes;  /* the classifier DFA is held dense ([S][|Pi|] int32) up to
                                            this size, above it sparse (per state a default target and
                                            the exceptions to it; a walk step reads one row) (0 = 512 MiB;
                                            negative: always sparse) */
} psc_options;

typedef struct {
    int32_t V, W;            /* vocabulary size, 32-bit words per mask row */
    int32_t n_lexer_states;  /* Q: lexer DFA states (the lexing transducer of Section 2.2) */
    int32_t n_parser_states; /* |Pi|: LALR(1) states = stack symbols (Section 2.4) */
    int32_t n_terminals;     /* grammar terminals + the end marker */
    int32_t n_classifier_states;  /* S: non-absorbing states of the classifier DFA (Eq. 9) */
    int32_t n_masks;         /* distinct precomputed masks A_s (Section 3.5) */
    int32_t eos_id;
    int64_t classifier_bytes;  /* device bytes of the classifier tables (cf. Table 7, DFA) */
    int64_t mask_bytes;        /* device bytes of the mask table (cf. Table 7, masks): each row is
                                  held as ids of 1024-token chunks, equal chunks stored once */
    int64_t states_built;      /* classifier states before minimisation */
    double compile_seconds;
    int64_t advance_table_bytes;  /* bytes psc_advance stages in shared memory (0: it reads global memory;
                                     a host_only handle: what a device upload would stage) */
    int64_t device_timeouts;      /* bounded in-kernel waits that gave up since the library was loaded
                                     (process-wide; non-zero means a pipeline fault; reading it synchronises) */
    int64_t bottom_up_states;     /* states of the bottom-up classifier (0: not built) */
    int64_t bottom_up_bytes;      /* its device bytes (blocks, edge slots, final table) */
    int64_t classifier_sparse;    /* 1: the classifier DFA is held in the sparse layout */
    int64_t advance_tables_packed;  /* 1: the staged parser tables are in the packed layout */
} psc_info_t;

/* Offline construction (Algorithm 1, Section 3).  Reads the grammar text (a
 * Lark-like notation, see the library's documentation), builds the lexer DFA,
 * the LALR(1) tables, the realizable terminal sequences R_q(v) of every token
 * from every lexer state (Section 3.1), the stack classifier of Eq. (9), its
 * bottom-up form (unless opts say otherwise) and the mask of every classifier
 * state, and uploads the tables to the current CUDA device unless
 * opts->host_only.
 *   grammar/grammar_len : grammar text (not NUL-terminated necessarily)
 *   vocab_bytes         : all token byte strings concatenated (host)
 *   vocab_offsets       : V+1 int64 offsets; token v = vocab_bytes[off[v], off[v+1])
 *   V, eos_id           : vocabulary size and the end-of-sequence id (its bytes are ignored;
 *                         -1 = no end-of-sequence token)
 *   opts                : NULL = defaults
 *   out                 : receives the handle (NULL on error)
 * Errors: PSC_ERR_GRAMMAR / _CONFLICT / _LEXER_AMBIGUOUS for the grammar,
 * PSC_ERR_LIMIT, PSC_ERR_OOM, PSC_ERR_CUDA, PSC_ERR_ARG. */
psc_status psc_compile(const char* grammar, size_t grammar_len, const uint8_t* vocab_bytes,
                       const int64_t* vocab_offsets, int32_t V, int32_t eos_id,
                       const psc_options* opts, psc_handle** out);

/* Frees the handle's host and device tables (NULL is a no-op).  No call that
 * uses the handle may still be running on any stream. */
void psc_destroy(psc_handle* h);

/* Writes the handle's compiled tables to a binary file (the paper ships its
 * preprocessing results to decoding users as zstd-compressed files, Section 5).
 * The file holds the lexer, parser, classifier (both forms) and mask tables and
 * the vocabulary, with a checksum, compressed in 16 MiB blocks by the system's
 * zstd library (libzstd.so.1) when it can be loaded at run time, else zlib
 * (libz.so.1), else stored as it is; the environment variable PSC_SAVE_CODEC
 * (none, zstd or zlib) chooses.  Errors: PSC_ERR_IO, PSC_ERR_ARG. */
psc_status psc_save(const psc_handle* h, const char* path);

/* Reads a file written by psc_save, checks its checksum and the consistency of
 * every table index, and uploads the tables to the current device (unless
 * opts->host_only; opts may be NULL).  Errors: PSC_ERR_IO (missing, truncated,
 * corrupt or inconsistent file, or compressed with a codec this host cannot
 * load), PSC_ERR_OOM, PSC_ERR_CUDA. */
psc_status psc_load(const char* path, const psc_options* opts, psc_handle** out);

/* Thread-local message of the last failed call on this thread ("" if none). */
const char* psc_last_error(void);

/* Table sizes of a compiled handle (Table 7 of the paper reports the same
 * quantities for its CPU implementation). */
psc_status psc_info(const psc_handle* h, psc_info_t* out);

/* A batch of B parser configurations on the device (Algorithm 2, steps 1-2:
 * the lexer state q and the parser stack alpha of each sequence, Section 3.2),
 * all at the empty prefix: q = the empty lexeme, alpha = [0], status OK.
 *   cap : stack capacity per row (>= 2); layout [B][cap] uint16, bottom first.
 * The states object owns its device arrays; initialisation is enqueued on stream. */
psc_status psc_state_init(const psc_handle* h, int32_t B, int32_t cap, void* stream, psc_states** out);

/* Resets rows to the empty prefix: the n row indices in d_rows (device int32),
 * or every row when d_rows is NULL. */
psc_status psc_state_reset(psc_states* st, const int32_t* d_rows, int32_t n, void* stream);

void psc_state_destroy(psc_states* st);

/* Copies every row of src into dst: lexer states, depths, statuses, stacks,
 * mask ids, pending greedy choices and the bottom-up classifier's kept states
 * (device-to-device, enqueued on stream).
 * Both objects must belong to the same handle and have the same B and cap
 * (else PSC_ERR_ARG).  The paper has no counterpart: it serves forking a batch
 * (beam search, speculative branches) and restoring a saved one, e.g. to
 * decode again from the same prefixes. */
psc_status psc_state_copy(psc_states* dst, const psc_states* src, void* stream);

/* Algorithm 2, steps 1-2, done incrementally on the device: for each row b with
 * d_tokens[b] >= 0, first checks the token against the row's current mask; a
 * token outside it sets PSC_ROW_REJECTED; the end-of-sequence token sets
 * PSC_ROW_DONE; any other allowed token is lexed from the row's lexer state and
 * the emitted terminals are fed to the LALR(1) parser on the row's stack.
 * Afterwards every row is classified (step 3) and its mask id kept in the
 * states object, so the next mask call reads it without walking the stack.
 * With the bottom-up classifier (psc_options.max_bottom_up_bytes >= 0, the
 * default) the classification re-reads only the stack entries the step
 * pushed; without it the stack is walked from the top.
 * d_tokens[b] < 0 leaves row b unchanged.  B must equal the batch size.
 *   d_row_status : optional device int32[B] copy of the statuses after the step. */
psc_status psc_advance(const psc_handle* h, psc_states* st, const int32_t* d_tokens, int32_t B,
                       int32_t* d_row_status, void* stream);

/* Algorithm 2, steps 3-4: classifies every row's (q, alpha) with the classifier
 * DFA (from the bottom-up classifier's kept state when it is built, else one
 * pass over the stack from the top, stopping at absorbing states; skipped when
 * the last psc_advance or decode step already did it) and writes the
 * precomputed mask of the resulting state as a packed bitmask.
 *   d_bitmask : device uint32 [B][W], W = ceil(V/32), row-contiguous.
 * Rows with status DONE get the end-of-sequence-only mask, failed rows the
 * empty mask. */
psc_status psc_fill_mask(const psc_handle* h, const psc_states* st, int32_t B, uint32_t* d_bitmask,
                         void* stream);

/* Applies packed bitmasks to logits in place: logits[b][v] = -inf where bit v
 * of row b is 0 (bf16 0xFF80, f32 0xFF800000); allowed logits keep their exact
 * bits.  Columns v >= V are not touched.  (The paper leaves this step to the
 * serving engine and excludes it from its timing, Section 4.3 "Metrics".)
 *   d_logits   : device [B] rows of row_stride elements of dtype
 *   row_stride : elements between rows, >= V
 *   d_bitmask  : device uint32 [B][ceil(V/32)] */
psc_status psc_apply_mask(void* d_logits, psc_dtype dtype, int64_t row_stride, const uint32_t* d_bitmask,
                          int32_t B, int32_t V, void* stream);

/* psc_fill_mask and psc_apply_mask fused: the row's classification (as in
 * psc_fill_mask) picks its mask row, which is applied to the logits straight from the device mask table
 * (the bitmask does not round-trip through memory).  V must equal the
 * handle's vocabulary size.
 *   d_bitmask_out : optional device uint32 [B][W] copy of the masks (NULL = none). */
psc_status psc_fill_apply(const psc_handle* h, const psc_states* st, int32_t B, void* d_logits,
                          psc_dtype dtype, int64_t row_stride, int32_t V, uint32_t* d_bitmask_out,
                          void* stream);

/* Greedy sampling over the allowed tokens: d_tokens[b] = the lowest index v
 * with the largest logits[b][v] among the tokens of row b's mask, or -1 when
 * the mask is empty.  Only allowed positions are read.  Rows are classified as
 * in psc_fill_mask (call it after psc_fill_apply and before psc_advance). */
psc_status psc_argmax_masked(const psc_handle* h, const psc_states* st, int32_t B, const void* d_logits,
                             psc_dtype dtype, int64_t row_stride, int32_t V, int32_t* d_tokens,
                             void* stream);

/* psc_fill_apply and psc_argmax_masked in one pass over the logits: each
 * 1024-token chunk holding an allowed position is read once (a chunk with none
 * is only written), every 32-byte sector that holds a masked position is
 * written once with -inf in the masked places, and the greedy choice among
 * allowed tokens is merged per row with a 64-bit atomic maximum (value order,
 * then the lowest index).  d_tokens[b] = chosen token or
 * -1 when row b allows nothing; d_bitmask_out as in psc_fill_apply.  The
 * per-row keys live in the states object; calls on the same states object
 * must not overlap. */
psc_status psc_fill_apply_argmax(const psc_handle* h, const psc_states* st, int32_t B, void* d_logits,
                                 psc_dtype dtype, int64_t row_stride, int32_t V, uint32_t* d_bitmask_out,
                                 int32_t* d_tokens, void* stream);

/* One whole decoding step on the device (Algorithm 2 steps 1-4 plus masking and
 * greedy sampling), in two kernels: the masking pass applies every row's mask
 * (step 4) to the logits in place, writes the optional bitmask copy and picks
 * the greedy token per row; the advance kernel then feeds that token to the
 * row's lexer and parser (steps 1-2) and classifies the new configuration
 * (step 3), so the next step's masking pass reads the mask ids directly.  The
 * masking pass classifies rows itself when the mask ids are not current (after
 * psc_state_init or psc_state_reset).
 *   d_tokens      : device int32 [B]; receives the chosen tokens (-1 = nothing allowed)
 *   d_row_status  : optional device int32 [B] statuses after the step
 * Other arguments as for psc_fill_apply_argmax.  Equivalent to
 * psc_decode_step_mask followed by psc_decode_step_advance. */
psc_status psc_decode_step(const psc_handle* h, psc_states* st, int32_t B, void* d_logits, psc_dtype dtype,
                           int64_t row_stride, int32_t V, uint32_t* d_bitmask_out, int32_t* d_tokens,
                           int32_t* d_row_status, void* stream);

/* The two halves of psc_decode_step, for callers that interleave work (or
 * timing) between them.  psc_decode_step_mask runs the masking pass and keeps
 * each row's greedy choice in the states object; psc_decode_step_advance
 * consumes those choices: writes them to d_tokens, advances every row and
 * classifies the new configurations.  Calling psc_decode_step_advance without
 * a preceding psc_decode_step_mask on the same states object finds no choices
 * (every token -1, rows unchanged).  Arguments as for psc_decode_step. */
psc_status psc_decode_step_mask(const psc_handle* h, psc_states* st, int32_t B, void* d_logits, psc_dtype dtype,
                                int64_t row_stride, int32_t V, uint32_t* d_bitmask_out, void* stream);
psc_status psc_decode_step_advance(const psc_handle* h, psc_states* st, int32_t B, int32_t* d_tokens,
                                   int32_t* d_row_status, void* stream);

/* Faults of the bounded in-kernel waits on this states object: every wait of
 * the masking pass and of the advance is bounded, and one that gives up (a
 * pipeline fault; the step's logits or rows may then be incomplete, rows whose
 * advance could not run get PSC_ROW_LIMIT) adds 1 to a counter kept in the
 * states object (zero after psc_state_init).  Copies the counter to *h_faults
 * and synchronises the stream; reset != 0 then zeroes it (enqueued on stream).
 * The paper has no counterpart: this is the per-batch error word a serving
 * loop checks between steps.  Errors: PSC_ERR_ARG, PSC_ERR_CUDA. */
psc_status psc_state_faults(psc_states* st, int32_t* h_faults, int32_t reset, void* stream);

/* Self-test of fault reporting: launches one CTA whose bounded wait, on an
 * mbarrier phase that no thread completes, gives up after `limit` polls
 * (1..2^24) and adds 1 to the states object's fault counter, the path a
 * pipeline wait that gives up takes.  Nothing faults and the device stays
 * usable.  Errors: PSC_ERR_ARG, PSC_ERR_CUDA. */
psc_status psc_check_wait(psc_states* st, int32_t limit, void* stream);

/* Copies the batch to host memory and synchronises the stream (tests and
 * debugging).  Any output pointer may be NULL.
 *   h_q, h_depth, h_status : int32 [B];  h_stack : uint16 [B][cap] */
psc_status psc_states_download(const psc_states* st, int32_t* h_q, int32_t* h_depth, uint16_t* h_stack,
                               int32_t* h_status, void* stream);

/* Host-side inspection of the compiled tables (no GPU needed):
 * psc_host_classify walks the classifier DFA for one configuration and
 * returns its mask id (or -1 on bad arguments); psc_host_mask_row copies mask
 * row `mask_id` (W words) to h_row. */
int32_t psc_host_classify(const psc_handle* h, int32_t q, const uint16_t* h_stack, int32_t depth,
                          int32_t status);

/* The same classification through the bottom-up classifier (the classifier
 * DFA reversed, reading the stack from the bottom; the regularity theorem of
 * Section 3.5 is what makes this automaton exist): returns the mask id, -1 on
 * bad arguments, or -2 when the handle has no bottom-up classifier or the
 * stack is not a path of the LR automaton (no parser builds such a stack).
 * States objects keep this automaton's state after every stack prefix of
 * every row, so a decode step re-reads only the stack entries it changed. */
int32_t psc_host_classify_bottom_up(const psc_handle* h, int32_t q, const uint16_t* h_stack, int32_t depth,
                                    int32_t status);
psc_status psc_host_mask_row(const psc_handle* h, int32_t mask_id, uint32_t* h_row);

/* Host-side lexer+parser step of one configuration (tests and prefix set-up
 * without a GPU): the same semantics as psc_advance for a single row held in
 * host memory.  *q, *depth, *status and h_stack[cap] are updated in place. */
psc_status psc_host_advance(const psc_handle* h, int32_t* q, uint16_t* h_stack, int32_t* depth, int32_t cap,
                            int32_t* status, int32_t token);

/* Allocation-free variant of psc_fill_apply.  The paper has no counterpart:
 * this entry point exists for callers that cannot allocate device memory at
 * the point where they apply the mask, for example code running while a
 * stream is being captured into a CUDA graph (cudaMalloc is not allowed
 * there), code inside a framework whose allocator owns all device memory, or
 * latency-critical loops where an allocation could synchronise the device.
 *
 * It does exactly what psc_fill_apply does, but the parser configurations
 * come from caller-owned device arrays instead of a psc_states object, and the
 * per-row mask ids it needs between the classifier walk and the masking pass
 * live in one library-owned scratch array of PSC_NOALLOC_MAX_ROWS int32 that
 * is part of the loaded module (a file-scope __device__ array, 64 KiB, held by
 * every GPU that loads the library until the process exits).  Nothing is
 * allocated or freed by the call.
 *   d_q, d_depth, d_status : device int32 [B] (lexer state, stack depth, row status)
 *   d_stack                : device uint16 [B][cap], bottom first (the layout psc_states_download returns);
 *                            a row whose lexer state, depth or stack symbols are out of range gets
 *                            the empty mask (its logits all -inf)
 *   other arguments        : as for psc_fill_apply
 * Errors: PSC_ERR_LIMIT when B > PSC_NOALLOC_MAX_ROWS; PSC_ERR_ARG for bad arguments.
 * The first call on a device looks up the scratch array's device address
 * (cudaGetSymbolAddress) with that device current; make that first call
 * before any stream capture.  The address is kept for the life of the
 * process: it does not survive cudaDeviceReset (which unloads the module), so
 * do not call this entry point after resetting the device.  Every call shares the same scratch array, which
 * keeps the last call's contents (each call writes every entry it reads, so
 * nothing needs clearing); calls that overlap on the GPU (different streams,
 * or host threads racing on one device) race on it and must be serialised by
 * the caller. */
#define PSC_NOALLOC_MAX_ROWS 16384
psc_status psc_fill_apply_noalloc(const psc_handle* h, const int32_t* d_q, const int32_t* d_depth,
                                  const int32_t* d_status, const uint16_t* d_stack, int32_t cap, int32_t B,
                                  void* d_logits, psc_dtype dtype, int64_t row_stride, int32_t V,
                                  uint32_t* d_bitmask_out, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* PSC_H */
