// C ABI of the PSC library (include/psc.h) and its CUDA kernels for sm_103a.
//
// Online step of the paper (Algorithm 2), per decoding step and batch row:
//   steps 1-2  incremental lexing and LR parsing of the sampled token on the
//              row's device-resident stack                      -> k_advance_warp
//   step 3     the classifier DFA over (q, stack from the top), O(|stack|),
//              stopping at absorbing states; kept incremental by the bottom-up
//              classifier (its state per stack prefix, so a step re-reads only
//              the entries it changed, then one lookup by q)    -> k_advance_warp / k_classify
//   step 4     the precomputed mask of the reached state         -> k_step_tma / k_fill / k_apply_rows
// plus applying the mask to the logits and greedy sampling over the allowed
// tokens (left to the serving engine in the paper).
//
// Memory layout on the device (all tables uploaded once by psc_compile):
//   dfa      int32 [S][n_lr]      next classifier state, or -(mask+1) when absorbing
//   mrows    uint32 [n_masks][nch] mask rows as ids of 1024-token chunks (nch = ceil(W / 32))
//   mchunks  uint32 [n_chunks][32] the distinct chunks (words past W zero)
//   bu       int32 [...]          bottom-up classifier blocks [final row, next block per edge slot]
//   bu_slot  int16 [n_lr][n_lr]   slot of the LR edge t -> u among t's successors, -1 none
//   bu_F     int32 [n_frow][nq]   mask id per final row and lexer state
//   stacks   uint16 [B][cap]      parser stacks, bottom first; depth[b] entries used
//   rmemo    int32 [B][cap]       bottom-up block of stack prefix [0, i] of every row
//   logits   [B][row_stride]      bf16 or f32, caller-owned, masked in place
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <memory>
#include <mutex>
#include <new>
#include <string>

#include "../../include/psc.h"
#include "psc_internal.h"

namespace {

thread_local std::string g_last_error;

psc_status fail_with(psc_status code, const std::string& msg) {
    g_last_error = msg;
    return code;
}

constexpr unsigned FULL = 0xffffffffu;
constexpr int ROW_OK = 0, ROW_DONE = 1, ROW_REJECTED = 2, ROW_OVERFLOW = 3, ROW_LIMIT = 4;

struct DevTables {
    const int16_t* lex_trans;
    const int32_t* lex_accept;
    const uint8_t* cls_ignored;
    const int32_t* action;
    const int32_t* go;
    const int32_t* rule_len;
    const int32_t* rule_lhs;
    const int16_t* resolve;
    const int32_t* dfa;        // dense [S][n_lr] (nullptr in the sparse layout)
    const int32_t* dfa_start;
    const int32_t* dfa_mask;
    // sparse layout (dfa_sparse = 1): one row per state, a state's id being its row's
    // offset: [exceptions n, default target, mask id, 0, (symbol, target) x n], symbols
    // ascending, targets row offsets or -(mask+1); dfa_start holds row offsets too
    const int32_t* dfa_rows;
    int dfa_sparse;
    const uint32_t* mchunks;   // distinct 32-word chunks of the mask rows [n_chunks][32]
    const uint32_t* mrows;     // mask rows as chunk ids [n_masks][nch]
    const uint8_t* vocab;
    const int64_t* vocab_off;
    const uint8_t* tok32;      // [V][32] the first 32 bytes of every token (zero-padded)
    int q0, nq, n_lr, n_terms, n_nts, end_term;
    int V, W, nch, eos_id, n_masks;
    // compact lexer/parser tables for k_advance_warp (adv_bytes = 0: not built)
    const uint8_t* adv;
    int adv_bytes, o_bc, o_trans, o_accept, o_ign, o_resolve, o_action, o_go, o_rlen, o_rlhs, nbc;
    int adv_packed;   // reduce entries of the compact ACTION hold (rule length << 10 | lhs) instead of the rule
    // packed (row-displaced) parser tables, for grammars whose dense compact tables do not
    // fit in shared memory: ACTION and GOTO each as a table of uint32 entries (row id << 16
    // | int16 entry) with equal rows stored once, and per state a word (row id << 17 | base):
    // the entry (s, x) is the one at base + x when its row id is the state's; lexeme
    // classes resolved through candidate terminal lists
    int adv_comb, o_cand, o_abase, o_gbase, o_acmb, o_gcmb, kc;
    // bottom-up classifier (bu = nullptr: not built; the root block, for the stack [0], is at 0)
    const int32_t* bu;        // blocks [final row, next block per successor slot]
    const int16_t* bu_slot;   // [n_lr][n_lr] slot of the LR edge t -> u, -1 none
    const int32_t* bu_F;      // [n_frow][nq] mask ids
    int bu_len, n_frow;
};

struct DevStates {
    int32_t* q;
    int32_t* depth;
    int32_t* status;
    uint16_t* stack;
    int32_t* mid;
    int B, cap;
    unsigned long long* best;   // per-row greedy-choice key (nullable)
    int32_t* rmemo;             // [B][cap] bottom-up classifier block after each stack prefix (nullable)
    int32_t* fault;             // bounded in-kernel waits on these states that gave up (nullable)
};

}  // namespace

struct psc_handle {
    psc::Tables t;
    bool host_only = true;
    int device = -1;
    DevTables d{};
    void* blocks[32] = {};
    int n_blocks = 0;
    int tma_ctas[2] = {1, 1};   // resident k_step_tma CTAs per SM (bf16, f32)
    int tables = 0;             // psc_options.global_tables the handle was made with
};

struct psc_states {
    const psc_handle* h = nullptr;
    DevStates d{};
    int device = -1;
    uint64_t gen = 1;        // bumped by every call that changes the rows
    uint64_t mid_gen = 0;    // generation the mask ids in d.mid were computed for
    bool after_mask = false; // the last work enqueued on these states is the TMA masking pass with
                             // the mask ids as they were (the advance may read the rows early)
};

namespace {

// ------------------------------------------------------------------ helpers
__device__ int g_pipeline_timeouts;   // bounded in-kernel waits that gave up (a fault if ever non-zero)

__device__ __forceinline__ void st_cs_v4(void* p, uint4 v) {
    asm volatile("st.global.cs.v4.b32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
                 "r"(v.w)
                 : "memory");
}

__device__ __forceinline__ uint4 ld_nc_v4(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.v4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// Word w of mask row `mid` (the mask of Section 3.5, held as chunk ids + chunks).
__device__ __forceinline__ uint32_t mask_word(const DevTables& T, int mid, int w) {
    uint32_t c = __ldg(T.mrows + (size_t)mid * T.nch + (w >> 5));
    return __ldg(T.mchunks + (size_t)c * 32 + (w & 31));
}

// Mask id of a configuration from the bottom-up classifier's block e for its
// whole stack (final table row, then the lexer state's column); -1 when e is
// not a usable block (the caller walks the stack instead).
__device__ __forceinline__ int memo_mask(const DevTables& T, int e, int q) {
    if (e < 0 || e >= T.bu_len) return -1;
    int fr = __ldg(T.bu + e);
    if (fr < 0 || fr >= T.n_frow) return -1;
    return __ldg(T.bu_F + (size_t)fr * T.nq + q);
}

// The row's mask id from its kept bottom-up state, or -1 (not kept / not built).
__device__ __forceinline__ int memo_classify(const DevTables& T, const DevStates& S, int b, int q, int depth) {
    if (!S.rmemo || !T.bu) return -1;
    return memo_mask(T, S.rmemo[(size_t)b * S.cap + depth - 1], q);
}

// One classifier transition in the sparse layout by a full warp (every lane with
// the same s and X): lane 0 loads the row's header, lane 1 the mask id, lanes
// 2-31 the first 30 exceptions; a ballot finds X; longer rows are scanned 32
// exceptions at a time.  Returns the target (row offset, or -(mask+1)).  The row
// array is padded so that these reads stay inside it.
__device__ __forceinline__ int sparse_step_warp(const int32_t* rows, int s, int X, int lane) {
    const int2* r2 = reinterpret_cast<const int2*>(rows + s);   // row offsets are even
    int2 v = __ldg(r2 + lane);
    int n = __shfl_sync(FULL, v.x, 0);
    int def = __shfl_sync(FULL, v.y, 0);
    unsigned hit = __ballot_sync(FULL, lane >= 2 && lane - 2 < n && v.x == X);
    if (hit) return __shfl_sync(FULL, v.y, __ffs(hit) - 1);
    for (int base = 30; base < n; base += 32) {
        int2 w = __ldg(r2 + 2 + base + lane);
        unsigned h2 = __ballot_sync(FULL, base + lane < n && w.x == X);
        if (h2) return __shfl_sync(FULL, w.y, __ffs(h2) - 1);
    }
    return def;
}

// The same transition by one thread (binary search over the row's exceptions).
__device__ __forceinline__ int sparse_step_thread(const int32_t* rows, int s, int X) {
    const int2* r2 = reinterpret_cast<const int2*>(rows + s);
    int2 h = __ldg(r2);
    int lo = 0, hi = h.x;
    while (lo < hi) {
        int m = (lo + hi) >> 1;
        int2 p = __ldg(r2 + 2 + m);
        if (p.x == X) return p.y;
        if (p.x < X) lo = m + 1;
        else hi = m;
    }
    return h.y;
}

// Mask id of the classifier state s when the stack ends there (either layout).
__device__ __forceinline__ int state_mask(const DevTables& T, int s) {
    return T.dfa_sparse ? __ldg(T.dfa_rows + s + 2) : __ldg(T.dfa_mask + s);
}

// Classification of one row (Algorithm 2 step 3) by a full warp: from the kept
// bottom-up block when there is one, else the walk of the classifier DFA: lanes
// load 32 stack symbols at a time (coalesced), the walk broadcasts them with
// shuffles and follows the DFA; every lane ends with the same mask id.  A stack
// symbol outside the LR states (only a caller-owned stack can hold one) gives
// the row the empty mask instead of a read outside the table.
__device__ int warp_classify(const DevTables& T, const DevStates& S, int b, int lane) {
    int status = S.status[b];
    if (status == ROW_DONE) return 1;
    if (status != ROW_OK) return 0;
    int q = S.q[b];
    int depth = S.depth[b];
    if (q < 0 || q >= T.nq || depth < 1 || depth > S.cap) return 0;
    int m = memo_classify(T, S, b, q, depth);
    if (m >= 0) return m;
    int s = __ldg(T.dfa_start + q);
    if (s < 0) return -s - 1;
    const uint16_t* st = S.stack + (size_t)b * S.cap;
    for (int top = depth - 1; top >= 0; top -= 32) {
        int i = top - lane;
        int x = i >= 0 ? st[i] : 0;
        int n = top + 1 < 32 ? top + 1 : 32;
        for (int j = 0; j < n; j++) {
            int X = __shfl_sync(FULL, x, j);   // the same in every lane: the warp returns together
            if ((unsigned)X >= (unsigned)T.n_lr) return 0;
            int nx = T.dfa_sparse ? sparse_step_warp(T.dfa_rows, s, X, lane) : __ldg(T.dfa + (size_t)s * T.n_lr + X);
            if (nx < 0) return -nx - 1;
            s = nx;
        }
    }
    return state_mask(T, s);
}

// the same classification by one thread (same guard on stack symbols)
__device__ int thread_classify(const DevTables& T, const DevStates& S, int b) {
    int status = S.status[b];
    if (status == ROW_DONE) return 1;
    if (status != ROW_OK) return 0;
    int q = S.q[b];
    int depth = S.depth[b];
    if (q < 0 || q >= T.nq || depth < 1 || depth > S.cap) return 0;
    int m = memo_classify(T, S, b, q, depth);
    if (m >= 0) return m;
    int s = __ldg(T.dfa_start + q);
    if (s < 0) return -s - 1;
    const uint16_t* st = S.stack + (size_t)b * S.cap;
    for (int i = depth - 1; i >= 0; i--) {
        int X = st[i];
        if (X >= T.n_lr) return 0;
        int nx = T.dfa_sparse ? sparse_step_thread(T.dfa_rows, s, X) : __ldg(T.dfa + (size_t)s * T.n_lr + X);
        if (nx < 0) return -nx - 1;
        s = nx;
    }
    return state_mask(T, s);
}

// ------------------------------------------------------------------ kernels
__global__ void k_state_init(DevStates S, int q0, const int32_t* rows, int n) {
    int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    int b = rows ? rows[i] : i;
    if (b < 0 || b >= S.B) return;
    S.q[b] = q0;
    S.depth[b] = 1;
    S.status[b] = ROW_OK;
    S.stack[(size_t)b * S.cap] = 0;
    S.mid[b] = 0;
    if (S.best) S.best[b] = 0ull;
    if (S.rmemo) S.rmemo[(size_t)b * S.cap] = 0;   // the bottom-up classifier's block for [0]
}

__global__ void k_classify(DevTables T, DevStates S, int B) {
    int warp = (int)((blockIdx.x * (size_t)blockDim.x + threadIdx.x) >> 5);
    int lane = threadIdx.x & 31;
    if (warp >= B) return;
    int mid = warp_classify(T, S, warp, lane);
    if (lane == 0) {
        S.mid[warp] = mid;
        if (S.best) S.best[warp] = 0ull;
    }
}

// out[b][:] = masks[mid[b]][:]   (16-byte vector copies when W % 4 == 0)
__global__ void k_fill(DevTables D, const int32_t* __restrict__ mid, int B, uint32_t* __restrict__ out, int vec) {
    size_t tid = blockIdx.x * (size_t)blockDim.x + threadIdx.x;
    size_t stride = (size_t)gridDim.x * blockDim.x;
    int W = D.W;
    if (vec) {
        int W4 = W >> 2;
        size_t total = (size_t)B * W4;
        for (size_t i = tid; i < total; i += stride) {
            int b = (int)(i / W4), w = (int)(i % W4);
            uint32_t c = __ldg(D.mrows + (size_t)__ldg(mid + b) * D.nch + ((4 * w) >> 5));
            uint4 v = ld_nc_v4(D.mchunks + (size_t)c * 32 + ((4 * w) & 31));
            st_cs_v4(out + (size_t)b * W + 4 * w, v);
        }
    } else {
        size_t total = (size_t)B * W;
        for (size_t i = tid; i < total; i += stride) {
            int b = (int)(i / W), w = (int)(i % W);
            out[i] = mask_word(D, __ldg(mid + b), w);
        }
    }
}

template <typename T>
struct NegInf;
template <>
struct NegInf<uint16_t> {
    static constexpr uint32_t pair = 0xFF80FF80u;
    static constexpr uint16_t one = 0xFF80u;
};
template <>
struct NegInf<uint32_t> {
    static constexpr uint32_t pair = 0xFF800000u;
    static constexpr uint32_t one = 0xFF800000u;
};

// Apply one 1024-column chunk of row b: `word` is this lane's mask word for
// columns [col0 + 32*lane, col0 + 32*lane + 32).  E = elements per 16 bytes.
template <typename T>
__device__ __forceinline__ void apply_chunk(T* row, int col0, uint32_t word, int lane) {
    constexpr int E = 16 / sizeof(T);
    constexpr int PASSES = 1024 / E / 32;
    constexpr uint32_t FULLBITS = (1u << E) - 1u;
    uint4 ninf = make_uint4(NegInf<T>::pair, NegInf<T>::pair, NegInf<T>::pair, NegInf<T>::pair);
#pragma unroll
    for (int k = 0; k < PASSES; k++) {
        int c = k * 32 + lane;                      // 16-byte chunk index within the 1024 columns
        int wsrc = (c * E) >> 5;
        int sh = (c * E) & 31;
        uint32_t bits = (__shfl_sync(FULL, word, wsrc) >> sh) & FULLBITS;
        // a 32-byte sector (this lane's 16 bytes and its neighbour's) is written whole or not
        // at all, so the L2 never holds a partly written sector (read-modify-write on eviction)
        bool keep = (bits & __shfl_xor_sync(FULL, bits, 1)) == FULLBITS;
        T* p = row + col0 + c * E;
        if (bits == 0) {
            st_cs_v4(p, ninf);
        } else if (!keep) {
            uint4 v = *reinterpret_cast<const uint4*>(p);
            uint32_t w[4] = {v.x, v.y, v.z, v.w};
            if (sizeof(T) == 2) {
#pragma unroll
                for (int e = 0; e < 8; e++)
                    if (!((bits >> e) & 1)) {
                        uint32_t& x = w[e >> 1];
                        x = (e & 1) ? ((x & 0x0000FFFFu) | 0xFF800000u) : ((x & 0xFFFF0000u) | 0x0000FF80u);
                    }
            } else {
#pragma unroll
                for (int e = 0; e < 4; e++)
                    if (!((bits >> e) & 1)) w[e] = 0xFF800000u;
            }
            *reinterpret_cast<uint4*>(p) = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
}

// element-by-element path for ragged chunks or unaligned rows: each lane
// handles the 32 columns of its own mask word
template <typename T>
__device__ __forceinline__ void apply_chunk_scalar(T* row, int col0, int ncols, uint32_t word, int lane) {
    int c0 = 32 * lane;
    for (int e = 0; e < 32; e++) {
        if (c0 + e >= ncols) break;
        if (!((word >> e) & 1)) row[col0 + c0 + e] = (T)NegInf<T>::one;
    }
}

// Mask source for the apply kernels: a caller bitmask [B][W], or the device
// mask table row picked by the classifier (mid[b]).
struct MaskSrc {
    const uint32_t* bitmask;   // nullable
    const uint32_t* chunks;    // the device mask table (chunk ids + chunks)
    const uint32_t* rows;
    const int32_t* mid;
    int W, nch;
    uint32_t* copy_out;        // nullable: also write the words here ([B][W])
    // word `lane` of 1024-column chunk j of row b (0 past W)
    __device__ __forceinline__ uint32_t word(int b, int j, int lane) const {
        int wi = j * 32 + lane;
        if (wi >= W) return 0u;
        if (bitmask) return __ldg(bitmask + (size_t)b * W + wi);
        uint32_t c = __ldg(rows + (size_t)__ldg(mid + b) * nch + j);
        return __ldg(chunks + (size_t)c * 32 + lane);
    }
};

template <typename T>
__global__ void __launch_bounds__(256) k_apply_rows(T* logits, int64_t stride, MaskSrc M, int B, int V, int vec) {
    int lane = threadIdx.x & 31;
    int gw = (int)((blockIdx.x * (size_t)blockDim.x + threadIdx.x) >> 5);
    int nw = (int)((gridDim.x * (size_t)blockDim.x) >> 5);
    int cpr = (V + 1023) >> 10;
    long total = (long)B * cpr;
    for (long c = gw; c < total; c += nw) {
        int b = (int)(c / cpr);
        int j = (int)(c - (long)b * cpr);
        int col0 = j << 10;
        int wi = (col0 >> 5) + lane;
        uint32_t word = M.word(b, j, lane);
        if (M.copy_out && wi < M.W) M.copy_out[(size_t)b * M.W + wi] = word;
        T* row = logits + (size_t)b * stride;
        int ncols = V - col0;
        if (vec && ncols >= 1024) apply_chunk<T>(row, col0, word, lane);
        else apply_chunk_scalar<T>(row, col0, ncols < 1024 ? ncols : 1024, word, lane);
    }
}

__device__ __forceinline__ float bf16_to_float(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }

// Greedy choice among allowed tokens: one block per row, reads only the
// 16-byte chunks that hold an allowed position.
template <typename T>
__global__ void __launch_bounds__(256) k_argmax_masked(const T* logits, int64_t stride, DevTables D,
                                                       const int32_t* mid, int B, int V, int vec,
                                                       int32_t* tokens) {
    int b = blockIdx.x;
    if (b >= B) return;
    int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarp = blockDim.x >> 5;
    const uint32_t* rowids = D.mrows + (size_t)mid[b] * D.nch;
    const T* row = logits + (size_t)b * stride;
    float best = 0.f;
    int bi = -1;
    auto consider = [&](float v, int i) {
        if (v != v) return;   // NaN never wins
        if (bi < 0 || v > best || (v == best && i < bi)) {
            best = v;
            bi = i;
        }
    };
    constexpr int E = 16 / sizeof(T);
    int cpr = (V + 1023) >> 10;
    for (int j = warp; j < cpr; j += nwarp) {
        int col0 = j << 10;
        int wi = (col0 >> 5) + lane;
        uint32_t word = wi < D.W ? __ldg(D.mchunks + (size_t)__ldg(rowids + j) * 32 + lane) : 0u;
        if (__ballot_sync(FULL, word != 0) == 0) continue;
        int ncols = V - col0;
        if (vec && ncols >= 1024) {
#pragma unroll
            for (int k = 0; k < 1024 / E / 32; k++) {
                int c = k * 32 + lane;
                uint32_t bits = (__shfl_sync(FULL, word, (c * E) >> 5) >> ((c * E) & 31)) & ((1u << E) - 1u);
                if (!bits) continue;
                uint4 v = ld_nc_v4(row + col0 + c * E);
                uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int e = 0; e < E; e++) {
                    if (!((bits >> e) & 1)) continue;
                    float f;
                    if (sizeof(T) == 2) f = bf16_to_float((uint16_t)((w[e >> 1] >> ((e & 1) * 16)) & 0xFFFF));
                    else f = __uint_as_float(w[e]);
                    consider(f, col0 + c * E + e);
                }
            }
        } else {
            for (int e = 0; e < 32; e++) {
                int col = col0 + 32 * lane + e;
                if (col >= V) break;
                if ((word >> e) & 1) {
                    float f = sizeof(T) == 2 ? bf16_to_float((uint16_t)row[col]) : __uint_as_float((uint32_t)row[col]);
                    consider(f, col);
                }
            }
        }
    }
    // warp then block reduction of (best, bi)
    for (int off = 16; off; off >>= 1) {
        float ov = __shfl_down_sync(FULL, best, off);
        int oi = __shfl_down_sync(FULL, bi, off);
        if (oi >= 0 && (bi < 0 || ov > best || (ov == best && oi < bi))) {
            best = ov;
            bi = oi;
        }
    }
    __shared__ float sv[32];
    __shared__ int si[32];
    if (lane == 0) {
        sv[warp] = best;
        si[warp] = bi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < nwarp; w++) {
            if (si[w] >= 0 && (bi < 0 || sv[w] > best || (sv[w] == best && si[w] < bi))) {
                best = sv[w];
                bi = si[w];
            }
        }
        tokens[b] = bi;
    }
}

// Feed one lexeme class to the parser on a row's stack: resolve the class to a
// terminal with the current top, reduce until it is shifted.  Returns a row
// status; `low` becomes the lowest stack index written.
__device__ int feed_class(const DevTables& T, uint16_t* st, int& depth, int cap, int cls, int& low) {
    int top = st[depth - 1];
    int t = T.resolve[(size_t)cls * T.n_lr + top];
    if (t < 0) return ROW_REJECTED;
    for (int guard = 0; guard < 4 * cap + 64; guard++) {
        int32_t a = T.action[(size_t)st[depth - 1] * T.n_terms + t];
        int kind = a & 3, val = a >> 2;
        if (kind == psc::ACT_SHIFT) {
            if (depth >= cap) return ROW_OVERFLOW;
            low = depth < low ? depth : low;
            st[depth++] = (uint16_t)val;
            return ROW_OK;
        }
        if (kind != psc::ACT_REDUCE) return ROW_REJECTED;
        int k = T.rule_len[val];
        if (depth - k < 1) return ROW_REJECTED;
        depth -= k;
        int go = T.go[(size_t)st[depth - 1] * T.n_nts + T.rule_lhs[val]];
        if (go < 0) return ROW_REJECTED;
        if (depth >= cap) return ROW_OVERFLOW;
        low = depth < low ? depth : low;
        st[depth++] = (uint16_t)go;
    }
    return ROW_LIMIT;
}

// Re-reads stack entries [from, depth) of one row through the bottom-up
// classifier, keeping its block after every prefix (memo[i]: stack [0, i]);
// returns the block of the whole stack, or -1 (unknown: the stack is then
// walked from the top).  Entries below `from` are unchanged since they were kept.
__device__ int memo_extend(const DevTables& T, const uint16_t* st, int32_t* memo, int from, int depth) {
    int e;
    if (from <= 0) {
        e = st[0] == 0 ? 0 : -1;
        memo[0] = e;
        from = 1;
    } else {
        e = memo[from - 1];
    }
    for (int i = from; i < depth; i++) {
        int t = st[i - 1], u = st[i];
        int k = t < T.n_lr && u < T.n_lr ? T.bu_slot[(size_t)t * T.n_lr + u] : -1;
        e = e >= 0 && k >= 0 && e + 1 + k < T.bu_len ? __ldg(T.bu + e + 1 + k) : -1;
        memo[i] = e;
    }
    return e;
}

// Algorithm 2 steps 1-2 for one row per thread.
__global__ void k_advance(DevTables T, DevStates S, const int32_t* tokens, int B, int use_mid,
                          int32_t* status_out, int from_keys, int32_t* tokens_out) {
    int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= B) return;
    int tok;
    if (from_keys) {   // the greedy choice of the fused masking pass
        unsigned long long k = S.best[b];
        S.best[b] = 0ull;
        tok = k ? (int32_t)(~(uint32_t)(k & 0xFFFFFFFFu)) : -1;
        tokens_out[b] = tok;
    } else {
        tok = tokens[b];
    }
    int status = S.status[b];
    if (tok >= 0) {
        if (status == ROW_DONE) {
            status = tok == T.eos_id ? ROW_DONE : ROW_REJECTED;
        } else if (status == ROW_OK) {
            if (tok >= T.V) {
                status = ROW_REJECTED;
            } else {
                int mid = use_mid ? S.mid[b] : thread_classify(T, S, b);
                bool allowed = (mask_word(T, mid, tok >> 5) >> (tok & 31)) & 1;
                if (!allowed) {
                    status = ROW_REJECTED;
                } else if (tok == T.eos_id) {
                    status = ROW_DONE;
                } else {
                    int q = S.q[b], depth = S.depth[b], low = 0x7FFFFFFF;
                    uint16_t* st = S.stack + (size_t)b * S.cap;
                    int64_t lo = T.vocab_off[tok], hi = T.vocab_off[tok + 1];
                    for (int64_t i = lo; i < hi && status == ROW_OK; i++) {
                        int c = T.vocab[i];
                        int nx = T.lex_trans[(size_t)q * 256 + c];
                        if (nx >= 0) {
                            q = nx;
                            continue;
                        }
                        int cls = q == T.q0 ? -1 : T.lex_accept[q];
                        if (cls < 0) {
                            status = ROW_REJECTED;
                            break;
                        }
                        if (!T.cls_ignored[cls]) status = feed_class(T, st, depth, S.cap, cls, low);
                        q = T.lex_trans[(size_t)T.q0 * 256 + c];
                        if (q < 0) status = ROW_REJECTED;
                    }
                    if (status == ROW_OK) {
                        S.q[b] = q;
                        S.depth[b] = depth;
                        if (S.rmemo && T.bu)
                            memo_extend(T, st, S.rmemo + (size_t)b * S.cap, low < depth ? low : depth, depth);
                    }
                }
            }
        }
        S.status[b] = status;
    }
    if (status_out) status_out[b] = status;
}


// ------------------------------------------------ fused masking + greedy choice
// Orderable 32-bit key of a float (larger float -> larger key; -0 == +0).
__device__ __forceinline__ uint32_t f32_order(uint32_t u) {
    if ((u & 0x7FFFFFFFu) == 0) u = 0;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// 64-bit greedy key: value order in the high word, then the lowest column wins.
__device__ __forceinline__ unsigned long long make_key(uint32_t ordered, int col) {
    return ((unsigned long long)ordered << 32) | (uint32_t)(~(uint32_t)col);
}

// Greedy state of one lane: the largest allowed value seen so far and the
// lowest column holding it (col < 0: nothing yet).  NaN never becomes best.
struct Best {
    float val;
    int col;
};

__device__ __forceinline__ void note_best(Best& best, float v, int col) {
    if (best.col < 0 || v > best.val || (v == best.val && col < best.col)) {
        best.val = v;
        best.col = col;
    }
}

__device__ __forceinline__ unsigned long long best_key_of(const Best& b) {
    return b.col >= 0 ? make_key(f32_order(__float_as_uint(b.val)), b.col) : 0ull;
}

// Allowed-position masks of one 16-byte piece, indexed by its mask bits:
// bf16 (8 bits -> 0xFFFF per allowed half of the 4 words), f32 (4 bits ->
// 0xFFFFFFFF per allowed word).  Built in shared memory by every CTA.
template <typename T>
__device__ __forceinline__ void build_allow_lut(uint4* lut) {
    constexpr int N = sizeof(T) == 2 ? 256 : 16;
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
        uint32_t w[4];
        for (int k = 0; k < 4; k++) {
            if (sizeof(T) == 2)
                w[k] = (((i >> (2 * k)) & 1) ? 0x0000FFFFu : 0u) | (((i >> (2 * k + 1)) & 1) ? 0xFFFF0000u : 0u);
            else
                w[k] = ((i >> k) & 1) ? 0xFFFFFFFFu : 0u;
        }
        lut[i] = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

__device__ __forceinline__ uint32_t sel_ninf(uint32_t w, uint32_t allow, uint32_t ninf) {
    return (w & allow) | (ninf & ~allow);
}

__device__ __forceinline__ float bf16_at(uint32_t w, int half) {
    return __uint_as_float(half ? (w & 0xFFFF0000u) : (w << 16));
}

// One 1024-column chunk of bf16: write -inf where masked (no read when the
// whole 16-byte piece is masked), read the pieces that hold an allowed
// position and fold their allowed values into the lane's best with packed
// bf16x2 maxima; the column is searched only when the piece can win.
__device__ __forceinline__ void apply_argmax_chunk_bf16(const uint16_t* src, uint16_t* row, int col0, uint32_t word, int lane,
                                                        Best& best, const uint4* lut) {
    const uint4 ninf = make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
    uint32_t bits[4];
    uint4 v[4];
#pragma unroll
    for (int k = 0; k < 4; k++) bits[k] = (__shfl_sync(FULL, word, k * 8 + (lane >> 2)) >> ((lane & 3) * 8)) & 0xFFu;
#pragma unroll
    for (int k = 0; k < 4; k++)   // issue every needed load before any store
        if (bits[k]) v[k] = *reinterpret_cast<const uint4*>(src + (k * 32 + lane) * 8);
#pragma unroll
    for (int k = 0; k < 4; k++) {
        uint16_t* p = row + col0 + (k * 32 + lane) * 8;
        uint32_t bk = bits[k];
        if (bk == 0) {
            st_cs_v4(p, ninf);
            continue;
        }
        uint4 am = lut[bk];
        uint32_t x0 = sel_ninf(v[k].x, am.x, 0xFF80FF80u), x1 = sel_ninf(v[k].y, am.y, 0xFF80FF80u);
        uint32_t x2 = sel_ninf(v[k].z, am.z, 0xFF80FF80u), x3 = sel_ninf(v[k].w, am.w, 0xFF80FF80u);
        __nv_bfloat162 m = __hmax2(__hmax2(*reinterpret_cast<__nv_bfloat162*>(&x0), *reinterpret_cast<__nv_bfloat162*>(&x1)),
                                   __hmax2(*reinterpret_cast<__nv_bfloat162*>(&x2), *reinterpret_cast<__nv_bfloat162*>(&x3)));
        float mf = fmaxf(__low2float(m), __high2float(m));
        if (best.col < 0 || mf >= best.val) {   // rare: this piece may hold the lane's best
            uint32_t w[4] = {v[k].x, v[k].y, v[k].z, v[k].w};
#pragma unroll
            for (int e = 0; e < 8; e++) {
                float f = bf16_at(w[e >> 1], e & 1);
                if (((bk >> e) & 1) && f == mf) {
                    note_best(best, f, col0 + (k * 32 + lane) * 8 + e);
                    break;
                }
            }
        }
        st_cs_v4(p, make_uint4(x0, x1, x2, x3));   // whole pieces: no partly written sectors
    }
}

// One 1024-column chunk of f32 (4 elements per 16-byte piece), in two halves of
// four pieces per lane (eight pieces and their bits at once exceed the register
// budget of three resident CTAs).
__device__ __forceinline__ void apply_argmax_chunk_f32(const uint32_t* src, uint32_t* row, int col0, uint32_t word, int lane,
                                                       Best& best, const uint4* lut) {
    const uint4 ninf = make_uint4(0xFF800000u, 0xFF800000u, 0xFF800000u, 0xFF800000u);
#pragma unroll 1
    for (int h = 0; h < 8; h += 4) {
        uint32_t bits[4];
        uint4 v[4];
#pragma unroll
        for (int k = 0; k < 4; k++)
            bits[k] = (__shfl_sync(FULL, word, (h + k) * 4 + (lane >> 3)) >> ((lane & 7) * 4)) & 0xFu;
#pragma unroll
        for (int k = 0; k < 4; k++)
            if (bits[k]) v[k] = *reinterpret_cast<const uint4*>(src + ((h + k) * 32 + lane) * 4);
#pragma unroll
        for (int k = 0; k < 4; k++) {
            uint32_t* p = row + col0 + ((h + k) * 32 + lane) * 4;
            uint32_t bk = bits[k];
            if (bk == 0) {
                st_cs_v4(p, ninf);
                continue;
            }
            uint4 am = lut[bk];
            uint32_t x0 = sel_ninf(v[k].x, am.x, 0xFF800000u), x1 = sel_ninf(v[k].y, am.y, 0xFF800000u);
            uint32_t x2 = sel_ninf(v[k].z, am.z, 0xFF800000u), x3 = sel_ninf(v[k].w, am.w, 0xFF800000u);
            float mf = fmaxf(fmaxf(__uint_as_float(x0), __uint_as_float(x1)), fmaxf(__uint_as_float(x2), __uint_as_float(x3)));
            if (best.col < 0 || mf >= best.val) {
                uint32_t w[4] = {v[k].x, v[k].y, v[k].z, v[k].w};
#pragma unroll
                for (int e = 0; e < 4; e++) {
                    float f = __uint_as_float(w[e]);
                    if (((bk >> e) & 1) && f == mf) {
                        note_best(best, f, col0 + ((h + k) * 32 + lane) * 4 + e);
                        break;
                    }
                }
            }
            st_cs_v4(p, make_uint4(x0, x1, x2, x3));
        }
    }
}

// Greedy state of a lane that streams bf16 chunks: the largest allowed value
// seen so far and the 16-byte piece holding its first occurrence (the piece's
// values and mask bits), resolved to a column once per work item.  The per-piece
// update is a handful of selects, so no lane diverges while it streams.
struct BestPiece {
    float val;       // -inf until an allowed value is seen
    int col;         // first column of the piece (-1: nothing yet)
    uint32_t bits;   // the piece's mask bits
    uint4 x;         // the piece's values
};

__device__ __forceinline__ BestPiece best_piece_none() {
    return BestPiece{-INFINITY, -1, 0u, make_uint4(0u, 0u, 0u, 0u)};
}

// Column and key of the piece's first allowed value equal to the best.
__device__ __forceinline__ unsigned long long best_piece_key_bf16(const BestPiece& bp) {
    if (bp.col < 0) return 0ull;
    uint32_t w[4] = {bp.x.x, bp.x.y, bp.x.z, bp.x.w};
    int at = 0;
#pragma unroll
    for (int e = 7; e >= 0; e--)
        if (((bp.bits >> e) & 1) && bf16_at(w[e >> 1], e & 1) == bp.val) at = e;
    return make_key(f32_order(__float_as_uint(bp.val)), bp.col + at);
}

// A lane's four 16-byte pieces of a bf16 chunk in registers: the mask bits of
// each piece and its values with -inf where masked.
struct ChunkRegs {
    uint32_t bits[4];
    uint4 x[4];
};

// Reads the lane's pieces of one 1024-column bf16 chunk from shared memory
// (pieces with nothing allowed are not read) and masks them.  The stage may be
// handed back as soon as this returns.
__device__ __forceinline__ void load_mask_chunk_bf16(const uint16_t* src, uint32_t word, int lane, const uint4* lut,
                                                     ChunkRegs& r) {
    uint4 v[4];
#pragma unroll
    for (int k = 0; k < 4; k++) r.bits[k] = (__shfl_sync(FULL, word, k * 8 + (lane >> 2)) >> ((lane & 3) * 8)) & 0xFFu;
#pragma unroll
    for (int k = 0; k < 4; k++)
        v[k] = r.bits[k] ? *reinterpret_cast<const uint4*>(src + (k * 32 + lane) * 8) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
    for (int k = 0; k < 4; k++) {
        uint4 am = lut[r.bits[k]];
        r.x[k] = make_uint4(sel_ninf(v[k].x, am.x, 0xFF80FF80u), sel_ninf(v[k].y, am.y, 0xFF80FF80u),
                            sel_ninf(v[k].z, am.z, 0xFF80FF80u), sel_ninf(v[k].w, am.w, 0xFF80FF80u));
    }
}

// Folds a masked chunk into the lane's best piece with packed bf16x2 maxima (NaN
// never wins: the maximum returns the other operand) and writes it to the row
// (32-byte sectors with every token allowed are left as they are).
// Every lane runs the same instructions for every piece; only a piece whose
// allowed values are all -inf or NaN, met before any other allowed value, takes
// a short scalar path.
__device__ __forceinline__ void fold_store_chunk_bf16(uint16_t* row, int col0, int lane, const ChunkRegs& r,
                                                      BestPiece& bp) {
#pragma unroll
    for (int k = 0; k < 4; k++) {
        uint32_t bk = r.bits[k];
        uint32_t x0 = r.x[k].x, x1 = r.x[k].y, x2 = r.x[k].z, x3 = r.x[k].w;
        __nv_bfloat162 m = __hmax2(__hmax2(*reinterpret_cast<__nv_bfloat162*>(&x0), *reinterpret_cast<__nv_bfloat162*>(&x1)),
                                   __hmax2(*reinterpret_cast<__nv_bfloat162*>(&x2), *reinterpret_cast<__nv_bfloat162*>(&x3)));
        float mf = fmaxf(__low2float(m), __high2float(m));
        int pc = col0 + (k * 32 + lane) * 8;
        bool upd = mf > bp.val;
        if (!upd && bk != 0u && bp.col < 0) {
            // nothing allowed seen yet and this piece's allowed values are -inf or NaN:
            // an allowed -inf is still a valid choice
#pragma unroll
            for (int e = 0; e < 8; e++) {
                uint32_t wv = e < 2 ? x0 : e < 4 ? x1 : e < 6 ? x2 : x3;
                if (((bk >> e) & 1) && bf16_at(wv, e & 1) == -INFINITY) upd = true;
            }
        }
        bp.val = upd ? mf : bp.val;
        bp.col = upd ? pc : bp.col;
        bp.bits = upd ? bk : bp.bits;
        bp.x.x = upd ? x0 : bp.x.x;
        bp.x.y = upd ? x1 : bp.x.y;
        bp.x.z = upd ? x2 : bp.x.z;
        bp.x.w = upd ? x3 : bp.x.w;
        // a 32-byte sector (this lane's piece and its neighbour's) is written whole or not
        // at all: a partly written sector costs a read-modify-write when the L2 evicts it.
        // Only sectors whose 16 tokens are all allowed stay as they are.
        uint32_t pair = bk & __shfl_xor_sync(FULL, bk, 1);
        if (pair != 0xFFu) st_cs_v4(row + pc, r.x[k]);
    }
}

template <typename T>
__device__ __forceinline__ void apply_argmax_chunk_scalar(T* row, int col0, int ncols, uint32_t word, int lane,
                                                          Best& best) {
    int c0 = 32 * lane;
    for (int e = 0; e < 32; e++) {
        if (c0 + e >= ncols) break;
        int col = col0 + c0 + e;
        if (!((word >> e) & 1)) {
            row[col] = (T)NegInf<T>::one;
        } else {
            float f = sizeof(T) == 2 ? __uint_as_float((uint32_t)row[col] << 16) : __uint_as_float((uint32_t)row[col]);
            if (!isnan(f)) note_best(best, f, col);
        }
    }
}

template <typename T>
__device__ __forceinline__ void apply_argmax_any(T* row, int col0, int V, uint32_t word, int lane, int vec, Best& best,
                                                 const uint4* lut) {
    int ncols = V - col0;
    if (vec && ncols >= 1024) {
        if (sizeof(T) == 2)
            apply_argmax_chunk_bf16(reinterpret_cast<uint16_t*>(row) + col0, reinterpret_cast<uint16_t*>(row), col0,
                                    word, lane, best, lut);
        else
            apply_argmax_chunk_f32(reinterpret_cast<uint32_t*>(row) + col0, reinterpret_cast<uint32_t*>(row), col0,
                                   word, lane, best, lut);
    } else {
        apply_argmax_chunk_scalar<T>(row, col0, ncols < 1024 ? ncols : 1024, word, lane, best);
    }
}

// Fused masking + greedy choice.  Work item = (row, segment of seg_chunks
// 1024-column chunks); the 8 warps of a CTA split a segment, reduce their keys
// in shared memory, and one 64-bit atomic max per item merges the row's best.
// WALK: the CTA classifies its rows itself (Algorithm 2 step 3): warp 0 walks
// the classifier for the next item's row while the CTA streams the current
// item, chunks being handed out through a shared counter so that warp 0 joins
// once its walk is done; the segment-0 CTA of a row records the row's mask id.
// Per-row keys must be zero on entry (state init, finalize and advance clear them).
template <typename T, bool WALK>
__global__ void __launch_bounds__(256, 4) k_apply_argmax(T* logits, int64_t stride, MaskSrc M, int B, int V, int vec,
                                                         int seg_chunks, unsigned long long* __restrict__ best_key,
                                                         DevTables D, DevStates S) {
    __shared__ unsigned long long red[8];
    __shared__ int s_mid[2];
    __shared__ int s_ctr;
    __shared__ uint4 s_lut[256];
    int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int cpr = (V + 1023) >> 10;
    int nseg = (cpr + seg_chunks - 1) / seg_chunks;
    long items = (long)B * nseg;
    int cur = 0;
    build_allow_lut<T>(s_lut);
    __syncthreads();
    if (WALK) {
        if (warp == 0 && (long)blockIdx.x < items) {
            int m = warp_classify(D, S, (int)(blockIdx.x / nseg), lane);
            if (lane == 0) s_mid[0] = m;
        }
        if (threadIdx.x == 0) s_ctr = 0;
        __syncthreads();
    }
    for (long it = blockIdx.x; it < items; it += gridDim.x) {
        int b = (int)(it / nseg);
        int sg = (int)(it - (long)b * nseg);
        int c0 = sg * seg_chunks;
        int c1 = min(c0 + seg_chunks, cpr);
        int wmid = 0;
        if (WALK) {
            wmid = s_mid[cur];
            if (sg == 0 && threadIdx.x == 0) S.mid[b] = wmid;
        }
        // word `lane` of chunk j of this row's mask
        auto word_at = [&](int j) -> uint32_t {
            if (!WALK) return M.word(b, j, lane);
            int wi = j * 32 + lane;
            return wi < D.W ? __ldg(D.mchunks + (size_t)__ldg(D.mrows + (size_t)wmid * D.nch + j) * 32 + lane) : 0u;
        };
        T* row = logits + (size_t)b * stride;
        Best best{0.f, -1};
        if (WALK) {
            long nx = it + gridDim.x;
            if (warp == 0 && nx < items) {
                int m = warp_classify(D, S, (int)(nx / nseg), lane);
                if (lane == 0) s_mid[cur ^ 1] = m;
            }
            for (;;) {
                int j = 0;
                if (lane == 0) j = atomicAdd(&s_ctr, 1);
                j = __shfl_sync(FULL, j, 0) + c0;
                if (j >= c1) break;
                int col0 = j << 10;
                int wi = (col0 >> 5) + lane;
                uint32_t word = word_at(j);
                if (M.copy_out && wi < M.W) M.copy_out[(size_t)b * M.W + wi] = word;
                apply_argmax_any<T>(row, col0, V, word, lane, vec, best, s_lut);
            }
        } else {
            for (int j = c0 + warp; j < c1; j += 8) {
                int col0 = j << 10;
                int wi = (col0 >> 5) + lane;
                uint32_t word = word_at(j);
                if (M.copy_out && wi < M.W) M.copy_out[(size_t)b * M.W + wi] = word;
                apply_argmax_any<T>(row, col0, V, word, lane, vec, best, s_lut);
            }
        }
        unsigned long long key = best_key_of(best);
#pragma unroll
        for (int off = 16; off; off >>= 1) {
            unsigned long long o = __shfl_xor_sync(FULL, key, off);
            key = o > key ? o : key;
        }
        if (lane == 0) red[warp] = key;
        __syncthreads();
        if (threadIdx.x == 0) {
            unsigned long long k = red[0];
            for (int w = 1; w < 8; w++) k = red[w] > k ? red[w] : k;
            if (k) atomicMax(best_key + b, k);
            if (WALK) s_ctr = 0;
        }
        cur ^= 1;
        __syncthreads();
    }
}

__global__ void k_finalize_tokens(unsigned long long* __restrict__ best_key, int B, int32_t* tokens) {
    int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= B) return;
    unsigned long long k = best_key[b];
    tokens[b] = k ? (int32_t)(~(uint32_t)(k & 0xFFFFFFFFu)) : -1;
    best_key[b] = 0ull;
}

// ------------------------------------------- advance with staged tables
// One warp per row.  The compact lexer/parser tables (int16 entries, byte
// classes for the lexer) are staged in shared memory by one bulk copy per CTA,
// and the top ADV_KEEP entries of the row's stack are copied into a per-warp
// window, so the parser's dependent reads are shared-memory reads.  After the
// token is consumed the warp classifies the new configuration (Algorithm 2 step
// 3: the bottom-up classifier from the lowest stack entry written, or a walk when
// it is not built) and stores the row's mask id for the next masking pass.
constexpr int ADV_WARPS = 8;     // rows per CTA
constexpr int ADV_WIN = 256;     // stack entries held per row
constexpr int ADV_KEEP = 192;    // entries copied in (the rest is room for pushes)
constexpr size_t ADV_TABLE_MAX = 200 * 1024;   // staged tables at most (one CTA of 8 rows per SM)

// Dynamic shared memory of k_advance_warp: the staged tables, then the stack windows.
int adv_smem(const DevTables& d) { return d.adv_bytes + ADV_WARPS * ADV_WIN * 2; }

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
// Global-window address of a device pointer, for the source operand of bulk copies
// (the same value for cudaMalloc memory; the conversion makes the state space explicit).
__device__ __forceinline__ uint64_t gmem_addr(const void* p) {
    return static_cast<uint64_t>(__cvta_generic_to_global(p));
}

// Programmatic dependent launch: the next kernel of the stream may be scheduled
// now (it waits for this grid's results with grid_dep_wait); and the wait for
// the previous kernel's results (returns at once when there is none to wait for).
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// psc_state_copy: every array of one batch's states into another's in one launch,
// once the previous kernel on the stream has completed (16-byte copies; a
// segment's bytes past its last whole 16 one by one; every segment starts on an
// allocation of its own, so 16-byte aligned).
struct CopySegs {
    const uint8_t* src[8];
    uint8_t* dst[8];
    unsigned long long bytes[8];
    int n;
};
__global__ void k_state_copy(CopySegs c) {
    grid_dep_wait();
    grid_dep_launch();
    const size_t tid = blockIdx.x * (size_t)blockDim.x + threadIdx.x, nt = (size_t)gridDim.x * blockDim.x;
    for (int k = 0; k < c.n; k++) {
        const size_t n16 = c.bytes[k] / 16;
        const uint4* src = reinterpret_cast<const uint4*>(c.src[k]);
        uint4* dst = reinterpret_cast<uint4*>(c.dst[k]);
        for (size_t i = tid; i < n16; i += nt) dst[i] = src[i];
        for (size_t i = n16 * 16 + tid; i < c.bytes[k]; i += nt) c.dst[k][i] = c.src[k][i];
    }
}

// Bounded wait on phase 0 of an mbarrier; returns false if it did not complete.
__device__ __forceinline__ bool mbar_wait0(uint32_t bar, int limit) {
    for (int it = 0; it < limit; it++) {
        uint32_t ok;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\n selp.u32 %0, 1, 0, p;\n}"
            : "=r"(ok)
            : "r"(bar)
            : "memory");
        if (ok) return true;
    }
    return false;
}

// Shared-memory loads and stores by 32-bit shared-window address.  The parser's
// table reads are chains of dependent loads, one lane at a time: naming the state
// space keeps each one a plain shared-memory access.
__device__ __forceinline__ int lds_s16(uint32_t a) {
    short v;
    asm volatile("ld.shared.s16 %0, [%1];" : "=h"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ int lds_u16(uint32_t a) {
    unsigned short v;
    asm volatile("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ int lds_u8(uint32_t a) {
    unsigned short v;
    asm volatile("ld.shared.u8 %0, [%1];" : "=h"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ int lds_s32(uint32_t a) {
    int v;
    asm volatile("ld.shared.s32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t lds_u32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ void sts_u16(uint32_t a, int v) {
    asm volatile("st.shared.u16 [%0], %1;" ::"r"(a), "h"((unsigned short)v) : "memory");
}

// A row's stack seen through its window: indices in [base, base + ADV_WIN) live
// in shared memory (at shared address wa), the others in global memory.  `lo`
// tracks the lowest index written (for the write-back and the bottom-up classifier).
struct StackView {
    uint16_t* win;
    uint16_t* st;
    int base;
    int lo;
    uint32_t wa;   // shared-window address of win
    __device__ __forceinline__ bool in_win(int i) const { return (unsigned)(i - base) < (unsigned)ADV_WIN; }
    __device__ __forceinline__ int get(int i) const { return in_win(i) ? lds_u16(wa + 2u * (i - base)) : st[i]; }
    __device__ __forceinline__ void set(int i, int v) {
        if (in_win(i)) sts_u16(wa + 2u * (i - base), v);
        else st[i] = (uint16_t)v;
        lo = i < lo ? i : lo;
    }
};

// Shared-window addresses of the compact lexer/parser tables staged by
// k_advance_warp, and their row strides in bytes.
struct AdvTabs {
    uint32_t bc, trans, acc, ign, res, act, go, rlen, rlhs;
    uint32_t trans_row, res_row, act_row, go_row;   // bytes per row: nbc, n_lr, n_terms, n_nts int16 entries
    uint32_t cand, abase, gbase, acmb, gcmb;       // packed layout
    int q0, kc;
    __device__ __forceinline__ AdvTabs(uint32_t sb, const DevTables& T)
        : bc(sb + T.o_bc), trans(sb + T.o_trans), acc(sb + T.o_accept), ign(sb + T.o_ign), res(sb + T.o_resolve),
          act(sb + T.o_action), go(sb + T.o_go), rlen(sb + T.o_rlen), rlhs(sb + T.o_rlhs),
          trans_row(2u * T.nbc), res_row(2u * T.n_lr), act_row(2u * T.n_terms), go_row(2u * T.n_nts),
          cand(sb + T.o_cand), abase(sb + T.o_abase), gbase(sb + T.o_gbase), acmb(sb + T.o_acmb),
          gcmb(sb + T.o_gcmb), q0(T.q0), kc(T.kc) {}
};

// Feed one lexeme class to the parser: resolve it to a terminal with the
// current top (contextual lexing), reduce until it is shifted.  Returns a row
// status.  `top` and `below` hold the two topmost entries in registers: a
// reduction of one symbol (the chains of unit rules) uncovers `below`, so it
// reads no stack entry; only a reduction of two or more symbols reads one.
// PACKED: reduce entries carry (rule length << 10 | left-hand side); then a run
// of one-symbol reductions takes a short loop (one action and one goto lookup
// each, the goto row of `below` fixed for the run) and the new top is written
// to the stack once, when the run ends (not at all when a longer reduction then
// pops it).
template <bool PACKED>
__device__ __forceinline__ int feed_class_win(const AdvTabs& A, StackView& sv, int& depth, int& top, int& below,
                                              int cap, int cls) {
    int t = lds_s16(A.res + cls * A.res_row + 2u * top);
    if (t < 0) return ROW_REJECTED;
    const uint32_t col = A.act + 2u * t;   // ACTION[.][t]
    bool dirty = false;                     // top changed by one-symbol reductions, not yet on the stack
    for (int guard = 0; guard < 4 * cap + 64; guard++) {
        int a = lds_s16(col + top * A.act_row);
        if (PACKED) {
            // packed unit reduction: kind REDUCE, rule length 1 (bits 12-15), lhs in bits 2-11
            const uint32_t go_below = A.go + below * A.go_row;
            while ((a & 0xF003) == 0x1002 && depth >= 2) {
                int g = lds_s16(go_below + ((a >> 1) & 0x7FE));   // GOTO[below][lhs], 2 * lhs = (a >> 1) & 0x7FE
                if (g < 0) return ROW_REJECTED;
                if (++guard >= 4 * cap + 64) return ROW_LIMIT;
                top = g;
                dirty = true;
                a = lds_s16(col + top * A.act_row);
            }
        }
        int kind = a & 3, val = (a >> 2) & 0x3FFF;
        if (kind == psc::ACT_SHIFT) {
            if (depth >= cap) return ROW_OVERFLOW;
            if (dirty) sv.set(depth - 1, top);
            sv.set(depth++, val);
            below = top;
            top = val;
            return ROW_OK;
        }
        if (kind != psc::ACT_REDUCE) return ROW_REJECTED;
        int k, lhs;
        if (PACKED) {
            k = val >> 10;
            lhs = val & 1023;
        } else {
            k = lds_u8(A.rlen + val);
            lhs = lds_s16(A.rlhs + 2u * val);
        }
        if (depth - k < 1) return ROW_REJECTED;
        if (k == 0 && dirty) sv.set(depth - 1, top);   // an empty rule pushes above the current top
        dirty = false;
        depth -= k;
        // the entry the reduction uncovers: the one below the top (k = 1), the top
        // itself (k = 0), else read from the stack
        int under;
        if (k == 1) under = below;
        else if (k == 0) under = top;
        else under = sv.get(depth - 1);
        int g = lds_s16(A.go + under * A.go_row + 2u * lhs);
        if (g < 0) return ROW_REJECTED;
        if (depth >= cap) return ROW_OVERFLOW;
        sv.set(depth++, g);
        below = under;
        top = g;
    }
    return ROW_LIMIT;
}

// Entry x of a packed table's row (w = the state's word, row id << 17 | base): the
// int16 entry when the slot belongs to the row, else `miss` (an ACTION error is 0,
// a missing GOTO -1).
__device__ __forceinline__ int comb_get(uint32_t tab, uint32_t w, int x, int miss) {
    uint32_t e = lds_u32(tab + 4u * ((w & 0x1FFFFu) + (uint32_t)x));
    return (e >> 16) == (w >> 17) ? (int)(int16_t)(e & 0xFFFFu) : miss;
}

// feed_class_win over the packed tables: the class is resolved by trying its
// candidate terminals in order (the first with an action in the top state); the
// ACTION word of the top stays in a register, each GOTO lookup first reads the
// word of the uncovered state (once per run of one-symbol reductions).
template <bool PACKED>
__device__ __forceinline__ int feed_class_comb(const AdvTabs& A, StackView& sv, int& depth, int& top, int& below,
                                               int cap, int cls) {
    uint32_t tw = lds_u32(A.abase + 4u * top);
    int t = -1, a = 0;
    for (int k = 0; k < A.kc; k++) {
        int c = lds_s16(A.cand + 2u * (cls * A.kc + k));
        if (c < 0) break;
        a = comb_get(A.acmb, tw, c, 0);
        if ((a & 3) != psc::ACT_ERR) {
            t = c;
            break;
        }
    }
    if (t < 0) return ROW_REJECTED;
    bool dirty = false;
    for (int guard = 0; guard < 4 * cap + 64; guard++) {
        if (guard > 0) a = comb_get(A.acmb, tw, t, 0);
        if (PACKED && (a & 0xF003) == 0x1002 && depth >= 2) {
            const uint32_t bw = lds_u32(A.gbase + 4u * below);
            do {   // one-symbol reductions: GOTO[below][lhs], lhs in bits 2-11
                int g = comb_get(A.gcmb, bw, (a >> 2) & 1023, -1);
                if (g < 0) return ROW_REJECTED;
                if (++guard >= 4 * cap + 64) return ROW_LIMIT;
                top = g;
                dirty = true;
                tw = lds_u32(A.abase + 4u * top);
                a = comb_get(A.acmb, tw, t, 0);
            } while ((a & 0xF003) == 0x1002);
        }
        int kind = a & 3, val = (a >> 2) & 0x3FFF;
        if (kind == psc::ACT_SHIFT) {
            if (depth >= cap) return ROW_OVERFLOW;
            if (dirty) sv.set(depth - 1, top);
            sv.set(depth++, val);
            below = top;
            top = val;
            return ROW_OK;
        }
        if (kind != psc::ACT_REDUCE) return ROW_REJECTED;
        int k, lhs;
        if (PACKED) {
            k = val >> 10;
            lhs = val & 1023;
        } else {
            k = lds_u8(A.rlen + val);
            lhs = lds_s16(A.rlhs + 2u * val);
        }
        if (depth - k < 1) return ROW_REJECTED;
        if (k == 0 && dirty) sv.set(depth - 1, top);
        dirty = false;
        depth -= k;
        int under;
        if (k == 1) under = below;
        else if (k == 0) under = top;
        else under = sv.get(depth - 1);
        int g = comb_get(A.gcmb, lds_u32(A.gbase + 4u * under), lhs, -1);
        if (g < 0) return ROW_REJECTED;
        if (depth >= cap) return ROW_OVERFLOW;
        sv.set(depth++, g);
        below = under;
        top = g;
        tw = lds_u32(A.abase + 4u * top);
    }
    return ROW_LIMIT;
}

template <bool PACKED, bool COMB>
__device__ __forceinline__ int feed_class(const AdvTabs& A, StackView& sv, int& depth, int& top, int& below, int cap,
                                          int cls) {
    if (COMB) return feed_class_comb<PACKED>(A, sv, depth, top, below, cap, cls);
    return feed_class_win<PACKED>(A, sv, depth, top, below, cap, cls);
}

// Classifier walk of a configuration (lexer state q, stack of the given depth
// read through the view) by a full warp: lanes fetch 32 stack symbols at a time,
// the walk broadcasts them with shuffles.  Every lane returns the mask id.
// 4-byte read-only load with an L2 cache policy (the classifier table: its lines are
// kept in L2 ahead of the logits the masking pass streams through it).
__device__ __forceinline__ int ld_keep(const int32_t* p, uint64_t pol) {
    int v;
    asm volatile("ld.global.nc.L2::cache_hint.b32 %0, [%1], %2;" : "=r"(v) : "l"(p), "l"(pol));
    return v;
}
__device__ __forceinline__ int warp_walk(const DevTables& T, const StackView& sv, int q, int depth, int lane) {
    if (q < 0 || q >= T.nq || depth < 1) return 0;
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    int s = __ldg(T.dfa_start + q);
    if (s < 0) return -s - 1;
    for (int top = depth - 1; top >= 0; top -= 32) {
        int i = top - lane;
        int x = i >= 0 ? sv.get(i) : 0;
        int n = top + 1 < 32 ? top + 1 : 32;
        for (int j = 0; j < n; j++) {
            int X = __shfl_sync(FULL, x, j);
            if ((unsigned)X >= (unsigned)T.n_lr) return 0;
            int nx = T.dfa_sparse ? sparse_step_warp(T.dfa_rows, s, X, lane) : ld_keep(T.dfa + (size_t)s * T.n_lr + X, pol);
            if (nx < 0) return -nx - 1;
            s = nx;
        }
    }
    return state_mask(T, s);
}

// memo_extend by a full warp: lanes fetch the edge slots of 32 entries at a
// time, the chain of block loads follows them (broadcast by shuffles), and each
// lane stores the block of its own entry.  e_below = block of stack [0, from-1]
// (ignored when from == 0).  Every lane returns the block of the whole stack.
__device__ __forceinline__ int warp_memo_extend(const DevTables& T, const StackView& sv, int32_t* memo, int from,
                                                int depth, int e_below, int lane) {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    int e = e_below;
    if (from <= 0) {
        e = sv.get(0) == 0 ? 0 : -1;
        if (lane == 0) memo[0] = e;
        from = 1;
    }
    for (int i0 = from; i0 < depth; i0 += 32) {
        int i = i0 + lane;
        int k = -1;
        if (i < depth) {
            int t = sv.get(i - 1), u = sv.get(i);
            k = t < T.n_lr && u < T.n_lr ? __ldg(T.bu_slot + (size_t)t * T.n_lr + u) : -1;
        }
        int n = depth - i0 < 32 ? depth - i0 : 32;
        int mine = -1;
        for (int j = 0; j < n; j++) {
            int kj = __shfl_sync(FULL, k, j);
            e = e >= 0 && kj >= 0 && e + 1 + kj < T.bu_len ? ld_keep(T.bu + e + 1 + kj, pol) : -1;
            mine = lane == j ? e : mine;
        }
        if (i < depth) memo[i] = mine;
    }
    return e;
}

// Algorithm 2 steps 1-3 for one row per warp: consume the row's token (the
// given one, or the greedy choice of the fused masking pass when from_keys),
// then classify the new configuration into S.mid.  Everything that needs only
// global memory (the row's state, its mask word, the token's bytes, the stack
// window) is loaded while the tables are still being staged.
// early: the row's state (lexer state, depth, status, mask id, stack window, kept
// bottom-up blocks) is read before waiting for the previous kernel.  Only the greedy
// keys come from that kernel (the masking pass), and the masking pass lets this
// kernel start only after its own wait for the advance before it, which wrote the
// rows; the host sets `early` only when the masking pass is the last work on
// these states and took the mask ids as they were.
template <bool PACKED, bool COMB>
__global__ void __launch_bounds__(ADV_WARPS * 32) k_advance_warp(DevTables T, DevStates S, const int32_t* tokens,
                                                                 int B, int use_mid, int32_t* status_out,
                                                                 int from_keys, int32_t* tokens_out, int early) {
    extern __shared__ uint4 smem4[];
    __shared__ __align__(8) uint64_t bar;
    __shared__ uint8_t tokc[ADV_WARPS][32];     // the lexer byte classes of each row's token (first 32 bytes)
    __shared__ uint16_t lexcls[ADV_WARPS][32];  // the lexeme classes the token emits (tokens up to 32 bytes)
    uint8_t* sm = reinterpret_cast<uint8_t*>(smem4);
    // one TMA bulk copy stages the compact tables (16-byte aligned, multiple of 16 bytes)
    uint32_t bar_a = smem_addr(&bar);
    if (threadIdx.x == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(bar_a) : "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar_a), "r"(T.adv_bytes) : "memory");
        asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                     ::"r"(smem_addr(sm)), "l"(gmem_addr(T.adv)), "r"(T.adv_bytes), "r"(bar_a)
                     : "memory");
    }
    grid_dep_launch();
    int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int b = blockIdx.x * ADV_WARPS + warp;
    bool active = b < B;   // warp-uniform
    StackView sv{reinterpret_cast<uint16_t*>(sm + T.adv_bytes) + warp * ADV_WIN,
                 S.stack + (size_t)(active ? b : 0) * S.cap, 0x40000000, 0x7FFFFFFF, 0u};
    sv.wa = smem_addr(sv.win);
    int tok = -1, status = ROW_OK, q = 0, depth = 0;
    bool parse = false;
    int32_t* memo = active && S.rmemo && T.bu ? S.rmemo + (size_t)b * S.cap : nullptr;
    int memo_top = -1, depth0 = 0;
    uint32_t mword = 0;
    int tbyte = 0;   // lane i: byte i of the token (first 32 bytes)
    int len = 0;
    int64_t vlo = 0;
    int cur_mid = 0;   // the mask the row's token is checked against
    bool live = false;
    // the row's state and the window of its stack top (for the parse and for the
    // classifier walk after it); read from L2 (an SM's L1 may still hold these lines
    // from an earlier kernel)
    auto load_row = [&]() {
        q = __ldcg(S.q + b);
        depth = __ldcg(S.depth + b);
        depth0 = depth;
        status = __ldcg(S.status + b);
        cur_mid = use_mid ? __ldcg(S.mid + b) : 0;
        live = status == ROW_OK && depth >= 1 && depth <= S.cap;
        if (live) {
            sv.base = depth > ADV_KEEP ? depth - ADV_KEEP : 0;
            for (int i = lane; i < depth - sv.base; i += 32) sv.win[i] = __ldcg(sv.st + sv.base + i);
            // the kept bottom-up blocks of the top 32 prefixes (lane l: stack [0, depth-1-l])
            if (memo && depth - 1 - lane >= 0) memo_top = __ldcg(memo + depth - 1 - lane);
        }
    };
    if (active && early) load_row();
    grid_dep_wait();   // the greedy keys (and, unless early, the rows) come from the previous kernel
    if (active) {
        if (!early) load_row();
        if (from_keys) {   // the greedy choice of the fused masking pass
            unsigned long long k = S.best[b];
            tok = k ? (int32_t)(~(uint32_t)(k & 0xFFFFFFFFu)) : -1;
            __syncwarp();
            if (lane == 0) {
                S.best[b] = 0ull;
                tokens_out[b] = tok;
            }
        } else {
            tok = tokens[b];
        }
        if (tok >= 0) {
            if (status == ROW_DONE) {
                status = tok == T.eos_id ? ROW_DONE : ROW_REJECTED;
            } else if (status == ROW_OK) {
                if (tok >= T.V) {
                    status = ROW_REJECTED;
                } else {
                    if (!use_mid) {   // the kept bottom-up block, else a walk of the stack in global memory
                        int e = __shfl_sync(FULL, memo_top, 0);
                        cur_mid = memo && live && q >= 0 && q < T.nq ? memo_mask(T, e, q) : -1;
                        StackView g{sv.win, sv.st, 0x40000000, 0x7FFFFFFF, sv.wa};
                        if (cur_mid < 0)
                            cur_mid = depth >= 1 && depth <= S.cap ? warp_walk(T, g, q, depth, lane) : 0;
                    }
                    // the token's mask bit (in flight while the token is parsed); the row is
                    // only committed (q, depth) when it is set
                    mword = mask_word(T, cur_mid, tok >> 5);
                    if (tok == T.eos_id) status = ((mword >> (tok & 31)) & 1) ? ROW_DONE : ROW_REJECTED;
                    else if (!live) status = ROW_REJECTED;
                    else parse = true;
                }
            }
        }
        if (parse) {   // the token's bytes: lane i holds byte i (loaded with the length, in parallel)
            tbyte = T.tok32[(size_t)tok * 32 + lane];
            vlo = T.vocab_off[tok];
            len = (int)(T.vocab_off[tok + 1] - vlo);
        }
    }
    __syncthreads();
    bool staged = __all_sync(FULL, mbar_wait0(bar_a, 1 << 24));
    // the tables are in: each lane turns its byte into a lexer byte class
    if (staged && active && parse && lane < len) tokc[warp][lane] = sm[T.o_bc + tbyte];
    __syncwarp();
    if (!staged) {
        // the copy did not land: give the rows a LIMIT status, wait (bounded) for the copy, return
        if (threadIdx.x == 0) {
            atomicAdd(&g_pipeline_timeouts, 1);
            if (S.fault) atomicAdd(S.fault, 1);
        }
        if (active && lane == 0) {
            if (status == ROW_OK) status = ROW_LIMIT;
            S.status[b] = status;
            if (status_out) status_out[b] = status;
            S.mid[b] = 0;
        }
        mbar_wait0(bar_a, 1 << 24);
        return;
    }
    if (!active) return;
    if (parse) {
        const AdvTabs A(smem_addr(sm), T);
        int nq = q, nd = depth;
        const uint32_t ca = smem_addr(&tokc[warp][0]);
        const uint32_t la = smem_addr(&lexcls[warp][0]);
        int ncls = -1;   // classes in lexcls; -1: the token is lexed by lane 0 (longer than 32 bytes)
        if (len <= 32) {
            // Lexing in parallel (the lexer does not depend on the parser): lane j runs the
            // lexer DFA over the lexeme that starts afresh at byte j, lane 0 over the
            // continuation of the row's pending lexeme; each records where its lexeme
            // ends (the byte it cannot take, or the end of the token) and the DFA state
            // there.  Then the lexemes are followed from one end to the next.
            int ls = lane == 0 ? q : A.q0;
            int le = lane;
            int pre = -2;   // class of the pending lexeme when the token's first byte ends it
            auto run = [&]() {
                while (le < len) {
                    int nx = lds_s16(A.trans + ls * A.trans_row + 2u * lds_u8(ca + le));
                    if (nx < 0) break;
                    ls = nx;
                    le++;
                }
            };
            if (lane < len) {
                run();
                if (lane == 0 && le == 0 && q != A.q0) {
                    pre = lds_s16(A.acc + 2u * q);
                    ls = A.q0;
                    run();
                }
            }
            pre = __shfl_sync(FULL, pre, 0);
            ncls = 0;
            if (pre != -2) {
                if (pre < 0) {
                    status = ROW_REJECTED;
                } else if (!lds_u8(A.ign + pre)) {
                    if (lane == 0) sts_u16(la, pre);
                    ncls = 1;
                }
            }
            int pos = 0;
            while (status == ROW_OK) {   // warp-uniform: pos and the lexeme ends come by shuffles
                int ep = __shfl_sync(FULL, le, pos), sp = __shfl_sync(FULL, ls, pos);
                if (ep == len) {   // the last lexeme stays pending
                    nq = sp;
                    break;
                }
                if (ep == pos) {   // the byte at pos starts no lexeme
                    status = ROW_REJECTED;
                    break;
                }
                int cls = sp == A.q0 ? -1 : lds_s16(A.acc + 2u * sp);
                if (cls < 0) {
                    status = ROW_REJECTED;
                    break;
                }
                if (!lds_u8(A.ign + cls)) {
                    if (lane == 0) sts_u16(la + 2u * ncls, cls);
                    ncls++;
                }
                pos = ep;
            }
        }
        __syncwarp();
        if (lane == 0) {
            int top = sv.get(depth - 1);
            int below = depth >= 2 ? sv.get(depth - 2) : 0;
            if (ncls >= 0) {
                for (int k = 0; k < ncls && status == ROW_OK; k++)
                    status = feed_class<PACKED, COMB>(A, sv, nd, top, below, S.cap, lds_u16(la + 2u * k));
            } else {
                // one byte (as its byte class) through the lexer DFA; a completed lexeme
                // goes to the parser
                auto lex = [&](int c) {
                    int nx = lds_s16(A.trans + nq * A.trans_row + 2u * c);
                    if (nx >= 0) {
                        nq = nx;
                        return;
                    }
                    int cls = nq == A.q0 ? -1 : lds_s16(A.acc + 2u * nq);
                    if (cls < 0) {
                        status = ROW_REJECTED;
                        return;
                    }
                    if (!lds_u8(A.ign + cls)) status = feed_class<PACKED, COMB>(A, sv, nd, top, below, S.cap, cls);
                    nq = lds_s16(A.trans + A.q0 * A.trans_row + 2u * c);
                    if (nq < 0) status = ROW_REJECTED;
                };
                for (int i = 0; i < 32 && status == ROW_OK; i++) lex(lds_u8(ca + i));
                for (int i = 32; i < len && status == ROW_OK; i++) lex(lds_u8(A.bc + T.vocab[vlo + i]));
            }
            if (!((mword >> (tok & 31)) & 1)) status = ROW_REJECTED;
            if (status == ROW_OK) {
                S.q[b] = nq;
                S.depth[b] = nd;
            }
        }
        status = __shfl_sync(FULL, status, 0);
        q = __shfl_sync(FULL, nq, 0);
        depth = __shfl_sync(FULL, nd, 0);
        sv.lo = __shfl_sync(FULL, sv.lo, 0);
        __syncwarp();
        if (status == ROW_OK) {
            // window entries from the lowest one written up to the new depth (lo stays
            // INT_MAX when nothing was written: clamp before adding the lane)
            int hi = depth < sv.base + ADV_WIN ? depth : sv.base + ADV_WIN;
            int from = sv.lo > sv.base ? sv.lo : sv.base;
            from = from < hi ? from : hi;
            for (int i = from + lane; i < hi; i += 32) sv.st[i] = sv.win[i - sv.base];
        }
    }
    if (lane == 0) {
        if (tok >= 0) S.status[b] = status;
        if (status_out) status_out[b] = status;
    }
    // the next masking pass's mask id (the window holds the stack top of every live
    // row; for the others sv.base still points past any stack index)
    int mid;
    if (status == ROW_DONE) {
        mid = 1;
    } else if (status != ROW_OK) {
        mid = 0;
    } else if (depth < 1 || depth > S.cap || q < 0 || q >= T.nq) {
        mid = 0;
    } else {
        mid = -1;
        if (memo) {
            // bottom-up classifier: re-read the entries from the lowest one written
            // (none written: the stack is as kept) and look the lexer state up
            int from = parse && sv.lo < depth ? sv.lo : depth;
            int below = from - 1;                    // block of stack [0, below] as kept
            int d = depth0 - 1 - below;              // its lane in the prefetched top
            int e_below = -1;
            if (below >= 0) e_below = d >= 0 && d < 32 ? __shfl_sync(FULL, memo_top, d) : memo[below];
            int e = warp_memo_extend(T, sv, memo, from, depth, e_below, lane);
            mid = memo_mask(T, e, q);
        }
        if (mid < 0) mid = warp_walk(T, sv, q, depth, lane);
    }
    if (lane == 0) S.mid[b] = mid;
}

// ------------------------------------------ TMA-pipelined decode masking pass
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
// Bounded wait for the phase with the given parity to complete (about a few
// seconds at most; a pipeline wait that gives up is counted and the kernel ends).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
    for (int it = 0; it < (1 << 22); it++) {
        uint32_t ok;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
            : "=r"(ok)
            : "r"(bar), "r"(parity)
            : "memory");
        if (ok) return true;
    }
    return false;
}
// 1-D bulk copy global -> shared, completing on the mbarrier (16-byte aligned, size a multiple of 16).
__device__ __forceinline__ void tma_load_1d(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(dst), "l"(gmem_addr(src)), "r"(bytes), "r"(bar)
                 : "memory");
}
// The same with an L2 cache policy (the streamed logits go first when L2 evicts,
// so the classifier table and mask rows the walks and the mask copies read stay).
__device__ __forceinline__ void tma_load_1d_hint(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar,
                                                 uint64_t policy) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;"
        ::"r"(dst), "l"(gmem_addr(src)), "r"(bytes), "r"(bar), "l"(policy)
        : "memory");
}
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}


constexpr long WARP_STEP_CHUNKS = 4096;   // batches of at most this many 1024-column chunks: k_step_warp
constexpr int TMA_SEG = 32;     // most 1024-column chunks per work item (one per lane of a warp)
constexpr int TMA_NCONS = 8;    // consumer warps; a ring stage holds one chunk for each of them
constexpr int TMA_WARPS = TMA_NCONS + 2;   // + producer + walker
constexpr int TMA_MIDS = 4;     // classified rows the walker may run ahead (it walks them together)
constexpr int TMA_MSLOTS = 3;   // mask-word buffers: the next item's words load while this item streams

// Shared-memory plan of the pipelined pass: NS ring stages of TMA_NCONS chunks,
// TMA_MSLOTS mask-word buffers (TMA_SEG x 32 words each), then the mbarriers.
template <typename T>
struct TmaShape {
    static constexpr int CHUNK = 1024 * (int)sizeof(T);   // bytes of one 1024-column chunk
    static constexpr int STAGE = TMA_NCONS * CHUNK;
    static constexpr int NS = sizeof(T) == 2 ? 3 : 2;
    static constexpr int NBARS = 2 * NS + 2 * TMA_MSLOTS + 2 * TMA_MIDS;
    static constexpr int SMEM = NS * STAGE + TMA_MSLOTS * TMA_SEG * 32 * 4 + NBARS * 8;
};

// The decode masking pass for small batches of bf16 rows whose mask ids are
// current, a warp per 1024-column chunk, eight chunks per CTA.  A lane loads its
// four 16-byte pieces of the chunk at once, whatever the mask (at these sizes the
// bytes are cheap and the latency is not), while the chunk's mask word comes
// through the row's mask id and chunk id; then the same masking, greedy fold,
// sector rule and keys as k_step_tma.  Requires 16-byte aligned rows.
__global__ void __launch_bounds__(256) k_step_warp(uint16_t* logits, int64_t stride, int B, int V, uint32_t* copy_out,
                                                   unsigned long long* __restrict__ best_key, DevTables D,
                                                   DevStates S) {
    __shared__ uint4 s_lut[256];
    build_allow_lut<uint16_t>(s_lut);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int cpr = (V + 1023) >> 10, cpb = (cpr + 7) >> 3;   // chunks per row, CTAs per row
    const int b = blockIdx.x / cpb, j = (blockIdx.x - b * cpb) * 8 + warp;
    grid_dep_wait();   // logits, mask ids and greedy keys come from earlier kernels
    grid_dep_launch();
    __syncthreads();   // the allow-mask table
    if (b >= B || j >= cpr) return;
    uint16_t* row = logits + (size_t)b * stride;
    const int col0 = j << 10;
    const bool whole = col0 + 1024 <= V;
    uint4 v[4];
    if (whole) {
#pragma unroll
        for (int k = 0; k < 4; k++) v[k] = *reinterpret_cast<const uint4*>(row + col0 + (k * 32 + lane) * 8);
    }
    const int mid = S.mid[b];
    const uint32_t cid = __ldg(D.mrows + (size_t)mid * D.nch + j);
    const uint32_t w = __ldg(D.mchunks + (size_t)cid * 32 + lane);
    if (copy_out) {
        int wi = j * 32 + lane;
        if (wi < D.W) copy_out[(size_t)b * D.W + wi] = w;
    }
    Best best{0.f, -1};
    BestPiece bp = best_piece_none();
    if (!whole) {
        apply_argmax_chunk_scalar<uint16_t>(row, col0, V - col0, w, lane, best);
    } else {
        ChunkRegs r;
#pragma unroll
        for (int k = 0; k < 4; k++) r.bits[k] = (__shfl_sync(FULL, w, k * 8 + (lane >> 2)) >> ((lane & 3) * 8)) & 0xFFu;
#pragma unroll
        for (int k = 0; k < 4; k++) {
            uint4 am = s_lut[r.bits[k]];
            r.x[k] = make_uint4(sel_ninf(v[k].x, am.x, 0xFF80FF80u), sel_ninf(v[k].y, am.y, 0xFF80FF80u),
                                sel_ninf(v[k].z, am.z, 0xFF80FF80u), sel_ninf(v[k].w, am.w, 0xFF80FF80u));
        }
        fold_store_chunk_bf16(row, col0, lane, r, bp);
    }
    unsigned long long key = best_key_of(best), kp = best_piece_key_bf16(bp);
    key = kp > key ? kp : key;
    uint32_t khi = (uint32_t)(key >> 32), klo = (uint32_t)key;
    uint32_t mhi = __reduce_max_sync(FULL, khi);
    uint32_t mlo = __reduce_max_sync(FULL, khi == mhi ? klo : 0u);
    key = ((unsigned long long)mhi << 32) | mlo;
    if (lane == 0 && key) atomicMax(best_key + b, key);
}

// One decode masking pass (classification, mask, apply, greedy key) with the
// logits streamed through shared memory by TMA bulk copies.  Work item = (row,
// segment of `seg` <= TMA_SEG chunks).  Warp 0 (producer) fetches each item's mask words
// one item ahead, then for every ring stage copies the stage's chunks that hold
// an allowed position (runs of neighbouring chunks in one copy; chunks with
// nothing allowed are not read); warp 1 reads (or, when they are not current,
// computes) the mask ids of the CTA's upcoming rows; consumer warp c takes chunk c of every stage, writes -inf where
// masked and folds allowed values into the row's greedy key.
// Requires 16-byte aligned rows; rows' mask rows padded to whole chunks.
template <typename T>
__global__ void __launch_bounds__(TMA_WARPS * 32, 3) k_step_tma(T* logits, int64_t stride, int B, int V,
                                                                uint32_t* copy_out,
                                                                unsigned long long* __restrict__ best_key,
                                                                DevTables D, DevStates S, int have_mid, int seg) {
    using Sh = TmaShape<T>;
    constexpr int NS = Sh::NS, CHUNK = Sh::CHUNK, STAGE = Sh::STAGE;
    static_assert(TMA_SEG == 32, "one lane per chunk of an item");
    static_assert(TMA_NCONS <= 32 && TMA_SEG % TMA_NCONS == 0, "whole stages per item");
    extern __shared__ __align__(128) uint8_t smem[];
    uint8_t* tiles = smem;
    uint32_t* mbuf = reinterpret_cast<uint32_t*>(smem + NS * STAGE);
    uint64_t* bars = reinterpret_cast<uint64_t*>(mbuf + TMA_MSLOTS * TMA_SEG * 32);
    __shared__ int s_mid[TMA_MIDS];
    __shared__ uint4 s_lut[256];
    int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int cpr = (V + 1023) >> 10;
    int nseg = (cpr + seg - 1) / seg;
    build_allow_lut<T>(s_lut);
    long items = (long)B * nseg;
    const uint32_t full0 = smem_addr(bars), empty0 = full0 + 8 * NS, mfull0 = empty0 + 8 * NS;
    const uint32_t mempty0 = mfull0 + 8 * TMA_MSLOTS, midf0 = mempty0 + 8 * TMA_MSLOTS, mide0 = midf0 + 8 * TMA_MIDS;
    if (threadIdx.x == 0) {
        for (int k = 0; k < NS; k++) {
            mbar_init(full0 + 8 * k, 1);
            mbar_init(empty0 + 8 * k, TMA_NCONS);
        }
        for (int k = 0; k < TMA_MSLOTS; k++) {
            mbar_init(mfull0 + 8 * k, 1);
            mbar_init(mempty0 + 8 * k, TMA_NCONS);
        }
        for (int k = 0; k < TMA_MIDS; k++) {
            mbar_init(midf0 + 8 * k, 1);
            mbar_init(mide0 + 8 * k, 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    __syncthreads();
    grid_dep_wait();   // mask ids, greedy keys and rows come from the previous kernel
    // the next kernel (the advance) may start now: the rows' writer before this pass
    // has completed, so the advance can read the rows before its own wait
    grid_dep_launch();
    bool failed = false;
    if (warp == 0) {
        // ---------------------------------------------------------- producer
        long s = 0;            // ring stages issued
        int issued = -1;       // last item whose mask words were requested
        const uint64_t stream_policy = l2_evict_first_policy();
        // request item ii's mask words (its row classified by the walker) into slot ii % TMA_MSLOTS
        auto fetch_mask = [&](int ii, long itm) -> bool {
            int b = (int)(itm / nseg), sg = (int)(itm - (long)b * nseg);
            int c0 = sg * seg, nch = min(seg, cpr - c0);
            int ms = ii % TMA_MIDS;
            if (!__shfl_sync(FULL, (int)mbar_wait(midf0 + 8 * ms, (uint32_t)((ii / TMA_MIDS) & 1)), 0)) return false;
            int mid = s_mid[ms];
            __syncwarp();
            int slot = ii % TMA_MSLOTS, use = ii / TMA_MSLOTS;
            if (lane == 0) {
                mbar_arrive(mide0 + 8 * ms);
                if (sg == 0 && !have_mid) S.mid[b] = mid;
            }
            if (use >= 1 && !__shfl_sync(FULL, (int)mbar_wait(mempty0 + 8 * slot, (uint32_t)((use - 1) & 1)), 0))
                return false;
            // the item's chunk ids, then one 128-byte bulk copy per chunk (lane k: chunk k)
            uint32_t cid = lane < nch ? __ldg(D.mrows + (size_t)mid * D.nch + c0 + lane) : 0u;
            if (lane == 0) mbar_arrive_tx(mfull0 + 8 * slot, nch * 128);
            __syncwarp();
            if (lane < nch)
                tma_load_1d(smem_addr(mbuf + slot * TMA_SEG * 32 + lane * 32), D.mchunks + (size_t)cid * 32, 128,
                            mfull0 + 8 * slot);
            issued = ii;
            return true;
        };
        int i = 0;
        if ((long)blockIdx.x < items && !fetch_mask(0, blockIdx.x)) failed = true;
        for (long it = blockIdx.x; it < items && !failed; it += gridDim.x, i++) {
            int b = (int)(it / nseg), sg = (int)(it - (long)b * nseg);
            int c0 = sg * seg, nch = min(seg, cpr - c0);
            if (it + gridDim.x < items && !fetch_mask(i + 1, it + gridDim.x)) { failed = true; break; }
            int slot = i % TMA_MSLOTS;
            if (!__shfl_sync(FULL, (int)mbar_wait(mfull0 + 8 * slot, (uint32_t)((i / TMA_MSLOTS) & 1)), 0)) {
                failed = true;
                break;
            }
            // lane k: does chunk k of the item hold an allowed position?  (rotated reads: no bank conflicts)
            const uint32_t* mb = mbuf + slot * TMA_SEG * 32;
            uint32_t acc = 0;
#pragma unroll 8
            for (int k = 0; k < 32; k++) acc |= mb[lane * 32 + ((k + lane) & 31)];
            uint32_t load = __ballot_sync(FULL, acc != 0u && lane < nch);
            if (c0 + nch == cpr && (V & 1023)) load &= ~(1u << (nch - 1));   // the ragged chunk is read directly
            const T* row = logits + (size_t)b * stride;
            for (int g = 0; g * TMA_NCONS < nch; g++, s++) {
                int stg = (int)(s % NS);
                if (s >= NS && !__shfl_sync(FULL, (int)mbar_wait(empty0 + 8 * stg, (uint32_t)(((s / NS) - 1) & 1)), 0)) {
                    failed = true;
                    break;
                }
                if (lane == 0) {
                    uint32_t f = (load >> (g * TMA_NCONS)) & ((1u << TMA_NCONS) - 1u);
                    if (f) {
                        mbar_arrive_tx(full0 + 8 * stg, (uint32_t)(__popc(f) * CHUNK));
                        while (f) {
                            int a = __ffs(f) - 1;
                            int len = __ffs(~(f >> a)) - 1;
                            tma_load_1d_hint(smem_addr(tiles + stg * STAGE + a * CHUNK),
                                             row + (size_t)(c0 + g * TMA_NCONS + a) * 1024, (uint32_t)(len * CHUNK),
                                             full0 + 8 * stg, stream_policy);
                            f &= ~(((1u << len) - 1u) << a);
                        }
                    } else {
                        mbar_arrive(full0 + 8 * stg);
                    }
                }
            }
        }
        if (failed && lane == 0) {
            // let this CTA's copies in flight land before it exits (bounded)
            for (long tt = s > NS ? s - NS : 0; tt < s; tt++) mbar_wait(full0 + 8 * (int)(tt % NS), (uint32_t)((tt / NS) & 1));
            for (int ii = issued > 0 ? issued - 1 : 0; ii <= issued; ii++)
                mbar_wait(mfull0 + 8 * (ii % TMA_MSLOTS), (uint32_t)((ii / TMA_MSLOTS) & 1));
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ walker
        // lanes 0..TMA_MIDS-1 each classify one of the next TMA_MIDS items' rows, so
        // the dependent table loads of those classifications overlap
        int i = 0;
        for (long it = blockIdx.x; it < items && !failed; it += (long)gridDim.x * TMA_MIDS, i += TMA_MIDS) {
            if (i >= TMA_MIDS && !__shfl_sync(FULL, (int)mbar_wait(mide0 + 8 * (TMA_MIDS - 1),
                                                                    ((i / TMA_MIDS) - 1) & 1), 0)) {
                failed = true;
                break;
            }
            long my = it + (long)lane * gridDim.x;
            int mid = 0;
            if (lane < TMA_MIDS && my < items) {
                int rb = (int)(my / nseg);
                mid = have_mid ? S.mid[rb] : thread_classify(D, S, rb);
            }
            if (lane < TMA_MIDS && my < items) {
                s_mid[lane] = mid;
                mbar_arrive(midf0 + 8 * lane);
            }
            __syncwarp();
        }
    } else {
        // --------------------------------------------------------- consumers
        int c = warp - 2;
        long s = 0;
        int i = 0;
        for (long it = blockIdx.x; it < items && !failed; it += gridDim.x, i++) {
            int b = (int)(it / nseg), sg = (int)(it - (long)b * nseg);
            int c0 = sg * seg, nch = min(seg, cpr - c0);
            int slot = i % TMA_MSLOTS;
            if (!__shfl_sync(FULL, (int)mbar_wait(mfull0 + 8 * slot, (uint32_t)((i / TMA_MSLOTS) & 1)), 0)) {
                failed = true;
                break;
            }
            const uint32_t* mb = mbuf + slot * TMA_SEG * 32;
            T* row = logits + (size_t)b * stride;
            Best best{0.f, -1};
            BestPiece bp = best_piece_none();
            for (int g = 0; g * TMA_NCONS < nch; g++, s++) {
                int stg = (int)(s % NS);
                if (!__shfl_sync(FULL, (int)mbar_wait(full0 + 8 * stg, (uint32_t)((s / NS) & 1)), 0)) {
                    failed = true;
                    break;
                }
                int k = g * TMA_NCONS + c;
                bool released = false;
                if (k < nch) {
                    int j = c0 + k;
                    uint32_t w = mb[k * 32 + lane];
                    if (copy_out) {
                        int wi = j * 32 + lane;
                        if (wi < D.W) copy_out[(size_t)b * D.W + wi] = w;
                    }
                    int col0 = j << 10;
                    const uint8_t* tile = tiles + stg * STAGE + c * CHUNK;
                    if ((j == cpr - 1) && (V & 1023)) {
                        apply_argmax_chunk_scalar<T>(row, col0, V - col0, w, lane, best);
                    } else if (__ballot_sync(FULL, w != 0u) == 0u) {
                        constexpr int PIECES = CHUNK / 16 / 32;
                        uint4 ninf = make_uint4(NegInf<T>::pair, NegInf<T>::pair, NegInf<T>::pair, NegInf<T>::pair);
#pragma unroll
                        for (int q = 0; q < PIECES; q++)
                            st_cs_v4(reinterpret_cast<uint8_t*>(row + col0) + (q * 32 + lane) * 16, ninf);
                    } else if constexpr (sizeof(T) == 2) {
                        // the chunk goes to registers and the stage back to the producer
                        // before the chunk is folded and written out
                        ChunkRegs r;
                        load_mask_chunk_bf16(reinterpret_cast<const uint16_t*>(tile), w, lane, s_lut, r);
                        __syncwarp();
                        if (lane == 0) mbar_arrive(empty0 + 8 * stg);
                        released = true;
                        fold_store_chunk_bf16(reinterpret_cast<uint16_t*>(row), col0, lane, r, bp);
                    } else {
                        apply_argmax_chunk_f32(reinterpret_cast<const uint32_t*>(tile), reinterpret_cast<uint32_t*>(row),
                                               col0, w, lane, best, s_lut);
                    }
                }
                if (!released) {
                    __syncwarp();
                    if (lane == 0) mbar_arrive(empty0 + 8 * stg);
                }
            }
            unsigned long long key = best_key_of(best);
            if constexpr (sizeof(T) == 2) {
                unsigned long long kp = best_piece_key_bf16(bp);
                key = kp > key ? kp : key;
            }
            // warp maximum of the 64-bit keys: the high words, then the low words of the lanes holding it
            uint32_t khi = (uint32_t)(key >> 32), klo = (uint32_t)key;
            uint32_t mhi = __reduce_max_sync(FULL, khi);
            uint32_t mlo = __reduce_max_sync(FULL, khi == mhi ? klo : 0u);
            key = ((unsigned long long)mhi << 32) | mlo;
            if (lane == 0) {
                if (key) atomicMax(best_key + b, key);
                mbar_arrive(mempty0 + 8 * slot);
            }
        }
    }
    if (failed && lane == 0) {
        atomicAdd(&g_pipeline_timeouts, 1);
        if (S.fault) atomicAdd(S.fault, 1);
    }
}

// A bounded wait on an mbarrier phase that nothing completes: gives up after
// `limit` polls and records it on the states object, as the pipeline's waits do
// (lets tests see fault reporting without any fault).
__global__ void k_wait_gives_up(DevStates S, int limit) {
    __shared__ __align__(8) uint64_t bar;
    uint32_t a = smem_addr(&bar);
    if (threadIdx.x == 0) {
        mbar_init(a, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    bool ok = mbar_wait0(a, limit);   // no thread arrives
    if (!ok && threadIdx.x == 0 && S.fault) atomicAdd(S.fault, 1);
}

// ----------------------------------------------------------------- host glue
psc_status cuda_check(cudaError_t e, const char* what) {
    if (e == cudaSuccess) return PSC_OK;
    return fail_with(e == cudaErrorMemoryAllocation ? PSC_ERR_OOM : PSC_ERR_CUDA,
                     std::string(what) + ": " + cudaGetErrorString(e));
}

psc_status launch_check(const char* what) { return cuda_check(cudaGetLastError(), what); }

int sm_count(int device) {
    int n = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, device);
    return n > 0 ? n : 1;
}

template <typename V>
psc_status upload(psc_handle* h, const std::vector<V>& v, const V** dst, size_t pad_bytes = 0) {
    size_t bytes = v.size() * sizeof(V) + pad_bytes;
    if (bytes == 0) bytes = 16;
    void* p = nullptr;
    psc_status s = cuda_check(cudaMalloc(&p, bytes), "cudaMalloc(tables)");
    if (s != PSC_OK) return s;
    if (h->n_blocks >= (int)(sizeof(h->blocks) / sizeof(h->blocks[0]))) {
        cudaFree(p);
        return fail_with(PSC_ERR_OOM, "too many device table blocks");
    }
    h->blocks[h->n_blocks++] = p;
    if (!v.empty()) {
        s = cuda_check(cudaMemcpy(p, v.data(), v.size() * sizeof(V), cudaMemcpyHostToDevice), "cudaMemcpy(tables)");
        if (s != PSC_OK) return s;
    }
    *dst = static_cast<const V*>(p);
    return PSC_OK;
}

psc_status check_device(const psc_handle* h, const char* what) {
    if (!h) return fail_with(PSC_ERR_ARG, std::string(what) + ": NULL handle");
    if (h->host_only) return fail_with(PSC_ERR_ARG, std::string(what) + ": handle was compiled host_only");
    int dev = -1;
    cudaGetDevice(&dev);
    if (dev != h->device)
        return fail_with(PSC_ERR_ARG, std::string(what) + ": current device differs from the handle's");
    return PSC_OK;
}

psc_status ensure_mid(const psc_handle* h, const psc_states* st, cudaStream_t s) {
    const_cast<psc_states*>(st)->after_mask = false;
    if (st->mid_gen == st->gen) return PSC_OK;
    int B = st->d.B;
    int threads = 256;
    int blocks = (int)(((size_t)B * 32 + threads - 1) / threads);
    k_classify<<<blocks, threads, 0, s>>>(h->d, st->d, B);
    psc_status r = launch_check("k_classify");
    if (r == PSC_OK) const_cast<psc_states*>(st)->mid_gen = st->gen;
    return r;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

psc_status launch_apply(void* logits, psc_dtype dtype, int64_t row_stride, const MaskSrc& M, int B, int V,
                        cudaStream_t s, int device) {
    size_t esz = dtype == PSC_BF16 ? 2 : 4;
    int vec = aligned16(logits) && ((row_stride * (int64_t)esz) % 16 == 0);
    long chunks = (long)B * ((V + 1023) / 1024);
    int threads = 256;
    long want = (chunks + 7) / 8;
    int blocks = (int)std::min<long>(want, (long)sm_count(device) * 8);
    if (blocks < 1) blocks = 1;
    if (dtype == PSC_BF16)
        k_apply_rows<uint16_t><<<blocks, threads, 0, s>>>((uint16_t*)logits, row_stride, M, B, V, vec);
    else
        k_apply_rows<uint32_t><<<blocks, threads, 0, s>>>((uint32_t*)logits, row_stride, M, B, V, vec);
    return launch_check("k_apply_rows");
}

// Masking + greedy choice with in-kernel classification; leaves each row's
// key in st->d.best and its mask id in st->d.mid.
// Launches a kernel that may start while the previous kernel of the stream finishes
// (programmatic dependent launch): it waits for that kernel's results itself.
template <typename... KArgs, typename... Args>
psc_status launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t cs, const char* what,
                      Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = cs;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cuda_check(cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...), what);
}

// Algorithm 2 steps 1-2 for every row (the token given, or the fused pass's greedy
// choice when d_tokens_out is set), then step 3 for the new configurations: the
// rows' mask ids are current afterwards.
using AdvanceKernel = void (*)(DevTables, DevStates, const int32_t*, int, int, int32_t*, int, int32_t*, int);
AdvanceKernel advance_kernel(const DevTables& d) {
    if (d.adv_comb) return d.adv_packed ? k_advance_warp<true, true> : k_advance_warp<false, true>;
    return d.adv_packed ? k_advance_warp<true, false> : k_advance_warp<false, false>;
}

psc_status launch_advance(const psc_handle* h, psc_states* st, const int32_t* d_tokens, int use_mid,
                          int32_t* d_row_status, int32_t* d_tokens_out, cudaStream_t cs) {
    int B = st->d.B;
    int from_keys = d_tokens_out ? 1 : 0;
    int early = from_keys && st->after_mask ? 1 : 0;
    st->after_mask = false;
    psc_status s;
    if (h->d.adv_bytes > 0) {
        s = launch_pdl(advance_kernel(h->d),
                       dim3((B + ADV_WARPS - 1) / ADV_WARPS), dim3(ADV_WARPS * 32), adv_smem(h->d), cs,
                       "k_advance_warp", h->d, st->d, d_tokens, B, use_mid, d_row_status, from_keys, d_tokens_out,
                       early);
    } else {
        k_advance<<<(B + 127) / 128, 128, 0, cs>>>(h->d, st->d, d_tokens, B, use_mid, d_row_status, from_keys,
                                                    d_tokens_out);
        s = launch_check("k_advance");
        if (s == PSC_OK) {
            int threads = 256;
            k_classify<<<(int)(((size_t)B * 32 + threads - 1) / threads), threads, 0, cs>>>(h->d, st->d, B);
            s = launch_check("k_classify");
        }
    }
    st->gen++;
    if (s == PSC_OK) st->mid_gen = st->gen;
    return s;
}

psc_status launch_fused(const psc_handle* h, const psc_states* st, void* d_logits, psc_dtype dtype, int64_t row_stride,
                        int V, uint32_t* d_bitmask_out, cudaStream_t cs) {
    int B = st->d.B;
    MaskSrc M{nullptr, h->d.mchunks, h->d.mrows, st->d.mid, h->d.W, h->d.nch, d_bitmask_out};
    size_t esz = dtype == PSC_BF16 ? 2 : 4;
    int vec = aligned16(d_logits) && ((row_stride * (int64_t)esz) % 16 == 0);
    int cpr = (V + 1023) / 1024;
    int have_mid = st->mid_gen == st->gen ? 1 : 0;   // mask ids current: no classifier walks
    psc_status s;
    if (vec) {
        // the pipelined pass (rows 16-byte aligned): as many CTAs as are resident at once;
        // items of 32 chunks; smaller (multiples of a stage) when the batch has too few
        // chunks to give every resident CTA work (one chunk per item instead of a stage
        // was measured no faster at batch 1: 8.3 us per graph-replayed step either way)
        long resident = (long)sm_count(h->device) * h->tma_ctas[dtype == PSC_BF16 ? 0 : 1];
        // small bf16 batches with current mask ids: a warp per chunk (measured on config 5's
        // tables, decode steps replayed from CUDA graphs: 7.5 instead of 9.2 us at batch 1,
        // 11.7 instead of 14.1 at 16).  Larger batches: the TMA pipeline below keeps more
        // bytes in flight (at batch 1024 the warp-per-chunk pass took 169.7 us per launch
        // against 157.6)
        if (dtype == PSC_BF16 && have_mid && (long)B * cpr <= WARP_STEP_CHUNKS) {
            s = launch_pdl(k_step_warp, dim3(B * ((cpr + 7) / 8)), dim3(256), 0, cs, "k_step_warp",
                           (uint16_t*)d_logits, row_stride, B, V, d_bitmask_out, st->d.best, h->d, st->d);
            if (s == PSC_OK) const_cast<psc_states*>(st)->mid_gen = st->gen;
            const_cast<psc_states*>(st)->after_mask = s == PSC_OK;
            return s;
        }
        long want = ((long)B * cpr + resident - 1) / resident;
        int seg = (int)std::min<long>(TMA_SEG, std::max<long>(TMA_NCONS, (want + TMA_NCONS - 1) / TMA_NCONS * TMA_NCONS));
        long titems = (long)B * ((cpr + seg - 1) / seg);
        int tgrid = (int)std::max(1L, std::min<long>(titems, resident));
        if (dtype == PSC_BF16)
            s = launch_pdl(k_step_tma<uint16_t>, dim3(tgrid), dim3(TMA_WARPS * 32), TmaShape<uint16_t>::SMEM, cs,
                           "k_step_tma", (uint16_t*)d_logits, row_stride, B, V, d_bitmask_out, st->d.best, h->d,
                           st->d, have_mid, seg);
        else
            s = launch_pdl(k_step_tma<uint32_t>, dim3(tgrid), dim3(TMA_WARPS * 32), TmaShape<uint32_t>::SMEM, cs,
                           "k_step_tma", (uint32_t*)d_logits, row_stride, B, V, d_bitmask_out, st->d.best, h->d,
                           st->d, have_mid, seg);
    } else {
        // rows not 16-byte aligned: warp-per-chunk pass, 4 resident CTAs of 256 threads per SM
        int slots = sm_count(h->device) * 4;
        long seg = ((long)cpr * B) / (2L * slots);
        int seg_chunks = (int)std::max(1L, std::min(32L, seg));
        long items = (long)B * ((cpr + seg_chunks - 1) / seg_chunks);
        int grid = (int)std::max(1L, std::min<long>(items, slots));
        if (dtype == PSC_BF16)
            k_apply_argmax<uint16_t, true><<<grid, 256, 0, cs>>>((uint16_t*)d_logits, row_stride, M, B, V, vec,
                                                                  seg_chunks, st->d.best, h->d, st->d);
        else
            k_apply_argmax<uint32_t, true><<<grid, 256, 0, cs>>>((uint32_t*)d_logits, row_stride, M, B, V, vec,
                                                                  seg_chunks, st->d.best, h->d, st->d);
        s = launch_check("k_apply_argmax");
    }
    if (s == PSC_OK) const_cast<psc_states*>(st)->mid_gen = st->gen;
    const_cast<psc_states*>(st)->after_mask = s == PSC_OK && vec && have_mid;
    return s;
}

// host-side parser step for psc_host_advance (same semantics as k_advance)
int host_feed(const psc::Tables& T, uint16_t* st, int& depth, int cap, int cls) {
    int t = T.resolve[(size_t)cls * T.n_lr + st[depth - 1]];
    if (t < 0) return ROW_REJECTED;
    for (int guard = 0; guard < 4 * cap + 64; guard++) {
        int32_t a = T.action[(size_t)st[depth - 1] * T.n_terms + t];
        int kind = a & 3, val = a >> 2;
        if (kind == psc::ACT_SHIFT) {
            if (depth >= cap) return ROW_OVERFLOW;
            st[depth++] = (uint16_t)val;
            return ROW_OK;
        }
        if (kind != psc::ACT_REDUCE) return ROW_REJECTED;
        int k = T.rule_len[val];
        if (depth - k < 1) return ROW_REJECTED;
        depth -= k;
        int go = T.go[(size_t)st[depth - 1] * T.n_nts + T.rule_lhs[val]];
        if (go < 0) return ROW_REJECTED;
        if (depth >= cap) return ROW_OVERFLOW;
        st[depth++] = (uint16_t)go;
    }
    return ROW_LIMIT;
}

}  // namespace

namespace {
// Compact int16 lexer/parser tables for k_advance_warp, or an empty blob when
// the grammar is too large for shared memory (k_advance then reads global memory).
// Candidate terminals of each lexeme class in an order such that, in every parser
// state s, the first candidate with an action in s is resolve[c][s] (or, where
// resolve gives -1 or a terminal without an action, none has one): resolution by
// trying the candidates in turn then picks what the resolve table picks.  Empty
// when no such order exists.
std::vector<std::vector<int>> class_candidates(const psc::Tables& t) {
    const int ncls = t.n_classes, n = t.n_lr;
    auto has = [&](int s, int x) { return psc::act_kind(t.action[(size_t)s * t.n_terms + x]) != psc::ACT_ERR; };
    std::vector<std::vector<int>> out(ncls);
    for (int c = 0; c < ncls; c++) {
        std::vector<int> L;
        for (int s = 0; s < n; s++) {
            int r = t.resolve[(size_t)c * n + s];
            if (r >= 0 && std::find(L.begin(), L.end(), r) == L.end()) L.push_back(r);
        }
        std::sort(L.begin(), L.end());
        const int m = (int)L.size();
        // r must come before x wherever resolve picks r while x has an action too
        std::vector<std::vector<char>> before(m, std::vector<char>(m, 0));
        for (int s = 0; s < n; s++) {
            int r = t.resolve[(size_t)c * n + s];
            if (r < 0) continue;
            int i = (int)(std::find(L.begin(), L.end(), r) - L.begin());
            for (int j = 0; j < m; j++)
                if (j != i && has(s, L[j])) before[i][j] = 1;
        }
        std::vector<char> done(m, 0);
        for (int k = 0; k < m; k++) {
            int pick = -1;
            for (int i = 0; i < m && pick < 0; i++) {
                if (done[i]) continue;
                bool free = true;
                for (int j = 0; j < m && free; j++) free = done[j] || j == i || !before[j][i];
                if (free) pick = i;
            }
            if (pick < 0) return {};   // a cycle: no order reproduces the table
            done[pick] = 1;
            out[c].push_back(L[pick]);
        }
        for (int s = 0; s < n; s++) {
            int r = t.resolve[(size_t)c * n + s], f = -1;
            for (int x : out[c])
                if (has(s, x)) {
                    f = x;
                    break;
                }
            if (!(r == f || (f < 0 && (r < 0 || !has(s, r))))) return {};
        }
    }
    return out;
}

// layout: 0 = the dense compact tables when they fit in shared memory, else the packed
// ones when those fit; 2 = the packed tables whenever they fit.
std::vector<uint8_t> build_advance_blob(const psc::Tables& t, DevTables& d, int layout) {
    std::vector<uint8_t> blob;
    d.adv_bytes = 0;
    d.adv_comb = 0;
    int n_rules = (int)t.rule_len.size();
    if (t.n_lr >= 8192 || n_rules >= 8192 || t.nq >= 32768 || t.n_terms >= 32768) return blob;
    for (int L : t.rule_len)
        if (L > 255) return blob;
    // byte classes of the lexer DFA
    std::vector<int> bc(256, -1);
    int nbc = 0;
    for (int b = 0; b < 256; b++) {
        if (bc[b] >= 0) continue;
        bc[b] = nbc;
        for (int b2 = b + 1; b2 < 256; b2++) {
            if (bc[b2] >= 0) continue;
            bool same = true;
            for (int q = 0; q < t.nq && same; q++) same = t.lex_trans[(size_t)q * 256 + b] == t.lex_trans[(size_t)q * 256 + b2];
            if (same) bc[b2] = nbc;
        }
        nbc++;
    }
    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t o = off;
        off = (off + bytes + 15) & ~(size_t)15;
        return (int)o;
    };
    int ncls = t.n_classes;
    d.o_bc = take(256);
    d.o_trans = take((size_t)t.nq * nbc * 2);
    d.o_accept = take((size_t)t.nq * 2);
    d.o_ign = take((size_t)std::max(ncls, 1));
    d.o_resolve = take((size_t)std::max(ncls, 1) * t.n_lr * 2);
    d.o_action = take((size_t)t.n_lr * t.n_terms * 2);
    d.o_go = take((size_t)t.n_lr * t.n_nts * 2);
    d.o_rlen = take((size_t)n_rules);
    d.o_rlhs = take((size_t)n_rules * 2);
    if (getenv("PSC_LOG"))
        fprintf(stderr, "psc: advance tables %zu B (lexer %d x %d classes, resolve %d x %d, action %d x %d, goto %d x %d)%s\n",
                off, t.nq, nbc, ncls, t.n_lr, t.n_lr, t.n_terms, t.n_lr, t.n_nts,
                off > ADV_TABLE_MAX ? ": too large for shared memory" : "");
    int max_len = 0;
    for (int L : t.rule_len) max_len = std::max(max_len, L);
    d.adv_packed = (max_len < 16 && t.n_nts <= 1024) ? 1 : 0;
    auto enc_action = [&](int32_t a) {
        int kind = psc::act_kind(a), val = psc::act_val(a);
        if (d.adv_packed && kind == psc::ACT_REDUCE) val = (t.rule_len[val] << 10) | t.rule_lhs[val];
        return (int16_t)(((val & 0x3FFF) << 2) | kind);
    };
    if (layout == 2 || off > ADV_TABLE_MAX) {
        // ---- packed layout: the lexer as above, then candidates, bases, the packed entries
        std::vector<std::vector<int>> cands = class_candidates(t);
        if (cands.empty() && ncls > 0) return blob;
        int kc = 1;
        for (auto& L : cands) kc = std::max(kc, (int)L.size());
        if (kc > 16) return blob;
        const int n = t.n_lr;
        // one packed table each for ACTION and GOTO: equal rows are stored once, rows are
        // placed first fit (fullest first) at the lowest base where all their entries land
        // on free slots; an entry records its row's id, so a lookup in another row misses.
        // Per state one word (row id << 17 | base).
        struct Packed {
            std::vector<uint32_t> slots;
            std::vector<uint32_t> word;   // per state
            int entries = 0;
        };
        auto pack = [&](int ncol, auto&& entry) -> Packed {   // entry(s, x, &v): has (s, x) an entry
            Packed P;
            std::vector<std::vector<std::pair<int, int16_t>>> rows;
            std::map<std::vector<std::pair<int, int16_t>>, int> ids;
            std::vector<int> rid(n);
            for (int s = 0; s < n; s++) {
                std::vector<std::pair<int, int16_t>> r;
                for (int x = 0; x < ncol; x++) {
                    int16_t v;
                    if (entry(s, x, &v)) r.push_back({x, v});
                }
                auto it = ids.find(r);
                if (it == ids.end()) {
                    it = ids.emplace(r, (int)rows.size()).first;
                    rows.push_back(r);
                }
                rid[s] = it->second;
            }
            const int nr = (int)rows.size();
            std::vector<int> order(nr), base(nr, 0);
            for (int r = 0; r < nr; r++) order[r] = r;
            std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return rows[a].size() > rows[b].size(); });
            std::vector<char> used;
            int len = ncol, first_free = 0;
            for (int r : order) {
                if (rows[r].empty()) continue;
                int lo = rows[r].front().first;
                for (int b = std::max(0, first_free - lo);; b++) {
                    if ((size_t)b + ncol > used.size()) used.resize((size_t)b + ncol + 4096, 0);
                    bool ok = true;
                    for (auto& e : rows[r])
                        if (used[b + e.first]) {
                            ok = false;
                            break;
                        }
                    if (!ok) continue;
                    for (auto& e : rows[r]) used[b + e.first] = 1;
                    base[r] = b;
                    len = std::max(len, b + ncol);
                    break;
                }
                while (first_free < (int)used.size() && used[first_free]) first_free++;
            }
            P.slots.assign((size_t)len, 0xFFFFFFFFu);
            for (int r = 0; r < nr; r++)
                for (auto& e : rows[r]) {
                    P.slots[(size_t)base[r] + e.first] = ((uint32_t)r << 16) | (uint16_t)e.second;
                    P.entries++;
                }
            if (nr >= (1 << 15) || len >= (1 << 17)) P.slots.clear();   // the state word cannot hold them
            P.word.resize(n);
            for (int s = 0; s < n; s++) P.word[s] = ((uint32_t)rid[s] << 17) | (uint32_t)base[rid[s]];
            return P;
        };
        Packed PA = pack(t.n_terms, [&](int s, int x, int16_t* v) {
            int32_t a = t.action[(size_t)s * t.n_terms + x];
            if (psc::act_kind(a) == psc::ACT_ERR) return false;
            *v = enc_action(a);
            return true;
        });
        Packed PG = pack(t.n_nts, [&](int s, int x, int16_t* v) {
            int32_t g = t.go[(size_t)s * t.n_nts + x];
            if (g < 0) return false;
            *v = (int16_t)g;
            return true;
        });
        if (PA.slots.empty() || PG.slots.empty()) return blob;
        // every lookup of the packed tables against the dense ones
        auto look = [](const Packed& P, int s, int x, int miss) {
            uint32_t w = P.word[s], e = P.slots[(size_t)(w & 0x1FFFFu) + x];
            return (e >> 16) == (w >> 17) ? (int)(int16_t)(e & 0xFFFFu) : miss;
        };
        for (int s = 0; s < n; s++) {
            for (int x = 0; x < t.n_terms; x++) {
                int32_t a = t.action[(size_t)s * t.n_terms + x];
                if (look(PA, s, x, 0) != (psc::act_kind(a) == psc::ACT_ERR ? 0 : (int)enc_action(a))) return blob;
            }
            for (int x = 0; x < t.n_nts; x++) {
                int32_t g = t.go[(size_t)s * t.n_nts + x];
                if (look(PG, s, x, -1) != (g >= 0 ? g : -1)) return blob;
            }
        }
        off = (size_t)d.o_resolve;   // the lexer parts stay where they are
        d.o_cand = take((size_t)std::max(ncls, 1) * kc * 2);
        d.o_abase = take((size_t)n * 4);
        d.o_gbase = take((size_t)n * 4);
        d.o_acmb = take(PA.slots.size() * 4);
        d.o_gcmb = take(PG.slots.size() * 4);
        d.o_rlen = take((size_t)n_rules);
        d.o_rlhs = take((size_t)n_rules * 2);
        d.o_resolve = d.o_action = d.o_go = 0;
        if (getenv("PSC_LOG"))
            fprintf(stderr, "psc: packed advance tables %zu B (ACTION %d entries in %zu slots, GOTO %d in %zu, "
                            "%d candidates per class)%s\n",
                    off, PA.entries, PA.slots.size(), PG.entries, PG.slots.size(), kc,
                    off > ADV_TABLE_MAX ? ": too large for shared memory" : "");
        if (off > ADV_TABLE_MAX) return blob;
        blob.assign(off, 0);
        for (int b = 0; b < 256; b++) blob[d.o_bc + b] = (uint8_t)bc[b];
        for (int q = 0; q < t.nq; q++) {
            for (int b = 0; b < 256; b++)
                reinterpret_cast<int16_t*>(blob.data() + d.o_trans)[(size_t)q * nbc + bc[b]] =
                    (int16_t)t.lex_trans[(size_t)q * 256 + b];
            reinterpret_cast<int16_t*>(blob.data() + d.o_accept)[q] = (int16_t)t.lex_accept[q];
        }
        for (int c = 0; c < ncls; c++) {
            blob[d.o_ign + c] = t.cls_ignored[c];
            for (int k = 0; k < kc; k++)
                reinterpret_cast<int16_t*>(blob.data() + d.o_cand)[(size_t)c * kc + k] =
                    (int16_t)(k < (int)cands[c].size() ? cands[c][k] : -1);
        }
        std::memcpy(blob.data() + d.o_abase, PA.word.data(), (size_t)n * 4);
        std::memcpy(blob.data() + d.o_gbase, PG.word.data(), (size_t)n * 4);
        std::memcpy(blob.data() + d.o_acmb, PA.slots.data(), PA.slots.size() * 4);
        std::memcpy(blob.data() + d.o_gcmb, PG.slots.data(), PG.slots.size() * 4);
        for (int r = 0; r < n_rules; r++) {
            blob[d.o_rlen + r] = (uint8_t)t.rule_len[r];
            reinterpret_cast<int16_t*>(blob.data() + d.o_rlhs)[r] = (int16_t)t.rule_lhs[r];
        }
        d.kc = kc;
        d.nbc = nbc;
        d.adv_comb = 1;
        d.adv_bytes = (int)off;
        return blob;
    }
    blob.assign(off, 0);
    auto put16 = [&](int o, size_t i, int v) { reinterpret_cast<int16_t*>(blob.data() + o)[i] = (int16_t)v; };
    for (int b = 0; b < 256; b++) blob[d.o_bc + b] = (uint8_t)bc[b];
    for (int q = 0; q < t.nq; q++) {
        for (int b = 0; b < 256; b++) put16(d.o_trans, (size_t)q * nbc + bc[b], t.lex_trans[(size_t)q * 256 + b]);
        put16(d.o_accept, q, t.lex_accept[q]);
    }
    for (int c = 0; c < ncls; c++) {
        blob[d.o_ign + c] = t.cls_ignored[c];
        for (int s = 0; s < t.n_lr; s++) put16(d.o_resolve, (size_t)c * t.n_lr + s, t.resolve[(size_t)c * t.n_lr + s]);
    }
    // a reduce entry carries its rule's length and left-hand side when they fit in 14 bits
    // (one dependent shared-memory read less per reduction)
    for (size_t i = 0; i < t.action.size(); i++) put16(d.o_action, i, enc_action(t.action[i]));
    for (size_t i = 0; i < t.go.size(); i++) put16(d.o_go, i, t.go[i]);
    for (int r = 0; r < n_rules; r++) {
        blob[d.o_rlen + r] = (uint8_t)t.rule_len[r];
        put16(d.o_rlhs, r, t.rule_lhs[r]);
    }
    d.nbc = nbc;
    d.adv_bytes = (int)off;
    return blob;
}

}  // namespace

// Scratch of psc_fill_apply_noalloc: per-row mask ids between the classifier
// walk and the masking pass, in the module itself so the call allocates nothing.
static __device__ __align__(256) int32_t g_noalloc_mid[PSC_NOALLOC_MAX_ROWS];

namespace {
std::mutex g_noalloc_mu;
int32_t* g_noalloc_ptr[256] = {};

// Device address of g_noalloc_mid on the current device (looked up once per device).
psc_status noalloc_scratch(int device, int32_t** out) {
    if (device < 0 || device >= 256) return fail_with(PSC_ERR_ARG, "psc_fill_apply_noalloc: bad device id");
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[device]) {
        void* p = nullptr;
        psc_status s = cuda_check(cudaGetSymbolAddress(&p, g_noalloc_mid), "cudaGetSymbolAddress(scratch)");
        if (s != PSC_OK) return s;
        g_noalloc_ptr[device] = static_cast<int32_t*>(p);
    }
    *out = g_noalloc_ptr[device];
    return PSC_OK;
}
}  // namespace

namespace {
// The first 32 bytes of every token, zero-padded to 32 ([V][32]): the advance loads a
// token's bytes with its length, instead of after its offset.
std::vector<uint8_t> token_prefixes(const psc::Tables& t) {
    std::vector<uint8_t> out((size_t)t.V * 32, 0);
    for (int v = 0; v < t.V; v++) {
        int64_t lo = t.vocab_off[v], n = std::min<int64_t>(32, t.vocab_off[v + 1] - lo);
        if (n > 0) std::memcpy(out.data() + (size_t)v * 32, t.vocab_bytes.data() + lo, (size_t)n);
    }
    return out;
}

// Uploads a handle's host tables to the current device (psc_compile, psc_load).
// tables: 0 = staged (dense compact tables when they fit, else packed ones), 1 = global
// memory, 2 = staged packed tables.
psc_status upload_tables(std::unique_ptr<psc_handle>& h, int tables) {
    const psc::Tables& t = h->t;
    psc_status s = cuda_check(cudaGetDevice(&h->device), "cudaGetDevice");
    if (s != PSC_OK) return s;
    DevTables& d = h->d;
    std::vector<int32_t> dfa = t.dfa;
    if (dfa.empty()) dfa.push_back(0);
    std::vector<int32_t> dfa_mask = t.dfa_mask;
    if (dfa_mask.empty()) dfa_mask.push_back(0);
    // sparse layout: the packed rows of the device, state ids replaced by row offsets
    std::vector<int32_t> rows, start = t.dfa_start;
    if (t.dfa_sparse) {
        std::vector<int64_t> off(t.S + 1, 0);
        for (int x = 0; x < t.S; x++) off[x + 1] = off[x] + 4 + 2 * (t.dfa_exc_off[x + 1] - t.dfa_exc_off[x]);
        if (off[t.S] + 128 > INT32_MAX) return fail_with(PSC_ERR_LIMIT, "sparse classifier exceeds 2^31 words");
        auto enc = [&](int32_t v) { return v >= 0 ? (int32_t)off[v] : v; };
        rows.assign((size_t)off[t.S] + 128, 0);   // padded: a warp reads 32 pairs past a row's header
        for (int x = 0; x < t.S; x++) {
            int32_t* r = rows.data() + off[x];
            int64_t e0 = t.dfa_exc_off[x], n = t.dfa_exc_off[x + 1] - e0;
            r[0] = (int32_t)n;
            r[1] = enc(t.dfa_def[x]);
            r[2] = t.dfa_mask[x];
            for (int64_t i = 0; i < n; i++) {
                r[4 + 2 * i] = t.dfa_exc_y[e0 + i];
                r[5 + 2 * i] = enc(t.dfa_exc_t[e0 + i]);
            }
        }
        for (int32_t& v : start) v = enc(v);
    } else {
        rows.push_back(0);
    }
    if ((s = upload(h.get(), t.lex_trans, &d.lex_trans)) || (s = upload(h.get(), t.lex_accept, &d.lex_accept)) ||
        (s = upload(h.get(), t.cls_ignored, &d.cls_ignored)) || (s = upload(h.get(), t.action, &d.action)) ||
        (s = upload(h.get(), t.go, &d.go)) || (s = upload(h.get(), t.rule_len, &d.rule_len)) ||
        (s = upload(h.get(), t.rule_lhs, &d.rule_lhs)) || (s = upload(h.get(), t.resolve, &d.resolve)) ||
        (s = upload(h.get(), dfa, &d.dfa)) || (s = upload(h.get(), start, &d.dfa_start)) ||
        (s = upload(h.get(), rows, &d.dfa_rows)) ||
        (s = upload(h.get(), dfa_mask, &d.dfa_mask)) || (s = upload(h.get(), t.mask_chunks, &d.mchunks)) ||
        (s = upload(h.get(), t.mask_rows, &d.mrows)) ||
        (s = upload(h.get(), t.vocab_bytes, &d.vocab, 16)) || (s = upload(h.get(), t.vocab_off, &d.vocab_off)) ||
        (s = upload(h.get(), token_prefixes(t), &d.tok32))) {
        for (int i = 0; i < h->n_blocks; i++) cudaFree(h->blocks[i]);
        return s;
    }
    d.bu = nullptr;
    d.bu_slot = nullptr;
    d.bu_F = nullptr;
    d.bu_len = d.n_frow = 0;
    if (t.n_bu > 0) {
        if ((s = upload(h.get(), t.bu, &d.bu)) || (s = upload(h.get(), t.bu_slot, &d.bu_slot)) ||
            (s = upload(h.get(), t.bu_F, &d.bu_F))) {
            for (int i = 0; i < h->n_blocks; i++) cudaFree(h->blocks[i]);
            return s;
        }
        d.bu_len = (int)t.bu.size();
        d.n_frow = t.n_frow;
    }
    std::vector<uint8_t> blob;
    d.adv_bytes = d.adv_comb = 0;
    if (tables != 1) blob = build_advance_blob(t, d, tables);
    if (!blob.empty()) {
        if ((s = upload(h.get(), blob, &d.adv)) != PSC_OK) {
            for (int i = 0; i < h->n_blocks; i++) cudaFree(h->blocks[i]);
            return s;
        }
        // the limit is per function and device, shared by every handle: raise it to the
        // device's opt-in maximum instead of to this handle's size
        int optin = 0;
        cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, h->device);
        cudaFuncAttributes fa{};
        auto kadv = advance_kernel(d);
        cudaFuncGetAttributes(&fa, kadv);
        optin -= (int)fa.sharedSizeBytes;   // the limit covers dynamic memory only
        if (optin < adv_smem(d)) {
            d.adv_bytes = 0;   // cannot stage: fall back to global tables
        } else if ((s = cuda_check(cudaFuncSetAttribute(kadv, cudaFuncAttributeMaxDynamicSharedMemorySize, optin),
                                   "cudaFuncSetAttribute(k_advance_warp)")) != PSC_OK) {
            for (int i = 0; i < h->n_blocks; i++) cudaFree(h->blocks[i]);
            return s;
        }
    }
    // the TMA masking pass uses more than the default 48 KiB of shared memory
    if ((s = cuda_check(cudaFuncSetAttribute(k_step_tma<uint16_t>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             TmaShape<uint16_t>::SMEM),
                        "cudaFuncSetAttribute(k_step_tma)")) != PSC_OK ||
        (s = cuda_check(cudaFuncSetAttribute(k_step_tma<uint32_t>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             TmaShape<uint32_t>::SMEM),
                        "cudaFuncSetAttribute(k_step_tma)")) != PSC_OK ||
        (s = cuda_check(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&h->tma_ctas[0], k_step_tma<uint16_t>,
                                                                      TMA_WARPS * 32, TmaShape<uint16_t>::SMEM),
                        "cudaOccupancyMaxActiveBlocksPerMultiprocessor(k_step_tma)")) != PSC_OK ||
        (s = cuda_check(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&h->tma_ctas[1], k_step_tma<uint32_t>,
                                                                      TMA_WARPS * 32, TmaShape<uint32_t>::SMEM),
                        "cudaOccupancyMaxActiveBlocksPerMultiprocessor(k_step_tma)")) != PSC_OK) {
        for (int i = 0; i < h->n_blocks; i++) cudaFree(h->blocks[i]);
        return s;
    }
    for (int k = 0; k < 2; k++) h->tma_ctas[k] = std::max(1, h->tma_ctas[k]);
    d.q0 = t.q0;
    d.nq = t.nq;
    d.n_lr = t.n_lr;
    d.n_terms = t.n_terms;
    d.n_nts = t.n_nts;
    d.end_term = t.end_term;
    d.V = t.V;
    d.W = t.W;
    d.nch = t.nch;
    d.dfa_sparse = t.dfa_sparse;
    if (t.dfa_sparse) d.dfa = nullptr;
    d.eos_id = t.eos_id;
    d.n_masks = t.n_masks;
    return PSC_OK;
}
}  // namespace

// ====================================================================== ABI
extern "C" {

const char* psc_last_error(void) { return g_last_error.c_str(); }

psc_status psc_compile(const char* grammar, size_t grammar_len, const uint8_t* vocab_bytes,
                       const int64_t* vocab_offsets, int32_t V, int32_t eos_id, const psc_options* opts,
                       psc_handle** out) {
    if (!out) return fail_with(PSC_ERR_ARG, "psc_compile: out is NULL");
    *out = nullptr;
    if (!grammar || !vocab_offsets || V <= 0 || (!vocab_bytes && vocab_offsets[V] > 0))
        return fail_with(PSC_ERR_ARG, "psc_compile: bad grammar or vocabulary arguments");
    if (eos_id >= V || eos_id < -1) return fail_with(PSC_ERR_ARG, "psc_compile: eos_id out of range");
    for (int v = 0; v < V; v++)
        if (vocab_offsets[v + 1] < vocab_offsets[v]) return fail_with(PSC_ERR_ARG, "psc_compile: offsets decrease");
    psc::Options o;
    bool host_only = false;
    int tables = 0;
    if (opts) {
        if (opts->max_states > 0) o.max_states = opts->max_states;
        if (opts->max_mask_bytes > 0) o.max_mask_bytes = opts->max_mask_bytes;
        o.threads = opts->threads;
        o.max_bottom_up_bytes = opts->max_bottom_up_bytes;
        o.max_dense_classifier_bytes = opts->max_dense_classifier_bytes;
        host_only = opts->host_only != 0;
        tables = opts->global_tables;
        if (tables < 0 || tables > 2) return fail_with(PSC_ERR_ARG, "psc_compile: global_tables must be 0, 1 or 2");
    }
    std::unique_ptr<psc_handle> h(new (std::nothrow) psc_handle());
    if (!h) return fail_with(PSC_ERR_OOM, "psc_compile: out of host memory");
    try {
        h->t = psc::compile_tables(std::string(grammar, grammar_len), vocab_bytes, vocab_offsets, V, eos_id, o);
    } catch (const psc::Error& e) {
        return fail_with((psc_status)e.code, e.what());
    } catch (const std::bad_alloc&) {
        return fail_with(PSC_ERR_OOM, "psc_compile: out of host memory");
    }
    h->host_only = host_only;
    h->tables = tables;
    if (!host_only) {
        psc_status s = upload_tables(h, tables);
        if (s != PSC_OK) return s;
    }
    *out = h.release();
    return PSC_OK;
}

void psc_destroy(psc_handle* h) {
    if (!h) return;
    for (int i = 0; i < h->n_blocks; i++) cudaFree(h->blocks[i]);
    delete h;
}

psc_status psc_info(const psc_handle* h, psc_info_t* out) {
    if (!h || !out) return fail_with(PSC_ERR_ARG, "psc_info: NULL argument");
    const psc::Tables& t = h->t;
    out->V = t.V;
    out->W = t.W;
    out->n_lexer_states = t.nq;
    out->n_parser_states = t.n_lr;
    out->n_terminals = t.n_terms;
    out->n_classifier_states = t.S;
    out->n_masks = t.n_masks;
    out->eos_id = t.eos_id;
    out->classifier_bytes = (int64_t)(t.dfa.size() + t.dfa_start.size() + t.dfa_mask.size()) * 4;
    if (t.dfa_sparse) out->classifier_bytes = (int64_t)(4 * (int64_t)t.S + 2 * (int64_t)t.dfa_exc_y.size() + t.nq) * 4;
    out->classifier_sparse = t.dfa_sparse;
    out->mask_bytes = (int64_t)(t.mask_rows.size() + t.mask_chunks.size()) * 4;
    out->states_built = t.n_dfa_states_built;
    out->compile_seconds = t.seconds_total;
    if (h->host_only) {   // what a device upload with the handle's placement would stage
        DevTables tmp{};
        if (h->tables != 1) build_advance_blob(t, tmp, h->tables);
        out->advance_table_bytes = tmp.adv_bytes;
        out->advance_tables_packed = tmp.adv_bytes > 0 && tmp.adv_comb;
    } else {
        out->advance_table_bytes = h->d.adv_bytes;
        out->advance_tables_packed = h->d.adv_bytes > 0 && h->d.adv_comb;
    }
    out->bottom_up_states = t.n_bu;
    out->bottom_up_bytes = (int64_t)(t.bu.size() + t.bu_F.size()) * 4 + (int64_t)t.bu_slot.size() * 2;
    out->device_timeouts = 0;
    if (!h->host_only) {
        int v = 0;
        if (cudaMemcpyFromSymbol(&v, g_pipeline_timeouts, sizeof(int)) == cudaSuccess) out->device_timeouts = v;
    }
    return PSC_OK;
}

psc_status psc_state_init(const psc_handle* h, int32_t B, int32_t cap, void* stream, psc_states** out) {
    if (!out) return fail_with(PSC_ERR_ARG, "psc_state_init: out is NULL");
    *out = nullptr;
    psc_status s = check_device(h, "psc_state_init");
    if (s != PSC_OK) return s;
    if (B <= 0 || cap < 2 || cap > (1 << 20)) return fail_with(PSC_ERR_ARG, "psc_state_init: bad B or cap");
    std::unique_ptr<psc_states> st(new (std::nothrow) psc_states());
    if (!st) return fail_with(PSC_ERR_OOM, "psc_state_init: out of host memory");
    st->h = h;
    st->device = h->device;
    DevStates& d = st->d;
    d.B = B;
    d.cap = cap;
    // the fault word, then the bottom-up classifier's kept blocks only when the handle has
    // that classifier
    const int n_arr = h->d.bu ? 8 : 7;
    void* p[8] = {};
    size_t sz[8] = {sizeof(int32_t) * B, sizeof(int32_t) * B, sizeof(int32_t) * B, sizeof(uint16_t) * (size_t)B * cap,
                    sizeof(int32_t) * B, sizeof(unsigned long long) * B, sizeof(int32_t),
                    sizeof(int32_t) * (size_t)B * cap};
    for (int i = 0; i < n_arr; i++) {
        s = cuda_check(cudaMalloc(&p[i], sz[i]), "cudaMalloc(states)");
        if (s != PSC_OK) {
            for (int j = 0; j < i; j++) cudaFree(p[j]);
            return s;
        }
    }
    d.q = (int32_t*)p[0];
    d.depth = (int32_t*)p[1];
    d.status = (int32_t*)p[2];
    d.stack = (uint16_t*)p[3];
    d.mid = (int32_t*)p[4];
    d.best = (unsigned long long*)p[5];
    d.fault = (int32_t*)p[6];
    d.rmemo = (int32_t*)p[7];
    cudaStream_t cs = (cudaStream_t)stream;
    s = cuda_check(cudaMemsetAsync(d.fault, 0, sizeof(int32_t), cs), "cudaMemsetAsync(fault)");
    if (s == PSC_OK) {
        k_state_init<<<(B + 255) / 256, 256, 0, cs>>>(d, h->d.q0, nullptr, B);
        s = launch_check("k_state_init");
    }
    if (s != PSC_OK) {
        for (int j = 0; j < n_arr; j++) cudaFree(p[j]);
        return s;
    }
    *out = st.release();
    return PSC_OK;
}

psc_status psc_state_copy(psc_states* dst, const psc_states* src, void* stream) {
    if (!dst || !src || dst->h != src->h || dst->d.B != src->d.B || dst->d.cap != src->d.cap)
        return fail_with(PSC_ERR_ARG, "psc_state_copy: states of different handles or shapes");
    if (dst == src) return PSC_OK;
    int dev = -1;
    cudaGetDevice(&dev);
    if (dev != dst->device) return fail_with(PSC_ERR_ARG, "psc_state_copy: current device differs from the states'");
    cudaStream_t cs = (cudaStream_t)stream;
    const DevStates& a = src->d;
    DevStates& b = dst->d;
    size_t B = (size_t)a.B;
    // one kernel for all the arrays (a copy per array costs a stream round trip each)
    CopySegs c{};
    auto add = [&](const void* src, void* dst, size_t bytes) {
        c.src[c.n] = static_cast<const uint8_t*>(src);
        c.dst[c.n] = static_cast<uint8_t*>(dst);
        c.bytes[c.n++] = bytes;
    };
    add(a.q, b.q, B * 4);
    add(a.depth, b.depth, B * 4);
    add(a.status, b.status, B * 4);
    add(a.stack, b.stack, B * (size_t)a.cap * 2);
    add(a.mid, b.mid, B * 4);
    if (a.best && b.best) add(a.best, b.best, B * 8);
    if (a.rmemo && b.rmemo) add(a.rmemo, b.rmemo, B * (size_t)a.cap * 4);
    size_t v16 = (B * (size_t)a.cap * 6 + B * 24) / 16;
    int grid = (int)std::max<size_t>(1, std::min<size_t>((v16 + 255) / 256, (size_t)sm_count(dev) * 4));
    psc_status s = launch_pdl(k_state_copy, dim3(grid), dim3(256), 0, cs, "k_state_copy", c);
    if (s != PSC_OK) return s;
    dst->gen++;
    dst->mid_gen = src->mid_gen == src->gen ? dst->gen : 0;   // the mask ids are as current as src's
    dst->after_mask = false;
    return PSC_OK;
}

psc_status psc_state_reset(psc_states* st, const int32_t* d_rows, int32_t n, void* stream) {
    if (!st) return fail_with(PSC_ERR_ARG, "psc_state_reset: NULL states");
    int cnt = d_rows ? n : st->d.B;
    if (cnt < 0) return fail_with(PSC_ERR_ARG, "psc_state_reset: negative count");
    st->gen++;
    st->after_mask = false;
    if (cnt == 0) return PSC_OK;
    k_state_init<<<(cnt + 255) / 256, 256, 0, (cudaStream_t)stream>>>(st->d, st->h->d.q0, d_rows, cnt);
    return launch_check("k_state_init");
}

void psc_state_destroy(psc_states* st) {
    if (!st) return;
    cudaFree(st->d.q);
    cudaFree(st->d.depth);
    cudaFree(st->d.status);
    cudaFree(st->d.stack);
    cudaFree(st->d.mid);
    cudaFree(st->d.best);
    cudaFree(st->d.fault);
    cudaFree(st->d.rmemo);
    delete st;
}

psc_status psc_advance(const psc_handle* h, psc_states* st, const int32_t* d_tokens, int32_t B,
                       int32_t* d_row_status, void* stream) {
    psc_status s = check_device(h, "psc_advance");
    if (s != PSC_OK) return s;
    if (!st || st->h != h || B != st->d.B || !d_tokens) return fail_with(PSC_ERR_ARG, "psc_advance: bad arguments");
    int use_mid = st->mid_gen == st->gen ? 1 : 0;
    return launch_advance(h, st, d_tokens, use_mid, d_row_status, nullptr, (cudaStream_t)stream);
}

psc_status psc_fill_mask(const psc_handle* h, const psc_states* st, int32_t B, uint32_t* d_bitmask, void* stream) {
    psc_status s = check_device(h, "psc_fill_mask");
    if (s != PSC_OK) return s;
    if (!st || st->h != h || B != st->d.B || !d_bitmask) return fail_with(PSC_ERR_ARG, "psc_fill_mask: bad arguments");
    cudaStream_t cs = (cudaStream_t)stream;
    if ((s = ensure_mid(h, st, cs)) != PSC_OK) return s;
    int vec = (h->d.W % 4 == 0) && aligned16(d_bitmask);
    size_t units = vec ? (size_t)B * (h->d.W / 4) : (size_t)B * h->d.W;
    int blocks = (int)std::min<size_t>((units + 255) / 256, (size_t)sm_count(h->device) * 8);
    if (blocks < 1) blocks = 1;
    k_fill<<<blocks, 256, 0, cs>>>(h->d, st->d.mid, B, d_bitmask, vec);
    return launch_check("k_fill");
}

psc_status psc_apply_mask(void* d_logits, psc_dtype dtype, int64_t row_stride, const uint32_t* d_bitmask, int32_t B,
                          int32_t V, void* stream) {
    if (!d_logits || !d_bitmask || B < 0 || V <= 0 || row_stride < V || (dtype != PSC_F32 && dtype != PSC_BF16))
        return fail_with(PSC_ERR_ARG, "psc_apply_mask: bad arguments");
    if (B == 0) return PSC_OK;
    int dev = 0;
    cudaGetDevice(&dev);
    MaskSrc M{d_bitmask, nullptr, nullptr, nullptr, (V + 31) / 32, 0, nullptr};
    return launch_apply(d_logits, dtype, row_stride, M, B, V, (cudaStream_t)stream, dev);
}

psc_status psc_fill_apply(const psc_handle* h, const psc_states* st, int32_t B, void* d_logits, psc_dtype dtype,
                          int64_t row_stride, int32_t V, uint32_t* d_bitmask_out, void* stream) {
    psc_status s = check_device(h, "psc_fill_apply");
    if (s != PSC_OK) return s;
    if (!st || st->h != h || B != st->d.B || !d_logits || V != h->d.V || row_stride < V ||
        (dtype != PSC_F32 && dtype != PSC_BF16))
        return fail_with(PSC_ERR_ARG, "psc_fill_apply: bad arguments");
    cudaStream_t cs = (cudaStream_t)stream;
    if ((s = ensure_mid(h, st, cs)) != PSC_OK) return s;
    MaskSrc M{nullptr, h->d.mchunks, h->d.mrows, st->d.mid, h->d.W, h->d.nch, d_bitmask_out};
    return launch_apply(d_logits, dtype, row_stride, M, B, V, cs, h->device);
}

psc_status psc_argmax_masked(const psc_handle* h, const psc_states* st, int32_t B, const void* d_logits,
                             psc_dtype dtype, int64_t row_stride, int32_t V, int32_t* d_tokens, void* stream) {
    psc_status s = check_device(h, "psc_argmax_masked");
    if (s != PSC_OK) return s;
    if (!st || st->h != h || B != st->d.B || !d_logits || !d_tokens || V != h->d.V || row_stride < V ||
        (dtype != PSC_F32 && dtype != PSC_BF16))
        return fail_with(PSC_ERR_ARG, "psc_argmax_masked: bad arguments");
    cudaStream_t cs = (cudaStream_t)stream;
    if ((s = ensure_mid(h, st, cs)) != PSC_OK) return s;
    size_t esz = dtype == PSC_BF16 ? 2 : 4;
    int vec = aligned16(d_logits) && ((row_stride * (int64_t)esz) % 16 == 0);
    if (dtype == PSC_BF16)
        k_argmax_masked<uint16_t><<<B, 256, 0, cs>>>((const uint16_t*)d_logits, row_stride, h->d, st->d.mid, B, V, vec,
                                                     d_tokens);
    else
        k_argmax_masked<uint32_t><<<B, 256, 0, cs>>>((const uint32_t*)d_logits, row_stride, h->d, st->d.mid, B, V, vec,
                                                     d_tokens);
    return launch_check("k_argmax_masked");
}

psc_status psc_fill_apply_argmax(const psc_handle* h, const psc_states* st, int32_t B, void* d_logits,
                                 psc_dtype dtype, int64_t row_stride, int32_t V, uint32_t* d_bitmask_out,
                                 int32_t* d_tokens, void* stream) {
    psc_status s = check_device(h, "psc_fill_apply_argmax");
    if (s != PSC_OK) return s;
    if (!st || st->h != h || B != st->d.B || !d_logits || !d_tokens || V != h->d.V || row_stride < V ||
        (dtype != PSC_F32 && dtype != PSC_BF16))
        return fail_with(PSC_ERR_ARG, "psc_fill_apply_argmax: bad arguments");
    cudaStream_t cs = (cudaStream_t)stream;
    if ((s = launch_fused(h, st, d_logits, dtype, row_stride, V, d_bitmask_out, cs)) != PSC_OK) return s;
    const_cast<psc_states*>(st)->after_mask = false;
    k_finalize_tokens<<<(B + 255) / 256, 256, 0, cs>>>(st->d.best, B, d_tokens);
    return launch_check("k_finalize_tokens");
}

psc_status psc_decode_step(const psc_handle* h, psc_states* st, int32_t B, void* d_logits, psc_dtype dtype,
                           int64_t row_stride, int32_t V, uint32_t* d_bitmask_out, int32_t* d_tokens,
                           int32_t* d_row_status, void* stream) {
    psc_status s = check_device(h, "psc_decode_step");
    if (s != PSC_OK) return s;
    if (!st || st->h != h || B != st->d.B || !d_logits || !d_tokens || V != h->d.V || row_stride < V ||
        (dtype != PSC_F32 && dtype != PSC_BF16))
        return fail_with(PSC_ERR_ARG, "psc_decode_step: bad arguments");
    cudaStream_t cs = (cudaStream_t)stream;
    if ((s = launch_fused(h, st, d_logits, dtype, row_stride, V, d_bitmask_out, cs)) != PSC_OK) return s;
    return launch_advance(h, st, nullptr, 1, d_row_status, d_tokens, cs);
}

psc_status psc_decode_step_mask(const psc_handle* h, psc_states* st, int32_t B, void* d_logits, psc_dtype dtype,
                                int64_t row_stride, int32_t V, uint32_t* d_bitmask_out, void* stream) {
    psc_status s = check_device(h, "psc_decode_step_mask");
    if (s != PSC_OK) return s;
    if (!st || st->h != h || B != st->d.B || !d_logits || V != h->d.V || row_stride < V ||
        (dtype != PSC_F32 && dtype != PSC_BF16))
        return fail_with(PSC_ERR_ARG, "psc_decode_step_mask: bad arguments");
    return launch_fused(h, st, d_logits, dtype, row_stride, V, d_bitmask_out, (cudaStream_t)stream);
}

psc_status psc_decode_step_advance(const psc_handle* h, psc_states* st, int32_t B, int32_t* d_tokens,
                                   int32_t* d_row_status, void* stream) {
    psc_status s = check_device(h, "psc_decode_step_advance");
    if (s != PSC_OK) return s;
    if (!st || st->h != h || B != st->d.B || !d_tokens)
        return fail_with(PSC_ERR_ARG, "psc_decode_step_advance: bad arguments");
    // the greedy keys were made for the mask ids the masking pass used (current
    // unless rows changed since): the advance checks tokens against those
    return launch_advance(h, st, nullptr, 1, d_row_status, d_tokens, (cudaStream_t)stream);
}

psc_status psc_states_download(const psc_states* st, int32_t* h_q, int32_t* h_depth, uint16_t* h_stack,
                               int32_t* h_status, void* stream) {
    if (!st) return fail_with(PSC_ERR_ARG, "psc_states_download: NULL states");
    cudaStream_t cs = (cudaStream_t)stream;
    const DevStates& d = st->d;
    psc_status s = PSC_OK;
    if (h_q && (s = cuda_check(cudaMemcpyAsync(h_q, d.q, sizeof(int32_t) * d.B, cudaMemcpyDeviceToHost, cs), "download q")))
        return s;
    if (h_depth && (s = cuda_check(cudaMemcpyAsync(h_depth, d.depth, sizeof(int32_t) * d.B, cudaMemcpyDeviceToHost, cs),
                                   "download depth")))
        return s;
    if (h_stack && (s = cuda_check(cudaMemcpyAsync(h_stack, d.stack, sizeof(uint16_t) * (size_t)d.B * d.cap,
                                                   cudaMemcpyDeviceToHost, cs),
                                   "download stack")))
        return s;
    if (h_status && (s = cuda_check(cudaMemcpyAsync(h_status, d.status, sizeof(int32_t) * d.B, cudaMemcpyDeviceToHost, cs),
                                    "download status")))
        return s;
    return cuda_check(cudaStreamSynchronize(cs), "cudaStreamSynchronize");
}

psc_status psc_state_faults(psc_states* st, int32_t* h_faults, int32_t reset, void* stream) {
    if (!st || !h_faults) return fail_with(PSC_ERR_ARG, "psc_state_faults: NULL argument");
    cudaStream_t cs = (cudaStream_t)stream;
    psc_status s = cuda_check(cudaMemcpyAsync(h_faults, st->d.fault, sizeof(int32_t), cudaMemcpyDeviceToHost, cs),
                              "psc_state_faults");
    if (s == PSC_OK) s = cuda_check(cudaStreamSynchronize(cs), "cudaStreamSynchronize");
    if (s == PSC_OK && reset)
        s = cuda_check(cudaMemsetAsync(st->d.fault, 0, sizeof(int32_t), cs), "cudaMemsetAsync(fault)");
    return s;
}

psc_status psc_check_wait(psc_states* st, int32_t limit, void* stream) {
    if (!st || limit < 1 || limit > (1 << 24)) return fail_with(PSC_ERR_ARG, "psc_check_wait: bad arguments");
    int dev = -1;
    cudaGetDevice(&dev);
    if (dev != st->device) return fail_with(PSC_ERR_ARG, "psc_check_wait: current device differs from the states'");
    k_wait_gives_up<<<1, 32, 0, (cudaStream_t)stream>>>(st->d, limit);
    return launch_check("k_wait_gives_up");
}

int32_t psc_host_classify(const psc_handle* h, int32_t q, const uint16_t* h_stack, int32_t depth, int32_t status) {
    if (!h || (depth > 0 && !h_stack) || depth < 0) return -1;
    for (int i = 0; i < depth; i++)
        if (h_stack[i] >= h->t.n_lr) return -1;
    return psc::classify_host(h->t, q, h_stack, depth, status);
}

int32_t psc_host_classify_bottom_up(const psc_handle* h, int32_t q, const uint16_t* h_stack, int32_t depth,
                                    int32_t status) {
    if (!h || (depth > 0 && !h_stack) || depth < 0) return -1;
    for (int i = 0; i < depth; i++)
        if (h_stack[i] >= h->t.n_lr) return -1;
    return psc::classify_host_bottom_up(h->t, q, h_stack, depth, status);
}

psc_status psc_host_mask_row(const psc_handle* h, int32_t mask_id, uint32_t* h_row) {
    if (!h || !h_row || mask_id < 0 || mask_id >= h->t.n_masks) return fail_with(PSC_ERR_ARG, "psc_host_mask_row: bad arguments");
    const psc::Tables& t = h->t;
    for (int c = 0; c < t.nch; c++) {   // chunk by chunk
        int nw = std::min(32, t.W - c * 32);
        std::memcpy(h_row + c * 32, t.mask_chunks.data() + (size_t)t.mask_rows[(size_t)mask_id * t.nch + c] * 32,
                    sizeof(uint32_t) * nw);
    }
    return PSC_OK;
}

psc_status psc_host_advance(const psc_handle* h, int32_t* q, uint16_t* h_stack, int32_t* depth, int32_t cap,
                            int32_t* status, int32_t tok) {
    if (!h || !q || !h_stack || !depth || !status || cap < 2 || *depth < 1 || *depth > cap)
        return fail_with(PSC_ERR_ARG, "psc_host_advance: bad arguments");
    const psc::Tables& T = h->t;
    if (*q < 0 || *q >= T.nq) return fail_with(PSC_ERR_ARG, "psc_host_advance: lexer state out of range");
    for (int i = 0; i < *depth; i++)
        if (h_stack[i] >= T.n_lr) return fail_with(PSC_ERR_ARG, "psc_host_advance: stack entry out of range");
    if (tok < 0) return PSC_OK;
    int st = *status;
    if (st == ROW_DONE) {
        *status = tok == T.eos_id ? ROW_DONE : ROW_REJECTED;
        return PSC_OK;
    }
    if (st != ROW_OK) return PSC_OK;
    if (tok >= T.V) {
        *status = ROW_REJECTED;
        return PSC_OK;
    }
    int mid = psc::classify_host(T, *q, h_stack, *depth, st);
    if (mid < 0 || !((psc::mask_word(T, mid, tok >> 5) >> (tok & 31)) & 1)) {
        *status = ROW_REJECTED;
        return PSC_OK;
    }
    if (tok == T.eos_id) {
        *status = ROW_DONE;
        return PSC_OK;
    }
    int cq = *q, d = *depth;
    for (int64_t i = T.vocab_off[tok]; i < T.vocab_off[tok + 1] && st == ROW_OK; i++) {
        int c = T.vocab_bytes[i];
        int nx = T.lex_trans[(size_t)cq * 256 + c];
        if (nx >= 0) {
            cq = nx;
            continue;
        }
        int cls = cq == T.q0 ? -1 : T.lex_accept[cq];
        if (cls < 0) {
            st = ROW_REJECTED;
            break;
        }
        if (!T.cls_ignored[cls]) st = host_feed(T, h_stack, d, cap, cls);
        cq = T.lex_trans[(size_t)T.q0 * 256 + c];
        if (cq < 0) st = ROW_REJECTED;
    }
    if (st == ROW_OK) {
        *q = cq;
        *depth = d;
    }
    *status = st;
    return PSC_OK;
}

psc_status psc_fill_apply_noalloc(const psc_handle* h, const int32_t* d_q, const int32_t* d_depth,
                                  const int32_t* d_status, const uint16_t* d_stack, int32_t cap, int32_t B,
                                  void* d_logits, psc_dtype dtype, int64_t row_stride, int32_t V,
                                  uint32_t* d_bitmask_out, void* stream) {
    psc_status s = check_device(h, "psc_fill_apply_noalloc");
    if (s != PSC_OK) return s;
    if (B > PSC_NOALLOC_MAX_ROWS)
        return fail_with(PSC_ERR_LIMIT, "psc_fill_apply_noalloc: B = " + std::to_string(B) +
                                            " exceeds PSC_NOALLOC_MAX_ROWS = " + std::to_string(PSC_NOALLOC_MAX_ROWS));
    if (B <= 0 || !d_q || !d_depth || !d_status || !d_stack || cap < 2 || !d_logits || V != h->d.V ||
        row_stride < V || (dtype != PSC_F32 && dtype != PSC_BF16))
        return fail_with(PSC_ERR_ARG, "psc_fill_apply_noalloc: bad arguments");
    int32_t* mid = nullptr;
    if ((s = noalloc_scratch(h->device, &mid)) != PSC_OK) return s;
    DevStates S{const_cast<int32_t*>(d_q), const_cast<int32_t*>(d_depth), const_cast<int32_t*>(d_status),
                const_cast<uint16_t*>(d_stack), mid, B, cap};
    cudaStream_t cs = (cudaStream_t)stream;
    int threads = 256;
    int blocks = (int)(((size_t)B * 32 + threads - 1) / threads);
    k_classify<<<blocks, threads, 0, cs>>>(h->d, S, B);
    if ((s = launch_check("k_classify")) != PSC_OK) return s;
    MaskSrc M{nullptr, h->d.mchunks, h->d.mrows, mid, h->d.W, h->d.nch, d_bitmask_out};
    return launch_apply(d_logits, dtype, row_stride, M, B, V, cs, h->device);
}

psc_status psc_save(const psc_handle* h, const char* path) {
    if (!h || !path) return fail_with(PSC_ERR_ARG, "psc_save: NULL argument");
    try {
        psc::save_tables(h->t, path);
    } catch (const psc::Error& e) {
        return fail_with((psc_status)e.code, e.what());
    } catch (const std::bad_alloc&) {
        return fail_with(PSC_ERR_OOM, "psc_save: out of host memory");
    }
    return PSC_OK;
}

psc_status psc_load(const char* path, const psc_options* opts, psc_handle** out) {
    if (!out || !path) return fail_with(PSC_ERR_ARG, "psc_load: NULL argument");
    *out = nullptr;
    std::unique_ptr<psc_handle> h(new (std::nothrow) psc_handle());
    if (!h) return fail_with(PSC_ERR_OOM, "psc_load: out of host memory");
    try {
        h->t = psc::load_tables(path);
    } catch (const psc::Error& e) {
        return fail_with((psc_status)e.code, e.what());
    } catch (const std::bad_alloc&) {
        return fail_with(PSC_ERR_OOM, "psc_load: out of host memory");
    }
    if (opts && opts->max_bottom_up_bytes < 0) {   // drop the bottom-up classifier
        psc::Tables& t = h->t;
        t.bu.clear();
        t.bu_slot.clear();
        t.bu_F.clear();
        t.bu_t.clear();
        t.bu_root = -1;
        t.n_bu = t.n_frow = 0;
    }
    h->host_only = opts && opts->host_only;
    h->tables = opts ? opts->global_tables : 0;
    if (h->tables < 0 || h->tables > 2) return fail_with(PSC_ERR_ARG, "psc_load: global_tables must be 0, 1 or 2");
    if (!h->host_only) {
        psc_status s = upload_tables(h, h->tables);
        if (s != PSC_OK) return s;
    }
    *out = h.release();
    return PSC_OK;
}

}  // extern "C"
