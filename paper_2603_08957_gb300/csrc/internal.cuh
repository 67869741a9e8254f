// internal.cuh -- declarations shared by the executor's translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <cstring>
#include <string>
#include <vector>

#include "ucl.h"

namespace ucl {

constexpr int kMaxCols = 15;     // key columns or tile dims of one operand
constexpr int kMaxLow = 30;      // lower labels of one binary EinSum

// Device status bits written by kernels (atomicOr into ctx->d_status).
enum : uint32_t {
    kStTimeout = 1u,     // a bounded wait ran out
    kStBadIndex = 2u,    // an index failed its bounds check; the access was skipped
    kStKeyRange = 4u,    // key outside [0, bound)
    kStUnsorted = 8u,    // keys not strictly ascending
    kStDupKey = 16u,     // two equal keys
};

// One key column copied into a bit field of a packed 64-bit key.
struct KeyField {
    int col;
    int shift;
    int bits;
    int rshift;   // the field holds the column's value >> rshift (0: the whole value)
};

// How to build one packed key from a relation's key row.
struct KeyPack {
    int nf;
    KeyField f[kMaxCols];
};

// Unpacking of the packed output key into the output relation's columns.
struct KeyUnpack {
    int uw;
    int shift[kMaxCols];
    int bits[kMaxCols];
};

// Generic lower-label contraction of one joined pair (FFMA path):
//   W[w] += sum_c U[offU(w) + cU(c)] * V[offV(w) + cV(c)] (* X[offX(w) + cX(c)])
// w runs over W's lower labels (row-major, W's order), c over the lower
// labels absent from W; X is the third input of a three-way EinSum.
struct LowerPlan {
    int nw;
    int w_ext[kMaxCols];
    int w_su[kMaxCols];
    int w_sv[kMaxCols];
    int w_sx[kMaxCols];
    int nc;
    int c_ext[kMaxLow];
    int c_su[kMaxLow];
    int c_sv[kMaxLow];
    int c_sx[kMaxLow];
    int64_t tile_u, tile_v, tile_x, tile_w, n_c;
};

// tcgen05 contraction shape: D[M x N] += A[M x K] * B[K x N] per pair, with
// D = the output tile up to a transpose.
struct TcPlan {
    int a_is_u;          // A operand tiles come from U (else from V)
    int M, N, K;         // M = 128 * m_blocks
    int m_blocks;
    int a_kmajor;        // A tile rows run over M (K contiguous) if 1, rows over K if 0
    int b_kmajor;        // B tile rows run over N (K contiguous) if 1, rows over K if 0
    int64_t sWm, sWn;    // output tile strides of the M and N indices
};

// tcgen05 three-way contraction of the MTTKRP shape (one label of each
// kind): W[i][r] += sum_{j,k} T[i][j][k] * E[j][r] * F[k][r], with the T
// tile laid out [i][j][k] and the F tile [k][r]; i = j = k = 16, r = 64.
struct Tc3Plan {
    int t, e, f;             // spec positions of T, the epilogue factor E, the MMA factor F
    bool t_mn;               // T tiles laid out [f][i][e] (else [i][e][f])
    int64_t sEj, sEr;        // E tile strides of j and r
    int64_t sWi, sWr;        // output tile strides of i and r
};

// Partition of the pair list into G contiguous units (one CTA each): unit u
// covers pairs [begin(u), begin(u + 1)) of the P pairs that start at `base`.
struct Units {
    int64_t P;
    int G;
    int64_t base;
    // Optional cut at segment boundaries: unit u starts at segment S * u / G
    // (seg: the S + 1 segment starts, device memory, seg[S] = the end), so no
    // segment spans two units and no partial or fixup is needed (G <= S).
    const int64_t *seg = nullptr;
    int64_t S = 0;
    __host__ __device__ int64_t begin(int u) const { return seg ? seg[S * u / G] : base + P * u / G; }
};

// Stream-ordered bump allocator over blocks obtained from the context hooks.
struct Arena {
    struct Block {
        char *ptr;
        size_t size;
    };
    std::vector<Block> blocks;
    size_t used = 0;   // bytes used in the last block
    size_t total() const {
        size_t t = 0;
        for (auto &b : blocks) t += b.size;
        return t;
    }
};

}  // namespace ucl

struct ucl_ctx {
    int device = 0;
    // Streams.  `main` is the caller's: relation storage, contractions and
    // results live in its order.  The key stage of ucl_einsum (joins, sorts,
    // sizing syncs) runs on `kstream`, so it overlaps the contractions still
    // queued on main; `stream` is the one launches go to right now.
    cudaStream_t stream = nullptr;
    cudaStream_t main = nullptr;
    cudaStream_t kstream = nullptr;
    cudaEvent_t ev_order = nullptr;   // scratch event for one-off stream ordering
    // Tile copies of ucl_relation_create run on `cstream`, so that the key
    // validation on main (and the next call's key stage) overlaps them;
    // ev_copy0 orders the copy after main's earlier work, ev_copy1 orders
    // main after the copy.
    cudaStream_t cstream = nullptr;
    cudaEvent_t ev_copy0 = nullptr, ev_copy1 = nullptr;
    ucl_alloc_fn alloc = nullptr;
    ucl_free_fn free_fn = nullptr;
    void *user = nullptr;
    int sm_count = 0;
    // Workspace arenas used by successive calls in turn; arena_done[i] is
    // recorded on main when the call using arena i has finished with it.
    static constexpr int kArenas = 4;
    ucl::Arena arenas[kArenas];
    cudaEvent_t arena_done[kArenas] = {};
    int arena_next = 0;
    ucl::Arena *arena = &arenas[0];
    // [1] validation flags (main), [2] sticky error bits of main-stream kernels,
    // words [16, 18): the fixup kernels' byte counter (64-bit)
    uint32_t *d_status = nullptr;
    static constexpr int kFixupCounterWord = 16;
    // pinned host scratch for sizing syncs: kPinnedRead int64 values, then the
    // device status words
    static constexpr int kPinnedRead = 36, kPinnedWords = 40;
    int64_t *h_pinned = nullptr;
    int timing = 0;
    // CUDA events of timed calls: six per call (stage boundaries on the key
    // stream and on main), reused
    // after ucl_ctx_timings(..., reset = 1)
    std::vector<cudaEvent_t> ev_pool;
    int ev_calls = 0;      // calls recorded since the last reset
    cudaEvent_t *cur_ev = nullptr;
    int launches = 0;
    ucl_stats last{};
    std::string err;
    int live_rels = 0;
    // Overrides read from the environment at creation, for measurement:
    // UCL_BANDS (unset: automatic; 0 or 1: no banding; 2..16: that many
    // bands where banding applies) and UCL_L2_HINTS (0: no L2 eviction hints).
    int tune_bands = -1;
    int tune_hints = 1;
    // UCL_TC_STAGES (pipeline stages of the binary tcgen05 kernel, 0: its own
    // choice), UCL_TC_MMA (1: one MMA warp; 0: its own choice) and
    // UCL_TC_PREFETCH (-1: its own rule; 0: no L2 prefetch; 1: prefetch the
    // streamed operand)
    int tune_tc_stages = 0;
    int tune_tc_mma = 0;
    // UCL_SEG_UNITS (0: always split pair lists evenly into work units, so
    // that segments may span units; else small lists are cut at segment
    // boundaries)
    int tune_seg_units = 1;
    int tune_tc_prefetch = -1;
    // UCL_WINDOW (-1 or unset: automatic; 0: no windows; n: windows of 2^n
    // output keys where the windowed tcgen05 kernel applies)
    int tune_window = -1;
    int l2_bytes = 0;
    // Bounded waits of the tcgen05 kernel: SM cycles before a role gives up
    // (0: the kernel's default of about a second), and the failure-detection
    // test hook that makes the next launch skip one stage fill (-1: none).
    long long wait_limit_cycles = 0;
    int withhold_fill = -1;
};

struct ucl_rel {
    ucl_ctx *ctx = nullptr;
    int64_t n = 0;
    int u = 0, r = 0;
    int64_t bounds[ucl::kMaxCols] = {};
    int64_t shape[ucl::kMaxCols] = {};
    ucl_dtype dtype = UCL_F32;
    int64_t tile = 1;            // elements per tile
    int32_t *keys = nullptr;     // device [n, u]
    void *tiles = nullptr;       // device [n, tile]
    void *own_block = nullptr;   // library-owned allocation (keys + tiles), or NULL
    size_t own_bytes = 0;
    int sorted = 0;              // keys strictly ascending lexicographically
    int key_bits = 0;            // sum of column bit widths
    cudaEvent_t ev_keys = nullptr;   // recorded on main once keys are valid (key-stream readers wait on it)
};

namespace ucl {

// ---- context helpers (api.cu)
void *ctx_alloc(ucl_ctx *ctx, size_t bytes);
void ctx_free(ucl_ctx *ctx, void *p, size_t bytes);
void *ws_get(ucl_ctx *ctx, size_t bytes);   // workspace of the current call's arena
// Order the stream in use after everything enqueued on main so far (no-op on main).
void order_after_main(ucl_ctx *ctx);
ucl_status fail(ucl_ctx *ctx, ucl_status st, const std::string &msg);
ucl_status cuda_check(ucl_ctx *ctx, cudaError_t e, const char *what);
int bit_width(int64_t bound);   // bits to store values in [0, bound)

// ---- key stage (keys.cu)
// Pack each row of keys[n, u] into a 64-bit key; optional second packing.
void launch_pack(ucl_ctx *ctx, const int32_t *keys, int u, int64_t n, KeyPack a, uint64_t *out_a, KeyPack b,
                 uint64_t *out_b);
// Validate keys of a relation: range check against bounds and strict ascending
// order of the packed full key (sets kStKeyRange / kStUnsorted).
void launch_check_keys(ucl_ctx *ctx, const int32_t *keys, int u, int64_t n, const int64_t *bounds, KeyPack full,
                       uint64_t *packed_out);
// Adjacent-equal check on a sorted array (sets kStDupKey).
void launch_check_dups(ucl_ctx *ctx, const uint64_t *sorted_keys, int64_t n);
// Stable LSD radix sort of (key, value) by the low `bits` bits of key.
// kin/vin and kalt/valt are ping-pong buffers; returns which holds the result
// (0: kin/vin, 1: kalt/valt).  vin may be NULL (keys only).
int radix_sort(ucl_ctx *ctx, uint64_t *kin, uint64_t *vin, uint64_t *kalt, uint64_t *valt, int64_t n, int bits,
               int lo = 0);
// Exclusive scan of n int64 values; writes total to *total_dev if non-NULL.
void scan_i64(ucl_ctx *ctx, const int64_t *in, int64_t *out, int64_t n, int64_t *total_dev);
// iota into u64
void launch_iota(ucl_ctx *ctx, uint64_t *out, int64_t n);
// Join count: for each U row i (sorted join keys jku), the matching range of V.
void launch_join_count(ucl_ctx *ctx, const uint64_t *jku, int64_t nu, const uint64_t *jkv, int64_t nv,
                       int64_t *cnt, uint32_t *lo);
// Expand pairs: pk = koU[u] | koV[v], pv = (u << 32) | v.
void launch_expand(ucl_ctx *ctx, const int64_t *off, int64_t nu, const uint32_t *lo, const uint64_t *perm_u,
                   const uint64_t *perm_v, const uint64_t *ko_u, const uint64_t *ko_v, int64_t P, uint64_t *pk,
                   uint64_t *pv);
// Unary: pairs = tuples of U.
void launch_unary_pairs(ucl_ctx *ctx, const uint64_t *ko_u, int64_t n, uint64_t *pk, uint64_t *pv);
// Segment heads (flag[p] = 1 where key >> shift changes), as int64 for the scan.
void launch_heads(ucl_ctx *ctx, const uint64_t *pk, int64_t P, int64_t *flag, int shift = 0);
// Banded pair lists, sorted by (band << out_bits | output key): band_start[b]
// = first pair of band b, band_seg[b] = its segment index (b = 0..B; B <= 63).
void launch_band_ranges(ucl_ctx *ctx, const uint64_t *pk, int64_t P, const int64_t *seg_excl, const int64_t *n_seg,
                        int out_bits, int B, int64_t *band_start, int64_t *band_seg);
// Small binary EinSums: the whole key stage in one CTA (28 KB of shared
// memory, so that it still fits beside a running contraction) with one
// result read: res[0] = pairs P, res[1] = segments S.  Applies when both
// inputs have at most kSmallTuples tuples and their product is at most 2^16
// (small_join_fits); when P exceeds kSmallPairs nothing but res[0] is
// written and the general path runs.
constexpr int kSmallTuples = 256;
constexpr int kSmallPairs = 1024;
bool small_join_fits(int64_t na, int64_t nb);
void launch_small_join(ucl_ctx *ctx, const int32_t *keys_a, int ua, int64_t na, const int32_t *keys_b, int ub,
                       int64_t nb, const KeyPack &join_a, const KeyPack &join_b, const KeyPack &out_a,
                       const KeyPack &out_b, const KeyUnpack &un, bool has_join, int64_t *res, int64_t *seg_start,
                       int32_t *out_keys, uint32_t *pu, uint32_t *pvi);
// Windows: slot[p] = output key & (2^wb - 1) and mask[ws] |= 1 << slot for
// each pair (flag/excl: window segment heads and their exclusive scan).
void launch_win_slots(ucl_ctx *ctx, const uint64_t *pk, int64_t P, int wb, const int64_t *flag, const int64_t *excl,
                      uint8_t *slot, uint32_t *mask);
// cnt[ws] = slots present in window segment ws.
void launch_win_count(ucl_ctx *ctx, const uint32_t *mask, int64_t Sw, int64_t *cnt);
// rowkey[wbase[ws] + i] = key of the i-th present slot of window segment ws.
void launch_win_rows(ucl_ctx *ctx, const uint64_t *pk, const int64_t *seg_start, int64_t Sw, const uint32_t *mask,
                     const int64_t *wbase, int wb, uint64_t *rowkey);
// out_keys[s] = the output key columns of packed key k[s].
void launch_unpack_keys(ucl_ctx *ctx, const uint64_t *k, int64_t n, KeyUnpack un, int32_t *out_keys);
// sk[s] = (output key << band_bits) | band of band segment s, sv[s] = s
// (the packed key of segment s is pk[seg_start[s]], or pk[s] if seg_start is NULL).
void launch_band_keys(ucl_ctx *ctx, const uint64_t *pk, const int64_t *seg_start, int64_t Sp, int out_bits,
                      int band_bits, uint64_t *sk, uint64_t *sv);
// After sorting sk: the S output keys and fstart[f] = first sorted band
// segment of output key f (fstart[S] = Sp).
void launch_band_outputs(ucl_ctx *ctx, const uint64_t *sk, const int64_t *excl, int64_t Sp, int64_t S, int band_bits,
                         KeyUnpack un, int32_t *out_keys, int64_t *fstart);
// Segment starts, output keys, pair index arrays.
void launch_segments(ucl_ctx *ctx, const uint64_t *pk, const uint64_t *pv, const int64_t *seg_excl, int64_t P,
                     int64_t S, KeyUnpack un, int32_t *out_keys, int64_t *seg_start, uint32_t *pu, uint32_t *pvi,
                     int shift = 0);
// Three-way join, second step.  pair_keys: jk[p] = jk_a[a] | jk_b[b] for
// each first-step pair pv1[p] = (a << 32) | b (either table may be NULL).
void launch_pair_keys(ucl_ctx *ctx, const uint64_t *pv1, int64_t P1, const uint64_t *jk_a, const uint64_t *jk_b,
                      uint64_t *jk);
// expand3: triple t of pair p (found in off2) and the third input's row c:
// pk[t] = pk1[p] | ko_c[c], pv[t] = (p << 32) | c.
void launch_expand3(ucl_ctx *ctx, const int64_t *off2, int64_t P1, const uint32_t *lo2, const uint64_t *perm_c,
                    const uint64_t *pk1, const uint64_t *ko_c, int64_t P, uint64_t *pk, uint64_t *pv);
// segments3: as launch_segments, with each triple's three row indices written
// in spec order: idx[ord[0]] = a, idx[ord[1]] = b, idx[ord[2]] = c.
void launch_segments3(ucl_ctx *ctx, const uint64_t *pk, const uint64_t *pv, const uint64_t *pv1,
                      const int64_t *seg_excl, int64_t P, int64_t S, KeyUnpack un, const int ord[3],
                      int32_t *out_keys, int64_t *seg_start, uint32_t *const idx[3]);

// ---- repartition (repartition.cu)
// Output key of slot r * np + p: field q (output order) is promoted label q's
// mixed-radix digit of p (p / pdiv % pext) or a kept label's field of the r-th
// distinct kept key (bits at ksh); it lands at osh in the packed output key.
struct RepartKeys {
    int uw;
    int promoted[kMaxCols];
    int ksh[kMaxCols], kbits[kMaxCols], osh[kMaxCols];
    int64_t pdiv[kMaxCols], pext[kMaxCols];
    int64_t np;
};
// Where an input element goes: per input tile dim its extent, its stride in
// the output tile (kept-lower labels) and its weight in p (promoted labels);
// per input key column its stride in the output tile (demoted labels, else 0).
struct RepartCopy {
    int r, u;
    int64_t ext[kMaxCols], ostride[kMaxCols], pstride[kMaxCols], kstride[kMaxCols];
    int64_t tile_in, tile_out, np;
};
void launch_kept_rank(ucl_ctx *ctx, const uint64_t *kk, const int64_t *flag, const int64_t *excl,
                      const uint64_t *perm, int64_t n, uint32_t *rank, uint64_t *dk);
void launch_out_keys(ucl_ctx *ctx, const uint64_t *dk, int64_t n_out, const RepartKeys &rk, uint64_t *okey,
                     uint64_t *iota);
void launch_out_place(ucl_ctx *ctx, const uint64_t *okey_sorted, const uint64_t *perm, int64_t n_out,
                      const KeyUnpack &un, uint32_t *pos, int32_t *out_keys);
void launch_repart_scatter(ucl_ctx *ctx, const void *in, ucl_dtype dt, const int32_t *keys, const uint32_t *rank,
                           const uint32_t *pos, int64_t n, const RepartCopy &pc, void *out);

// ---- statistics (stats.cu)
// Bitmap layout of one statistics pass: one bitmap per key column (bound
// bits) then one per tile dim (extent bits), at the given word offsets.
struct StatsGeom {
    int u, r;
    int64_t E;                      // elements per tile
    int64_t ext[kMaxCols];          // tile extents
    int64_t key_off[kMaxCols];      // word offset of key column c's bitmap
    int64_t dim_off[kMaxCols];      // word offset of tile dim q's bitmap (dim_off[0] = end of keys if r = 0)
    int64_t words, dim_words;       // all words; words of the tile-dim bitmaps
    int smem_dims;                  // tile-dim bitmaps gathered in shared memory first
};
bool stats_geometry(const ucl_rel *R, StatsGeom &g);
// One pass over R's tiles: count non-zeros into *nnz, mark bitmaps in bits
// (NULL: none), set tuple_nz[t] = 1 for tuples with a non-zero (NULL: none).
void launch_relation_stats(ucl_ctx *ctx, const ucl_rel *R, const StatsGeom &g, uint32_t *bits,
                           unsigned long long *nnz, int64_t *tuple_nz);
// out[c] = set bits of bitmap c (key columns, then tile dims).
void launch_popc(ucl_ctx *ctx, const uint32_t *bits, const StatsGeom &g, int64_t *out);
// Copy tuple t of R to position excl[t] where flag[t] is set.
void launch_compact(ucl_ctx *ctx, const ucl_rel *R, const int64_t *flag, const int64_t *excl, void *out_tiles,
                    int32_t *out_keys);

// ---- contraction (contract_simt.cu / contract_tc.cu)
struct ContractArgs {
    const void *U;
    const void *V;         // NULL for a unary EinSum
    ucl_dtype du, dv;
    int64_t nU, nV;
    const uint32_t *pu;    // [P] U tuple of each pair
    const uint32_t *pv;    // [P] V tuple of each pair
    const void *X;         // third input of a three-way EinSum, else NULL
    ucl_dtype dx;
    int64_t nX;
    const uint32_t *px;    // [P] X tuple of each triple
    const int64_t *seg_start;  // [S + 1]
    int64_t S;
    Units units;
    void *out;             // [S, tile_w]
    ucl_dtype dout;
    int epi;
    float scale;
    int agg, comb, map;    // extended EinSum (ucl_agg / ucl_comb / ucl_map); 0, 0, 0 = sum of products
    float *partials;       // [G, 2, tile_w]
    int64_t tile_w;
    unsigned long long *fixup_bytes;   // device counter the fixup kernel adds its bytes to (may be NULL)
    // windowed tcgen05 kernel (win_bits > 0): segments are windows of
    // 2^win_bits output keys; per pair its slot and A-tile run (see
    // contract_tc.cu); per window its present slots and first output row
    int win_bits;
    const uint8_t *slot;
    const uint8_t *arun;
    const uint32_t *wmask;
    const int64_t *wbase;
    int share_cap;
    int bands;             // > 1: U's tuples are split into this many bands of its join label (one launch each)
    int l2_hints;          // TMA loads carry L2 eviction hints (streamed operand first, reused operand last)
};
void launch_contract_simt(ucl_ctx *ctx, const ContractArgs &a, const LowerPlan &lp);
void launch_fixup(ucl_ctx *ctx, const ContractArgs &a);
// Band sum of a banded EinSum (see launch_band_outputs): out[f] = epilogue(sum
// over r in [fstart[f], fstart[f + 1]) of part[order[r]]), cast to dout; adds
// its bytes (partials read, outputs written) to *bytes if not NULL.
void launch_band_sum(ucl_ctx *ctx, const float *part, const uint64_t *order, const int64_t *fstart, int64_t S,
                     int64_t tile_w, void *out, ucl_dtype dout, int epi, float scale, unsigned long long *bytes);
// tcgen05 path; returns false (nothing launched) if the shapes do not fit.
bool tc_supported(const TcPlan &tp, const ContractArgs &a, std::string *why);
ucl_status launch_contract_tc(ucl_ctx *ctx, const ContractArgs &a, const TcPlan &tp, const ucl_rel *ra,
                              const ucl_rel *rb);
int tc_units(ucl_ctx *ctx, const TcPlan &tp, int64_t P);
// Longest run of pairs sharing one loaded A tile in the windowed tcgen05
// kernel for this shape and window size (0: the windowed kernel does not apply).
int tc_window_cap(const TcPlan &tp, int win_bits);
// arun[p] for the windowed kernel: low nibble = pairs back to the pair that
// loads p's A tile (a run of equal pa[] is cut every cap positions), high
// nibble (at that pair) = pairs after it sharing the tile.
void launch_arun(ucl_ctx *ctx, const uint32_t *pa, int64_t P, int cap, uint8_t *arun);
// Windowed fixup: a window split across units sums its present slots'
// partials in unit order into their output rows.
void launch_fixup_window(ucl_ctx *ctx, const ContractArgs &a);
ucl_status launch_contract_tc3(ucl_ctx *ctx, const ContractArgs &a, const Tc3Plan &tp, const ucl_rel *const *in);
int tc3_units(ucl_ctx *ctx, int64_t P);

}  // namespace ucl
