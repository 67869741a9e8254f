/*
 * ucl.h -- C ABI of the GB300 executor for upper-case-lower-case (UCL) EinSum
 * over tensor-relations.
 *
 * A tensor-relation (paper Sec. 4.2) is a set of tuples (key, tile): the key is
 * the vector of values of the operand's upper-case (promoted) labels, the tile
 * is the dense sub-tensor over its lower-case (demoted) labels.  One binary
 * UCL EinSum is evaluated as the TR-SQL template of Sec. 5 (Eq. eqn-TRA):
 *
 *     SELECT up(W), SUM(K(valU, valV)) FROM U NATURAL JOIN V GROUP BY up(W)
 *
 * where K is the lower-case EinSum applied to the two joined tiles.  The
 * executor runs every step on the GPU: key packing, radix sort and merge-join
 * of the keys, a batched tile contraction (tcgen05 tensor cores for bf16
 * GEMM-shaped kernels, FFMA otherwise) whose epilogue performs the segmented
 * group-by sum, and compaction of the output relation.
 *
 * Conventions shared by every call:
 *   - Every call returns a ucl_status and never aborts.  On error an output
 *     handle is set to NULL and inputs are left untouched; ucl_last_error()
 *     gives a one-line reason.
 *   - Device pointers are CUDA device addresses on the context's device.
 *   - All GPU work is asynchronous on the context's stream, except where a
 *     call documents a host synchronisation.
 *   - Not thread-safe: one context is used by one host thread at a time.
 */
#ifndef UCL_H
#define UCL_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    UCL_OK = 0,
    UCL_ERR_ARG = 1,         /* NULL handle, bad pointer, n < 0, unknown enum */
    UCL_ERR_SPEC = 2,        /* malformed spec string (grammar below) */
    UCL_ERR_SHAPE = 3,       /* arity or extents disagree with the spec */
    UCL_ERR_DUP_KEY = 4,     /* two tuples of one relation share a key (Sec. 4.2: one tuple per key) */
    UCL_ERR_KEY_RANGE = 5,   /* a key value outside [0, bound) */
    UCL_ERR_OOM = 6,         /* the allocator returned NULL */
    UCL_ERR_CUDA = 7,        /* a CUDA runtime call failed */
    UCL_ERR_UNSUPPORTED = 8, /* valid but outside this build (e.g. > 64 key bits) */
    UCL_ERR_TIMEOUT = 9      /* a device-side wait ran out; the context stays usable */
} ucl_status;

typedef enum { UCL_BF16 = 0, UCL_F32 = 1 } ucl_dtype;

typedef enum { UCL_EPI_NONE = 0, UCL_EPI_RELU = 1 } ucl_epilogue;

/* Where ucl_relation_create reads keys and tiles from. */
typedef enum {
    UCL_MEM_DEVICE_BORROW = 0, /* device memory the caller keeps alive and unchanged while the relation lives */
    UCL_MEM_DEVICE_COPY = 1,   /* device memory copied into library-owned buffers */
    UCL_MEM_HOST_COPY = 2      /* host memory (pinned or pageable) copied to the device */
} ucl_mem;

/* Contraction kernel choice; AUTO picks tcgen05 when the tile kernel is a
 * bf16 GEMM that fits it, FFMA otherwise. */
typedef enum { UCL_PATH_AUTO = 0, UCL_PATH_SIMT = 1, UCL_PATH_TC = 2 } ucl_path;

typedef struct ucl_ctx ucl_ctx;
typedef struct ucl_rel ucl_rel;

/* Allocator hooks.  alloc returns device memory of at least `bytes` bytes
 * (256-byte aligned) or NULL; free releases it.  Both must be ordered on the
 * context's stream (a caching allocator bound to that stream, or
 * cudaMallocAsync/cudaFreeAsync on it).  NULL hooks select
 * cudaMallocAsync/cudaFreeAsync on the context's stream. */
typedef void *(*ucl_alloc_fn)(size_t bytes, void *user);
typedef void (*ucl_free_fn)(void *ptr, size_t bytes, void *user);

/* Extended EinSum (Sec. 3, the general form of Eq. Einsum: an aggregate ⊕
 * over the joined values of a scalar function ⊗).  The term of one joined
 * tuple and one lower-index combination is map(comb(u, v)) -- map(u) for a
 * unary EinSum -- and terms are folded with agg.  Sec. 3's example
 * W_i = max_j (U_ij - V_ij)^2 is {MAX, SUB, SQUARE}; softmax is four calls
 * ({MAX}, {SUM, SUB, EXP}, {SUM}, {SUM, DIV}).  Aggregation ranges over the
 * tuples present, as SQL GROUP BY does: an absent tuple contributes nothing,
 * also to MAX and MIN. */
typedef enum { UCL_AGG_SUM = 0, UCL_AGG_MAX = 1, UCL_AGG_MIN = 2 } ucl_agg;
typedef enum { UCL_COMB_MUL = 0, UCL_COMB_ADD = 1, UCL_COMB_SUB = 2, UCL_COMB_DIV = 3 } ucl_comb;
typedef enum { UCL_MAP_IDENT = 0, UCL_MAP_RELU = 1, UCL_MAP_EXP = 2, UCL_MAP_SQUARE = 3 } ucl_map;

typedef struct {
    ucl_dtype out_dtype;  /* dtype of the output tiles */
    ucl_epilogue epi;     /* applied after the full aggregate */
    float scale;          /* out = epi(scale * aggregate); 1.0f for a plain sum */
    int path;             /* ucl_path */
    int agg;              /* ucl_agg; UCL_AGG_SUM for the plain EinSum */
    int comb;             /* ucl_comb; UCL_COMB_MUL for the plain EinSum */
    int map;              /* ucl_map; UCL_MAP_IDENT for the plain EinSum */
} ucl_einsum_opts;

#define UCL_NSTAGES 4

/* Counters and stage timings of the last ucl_einsum on a context. */
typedef struct {
    int64_t n_pairs;       /* joined tuple pairs (one kernel invocation each) */
    int64_t n_segments;    /* output tuples = distinct output keys */
    double flops;          /* 2 * n_pairs * prod(all lower extents of the kernel) */
    double bytes_contract; /* algorithmic bytes of the contraction stage */
    int path;              /* ucl_path actually used (SIMT or TC) */
    int launches;          /* GPU kernels launched by the call */
    int timed;             /* 1 if stage_ms is valid (timing enabled) */
    int n_units;           /* work units (CTAs) the pair list was cut into for the contraction */
    int n_bands;           /* bands of the contracted label (1: not banded; see ucl_einsum) */
    int64_t n_band_segments; /* (band, output key) groups of a banded EinSum, else n_segments */
    /* stage_ms: [0] key pack/sort/join count, [1] pair expansion, pair sort,
     * segments, [2] tile contraction + fused group-by, [3] split-segment fixup
     * and output key compaction.  CUDA-event times on the context stream. */
    float stage_ms[UCL_NSTAGES];
} ucl_stats;

/* --------------------------------------------------------------- context */

/* Create a context on `device` that issues work on `stream` (a cudaStream_t,
 * NULL = the legacy default stream).  Allocates a small device status word
 * and pinned host scratch; device workspace grows on demand through the
 * allocator hooks and is reused across calls. */
ucl_status ucl_ctx_create(int device, void *stream, ucl_alloc_fn alloc, ucl_free_fn free_fn, void *user,
                          ucl_ctx **out);

/* Synchronises the stream, then frees the workspace.  Relations created on
 * the context must be destroyed first. */
ucl_status ucl_ctx_destroy(ucl_ctx *ctx);

/* Drain the context's stream and report device-side failures (a bounded wait
 * that ran out: UCL_ERR_TIMEOUT; a failed bounds check: UCL_ERR_CUDA) raised
 * by kernels of earlier calls.  Such failures are sticky: if not collected
 * here they surface at the next synchronising call of the context. */
ucl_status ucl_ctx_synchronize(ucl_ctx *ctx);

/* Enable (1) or disable (0) CUDA-event stage timing for later calls. */
ucl_status ucl_ctx_set_timing(ucl_ctx *ctx, int enable);

/* Statistics of the last ucl_einsum; synchronises on its last event when
 * timing is enabled. */
ucl_status ucl_get_last_stats(ucl_ctx *ctx, ucl_stats *out);

/* Stage times of every ucl_einsum made with timing enabled since the last
 * reset, so that a caller can time many calls without synchronising between
 * them: ms[c * UCL_NSTAGES + s] receives stage s of call c (the stages of
 * ucl_stats.stage_ms) for c < max_calls; *n_calls (if not NULL) the number of
 * calls recorded.  Synchronises on the last recorded event.  reset != 0
 * forgets the recorded calls and recycles their events. */
ucl_status ucl_ctx_timings(ucl_ctx *ctx, float *ms, int max_calls, int *n_calls, int reset);

/* Bytes moved by the fixup kernels of every ucl_einsum on this context since
 * the last reset: the fp32 partials of output keys whose pairs straddle work
 * units, read once, plus those keys' output tiles, written once -- the
 * algorithmic bytes of the cross-unit part of the group-by sum (Sec. 5's
 * SUM ... GROUP BY).  Counted on the device by the fixup kernels themselves.
 * Synchronises the context's stream.  reset != 0 zeroes the counter. */
ucl_status ucl_ctx_fixup_bytes(ucl_ctx *ctx, int64_t *bytes, int reset);

/* Failure detection.  Every wait of a tcgen05 contraction on a barrier phase
 * is bounded: after `cycles` SM clock cycles (0 restores the default of about
 * 2.5e9, a little over a second) the waiting role aborts its CTA, which
 * drains its copies and tensor-core work in flight, frees its tensor memory
 * and returns; the context then reports UCL_ERR_TIMEOUT at its next
 * synchronising call (ucl_ctx_synchronize) and stays usable.  The paper has no
 * counterpart; it is a service of this library.  Errors: UCL_ERR_ARG. */
ucl_status ucl_ctx_set_wait_limit(ucl_ctx *ctx, int64_t cycles);

/* Test hook for the failure path above: the next binary tcgen05 contraction
 * on this context skips pipeline stage fill `fill` (no copy is issued and no
 * arrival posted), so that the roles waiting on it run into their limit.
 * One launch only; -1 cancels.  Errors: UCL_ERR_ARG. */
ucl_status ucl_ctx_withhold_stage(ucl_ctx *ctx, int fill);

/* ------------------------------------------------------------- relations */

/* Create a tensor-relation (Sec. 4.2, schema (INT up[1], ..., TENSOR val)).
 *   n          number of tuples (>= 0)
 *   u          number of key columns = promoted labels (0..15)
 *   keys       int32 [n, u] row-major; column c holds values in [0, key_bounds[c])
 *   key_bounds int64 [u], each >= 1 (host memory)
 *   r          number of tile dimensions = demoted labels (0..15; 0 = scalar tiles)
 *   tile_shape int64 [r], each >= 1 (host memory)
 *   dtype      element type of the tiles
 *   tiles      [n, prod(tile_shape)] row-major tiles, last dimension fastest
 *   mem        where keys and tiles live (ucl_mem); with BORROW the tiles
 *              must be 16-byte aligned for the tensor-core path to apply
 * Validates on the GPU that every key is in range (UCL_ERR_KEY_RANGE) and that
 * no key repeats (UCL_ERR_DUP_KEY), and records whether the keys are already
 * in ascending order; synchronises the stream once (twice if unsorted).
 * With a COPY mode the tile copy runs on a stream of the context, overlapping
 * the key copy and validation, and the context's stream is ordered after it.
 * HOST_COPY returns once the copy is complete, so host memory may be reused
 * at once; DEVICE_COPY returns without waiting (the source must stay unchanged
 * until the context's stream passes this call, as for any stream-ordered
 * copy).
 * Returns UCL_ERR_UNSUPPORTED if the key bit widths, ceil(log2(bound)) per
 * column, sum to more than 64. */
ucl_status ucl_relation_create(ucl_ctx *ctx, int64_t n, int u, const int32_t *keys, const int64_t *key_bounds,
                               int r, const int64_t *tile_shape, ucl_dtype dtype, const void *tiles, ucl_mem mem,
                               ucl_rel **out);

/* Frees library-owned buffers (stream-ordered).  Borrowed memory is untouched. */
ucl_status ucl_relation_destroy(ucl_rel *rel);

/* Shape of a relation.  key_bounds / tile_shape may be NULL; otherwise they
 * receive u / r entries. */
ucl_status ucl_relation_info(const ucl_rel *rel, int64_t *n, int *u, int *r, int64_t *key_bounds,
                             int64_t *tile_shape, ucl_dtype *dtype);

/* Device addresses of the key array [n, u] and tile array [n, tile]. */
ucl_status ucl_relation_data(const ucl_rel *rel, const int32_t **keys, const void **tiles);

/* Copy keys (int32 [n, u]) and tiles ([n, tile] in the relation's dtype) to
 * host memory; either destination may be NULL.  Synchronises the stream. */
ucl_status ucl_relation_download(const ucl_rel *rel, int32_t *keys_host, void *tiles_host);

/* ----------------------------------------------------------------- einsum */

/* Evaluate one UCL EinSum (Sec. 4.3 notation, Sec. 5 Eq. eqn-TRA).
 *
 * Spec grammar: "<op>,<op>->" "<out>" with 1, 2 or 3 input operands (n_in).
 * Each operand is a string of letters, one letter per label; an upper-case
 * letter is a promoted label (a key column, in the order the upper-case
 * letters appear), a lower-case letter a demoted label (a tile dimension, in
 * the order the lower-case letters appear).  Letters are case-sensitive
 * labels: 'J' and 'j' are two labels, as in a tile index J and an offset j of
 * one reshaped dense index.  A label appears at most once per operand; every
 * output label appears in some input; a label has one extent everywhere.
 * Labels absent from the output are summed: upper ones by the group-by, lower
 * ones inside the tile kernel.  Shared upper labels are the join attributes;
 * with none the join is a cross product (Sec. 7.2).  n_in = 1 is a unary
 * EinSum (a group-by sum over one relation, e.g. with the relu epilogue).
 * n_in = 3 joins all three inputs (tuples agree on every shared upper label)
 * and multiplies the three tiles' entries, as in MTTKRP
 * "IJKijk,Jjr,Kkr->Iir"; the two inputs sharing the most key bits are joined
 * first, so a star join never forms a cross product of its factors.
 *
 * Output: a new relation owned by the library (destroy it with
 * ucl_relation_destroy), one tuple per distinct output key produced by at
 * least one joined pair -- also when its sum is zero -- in ascending
 * lexicographic key order; tiles row-major over the output's lower labels.
 *
 * opts (NULL: fp32 output, plain sum of products, automatic path) selects the
 * extended EinSum (ucl_agg / ucl_comb / ucl_map).  Anything but {SUM, MUL,
 * IDENT} runs on the FFMA path (UCL_PATH_TC gives UCL_ERR_UNSUPPORTED) and,
 * with three inputs, is UCL_ERR_UNSUPPORTED.  MAX / MIN fold in any order,
 * exactly; exp is CUDA's expf; DIV is IEEE division (a zero divisor gives
 * inf or NaN, as in IEEE arithmetic).
 *
 * Synchronises the stream twice (after the join count and after the segment
 * count: both sizes depend on the data; three inputs add one sync after the
 * first join's count).  The contraction is deterministic:
 * pairs of one output key are summed in a fixed order.
 * Errors: UCL_ERR_SPEC / SHAPE for spec-relation mismatches, UCL_ERR_OOM,
 * UCL_ERR_UNSUPPORTED (more than 2^31-1 joined pairs, > 64 key bits),
 * UCL_ERR_TIMEOUT / UCL_ERR_CUDA for device failures. */
ucl_status ucl_einsum(ucl_ctx *ctx, const char *spec, int n_in, ucl_rel *const *in, const ucl_einsum_opts *opts,
                      ucl_rel **out);

/* ------------------------------------------------------------ repartition */

/* Change a relation's upper/lower split without changing the tensor it
 * denotes (Sec. 6, the representation change between two EinSums whose
 * decompositions of a tensor differ: decompose every tuple over the full
 * range of each label that becomes upper -- the ALLINTS step -- then stack
 * the labels that become lower, grouped by the new upper labels -- the STACK
 * aggregate).
 *
 * Spec: "<input labels>-><output>".  The input side lists the relation's
 * labels, one letter each, upper case for key columns and lower case for tile
 * dimensions, in order.  The output side is either
 *   "<keys>|<tile dims>", the input's letters as written, or
 *   the same letters with their case changed to give the new class (letters
 *   then compare without case, so this form cannot tell J from j).
 * Examples: "Ki->kI" (or "Ki->i|K") turns row vectors keyed by the row index
 * into column vectors keyed by the column index; "Jfj->fJ|j" splits [f][j]
 * tiles keyed by J into j-vectors keyed by (f, J).
 *
 * Output (owned by the library, destroy with ucl_relation_destroy): one tuple
 * for every combination of a distinct value of the labels upper on both
 * sides (as present in the input) with every index of the labels that become
 * upper, in ascending key order; tiles row-major over the output's lower
 * labels, the input's dtype, positions no input element maps to set to 0
 * (tuples are never dropped, as the decompose step keeps every index).
 * Values are copied, never rounded.  Synchronises the stream once when the
 * input has key labels that stay upper.
 * Errors: UCL_ERR_ARG, UCL_ERR_SPEC (labels), UCL_ERR_SHAPE (arity),
 * UCL_ERR_UNSUPPORTED (> 64 output key bits, a tile or count of 2^31 or
 * more), UCL_ERR_OOM, UCL_ERR_CUDA. */
ucl_status ucl_repartition(ucl_ctx *ctx, const char *spec, const ucl_rel *in, ucl_rel **out);

/* ------------------------------------------------------------ statistics */

/* Statistics of the tensor a relation stores (Sec. 7.1), which the planner
 * (ucl_plan) needs for every input tensor:
 *   nnz       optional; receives T, the number of non-zero tile elements
 *             (bf16/fp32 ±0 is zero; NaN counts as non-zero)
 *   distinct  optional, int64 [u + r]; receives V for each key column (the
 *             number of its values carried by a tuple with a non-zero
 *             element) and then for each tile dim (the number of its indices
 *             at which some tuple has a non-zero element)
 * Reads every tile once.  Works on one bitmap per key column (bound / 8
 * bytes) and per tile dim in the context's workspace.  Synchronises the
 * stream once.
 * Errors: UCL_ERR_ARG, UCL_ERR_OOM, UCL_ERR_CUDA. */
ucl_status ucl_relation_stats(ucl_ctx *ctx, const ucl_rel *rel, int64_t *nnz, int64_t *distinct);

/* A new relation with the tuples of `in` whose tile holds a non-zero element,
 * in the same (key) order: the elimination of all-zero tuples that Sec. 4.2
 * allows.  Output owned by the library (ucl_relation_destroy).  Synchronises
 * the stream once.
 * Errors: UCL_ERR_ARG, UCL_ERR_OOM, UCL_ERR_CUDA. */
ucl_status ucl_drop_zero_tiles(ucl_ctx *ctx, const ucl_rel *in, ucl_rel **out);

/* ---------------------------------------------------------------- planner */

#define UCL_PLAN_MAX_VERTICES 64

/* One vertex of a tree of binary EinSums (Sec. 8.1): an input tensor
 * (left = right = -1) or W = sum U x V over the labels W does not keep, U
 * and V being the tensors of vertices `left` and `right`.  Vertices come in
 * topological order, the last is the root, and every tensor but the root is
 * consumed exactly once. */
typedef struct {
    int left, right;          /* producer vertices of the two inputs, or -1, -1 */
    const char *labels;       /* the labels of the tensor this vertex produces: one
                                 byte each, distinct, NUL-terminated, at most 12 */
    int dtype_bytes;          /* bytes per element of that tensor */
    double nnz;               /* T of the tensor: required for inputs; for an EinSum
                                 vertex, measured statistics or < 0 to estimate */
    const double *distinct;   /* V per label in `labels` order: required for inputs;
                                 for an EinSum vertex NULL to estimate (Alg. 2) */
} ucl_plan_vertex;

/* Per-unit costs of Sec. 7.2, in any one unit of time: per byte moved into a
 * join or an aggregation (C_xfer), per kernel flop (C_krnel = flop x the
 * kernel's 2 x multiply-adds), per added output-tile element (C_add = add x
 * tile elements), per tuple (C_fixed); key_bytes = bytes per key column.
 * max_call_bytes > 0 is the memory constraint of Sec. 8.2: a split is only
 * considered when the three tiles of one kernel call (U's, V's and W's, at
 * their element sizes) total at most that many bytes. */
typedef struct {
    double xfer, flop, add, fixed;
    int key_bytes;
    double max_call_bytes;
} ucl_cost_model;

/* One plan: for every vertex the promoted labels of its output (bit q = its
 * q-th label; an input tensor's is the split its consumer reads), and for
 * every EinSum vertex the promoted labels of its left and right input as it
 * reads them (bits over that input's labels).  Where a producer's output split
 * differs from its consumer's read split, the plan repartitions the tensor
 * between them (ucl_repartition). */
typedef struct {
    double cost;
    uint32_t up[UCL_PLAN_MAX_VERTICES];
    uint32_t in_up[UCL_PLAN_MAX_VERTICES][2];
} ucl_plan_choice;

/* The k cheapest plans of an EinSum tree under the cost model of Sec. 7.2,
 * by the dynamic programme of Alg. 1 extended to keep the k cheapest entries
 * per vertex and output split.  Host only: no GPU work, no context.
 *   vertices                  [n_vertices] the tree
 *   label_names, label_bounds [n_labels] each label's extent
 *   k                         plans wanted (>= 1)
 *   out                       [k] receives the plans, cheapest first
 *   n_out                     receives how many plans were written (<= k)
 * A label takes one class within an EinSum: upper in every operand that has
 * it, or lower in all.  Input tensors cost nothing in any split.
 * Errors: UCL_ERR_ARG (counts, pointers, not a tree in topological order),
 * UCL_ERR_SPEC (a label twice in a tensor, an output label in no input),
 * UCL_ERR_SHAPE (a label without a bound), UCL_ERR_UNSUPPORTED (more than
 * 12 labels in one tensor). */
ucl_status ucl_plan(int n_vertices, const ucl_plan_vertex *vertices, const char *label_names,
                    const int64_t *label_bounds, int n_labels, const ucl_cost_model *cost_model, int k,
                    ucl_plan_choice *out, int *n_out);

/* One plan for an EinSum program whose tensors may be consumed more than once
 * (a DAG), by the heuristic of Sec. 8.2 ("when results are consumed more than
 * once").  The DAG is cut into trees at every EinSum result used more than
 * once and at every result no EinSum uses (an output): such a result roots a
 * tree, every other EinSum vertex joins the tree of its one consumer.  Trees
 * are optimised one after another in increasing order of their root, each by
 * the dynamic programme of Alg. 1; a result an earlier tree decided is read as
 * an input whose split is fixed (reading it in another split costs C_repart),
 * and the program's input tensors stay free in any split.  Not globally
 * optimal: a result used twice is decided for its own tree alone.  Host only.
 *   vertices   [n_vertices] in topological order, as for ucl_plan, except that
 *              any tensor may be consumed any number of times (an EinSum may
 *              read one tensor as both operands) and several vertices may be
 *              outputs
 *   out        receives the plan: cost = the sum of the trees' costs; up[i]
 *              an EinSum's output split, or for an input tensor the split its
 *              first consumer (lowest index, left operand first) reads; in_up
 *              every EinSum's read splits
 *   tree_root  optional [n_vertices]; receives the root of each EinSum
 *              vertex's tree, -1 for inputs
 * Errors: as ucl_plan (no tree condition), and UCL_ERR_UNSUPPORTED when no
 * split of some tree satisfies the memory bound. */
ucl_status ucl_plan_dag(int n_vertices, const ucl_plan_vertex *vertices, const char *label_names,
                        const int64_t *label_bounds, int n_labels, const ucl_cost_model *cost_model,
                        ucl_plan_choice *out, int *tree_root);

/* ------------------------------------------------------- no allocation */

/* Largest key array ucl_keys_check_noalloc accepts (tuples). */
#define UCL_NOALLOC_MAX_TUPLES (1 << 20)

/* The key checks of ucl_relation_create -- every key in [0, bound), no key
 * twice (UCL_ERR_KEY_RANGE / UCL_ERR_DUP_KEY), ascending order reported in
 * *sorted -- for callers that cannot allocate device memory: code that runs
 * under a device-memory budget owned by another component, or that must
 * never call cudaMalloc because it can synchronise the device.  This call
 * allocates nothing and needs no context: its scratch is a fixed array of
 * about 16.3 MiB in the library's own device memory, which every GPU that
 * loads the library holds until the process exits.  The paper has no
 * counterpart; this is a service of this library.
 *   device, stream  where the work runs (stream NULL = legacy default stream)
 *   n, u, keys      int32 [n, u] key array in device memory, n <= UCL_NOALLOC_MAX_TUPLES
 *   key_bounds      int64 [u] bounds (host memory)
 *   sorted          optional; receives 1 if the keys are strictly ascending
 * Returns UCL_ERR_UNSUPPORTED for n > UCL_NOALLOC_MAX_TUPLES or more than 64
 * key bits.  Synchronises `stream` (once, or twice for unsorted keys).  The
 * calling thread's current device is the same on return as on entry.  The
 * first call on a device looks up the scratch array's device address for
 * that device and keeps it for the life of the process; make that first
 * call before any stream capture, and do not use this call on a device after
 * cudaDeviceReset (the kept address would be stale).  Every call shares the
 * one scratch array: calls whose GPU work overlaps (e.g. on two streams) race
 * on it and must be serialised by the caller. */
ucl_status ucl_keys_check_noalloc(int device, void *stream, int64_t n, int u, const int32_t *keys,
                                  const int64_t *key_bounds, int *sorted);

/* ------------------------------------------------------------ diagnostics */

const char *ucl_status_str(ucl_status st);

/* One-line description of the last error on this context ("" if none). */
const char *ucl_last_error(const ucl_ctx *ctx);

#ifdef __cplusplus
}
#endif

#endif /* UCL_H */
