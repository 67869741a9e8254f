// repartition.cu -- kernels that change a tensor-relation's upper/lower
// split (paper Sec. 6: between two EinSums whose decompositions of a tensor
// differ, every tuple is decomposed along the labels that become upper, over
// their whole range, and the pieces are stacked along the labels that become
// lower, grouped by the new upper labels).
//
// The executor does both steps at once: the output keys are every distinct
// value of the kept upper labels combined with every index of the promoted
// labels; each input element is copied once to its place in its output tile,
// and output positions no input element maps to stay zero.  All kernels are
// grid-stride and wait on nothing.
#include "internal.cuh"

namespace ucl {

namespace {

constexpr int kThreads = 256;

int grid_for(ucl_ctx *ctx, int64_t n) {
    int64_t want = (n + kThreads - 1) / kThreads;
    int64_t cap = (int64_t)ctx->sm_count * 16;
    if (want < 1) want = 1;
    return (int)(want < cap ? want : cap);
}

// Rank of every input tuple among the distinct kept keys, and the distinct
// kept keys themselves.  kk is the (sorted) packed kept key, flag its head
// flags and excl their exclusive scan; perm maps sorted positions back to
// input tuples (NULL: kk is in input order).
__global__ void kept_rank_kernel(const uint64_t *__restrict__ kk, const int64_t *__restrict__ flag,
                                 const int64_t *__restrict__ excl, const uint64_t *__restrict__ perm, int64_t n,
                                 uint32_t *rank, uint64_t *dk) {
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = excl[i] + flag[i] - 1;
        rank[perm ? perm[i] : (uint64_t)i] = (uint32_t)r;
        if (flag[i]) dk[r] = kk[i];
    }
}

// Packed output key of output slot o = r * NP + p: kept fields from the r-th
// distinct kept key, promoted fields from the mixed-radix digits of p.
__global__ void out_key_kernel(const uint64_t *__restrict__ dk, int64_t n_out, RepartKeys rk, uint64_t *okey,
                               uint64_t *iota) {
    for (int64_t o = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; o < n_out;
         o += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = o / rk.np, p = o % rk.np;
        const uint64_t kv = dk ? dk[r] : 0ull;
        uint64_t key = 0;
        for (int q = 0; q < rk.uw; ++q) {
            uint64_t v;
            if (rk.promoted[q])
                v = (uint64_t)((p / rk.pdiv[q]) % rk.pext[q]);
            else
                v = (kv >> rk.ksh[q]) & ((rk.kbits[q] ? (~0ull >> (64 - rk.kbits[q])) : 0ull));
            key |= v << rk.osh[q];
        }
        okey[o] = key;
        if (iota) iota[o] = (uint64_t)o;
    }
}

// Output position of each slot after the sort, and the output key columns.
__global__ void out_place_kernel(const uint64_t *__restrict__ okey_sorted, const uint64_t *__restrict__ perm,
                                 int64_t n_out, KeyUnpack un, uint32_t *pos, int32_t *out_keys) {
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n_out;
         i += (int64_t)gridDim.x * blockDim.x) {
        if (pos) pos[perm[i]] = (uint32_t)i;
        const uint64_t k = okey_sorted[i];
        for (int c = 0; c < un.uw; ++c) {
            const uint64_t mask = un.bits[c] ? ((~0ull) >> (64 - un.bits[c])) : 0ull;
            out_keys[i * un.uw + c] = (int32_t)((k >> un.shift[c]) & mask);
        }
    }
}

// One thread per input element: element e of tuple t goes to output slot
// rank[t] * NP + p(e), at the offset given by its kept-lower coordinates and
// the tuple's demoted key values.
template <typename T>
__global__ void scatter_kernel(const T *__restrict__ in, const int32_t *__restrict__ keys,
                               const uint32_t *__restrict__ rank, const uint32_t *__restrict__ pos, int64_t n,
                               RepartCopy pc, T *out) {
    const int64_t total = n * pc.tile_in;
    for (int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; g < total;
         g += (int64_t)gridDim.x * blockDim.x) {
        const int64_t t = g / pc.tile_in;
        int64_t rem = g - t * pc.tile_in, off = 0, p = 0;
        for (int d = pc.r - 1; d >= 0; --d) {
            const int64_t idx = rem % pc.ext[d];
            rem /= pc.ext[d];
            off += idx * pc.ostride[d];
            p += idx * pc.pstride[d];
        }
        for (int c = 0; c < pc.u; ++c) off += (int64_t)keys[t * pc.u + c] * pc.kstride[c];
        const int64_t slot = (int64_t)rank[t] * pc.np + p;
        const int64_t o = pos ? (int64_t)pos[slot] : slot;
        out[o * pc.tile_out + off] = in[g];
    }
}

// Fast path when the input's innermost tile dim stays the output's innermost
// one: its runs of E elements are contiguous on both sides, so they move as
// V-element vectors (VT).  A group of G lanes takes one tuple at a time: the
// tuple's key offset and slot base are read once, then the lanes walk the
// tile's vectors (32-bit index math inside a tile).
template <typename VT, int G>
__global__ void scatter_runs_kernel(const VT *__restrict__ in, const int32_t *__restrict__ keys,
                                    const uint32_t *__restrict__ rank, const uint32_t *__restrict__ pos, int64_t n,
                                    RepartCopy pc, int vpr, VT *out) {
    const int sub = threadIdx.x % G;
    const int64_t groups = ((int64_t)gridDim.x * blockDim.x) / G;
    const uint32_t vecs = (uint32_t)(pc.tile_in / (pc.ext[pc.r - 1] / vpr));   // vectors per input tile
    const int64_t vpo = pc.tile_out / (pc.ext[pc.r - 1] / vpr);                // vectors per output tile
    const int64_t V = pc.ext[pc.r - 1] / vpr;                                  // elements per vector
    for (int64_t t = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) / G; t < n; t += groups) {
        int64_t koff = 0;
        for (int c = 0; c < pc.u; ++c) koff += (int64_t)keys[t * pc.u + c] * pc.kstride[c];
        const int64_t base = (int64_t)rank[t] * pc.np;
        const VT *src = in + t * (int64_t)vecs;
        for (uint32_t v = sub; v < vecs; v += G) {
            uint32_t run = v / (uint32_t)vpr;
            const uint32_t w = v - run * (uint32_t)vpr;
            int64_t off = koff, p = 0;
            for (int d = pc.r - 2; d >= 0; --d) {
                const uint32_t e = (uint32_t)pc.ext[d];
                const uint32_t idx = run % e;
                run /= e;
                off += (int64_t)idx * pc.ostride[d];
                p += (int64_t)idx * pc.pstride[d];
            }
            const int64_t o = pos ? (int64_t)pos[base + p] : base + p;
            out[o * vpo + off / V + w] = src[v];
        }
    }
}

}  // namespace

void launch_kept_rank(ucl_ctx *ctx, const uint64_t *kk, const int64_t *flag, const int64_t *excl,
                      const uint64_t *perm, int64_t n, uint32_t *rank, uint64_t *dk) {
    if (n <= 0) return;
    kept_rank_kernel<<<grid_for(ctx, n), kThreads, 0, ctx->stream>>>(kk, flag, excl, perm, n, rank, dk);
    ctx->launches++;
}

void launch_out_keys(ucl_ctx *ctx, const uint64_t *dk, int64_t n_out, const RepartKeys &rk, uint64_t *okey,
                     uint64_t *iota) {
    if (n_out <= 0) return;
    out_key_kernel<<<grid_for(ctx, n_out), kThreads, 0, ctx->stream>>>(dk, n_out, rk, okey, iota);
    ctx->launches++;
}

void launch_out_place(ucl_ctx *ctx, const uint64_t *okey_sorted, const uint64_t *perm, int64_t n_out,
                      const KeyUnpack &un, uint32_t *pos, int32_t *out_keys) {
    if (n_out <= 0) return;
    out_place_kernel<<<grid_for(ctx, n_out), kThreads, 0, ctx->stream>>>(okey_sorted, perm, n_out, un, pos,
                                                                        out_keys);
    ctx->launches++;
}

void launch_repart_scatter(ucl_ctx *ctx, const void *in, ucl_dtype dt, const int32_t *keys, const uint32_t *rank,
                           const uint32_t *pos, int64_t n, const RepartCopy &pc, void *out) {
    if (n <= 0 || pc.tile_in <= 0) return;
    if (pc.r > 0 && pc.ostride[pc.r - 1] == 1 && pc.pstride[pc.r - 1] == 0) {
        // runs of the innermost dim: widest vector dividing the run (in bytes)
        // that both tile arrays' alignment allows
        const int es = dt == UCL_BF16 ? 2 : 4;
        const int64_t run_bytes = pc.ext[pc.r - 1] * es;
        const uintptr_t al = reinterpret_cast<uintptr_t>(in) | reinterpret_cast<uintptr_t>(out);
        int vb = 16;
        while (vb > es && (run_bytes % vb || al % vb)) vb >>= 1;
        const int vpr = (int)(run_bytes / vb);   // vectors per run
        const int64_t vecs = pc.tile_in * es / vb;
        const int G = vecs >= 32 ? 32 : (vecs >= 16 ? 16 : (vecs >= 8 ? 8 : (vecs >= 4 ? 4 : (vecs >= 2 ? 2 : 1))));
        const int64_t want = (n * G + kThreads - 1) / kThreads;
        const int g = (int)(want < (int64_t)ctx->sm_count * 32 ? (want < 1 ? 1 : want) : (int64_t)ctx->sm_count * 32);
#define UCL_RUNS(VT)                                                                                             \
    switch (G) {                                                                                                 \
        case 32: scatter_runs_kernel<VT, 32><<<g, kThreads, 0, ctx->stream>>>(                                   \
            static_cast<const VT *>(in), keys, rank, pos, n, pc, vpr, static_cast<VT *>(out)); break;            \
        case 16: scatter_runs_kernel<VT, 16><<<g, kThreads, 0, ctx->stream>>>(                                   \
            static_cast<const VT *>(in), keys, rank, pos, n, pc, vpr, static_cast<VT *>(out)); break;            \
        case 8: scatter_runs_kernel<VT, 8><<<g, kThreads, 0, ctx->stream>>>(                                     \
            static_cast<const VT *>(in), keys, rank, pos, n, pc, vpr, static_cast<VT *>(out)); break;            \
        case 4: scatter_runs_kernel<VT, 4><<<g, kThreads, 0, ctx->stream>>>(                                     \
            static_cast<const VT *>(in), keys, rank, pos, n, pc, vpr, static_cast<VT *>(out)); break;            \
        case 2: scatter_runs_kernel<VT, 2><<<g, kThreads, 0, ctx->stream>>>(                                     \
            static_cast<const VT *>(in), keys, rank, pos, n, pc, vpr, static_cast<VT *>(out)); break;            \
        default: scatter_runs_kernel<VT, 1><<<g, kThreads, 0, ctx->stream>>>(                                    \
            static_cast<const VT *>(in), keys, rank, pos, n, pc, vpr, static_cast<VT *>(out)); break;            \
    }
        switch (vb) {
            case 16: UCL_RUNS(uint4) break;
            case 8: UCL_RUNS(uint2) break;
            case 4: UCL_RUNS(uint32_t) break;
            default: UCL_RUNS(uint16_t) break;
        }
#undef UCL_RUNS
        ctx->launches++;
        return;
    }
    const int g = grid_for(ctx, n * pc.tile_in);
    if (dt == UCL_BF16)
        scatter_kernel<uint16_t><<<g, kThreads, 0, ctx->stream>>>(static_cast<const uint16_t *>(in), keys, rank, pos,
                                                                 n, pc, static_cast<uint16_t *>(out));
    else
        scatter_kernel<uint32_t><<<g, kThreads, 0, ctx->stream>>>(static_cast<const uint32_t *>(in), keys, rank, pos,
                                                                 n, pc, static_cast<uint32_t *>(out));
    ctx->launches++;
}

}  // namespace ucl
