// repartition.cu -- kernels that change a tensor-relation's upper/lower
// split (paper Sec. 5: between two EinSums whose decompositions of a tensor
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
