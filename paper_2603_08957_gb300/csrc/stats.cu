// stats.cu -- statistics of the tensor a tensor-relation stores (paper
// Sec. 7.1: T(U), its non-zero entries, and V(l, U), the number of slices
// along label l that hold a non-zero), and the optional elimination of tuples
// whose tile is all zero (Sec. 4.2).
//
// One streaming pass reads every tile once.  Each thread takes 16-byte
// vectors of one tile row; a vector with a non-zero element marks, with
// check-before-set atomics, the tuple's key values in one bitmap per key
// column and the element's tile coordinates in one bitmap per tile dimension
// (in shared memory while those fit).  Distinct counts are popcounts of the
// bitmaps.  No kernel waits on another CTA.
#include "internal.cuh"

namespace ucl {

namespace {

constexpr int kThreads = 256;
constexpr int64_t kSmemWords = 12288;   // 48 KB of tile-dimension bitmaps per CTA

__device__ __forceinline__ void mark(uint32_t *words, int64_t idx) {
    uint32_t *w = words + (idx >> 5);
    const uint32_t b = 1u << (idx & 31);
    if (!(*w & b)) atomicOr(w, b);
}

// Non-zero mask of V raw elements (bf16 or f32 bit patterns; ±0 is zero).
template <typename W>
__device__ __forceinline__ bool nonzero(W x);
template <>
__device__ __forceinline__ bool nonzero<uint16_t>(uint16_t x) { return (x & 0x7fffu) != 0; }
template <>
__device__ __forceinline__ bool nonzero<uint32_t>(uint32_t x) { return (x & 0x7fffffffu) != 0; }

template <typename W, int V>
struct Vec {
    W e[V];
};

template <typename W, int V>
__global__ void __launch_bounds__(kThreads, 1) stats_kernel(const Vec<W, V> *__restrict__ tiles,
                                                         const int32_t *__restrict__ keys, int64_t n, StatsGeom g,
                                                         uint32_t *bits, unsigned long long *nnz, int64_t *tuple_nz) {
    extern __shared__ uint32_t sbits[];
    uint32_t *dimbits = g.smem_dims ? sbits : bits + g.dim_off[0];
    if (g.smem_dims) {
        for (int64_t i = threadIdx.x; i < g.dim_words; i += blockDim.x) sbits[i] = 0;
        __syncthreads();
    }
    const int64_t nvec = n * (g.E / V);
    const int last = g.r - 1;
    unsigned long long cnt = 0;
    for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < nvec; v += (int64_t)gridDim.x * blockDim.x) {
        const Vec<W, V> x = tiles[v];
        uint32_t m = 0;
#pragma unroll
        for (int i = 0; i < V; ++i) m |= nonzero<W>(x.e[i]) ? (1u << i) : 0u;
        if (!m) continue;
        cnt += __popc(m);
        const int64_t g0 = v * V;
        const int64_t t = g0 / g.E;
        uint32_t rem = (uint32_t)(g0 - t * g.E);
        if (tuple_nz) tuple_nz[t] = 1;
        if (bits) {
            for (int c = 0; c < g.u; ++c) mark(bits + g.key_off[c], keys[t * g.u + c]);
            if (g.r > 0) {
                // the V elements share every coordinate but the innermost one
                const uint32_t in0 = rem % (uint32_t)g.ext[last];
                rem /= (uint32_t)g.ext[last];
                for (int q = last - 1; q >= 0; --q) {
                    const uint32_t e = (uint32_t)g.ext[q];
                    mark(dimbits + (g.dim_off[q] - g.dim_off[0]), rem % e);
                    rem /= e;
                }
                for (uint32_t mm = m; mm; mm &= mm - 1)
                    mark(dimbits + (g.dim_off[last] - g.dim_off[0]), in0 + (uint32_t)(__ffs(mm) - 1));
            }
        }
    }
    if (nnz) {
        for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
        if ((threadIdx.x & 31) == 0 && cnt) atomicAdd(nnz, cnt);
    }
    if (g.smem_dims) {
        __syncthreads();
        for (int64_t i = threadIdx.x; i < g.dim_words; i += blockDim.x)
            if (sbits[i]) atomicOr(bits + g.dim_off[0] + i, sbits[i]);
    }
}

// Popcount of bitmap c (words [off[c], off[c + 1])), one CTA per bitmap.
__global__ void __launch_bounds__(kThreads) popc_kernel(const uint32_t *__restrict__ bits, StatsGeom g,
                                                        int64_t *out) {
    const int c = blockIdx.x;
    const int64_t lo = c < g.u ? g.key_off[c] : g.dim_off[c - g.u];
    const int64_t hi = c + 1 < g.u ? g.key_off[c + 1] : (c + 1 - g.u < g.r ? g.dim_off[c + 1 - g.u] : g.words);
    int64_t s = 0;
    for (int64_t i = lo + threadIdx.x; i < hi; i += blockDim.x) s += __popc(bits[i]);
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    __shared__ int64_t part[kThreads / 32];
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        int64_t tot = 0;
        for (int w = 0; w < kThreads / 32; ++w) tot += part[w];
        out[c] = tot;
    }
}

// Gather the tuples whose flag is set: tuple t goes to position excl[t].  One
// warp per tuple; tiles move as 16-byte vectors when their size allows.
template <typename VT>
__global__ void __launch_bounds__(kThreads) compact_kernel(const VT *__restrict__ tiles, const int32_t *__restrict__ keys,
                                                           const int64_t *__restrict__ flag,
                                                           const int64_t *__restrict__ excl, int64_t n, int u,
                                                           int64_t vecs, VT *out_tiles, int32_t *out_keys) {
    const int lane = threadIdx.x & 31;
    const int64_t warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t t = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; t < n; t += warps) {
        if (!flag[t]) continue;
        const int64_t o = excl[t];
        if (lane < u) out_keys[o * u + lane] = keys[t * u + lane];
        const VT *src = tiles + t * vecs;
        VT *dst = out_tiles + o * vecs;
        for (int64_t i = lane; i < vecs; i += 32) dst[i] = src[i];
    }
}

int grid_for(ucl_ctx *ctx, int64_t work, int per_block) {
    int64_t want = (work + per_block - 1) / per_block;
    const int64_t cap = (int64_t)ctx->sm_count * 8;
    if (want < 1) want = 1;
    return (int)(want < cap ? want : cap);
}

template <typename W, int V>
void launch_stats_v(ucl_ctx *ctx, const void *tiles, const int32_t *keys, int64_t n, const StatsGeom &g,
                    uint32_t *bits, unsigned long long *nnz, int64_t *tuple_nz) {
    const int64_t nvec = n * (g.E / V);
    const int grid = grid_for(ctx, nvec, kThreads);
    const size_t smem = g.smem_dims ? (size_t)g.dim_words * 4 : 0;
    auto kern = stats_kernel<W, V>;
    if (smem > 48 * 1024) cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    kern<<<grid, kThreads, smem, ctx->stream>>>(static_cast<const Vec<W, V> *>(tiles), keys, n, g, bits, nnz,
                                                tuple_nz);
}

}  // namespace

bool stats_geometry(const ucl_rel *R, StatsGeom &g) {
    g = StatsGeom{};
    g.u = R->u;
    g.r = R->r;
    g.E = R->tile;
    int64_t w = 0;
    for (int c = 0; c < R->u; ++c) {
        g.key_off[c] = w;
        w += (R->bounds[c] + 31) / 32;
    }
    for (int q = 0; q < R->r; ++q) {
        g.ext[q] = R->shape[q];
        g.dim_off[q] = w;
        w += (R->shape[q] + 31) / 32;
    }
    if (R->r == 0) g.dim_off[0] = w;
    g.words = w;
    g.dim_words = w - g.dim_off[0];
    g.smem_dims = R->r > 0 && g.dim_words <= kSmemWords;
    return true;
}

void launch_relation_stats(ucl_ctx *ctx, const ucl_rel *R, const StatsGeom &g, uint32_t *bits,
                           unsigned long long *nnz, int64_t *tuple_nz) {
    if (R->n <= 0 || R->tile <= 0) return;
    // vector width: the widest of 16/8/4/2 bytes (or one element) that divides
    // the innermost tile extent, with an aligned tile base
    const int es = R->dtype == UCL_BF16 ? 2 : 4;
    const int64_t inner = R->r > 0 ? R->shape[R->r - 1] : 1;
    const uintptr_t al = reinterpret_cast<uintptr_t>(R->tiles);
    int vb = 16;
    while (vb > es && ((inner * es) % vb || al % vb)) vb >>= 1;
    const int V = vb / es;
    if (R->dtype == UCL_BF16) {
        switch (V) {
            case 8: launch_stats_v<uint16_t, 8>(ctx, R->tiles, R->keys, R->n, g, bits, nnz, tuple_nz); break;
            case 4: launch_stats_v<uint16_t, 4>(ctx, R->tiles, R->keys, R->n, g, bits, nnz, tuple_nz); break;
            case 2: launch_stats_v<uint16_t, 2>(ctx, R->tiles, R->keys, R->n, g, bits, nnz, tuple_nz); break;
            default: launch_stats_v<uint16_t, 1>(ctx, R->tiles, R->keys, R->n, g, bits, nnz, tuple_nz); break;
        }
    } else {
        switch (V) {
            case 4: launch_stats_v<uint32_t, 4>(ctx, R->tiles, R->keys, R->n, g, bits, nnz, tuple_nz); break;
            case 2: launch_stats_v<uint32_t, 2>(ctx, R->tiles, R->keys, R->n, g, bits, nnz, tuple_nz); break;
            default: launch_stats_v<uint32_t, 1>(ctx, R->tiles, R->keys, R->n, g, bits, nnz, tuple_nz); break;
        }
    }
    ctx->launches++;
}

void launch_popc(ucl_ctx *ctx, const uint32_t *bits, const StatsGeom &g, int64_t *out) {
    if (g.u + g.r == 0) return;
    popc_kernel<<<g.u + g.r, kThreads, 0, ctx->stream>>>(bits, g, out);
    ctx->launches++;
}

void launch_compact(ucl_ctx *ctx, const ucl_rel *R, const int64_t *flag, const int64_t *excl, void *out_tiles,
                    int32_t *out_keys) {
    if (R->n <= 0) return;
    const int64_t bytes = R->tile * (R->dtype == UCL_BF16 ? 2 : 4);
    const uintptr_t al = reinterpret_cast<uintptr_t>(R->tiles) | reinterpret_cast<uintptr_t>(out_tiles);
    const int grid = grid_for(ctx, R->n * 32, kThreads);
    if (bytes % 16 == 0 && al % 16 == 0)
        compact_kernel<uint4><<<grid, kThreads, 0, ctx->stream>>>(static_cast<const uint4 *>(R->tiles), R->keys,
                                                                  flag, excl, R->n, R->u, bytes / 16,
                                                                  static_cast<uint4 *>(out_tiles), out_keys);
    else if (bytes % 4 == 0 && al % 4 == 0)
        compact_kernel<uint32_t><<<grid, kThreads, 0, ctx->stream>>>(static_cast<const uint32_t *>(R->tiles),
                                                                     R->keys, flag, excl, R->n, R->u, bytes / 4,
                                                                     static_cast<uint32_t *>(out_tiles), out_keys);
    else
        compact_kernel<uint16_t><<<grid, kThreads, 0, ctx->stream>>>(static_cast<const uint16_t *>(R->tiles),
                                                                     R->keys, flag, excl, R->n, R->u, bytes / 2,
                                                                     static_cast<uint16_t *>(out_tiles), out_keys);
    ctx->launches++;
}

}  // namespace ucl
