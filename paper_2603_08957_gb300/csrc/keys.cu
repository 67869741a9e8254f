// keys.cu -- the relational half of one UCL EinSum on the GPU: key packing,
// key validation, LSD radix sort, the merge-join (count + expand) and the
// group-by segmentation of the pair list (paper Sec. 5, the NATURAL JOIN and
// GROUP BY of the TR-SQL template).
//
// Every kernel is a plain grid-stride or reduce-then-scan kernel: no kernel
// waits on another CTA, so nothing here can spin.
#include "internal.cuh"

namespace ucl {

namespace {

constexpr int kThreads = 256;

int grid_for(ucl_ctx *ctx, int64_t n, int per_thread = 1) {
    int64_t want = (n + (int64_t)kThreads * per_thread - 1) / ((int64_t)kThreads * per_thread);
    int64_t cap = (int64_t)ctx->sm_count * 8;
    if (want < 1) want = 1;
    return (int)(want < cap ? want : cap);
}

__device__ __forceinline__ uint64_t pack_row(const int32_t *row, const KeyPack &kp) {
    uint64_t k = 0;
    for (int i = 0; i < kp.nf; ++i) {
        uint64_t v = (uint32_t)row[kp.f[i].col] >> kp.f[i].rshift;
        k |= v << kp.f[i].shift;
    }
    return k;
}

__global__ void pack_kernel(const int32_t *__restrict__ keys, int u, int64_t n, KeyPack a, uint64_t *out_a,
                            KeyPack b, uint64_t *out_b) {
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int32_t *row = keys + i * u;
        if (out_a) out_a[i] = pack_row(row, a);
        if (out_b) out_b[i] = pack_row(row, b);
    }
}

struct Bounds {
    int64_t b[kMaxCols];
};

__global__ void check_keys_kernel(const int32_t *__restrict__ keys, int u, int64_t n, Bounds bd, KeyPack full,
                                  uint64_t *packed, uint32_t *status) {
    uint32_t st = 0;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int32_t *row = keys + i * u;
        for (int c = 0; c < u; ++c) {
            int32_t v = row[c];
            if (v < 0 || (int64_t)v >= bd.b[c]) st |= kStKeyRange;
        }
        uint64_t k = pack_row(row, full);
        if (i > 0 && pack_row(row - u, full) >= k) st |= kStUnsorted;
        if (packed) packed[i] = k;
    }
    if (st) atomicOr(status, st);
}

__global__ void check_dups_kernel(const uint64_t *__restrict__ k, int64_t n, uint32_t *status) {
    for (int64_t i = 1 + blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        if (k[i] == k[i - 1]) {
            atomicOr(status, kStDupKey);
            return;
        }
}

__global__ void iota_kernel(uint64_t *out, int64_t n) {
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        out[i] = (uint64_t)i;
}

// ------------------------------------------------------------------ scan

constexpr int kScanThreads = 512;
constexpr int kScanItems = 8;
constexpr int kScanTile = kScanThreads * kScanItems;

template <typename T>
__device__ T block_excl_scan(T v, T *total) {
    __shared__ T warp_sums[kScanThreads / 32];
    int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    T x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        T y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[w] = x;
    __syncthreads();
    if (w == 0) {
        T s = lane < kScanThreads / 32 ? warp_sums[lane] : T(0);
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            T y = __shfl_up_sync(0xffffffffu, s, o);
            if (lane >= o) s += y;
        }
        if (lane < kScanThreads / 32) warp_sums[lane] = s;
    }
    __syncthreads();
    T before = (w > 0 ? warp_sums[w - 1] : T(0)) + x - v;
    *total = warp_sums[kScanThreads / 32 - 1];
    __syncthreads();
    return before;
}

template <typename T>
__global__ void __launch_bounds__(kScanThreads) scan_reduce_kernel(const T *__restrict__ in, int64_t n, T *sums) {
    int64_t base = (int64_t)blockIdx.x * kScanTile + (int64_t)threadIdx.x * kScanItems;
    T s = 0;
#pragma unroll
    for (int j = 0; j < kScanItems; ++j)
        if (base + j < n) s += in[base + j];
    T tot;
    block_excl_scan<T>(s, &tot);
    if (threadIdx.x == 0) sums[blockIdx.x] = tot;
}

template <typename T>
__global__ void __launch_bounds__(kScanThreads) scan_tile_kernel(const T *in, T *out, int64_t n, const T *offsets,
                                                                 T *total_dev) {
    int64_t base = (int64_t)blockIdx.x * kScanTile + (int64_t)threadIdx.x * kScanItems;
    T v[kScanItems];
    T s = 0;
#pragma unroll
    for (int j = 0; j < kScanItems; ++j) {
        v[j] = base + j < n ? in[base + j] : T(0);
        s += v[j];
    }
    T tot;
    T run = block_excl_scan<T>(s, &tot) + (offsets ? offsets[blockIdx.x] : T(0));
#pragma unroll
    for (int j = 0; j < kScanItems; ++j) {
        if (base + j < n) out[base + j] = run;
        run += v[j];
    }
    if (total_dev && blockIdx.x == gridDim.x - 1 && threadIdx.x == kScanThreads - 1) *total_dev = run;
}

template <typename T>
void scan_excl(ucl_ctx *ctx, const T *in, T *out, int64_t n, T *total_dev) {
    if (n <= 0) {
        if (total_dev) cudaMemsetAsync(total_dev, 0, sizeof(T), ctx->stream);
        return;
    }
    int64_t nb = (n + kScanTile - 1) / kScanTile;
    T *sums = nullptr;
    if (nb > 1) {
        sums = (T *)ws_get(ctx, sizeof(T) * nb);
        scan_reduce_kernel<T><<<(unsigned)nb, kScanThreads, 0, ctx->stream>>>(in, n, sums);
        ctx->launches++;
        scan_excl<T>(ctx, sums, sums, nb, nullptr);
    }
    scan_tile_kernel<T><<<(unsigned)nb, kScanThreads, 0, ctx->stream>>>(in, out, n, sums, total_dev);
    ctx->launches++;
}

// ------------------------------------------------------------ radix sort

constexpr int kRadixBits = 8;
constexpr int kBuckets = 1 << kRadixBits;
constexpr int kSortThreads = 256;
constexpr int kSortItems = 16;
constexpr int kSortTile = kSortThreads * kSortItems;
static_assert(kSortThreads == kBuckets, "the scatter kernels keep one bucket per thread");

__global__ void __launch_bounds__(kSortThreads) radix_hist_kernel(const uint64_t *__restrict__ k, int64_t n,
                                                                  int shift, uint32_t *hist, int nblocks) {
    __shared__ uint32_t h[kBuckets];
    h[threadIdx.x] = 0;
    __syncthreads();
    int64_t start = (int64_t)blockIdx.x * kSortTile;
    int64_t end = start + kSortTile < n ? start + kSortTile : n;
    for (int64_t i = start + threadIdx.x; i < end; i += kSortThreads)
        atomicAdd(&h[(uint32_t)(k[i] >> shift) & (kBuckets - 1)], 1u);
    __syncthreads();
    hist[(int64_t)threadIdx.x * nblocks + blockIdx.x] = h[threadIdx.x];
}

// Stable scatter: items of the block are ranked in index order, one round of
// 256 at a time; within a warp equal digits are ranked by __match_any_sync,
// across warps by a per-digit prefix over the warps' counts.
__global__ void __launch_bounds__(kSortThreads) radix_scatter_kernel(const uint64_t *__restrict__ kin,
                                                                     const uint64_t *__restrict__ vin,
                                                                     uint64_t *__restrict__ kout,
                                                                     uint64_t *__restrict__ vout, int64_t n,
                                                                     int shift, const uint32_t *__restrict__ offs,
                                                                     int nblocks) {
    constexpr int kWarps = kSortThreads / 32;
    __shared__ uint32_t base[kBuckets];
    __shared__ uint32_t wcnt[kWarps][kBuckets];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    base[tid] = offs[(int64_t)tid * nblocks + blockIdx.x];
    int64_t start = (int64_t)blockIdx.x * kSortTile;
    int64_t end = start + kSortTile < n ? start + kSortTile : n;
    for (int64_t r = start; r < end; r += kSortThreads) {
        for (int i = tid; i < kWarps * kBuckets; i += kSortThreads) (&wcnt[0][0])[i] = 0;
        __syncthreads();
        int64_t i = r + tid;
        bool valid = i < end;
        uint64_t key = valid ? kin[i] : 0;
        uint64_t val = (valid && vin) ? vin[i] : 0;
        uint32_t d = valid ? (uint32_t)(key >> shift) & (kBuckets - 1) : (uint32_t)kBuckets;
        uint32_t peers = __match_any_sync(0xffffffffu, d);
        uint32_t below = peers & ((1u << lane) - 1u);
        if (valid && below == 0) wcnt[warp][d] = __popc(peers);
        __syncthreads();
        {
            uint32_t run = base[tid];
#pragma unroll
            for (int w = 0; w < kWarps; ++w) {
                uint32_t c = wcnt[w][tid];
                wcnt[w][tid] = run;
                run += c;
            }
            base[tid] = run;
        }
        __syncthreads();
        if (valid) {
            uint32_t dst = wcnt[warp][d] + __popc(below);
            kout[dst] = key;
            if (vin) vout[dst] = val;
        }
        __syncthreads();
    }
}

// A whole LSD radix sort of at most kSortTile items in one CTA, for the short
// arrays of small EinSums: per 8-bit pass each thread loads its kSortItems
// items once, then a shared-memory histogram, its exclusive scan and the
// stable scatter of radix_scatter_kernel (ranks in index order, 256 items a
// round); passes alternate between the two buffers, with a block barrier
// between them.  The buffers are read and written in the same launch, so they
// are plain (coherent) pointers.
__global__ void __launch_bounds__(kSortThreads) radix_sort_small_kernel(uint64_t *k0, uint64_t *v0, uint64_t *k1,
                                                                        uint64_t *v1, int n, int lo, int bits) {
    constexpr int kWarps = kSortThreads / 32;
    __shared__ uint32_t base[kBuckets];
    __shared__ uint32_t wcnt[kWarps][kBuckets];
    __shared__ uint32_t wsum[kWarps];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool has_v = v0 != nullptr;
    uint64_t *ks = k0, *vs = v0, *kd = k1, *vd = v1;
    for (int shift = lo; shift < lo + bits; shift += kRadixBits) {
        // this thread's items (round j holds item j * 256 + tid), loaded once per pass
        uint64_t kk[kSortItems], vv[kSortItems];
#pragma unroll
        for (int j = 0; j < kSortItems; ++j) {
            const int i = j * kSortThreads + tid;
            kk[j] = i < n ? ks[i] : 0;
            vv[j] = (i < n && has_v) ? vs[i] : 0;
        }
        base[tid] = 0;
        __syncthreads();
#pragma unroll
        for (int j = 0; j < kSortItems; ++j)
            if (j * kSortThreads + tid < n) atomicAdd(&base[(uint32_t)(kk[j] >> shift) & (kBuckets - 1)], 1u);
        __syncthreads();
        // exclusive scan of the 256 bucket counts: within warps, then over the warps' totals
        const uint32_t c = base[tid];
        uint32_t x = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) wsum[warp] = x;
        __syncthreads();
        uint32_t before = 0;
        for (int w = 0; w < warp; ++w) before += wsum[w];
        base[tid] = before + x - c;
        __syncthreads();
#pragma unroll
        for (int j = 0; j < kSortItems; ++j) {
            if (j * kSortThreads >= n) break;   // uniform
            for (int q = tid; q < kWarps * kBuckets; q += kSortThreads) (&wcnt[0][0])[q] = 0;
            __syncthreads();
            const bool valid = j * kSortThreads + tid < n;
            const uint32_t d = valid ? (uint32_t)(kk[j] >> shift) & (kBuckets - 1) : (uint32_t)kBuckets;
            const uint32_t peers = __match_any_sync(0xffffffffu, d);
            const uint32_t below = peers & ((1u << lane) - 1u);
            if (valid && below == 0) wcnt[warp][d] = __popc(peers);
            __syncthreads();
            {
                uint32_t run = base[tid];
#pragma unroll
                for (int w = 0; w < kWarps; ++w) {
                    const uint32_t cw = wcnt[w][tid];
                    wcnt[w][tid] = run;
                    run += cw;
                }
                base[tid] = run;
            }
            __syncthreads();
            if (valid) {
                const uint32_t dst = wcnt[warp][d] + __popc(below);
                kd[dst] = kk[j];
                if (has_v) vd[dst] = vv[j];
            }
            __syncthreads();
        }
        uint64_t *t = ks;
        ks = kd;
        kd = t;
        t = vs;
        vs = vd;
        vd = t;
    }
}

// ------------------------------------------------------------------ join

__device__ __forceinline__ int64_t lower_bound_u64(const uint64_t *a, int64_t n, uint64_t k) {
    int64_t lo = 0, hi = n;
    while (lo < hi) {
        int64_t mid = (lo + hi) >> 1;
        if (a[mid] < k) lo = mid + 1; else hi = mid;
    }
    return lo;
}

__device__ __forceinline__ int64_t upper_bound_u64(const uint64_t *a, int64_t n, uint64_t k) {
    int64_t lo = 0, hi = n;
    while (lo < hi) {
        int64_t mid = (lo + hi) >> 1;
        if (a[mid] <= k) lo = mid + 1; else hi = mid;
    }
    return lo;
}

__global__ void join_count_kernel(const uint64_t *__restrict__ jku, int64_t nu, const uint64_t *__restrict__ jkv,
                                  int64_t nv, int64_t *cnt, uint32_t *lo) {
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < nu; i += (int64_t)gridDim.x * blockDim.x) {
        int64_t l = 0, h = nv;
        if (jkv) {
            uint64_t k = jku[i];
            l = lower_bound_u64(jkv, nv, k);
            h = upper_bound_u64(jkv + l, nv - l, k) + l;
        }
        cnt[i] = h - l;
        lo[i] = (uint32_t)l;
    }
}

__global__ void expand_kernel(const int64_t *__restrict__ off, int64_t nu, const uint32_t *__restrict__ lo,
                              const uint64_t *__restrict__ perm_u, const uint64_t *__restrict__ perm_v,
                              const uint64_t *__restrict__ ko_u, const uint64_t *__restrict__ ko_v, int64_t P,
                              uint64_t *pk, uint64_t *pv) {
    for (int64_t p = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; p < P; p += (int64_t)gridDim.x * blockDim.x) {
        // last row i with off[i] <= p
        int64_t a = 0, b = nu;
        while (a < b) {
            int64_t mid = (a + b) >> 1;
            if (off[mid] <= p) a = mid + 1; else b = mid;
        }
        int64_t i = a - 1;
        int64_t vpos = (int64_t)lo[i] + (p - off[i]);
        uint64_t u = perm_u ? perm_u[i] : (uint64_t)i;
        uint64_t v = perm_v ? perm_v[vpos] : (uint64_t)vpos;
        pk[p] = ko_u[u] | (ko_v ? ko_v[v] : 0ull);
        pv[p] = (u << 32) | v;
    }
}

__global__ void unary_pairs_kernel(const uint64_t *__restrict__ ko_u, int64_t n, uint64_t *pk, uint64_t *pv) {
    for (int64_t p = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; p < n; p += (int64_t)gridDim.x * blockDim.x) {
        pk[p] = ko_u[p];
        pv[p] = (uint64_t)p << 32;
    }
}

__global__ void heads_kernel(const uint64_t *__restrict__ pk, int64_t P, int shift, int64_t *flag) {
    for (int64_t p = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; p < P; p += (int64_t)gridDim.x * blockDim.x)
        flag[p] = (p == 0 || (pk[p] >> shift) != (pk[p - 1] >> shift)) ? 1 : 0;
}

// Banded pair lists (pairs sorted by (band, output key)): thread b finds the
// first pair of band b (b = B: P) and the index of its segment.
__global__ void band_ranges_kernel(const uint64_t *__restrict__ pk, int64_t P, const int64_t *__restrict__ seg_excl,
                                   const int64_t *__restrict__ n_seg, int out_bits, int B, int64_t *band_start,
                                   int64_t *band_seg) {
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b > B) return;
    int64_t lo = 0, hi = P;
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if ((int64_t)(pk[mid] >> out_bits) < b) lo = mid + 1; else hi = mid;
    }
    band_start[b] = lo;
    band_seg[b] = lo < P ? seg_excl[lo] : *n_seg;
}

// Key of each band segment for the band sum: (output key, band), so that a
// sort groups every output key's band partials in band order.
__global__ void band_keys_kernel(const uint64_t *__restrict__ pk, const int64_t *__restrict__ seg_start, int64_t Sp,
                                 int out_bits, int band_bits, uint64_t *sk, uint64_t *sv) {
    const uint64_t omask = out_bits ? (~0ull >> (64 - out_bits)) : 0ull;
    for (int64_t s = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; s < Sp; s += (int64_t)gridDim.x * blockDim.x) {
        const uint64_t k = seg_start ? pk[seg_start[s]] : pk[s];
        sk[s] = ((k & omask) << band_bits) | (k >> out_bits);
        sv[s] = (uint64_t)s;
    }
}

// Output keys and the first sorted band segment of each output key.
__global__ void band_outputs_kernel(const uint64_t *__restrict__ sk, const int64_t *__restrict__ excl, int64_t Sp,
                                    int64_t S, int band_bits, KeyUnpack un, int32_t *out_keys, int64_t *fstart) {
    for (int64_t p = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; p < Sp; p += (int64_t)gridDim.x * blockDim.x) {
        const uint64_t k = sk[p] >> band_bits;
        if (p == 0 || k != (sk[p - 1] >> band_bits)) {
            const int64_t f = excl[p];
            fstart[f] = p;
            for (int c = 0; c < un.uw; ++c) {
                uint64_t mask = un.bits[c] ? ((~0ull) >> (64 - un.bits[c])) : 0ull;
                out_keys[f * un.uw + c] = (int32_t)((k >> un.shift[c]) & mask);
            }
        }
        if (p == 0) fstart[S] = Sp;
    }
}

__global__ void segments_kernel(const uint64_t *__restrict__ pk, const uint64_t *__restrict__ pv,
                                const int64_t *__restrict__ seg_excl, int64_t P, int64_t S, KeyUnpack un,
                                int32_t *out_keys, int64_t *seg_start, uint32_t *pu, uint32_t *pvi, int shift) {
    for (int64_t p = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; p < P; p += (int64_t)gridDim.x * blockDim.x) {
        uint64_t v = pv[p];
        pu[p] = (uint32_t)(v >> 32);
        pvi[p] = (uint32_t)v;
        uint64_t k = pk[p];
        if (p == 0 || (k >> shift) != (pk[p - 1] >> shift)) {
            int64_t s = seg_excl[p];
            seg_start[s] = p;
            for (int c = 0; c < un.uw; ++c) {
                uint64_t mask = un.bits[c] ? ((~0ull) >> (64 - un.bits[c])) : 0ull;
                out_keys[s * un.uw + c] = (int32_t)((k >> un.shift[c]) & mask);
            }
        }
        if (p == 0) seg_start[S] = P;
    }
}

// Last row i of a monotone offset table with off[i] <= p.
__device__ __forceinline__ int64_t owner_row(const int64_t *off, int64_t n, int64_t p) {
    int64_t a = 0, b = n;
    while (a < b) {
        int64_t mid = (a + b) >> 1;
        if (off[mid] <= p) a = mid + 1; else b = mid;
    }
    return a - 1;
}

__global__ void pair_keys_kernel(const uint64_t *__restrict__ pv1, int64_t P1, const uint64_t *__restrict__ jk_a,
                                 const uint64_t *__restrict__ jk_b, uint64_t *jk) {
    for (int64_t p = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; p < P1; p += (int64_t)gridDim.x * blockDim.x) {
        const uint64_t v = pv1[p];
        jk[p] = (jk_a ? jk_a[v >> 32] : 0ull) | (jk_b ? jk_b[(uint32_t)v] : 0ull);
    }
}

__global__ void expand3_kernel(const int64_t *__restrict__ off2, int64_t P1, const uint32_t *__restrict__ lo2,
                               const uint64_t *__restrict__ perm_c, const uint64_t *__restrict__ pk1,
                               const uint64_t *__restrict__ ko_c, int64_t P, uint64_t *pk, uint64_t *pv) {
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < P; t += (int64_t)gridDim.x * blockDim.x) {
        const int64_t p = owner_row(off2, P1, t);
        const int64_t cpos = (int64_t)lo2[p] + (t - off2[p]);
        const uint64_t c = perm_c ? perm_c[cpos] : (uint64_t)cpos;
        pk[t] = pk1[p] | ko_c[c];
        pv[t] = ((uint64_t)p << 32) | c;
    }
}

struct Ord3 {
    int o[3];
};

__global__ void segments3_kernel(const uint64_t *__restrict__ pk, const uint64_t *__restrict__ pv,
                                 const uint64_t *__restrict__ pv1, const int64_t *__restrict__ seg_excl, int64_t P,
                                 int64_t S, KeyUnpack un, Ord3 ord, int32_t *out_keys, int64_t *seg_start,
                                 uint32_t *i0, uint32_t *i1, uint32_t *i2) {
    uint32_t *idx[3] = {i0, i1, i2};
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < P; t += (int64_t)gridDim.x * blockDim.x) {
        const uint64_t v = pv[t];
        const uint64_t ab = pv1[v >> 32];
        idx[ord.o[0]][t] = (uint32_t)(ab >> 32);
        idx[ord.o[1]][t] = (uint32_t)ab;
        idx[ord.o[2]][t] = (uint32_t)v;
        const uint64_t k = pk[t];
        if (t == 0 || k != pk[t - 1]) {
            const int64_t s = seg_excl[t];
            seg_start[s] = t;
            for (int c = 0; c < un.uw; ++c) {
                uint64_t mask = un.bits[c] ? ((~0ull) >> (64 - un.bits[c])) : 0ull;
                out_keys[s * un.uw + c] = (int32_t)((k >> un.shift[c]) & mask);
            }
        }
        if (t == 0) seg_start[S] = P;
    }
}

}  // namespace

// ------------------------------------------------------------ launchers

void launch_pack(ucl_ctx *ctx, const int32_t *keys, int u, int64_t n, KeyPack a, uint64_t *out_a, KeyPack b,
                 uint64_t *out_b) {
    if (n <= 0) return;
    pack_kernel<<<grid_for(ctx, n), kThreads, 0, ctx->stream>>>(keys, u, n, a, out_a, b, out_b);
    ctx->launches++;
}

void launch_check_keys(ucl_ctx *ctx, const int32_t *keys, int u, int64_t n, const int64_t *bounds, KeyPack full,
                       uint64_t *packed_out) {
    if (n <= 0) return;
    Bounds bd{};
    for (int c = 0; c < u; ++c) bd.b[c] = bounds[c];
    check_keys_kernel<<<grid_for(ctx, n), kThreads, 0, ctx->stream>>>(keys, u, n, bd, full, packed_out,
                                                                      ctx->d_status + 1);
    ctx->launches++;
}

void launch_check_dups(ucl_ctx *ctx, const uint64_t *sorted_keys, int64_t n) {
    if (n <= 1) return;
    check_dups_kernel<<<grid_for(ctx, n), kThreads, 0, ctx->stream>>>(sorted_keys, n, ctx->d_status + 1);
    ctx->launches++;
}

void launch_iota(ucl_ctx *ctx, uint64_t *out, int64_t n) {
    if (n <= 0) return;
    iota_kernel<<<grid_for(ctx, n), kThreads, 0, ctx->stream>>>(out, n);
    ctx->launches++;
}

void scan_i64(ucl_ctx *ctx, const int64_t *in, int64_t *out, int64_t n, int64_t *total_dev) {
    scan_excl<int64_t>(ctx, in, out, n, total_dev);
}

int radix_sort(ucl_ctx *ctx, uint64_t *kin, uint64_t *vin, uint64_t *kalt, uint64_t *valt, int64_t n, int bits,
               int lo) {
    if (bits <= 0 || n <= 1) return 0;
    if (n <= kSortTile) {
        // one launch for every pass
        radix_sort_small_kernel<<<1, kSortThreads, 0, ctx->stream>>>(kin, vin, kalt, valt, (int)n, lo, bits);
        ctx->launches++;
        return ((bits + kRadixBits - 1) / kRadixBits) & 1;
    }
    int nblocks = (int)((n + kSortTile - 1) / kSortTile);
    uint32_t *hist = (uint32_t *)ws_get(ctx, sizeof(uint32_t) * (size_t)kBuckets * nblocks);
    uint64_t *ks = kin, *vs = vin, *kd = kalt, *vd = valt;
    int which = 0;
    for (int shift = lo; shift < lo + bits; shift += kRadixBits) {
        radix_hist_kernel<<<nblocks, kSortThreads, 0, ctx->stream>>>(ks, n, shift, hist, nblocks);
        ctx->launches++;
        scan_excl<uint32_t>(ctx, hist, hist, (int64_t)kBuckets * nblocks, nullptr);
        radix_scatter_kernel<<<nblocks, kSortThreads, 0, ctx->stream>>>(ks, vs, kd, vd, n, shift, hist, nblocks);
        ctx->launches++;
        uint64_t *t = ks; ks = kd; kd = t;
        t = vs; vs = vd; vd = t;
        which ^= 1;
    }
    return which;
}

void launch_join_count(ucl_ctx *ctx, const uint64_t *jku, int64_t nu, const uint64_t *jkv, int64_t nv,
                       int64_t *cnt, uint32_t *lo) {
    if (nu <= 0) return;
    join_count_kernel<<<grid_for(ctx, nu), kThreads, 0, ctx->stream>>>(jku, nu, jkv, nv, cnt, lo);
    ctx->launches++;
}

void launch_expand(ucl_ctx *ctx, const int64_t *off, int64_t nu, const uint32_t *lo, const uint64_t *perm_u,
                   const uint64_t *perm_v, const uint64_t *ko_u, const uint64_t *ko_v, int64_t P, uint64_t *pk,
                   uint64_t *pv) {
    if (P <= 0) return;
    expand_kernel<<<grid_for(ctx, P), kThreads, 0, ctx->stream>>>(off, nu, lo, perm_u, perm_v, ko_u, ko_v, P, pk,
                                                                  pv);
    ctx->launches++;
}

void launch_unary_pairs(ucl_ctx *ctx, const uint64_t *ko_u, int64_t n, uint64_t *pk, uint64_t *pv) {
    if (n <= 0) return;
    unary_pairs_kernel<<<grid_for(ctx, n), kThreads, 0, ctx->stream>>>(ko_u, n, pk, pv);
    ctx->launches++;
}

void launch_heads(ucl_ctx *ctx, const uint64_t *pk, int64_t P, int64_t *flag, int shift) {
    if (P <= 0) return;
    heads_kernel<<<grid_for(ctx, P), kThreads, 0, ctx->stream>>>(pk, P, shift, flag);
    ctx->launches++;
}

// ---------------------------------------------------------------- windows
// Windowed pair lists: pairs sorted by (band, output key >> wb), so that the
// pairs of 2^wb consecutive output keys (a window) are contiguous and those
// of one tuple of the first input stay together.  Per pair its slot (output
// key & (2^wb - 1)); per window segment the mask of slots present.

__global__ void win_slots_kernel(const uint64_t *__restrict__ pk, int64_t P, int wb, const int64_t *__restrict__ flag,
                                 const int64_t *__restrict__ excl, uint8_t *slot, uint32_t *mask) {
    const uint64_t qm = (1ull << wb) - 1ull;
    for (int64_t p = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; p < P; p += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t q = (uint32_t)(pk[p] & qm);
        slot[p] = (uint8_t)q;
        const int64_t ws = excl[p] + flag[p] - 1;
        atomicOr(&mask[ws], 1u << q);
    }
}

__global__ void win_count_kernel(const uint32_t *__restrict__ mask, int64_t Sw, int64_t *cnt) {
    for (int64_t s = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; s < Sw; s += (int64_t)gridDim.x * blockDim.x)
        cnt[s] = __popc(mask[s]);
}

// Row r of the output (or of the band partials) for each present slot of a
// window segment, in slot order: rowkey = (window's full key) | slot.
__global__ void win_rows_kernel(const uint64_t *__restrict__ pk, const int64_t *__restrict__ seg_start, int64_t Sw,
                                const uint32_t *__restrict__ mask, const int64_t *__restrict__ wbase, int wb,
                                uint64_t *rowkey) {
    for (int64_t s = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; s < Sw; s += (int64_t)gridDim.x * blockDim.x) {
        const uint64_t base = (pk[seg_start[s]] >> wb) << wb;
        uint32_t m = mask[s];
        int64_t r = wbase[s];
        while (m) {
            const int q = __ffs(m) - 1;
            m &= m - 1;
            rowkey[r++] = base | (uint64_t)q;
        }
    }
}

__global__ void unpack_keys_kernel(const uint64_t *__restrict__ k, int64_t n, KeyUnpack un, int32_t *out_keys) {
    for (int64_t s = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; s < n; s += (int64_t)gridDim.x * blockDim.x)
        for (int c = 0; c < un.uw; ++c) {
            uint64_t mask = un.bits[c] ? ((~0ull) >> (64 - un.bits[c])) : 0ull;
            out_keys[s * un.uw + c] = (int32_t)((k[s] >> un.shift[c]) & mask);
        }
}

// ------------------------------------------------------------ small join
// The whole key stage of a small binary EinSum in one CTA of 1024 threads,
// in shared memory: pack both inputs' keys, join by comparing every A tuple
// with every B tuple (A in row order, B in row order), expand the pairs,
// sort them by output key (stable: bitonic on (key, expansion index)), find
// the segments and write seg_start, the output keys and each pair's rows.
// res[0] = P (pair count; when above kSmallPairs nothing else is written and
// the caller runs the general key stage), res[1] = S.
constexpr int kSmallThreads = 1024;

__device__ __forceinline__ uint64_t pack_col(const int32_t *row, const KeyPack &kp) { return pack_row(row, kp); }

__global__ void __launch_bounds__(kSmallThreads) small_join_kernel(
    const int32_t *__restrict__ keys_a, int ua, int na, const int32_t *__restrict__ keys_b, int ub, int nb,
    KeyPack join_a, KeyPack join_b, KeyPack out_a, KeyPack out_b, KeyUnpack un, int has_join, int64_t *res,
    int64_t *seg_start, int32_t *out_keys, uint32_t *pu, uint32_t *pvi) {
    extern __shared__ uint64_t sm[];
    uint64_t *ja = sm, *oa = ja + kSmallTuples, *jb = oa + kSmallTuples, *ob = jb + kSmallTuples;
    uint64_t *pk = ob + kSmallTuples, *pv = pk + kSmallPairs;
    uint32_t *ord = reinterpret_cast<uint32_t *>(pv + kSmallPairs);   // expansion index, then scan scratch
    __shared__ int32_t cnt[kSmallTuples];
    __shared__ int32_t wsum[kSmallThreads / 32];
    __shared__ int32_t total;
    const int tid = threadIdx.x;
    for (int i = tid; i < na; i += kSmallThreads) {
        ja[i] = has_join ? pack_col(keys_a + (int64_t)i * ua, join_a) : 0ull;
        oa[i] = pack_col(keys_a + (int64_t)i * ua, out_a);
    }
    for (int i = tid; i < nb; i += kSmallThreads) {
        jb[i] = has_join ? pack_col(keys_b + (int64_t)i * ub, join_b) : 0ull;
        ob[i] = pack_col(keys_b + (int64_t)i * ub, out_b);
    }
    __syncthreads();
    // matches per A tuple
    for (int i = tid; i < na; i += kSmallThreads) {
        int c = 0;
        const uint64_t k = ja[i];
        for (int j = 0; j < nb; ++j) c += jb[j] == k;
        cnt[i] = c;
    }
    __syncthreads();
    // exclusive scan of cnt[0, na) (na <= 4 * kSmallThreads: four per thread)
    {
        int v[4], run = 0;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int i = tid * 4 + q;
            v[q] = i < na ? cnt[i] : 0;
            run += v[q];
        }
        int x = run;
        const int lane = tid & 31, w = tid >> 5;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) wsum[w] = x;
        __syncthreads();
        if (tid == 0) {
            int r = 0;
            for (int q = 0; q < kSmallThreads / 32; ++q) {
                const int t = wsum[q];
                wsum[q] = r;
                r += t;
            }
            total = r;
        }
        __syncthreads();
        int base = wsum[w] + x - run;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int i = tid * 4 + q;
            if (i < na) cnt[i] = base;
            base += v[q];
        }
    }
    __syncthreads();
    const int P = total;
    if (tid == 0) res[0] = P;
    if (P > kSmallPairs || P == 0) {
        if (tid == 0) res[1] = 0;
        return;
    }
    // expand: A row order, then B row order
    for (int i = tid; i < na; i += kSmallThreads) {
        int o = cnt[i];
        const uint64_t k = ja[i];
        for (int j = 0; j < nb; ++j)
            if (jb[j] == k) {
                pk[o] = oa[i] | ob[j];
                pv[o] = ((uint64_t)i << 32) | (uint32_t)j;
                ord[o] = (uint32_t)o;
                ++o;
            }
    }
    int n2 = 1;
    while (n2 < P) n2 <<= 1;
    for (int i = P + tid; i < n2; i += kSmallThreads) {
        pk[i] = ~0ull;
        pv[i] = 0;
        ord[i] = 0xFFFFFFFFu;
    }
    __syncthreads();
    // bitonic sort by (output key, expansion index): unique, so stable
    for (int k = 2; k <= n2; k <<= 1)
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = tid; i < n2; i += kSmallThreads) {
                const int l = i ^ j;
                if (l > i) {
                    const bool up = (i & k) == 0;
                    const bool gt = pk[i] > pk[l] || (pk[i] == pk[l] && ord[i] > ord[l]);
                    if (gt == up) {
                        uint64_t t = pk[i]; pk[i] = pk[l]; pk[l] = t;
                        t = pv[i]; pv[i] = pv[l]; pv[l] = t;
                        const uint32_t u = ord[i]; ord[i] = ord[l]; ord[l] = u;
                    }
                }
            }
            __syncthreads();
        }
    // segment heads and their exclusive scan (reusing ord as scratch)
    {
        int v[4], run = 0;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int p = tid * 4 + q;
            v[q] = p < P && (p == 0 || pk[p] != pk[p - 1]) ? 1 : 0;
            run += v[q];
        }
        int x = run;
        const int lane = tid & 31, w = tid >> 5;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        __syncthreads();
        if (lane == 31) wsum[w] = x;
        __syncthreads();
        if (tid == 0) {
            int r = 0;
            for (int q = 0; q < kSmallThreads / 32; ++q) {
                const int t = wsum[q];
                wsum[q] = r;
                r += t;
            }
            total = r;
        }
        __syncthreads();
        int base = wsum[w] + x - run;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int p = tid * 4 + q;
            if (p < P) {
                if (v[q]) {
                    seg_start[base] = p;
                    const uint64_t key = pk[p];
                    for (int c = 0; c < un.uw; ++c) {
                        const uint64_t m = un.bits[c] ? ((~0ull) >> (64 - un.bits[c])) : 0ull;
                        out_keys[(int64_t)base * un.uw + c] = (int32_t)((key >> un.shift[c]) & m);
                    }
                }
                pu[p] = (uint32_t)(pv[p] >> 32);
                pvi[p] = (uint32_t)pv[p];
            }
            base += v[q];
        }
    }
    __syncthreads();
    if (tid == 0) {
        seg_start[total] = P;
        res[1] = total;
    }
}

bool small_join_fits(int64_t na, int64_t nb) {
    return na >= 1 && nb >= 1 && na <= kSmallTuples && nb <= kSmallTuples && na * nb <= (int64_t)1 << 16;
}

void launch_small_join(ucl_ctx *ctx, const int32_t *keys_a, int ua, int64_t na, const int32_t *keys_b, int ub,
                       int64_t nb, const KeyPack &join_a, const KeyPack &join_b, const KeyPack &out_a,
                       const KeyPack &out_b, const KeyUnpack &un, bool has_join, int64_t *res, int64_t *seg_start,
                       int32_t *out_keys, uint32_t *pu, uint32_t *pvi) {
    const size_t smem = sizeof(uint64_t) * (4 * (size_t)kSmallTuples + 2 * (size_t)kSmallPairs) +
                        sizeof(uint32_t) * (size_t)kSmallPairs;
    static bool attr[64] = {};   // the attribute is set once per device
    const int d = ctx->device >= 0 && ctx->device < 64 ? ctx->device : 0;
    if (!attr[d]) {
        cudaFuncSetAttribute(small_join_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        attr[d] = true;
    }
    small_join_kernel<<<1, kSmallThreads, smem, ctx->stream>>>(keys_a, ua, (int)na, keys_b, ub, (int)nb, join_a,
                                                                join_b, out_a, out_b, un, has_join ? 1 : 0, res,
                                                                seg_start, out_keys, pu, pvi);
    ctx->launches++;
}

// A-tile runs for the windowed kernel (see internal.cuh, launch_arun).
__global__ void arun_kernel(const uint32_t *__restrict__ pa, int64_t P, int cap, uint8_t *arun) {
    for (int64_t p = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; p < P; p += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t me = pa[p];
        int back = 0;
        while (back < cap - 1) {
            const int64_t x = p - back;   // x is in the run of p; does x load?
            if (x == 0 || x % cap == 0 || pa[x - 1] != me) break;
            ++back;
        }
        int fwd = 0;
        if (back == 0)
            while (fwd < cap - 1 && p + fwd + 1 < P && (p + fwd + 1) % cap != 0 && pa[p + fwd + 1] == me) ++fwd;
        arun[p] = (uint8_t)(back | (fwd << 4));
    }
}

void launch_arun(ucl_ctx *ctx, const uint32_t *pa, int64_t P, int cap, uint8_t *arun) {
    if (P <= 0) return;
    arun_kernel<<<grid_for(ctx, P), kThreads, 0, ctx->stream>>>(pa, P, cap, arun);
    ctx->launches++;
}

void launch_win_slots(ucl_ctx *ctx, const uint64_t *pk, int64_t P, int wb, const int64_t *flag, const int64_t *excl,
                      uint8_t *slot, uint32_t *mask) {
    if (P <= 0) return;
    win_slots_kernel<<<grid_for(ctx, P), kThreads, 0, ctx->stream>>>(pk, P, wb, flag, excl, slot, mask);
    ctx->launches++;
}

void launch_win_count(ucl_ctx *ctx, const uint32_t *mask, int64_t Sw, int64_t *cnt) {
    if (Sw <= 0) return;
    win_count_kernel<<<grid_for(ctx, Sw), kThreads, 0, ctx->stream>>>(mask, Sw, cnt);
    ctx->launches++;
}

void launch_win_rows(ucl_ctx *ctx, const uint64_t *pk, const int64_t *seg_start, int64_t Sw, const uint32_t *mask,
                     const int64_t *wbase, int wb, uint64_t *rowkey) {
    if (Sw <= 0) return;
    win_rows_kernel<<<grid_for(ctx, Sw), kThreads, 0, ctx->stream>>>(pk, seg_start, Sw, mask, wbase, wb, rowkey);
    ctx->launches++;
}

void launch_unpack_keys(ucl_ctx *ctx, const uint64_t *k, int64_t n, KeyUnpack un, int32_t *out_keys) {
    if (n <= 0 || un.uw == 0) return;
    unpack_keys_kernel<<<grid_for(ctx, n), kThreads, 0, ctx->stream>>>(k, n, un, out_keys);
    ctx->launches++;
}

void launch_band_ranges(ucl_ctx *ctx, const uint64_t *pk, int64_t P, const int64_t *seg_excl, const int64_t *n_seg,
                        int out_bits, int B, int64_t *band_start, int64_t *band_seg) {
    band_ranges_kernel<<<1, 64, 0, ctx->stream>>>(pk, P, seg_excl, n_seg, out_bits, B, band_start, band_seg);
    ctx->launches++;
}

void launch_band_keys(ucl_ctx *ctx, const uint64_t *pk, const int64_t *seg_start, int64_t Sp, int out_bits,
                      int band_bits, uint64_t *sk, uint64_t *sv) {
    if (Sp <= 0) return;
    band_keys_kernel<<<grid_for(ctx, Sp), kThreads, 0, ctx->stream>>>(pk, seg_start, Sp, out_bits, band_bits, sk, sv);
    ctx->launches++;
}

void launch_band_outputs(ucl_ctx *ctx, const uint64_t *sk, const int64_t *excl, int64_t Sp, int64_t S, int band_bits,
                         KeyUnpack un, int32_t *out_keys, int64_t *fstart) {
    if (Sp <= 0) return;
    band_outputs_kernel<<<grid_for(ctx, Sp), kThreads, 0, ctx->stream>>>(sk, excl, Sp, S, band_bits, un, out_keys,
                                                                         fstart);
    ctx->launches++;
}

void launch_segments(ucl_ctx *ctx, const uint64_t *pk, const uint64_t *pv, const int64_t *seg_excl, int64_t P,
                     int64_t S, KeyUnpack un, int32_t *out_keys, int64_t *seg_start, uint32_t *pu, uint32_t *pvi,
                     int shift) {
    if (P <= 0) return;
    segments_kernel<<<grid_for(ctx, P), kThreads, 0, ctx->stream>>>(pk, pv, seg_excl, P, S, un, out_keys,
                                                                    seg_start, pu, pvi, shift);
    ctx->launches++;
}

void launch_pair_keys(ucl_ctx *ctx, const uint64_t *pv1, int64_t P1, const uint64_t *jk_a, const uint64_t *jk_b,
                      uint64_t *jk) {
    if (P1 <= 0) return;
    pair_keys_kernel<<<grid_for(ctx, P1), kThreads, 0, ctx->stream>>>(pv1, P1, jk_a, jk_b, jk);
    ctx->launches++;
}

void launch_expand3(ucl_ctx *ctx, const int64_t *off2, int64_t P1, const uint32_t *lo2, const uint64_t *perm_c,
                    const uint64_t *pk1, const uint64_t *ko_c, int64_t P, uint64_t *pk, uint64_t *pv) {
    if (P <= 0) return;
    expand3_kernel<<<grid_for(ctx, P), kThreads, 0, ctx->stream>>>(off2, P1, lo2, perm_c, pk1, ko_c, P, pk, pv);
    ctx->launches++;
}

void launch_segments3(ucl_ctx *ctx, const uint64_t *pk, const uint64_t *pv, const uint64_t *pv1,
                      const int64_t *seg_excl, int64_t P, int64_t S, KeyUnpack un, const int ord[3],
                      int32_t *out_keys, int64_t *seg_start, uint32_t *const idx[3]) {
    if (P <= 0) return;
    Ord3 o{{ord[0], ord[1], ord[2]}};
    segments3_kernel<<<grid_for(ctx, P), kThreads, 0, ctx->stream>>>(pk, pv, pv1, seg_excl, P, S, un, o, out_keys,
                                                                     seg_start, idx[0], idx[1], idx[2]);
    ctx->launches++;
}

}  // namespace ucl
