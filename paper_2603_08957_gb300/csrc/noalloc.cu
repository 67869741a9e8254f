// noalloc.cu -- key validation that allocates nothing.
//
// ucl_relation_create validates keys with workspace obtained from the
// context's allocator.  Some callers cannot allocate device memory at all --
// for example code that runs under a device-memory budget owned by another
// component, or that must never call cudaMalloc because that call can
// synchronise the device.  ucl_keys_check_noalloc gives them the same checks
// (key range, one tuple per key, ascending order) using only a fixed scratch
// array that lives in this file: every GPU that loads the library holds it
// until the process exits.
//
// The scratch is file-scope device memory.  In host code its name is only a
// host-side stand-in, so its device address is looked up once per device with
// cudaGetSymbolAddress (with that device current) and passed to the kernels.
// Every call shares the one array: calls whose GPU work overlaps (on
// different streams) race on it.
#include <mutex>

#include "internal.cuh"

namespace {

constexpr int64_t kMaxTuples = UCL_NOALLOC_MAX_TUPLES;
constexpr int kThreads = 256;
constexpr int kBuckets = 256;
constexpr int kItems = 4096;                                   // tuples per sort block
constexpr int kMaxBlocks = (int)((kMaxTuples + kItems - 1) / kItems);

// [0, 2 kMaxTuples) two packed-key buffers, then the digit histogram
// [kBuckets * kMaxBlocks], then 4 flag words.
constexpr size_t kScratchWords = 2 * (size_t)kMaxTuples + (kBuckets * (size_t)kMaxBlocks + 4 + 1) / 2;
static __device__ __align__(256) unsigned long long g_noalloc_scratch[kScratchWords];

enum : uint32_t { kRange = 1u, kUnsorted = 2u, kDup = 4u };

struct Bounds {
    int64_t b[ucl::kMaxCols];
    int shift[ucl::kMaxCols];
};

__global__ void nk_check(const int32_t *__restrict__ keys, int u, int64_t n, Bounds bd, uint64_t *packed,
                         uint32_t *flags) {
    uint32_t f = 0;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        uint64_t k = 0, prev = 0;
        for (int c = 0; c < u; ++c) {
            const int32_t v = keys[i * u + c];
            if (v < 0 || (int64_t)v >= bd.b[c]) f |= kRange;
            k |= (uint64_t)(uint32_t)v << bd.shift[c];
            if (i > 0) prev |= (uint64_t)(uint32_t)keys[(i - 1) * u + c] << bd.shift[c];
        }
        if (i > 0 && prev >= k) f |= kUnsorted;
        packed[i] = k;
    }
    if (f) atomicOr(flags, f);
}

__global__ void nk_hist(const uint64_t *__restrict__ k, int64_t n, int shift, uint32_t *hist, int nblocks) {
    __shared__ uint32_t h[kBuckets];
    h[threadIdx.x] = 0;
    __syncthreads();
    const int64_t start = (int64_t)blockIdx.x * kItems, end = start + kItems < n ? start + kItems : n;
    for (int64_t i = start + threadIdx.x; i < end; i += kThreads) atomicAdd(&h[(uint32_t)(k[i] >> shift) & 255u], 1u);
    __syncthreads();
    hist[(int64_t)threadIdx.x * nblocks + blockIdx.x] = h[threadIdx.x];
}

// Exclusive scan of the histogram by one block (at most kBuckets * kMaxBlocks entries).
__global__ void nk_scan(uint32_t *hist, int count) {
    __shared__ uint32_t part[kThreads];
    const int per = (count + kThreads - 1) / kThreads;
    const int b0 = threadIdx.x * per, b1 = b0 + per < count ? b0 + per : count;
    uint32_t s = 0;
    for (int i = b0; i < b1; ++i) s += hist[i];
    part[threadIdx.x] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t run = 0;
        for (int t = 0; t < kThreads; ++t) {
            const uint32_t v = part[t];
            part[t] = run;
            run += v;
        }
    }
    __syncthreads();
    uint32_t run = part[threadIdx.x];
    for (int i = b0; i < b1; ++i) {
        const uint32_t v = hist[i];
        hist[i] = run;
        run += v;
    }
}

// Stable scatter: each round of kThreads items is ranked with a shared-memory
// counting pass in item order (one thread per digit value walks the round).
__global__ void nk_scatter(const uint64_t *__restrict__ kin, uint64_t *__restrict__ kout, int64_t n, int shift,
                           const uint32_t *__restrict__ offs, int nblocks) {
    __shared__ uint32_t base[kBuckets];
    __shared__ uint32_t digit[kThreads];
    __shared__ uint32_t rank[kThreads];
    base[threadIdx.x] = offs[(int64_t)threadIdx.x * nblocks + blockIdx.x];
    const int64_t start = (int64_t)blockIdx.x * kItems, end = start + kItems < n ? start + kItems : n;
    for (int64_t r = start; r < end; r += kThreads) {
        const int64_t i = r + threadIdx.x;
        const bool valid = i < end;
        const uint64_t key = valid ? kin[i] : 0;
        digit[threadIdx.x] = valid ? (uint32_t)(key >> shift) & 255u : kBuckets;
        __syncthreads();
        // thread d ranks the items of digit d in this round, in item order
        {
            const uint32_t d = threadIdx.x;
            uint32_t c = base[d];
            for (int t = 0; t < kThreads; ++t)
                if (digit[t] == d) rank[t] = c++;
            base[d] = c;
        }
        __syncthreads();
        if (valid) kout[rank[threadIdx.x]] = key;
        __syncthreads();
    }
}

__global__ void nk_dups(const uint64_t *__restrict__ k, int64_t n, uint32_t *flags) {
    for (int64_t i = 1 + blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        if (k[i] == k[i - 1]) {
            atomicOr(flags, kDup);
            return;
        }
}

// Device address of the scratch array, looked up once per device.
std::mutex g_mu;
void *g_addr[64];

cudaError_t scratch_for(int device, void **out) {
    std::lock_guard<std::mutex> lk(g_mu);
    if (device < 0 || device >= 64) return cudaErrorInvalidDevice;
    if (!g_addr[device]) {
        int prev = 0;
        cudaError_t e = cudaGetDevice(&prev);
        if (e != cudaSuccess) return e;
        e = cudaSetDevice(device);
        if (e != cudaSuccess) return e;
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        cudaSetDevice(prev);
        if (e != cudaSuccess) return e;
        g_addr[device] = p;
    }
    *out = g_addr[device];
    return cudaSuccess;
}

// Restores the calling thread's current device on every return path.
struct DeviceGuard {
    int prev = -1;
    DeviceGuard() {
        if (cudaGetDevice(&prev) != cudaSuccess) {
            cudaGetLastError();
            prev = -1;
        }
    }
    ~DeviceGuard() {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

ucl_status check_keys(int device, void *stream, int64_t n, int u, const int32_t *keys, const int64_t *key_bounds,
                      int *sorted) {
    if (sorted) *sorted = 0;
    if (n < 0 || u < 0 || u > ucl::kMaxCols || (n > 0 && u > 0 && !keys) || (u > 0 && !key_bounds))
        return UCL_ERR_ARG;
    if (n > kMaxTuples) return UCL_ERR_UNSUPPORTED;
    Bounds bd{};
    int total = 0;
    for (int c = 0; c < u; ++c) {
        if (key_bounds[c] < 1 || key_bounds[c] > (1ll << 31)) return UCL_ERR_ARG;
        bd.b[c] = key_bounds[c];
        total += ucl::bit_width(key_bounds[c]);
    }
    if (total > 64) return UCL_ERR_UNSUPPORTED;
    int shift = total;
    for (int c = 0; c < u; ++c) {
        shift -= ucl::bit_width(key_bounds[c]);
        bd.shift[c] = shift;
    }
    if (u == 0) {
        if (sorted) *sorted = 1;
        return n > 1 ? UCL_ERR_DUP_KEY : UCL_OK;
    }
    if (n == 0) {
        if (sorted) *sorted = 1;
        return UCL_OK;
    }
    DeviceGuard guard;
    cudaError_t e = cudaSetDevice(device);
    if (e != cudaSuccess) return UCL_ERR_CUDA;
    void *base = nullptr;
    if ((e = scratch_for(device, &base)) != cudaSuccess) return UCL_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    uint64_t *k0 = static_cast<uint64_t *>(base), *k1 = k0 + kMaxTuples;
    uint32_t *hist = reinterpret_cast<uint32_t *>(k1 + kMaxTuples);
    uint32_t *flags = hist + (size_t)kBuckets * kMaxBlocks;
    uint32_t host_flags = 0;
    const int grid = (int)((n + kThreads - 1) / kThreads < 1024 ? (n + kThreads - 1) / kThreads : 1024);
    // the flag word keeps the previous call's value: clear it first
    e = cudaMemsetAsync(flags, 0, sizeof(uint32_t), s);
    if (e == cudaSuccess) {
        nk_check<<<grid, kThreads, 0, s>>>(keys, u, n, bd, k0, flags);
        // a launch that failed leaves the flags at 0: never read them then
        e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaMemcpyAsync(&host_flags, flags, sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return UCL_ERR_CUDA;
    if (host_flags & kRange) return UCL_ERR_KEY_RANGE;
    if (!(host_flags & kUnsorted)) {
        if (sorted) *sorted = 1;
        return UCL_OK;
    }
    // unsorted: LSD radix sort of the packed keys, then an adjacent-equal check
    const int nblocks = (int)((n + kItems - 1) / kItems);
    uint64_t *src = k0, *dst = k1;
    for (int sh = 0; sh < total && e == cudaSuccess; sh += 8) {
        nk_hist<<<nblocks, kThreads, 0, s>>>(src, n, sh, hist, nblocks);
        nk_scan<<<1, kThreads, 0, s>>>(hist, kBuckets * nblocks);
        nk_scatter<<<nblocks, kThreads, 0, s>>>(src, dst, n, sh, hist, nblocks);
        e = cudaGetLastError();
        uint64_t *t = src;
        src = dst;
        dst = t;
    }
    if (e == cudaSuccess) {
        nk_dups<<<grid, kThreads, 0, s>>>(src, n, flags);
        e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaMemcpyAsync(&host_flags, flags, sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return UCL_ERR_CUDA;
    return (host_flags & kDup) ? UCL_ERR_DUP_KEY : UCL_OK;
}

}  // namespace

extern "C" ucl_status ucl_keys_check_noalloc(int device, void *stream, int64_t n, int u, const int32_t *keys,
                                             const int64_t *key_bounds, int *sorted) {
    return check_keys(device, stream, n, u, keys, key_bounds, sorted);
}
