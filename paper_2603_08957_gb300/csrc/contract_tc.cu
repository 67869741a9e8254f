// contract_tc.cu -- tcgen05 tile contraction with the segmented group-by sum
// fused into its epilogue (paper Sec. 5: the kernel K applied to every joined
// pair, then SUM ... GROUP BY up(W)).
//
// Applies when the lower-case EinSum of one pair is a bf16 GEMM,
//     D[M x N] += A[M x K] * B[K x N],
// with A and B the two joined tiles (either operand order) and the output
// tile equal to D up to a transpose.  One CTA per SM processes a contiguous
// unit of the pair list, which is ordered by output key:
//
//   warp 0      TMA producer: gathers the A and B tiles of consecutive pairs
//               (tile index = tuple index, from the pair list) into a ring of
//               shared-memory stages, 128B/64B/32B-swizzled;
//   warp 1      MMA issuer: one thread issues tcgen05.mma per 16-deep K step
//               into a TMEM accumulator, accumulating across all pairs of one
//               output key (one segment); the warp owns the TMEM allocation;
//   warps 2-5   epilogue: when a segment's accumulator is complete, drain it
//               from TMEM (tcgen05.ld), apply scale / relu, cast and store the
//               output tile -- or, for a segment that continues in another
//               unit, store an fp32 partial for the fixup kernel.
//
// Accumulators are multi-buffered in TMEM so the epilogue of one segment
// overlaps the MMAs of the next.  Tiles too large for a deep enough ring of
// whole pairs are streamed in K chunks: a stage then holds one chunk of one
// pair, and the pipeline runs over (pair, chunk) positions, kc per pair; all
// chunks of a segment's pairs accumulate into its buffer.  A pipeline stage holds the tiles of `pps`
// consecutive pairs, so that barrier traffic is paid once per stage.  The
// producer and MMA warps run warp-uniform loops and issue through one elected
// lane; descriptors are precomputed so that one MMA costs a few integer adds.
// Every wait on an mbarrier is bounded (about 1 s of SM clock); on expiry the
// CTA raises kStTimeout, every role leaves its loop, in-flight TMA copies and
// MMAs are drained (again with a bound), TMEM is freed and the kernel returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstdlib>
#include <mutex>

#include "internal.cuh"

namespace ucl {

namespace {

constexpr int kProducers = 2;                                 // TMA warps
constexpr int kMmaWarps = 2;                                  // MMA-issuing warps (the first also owns TMEM)
constexpr int kTcThreads = 32 * (kProducers + kMmaWarps + 4);  // + 4 epilogue warps
constexpr long long kWaitLimitCycles = 2500000000ll;   // ~1.2 s at 2.07 GHz
constexpr int kMaxStages = 8;
constexpr int kMaxAcc = 4;
constexpr uint32_t kSmemLimit = 227 * 1024;
// barriers, then 16 misc words, then (windowed kernel) 4 pair words and a
// release word per stage, with room to spare
constexpr uint32_t kBarBytes = 8u * (2 * kMaxStages + 2 * kMaxAcc + 1) + 64 + 64 + 256;

struct TcArgs {
    const uint32_t *pa;   // [P] A tuple of each pair
    const uint32_t *pb;   // [P] B tuple of each pair
    int64_t nA, nB;
    const int64_t *seg_start;
    int64_t S;
    Units units;
    void *out;
    int dout, epi;
    float scale;
    float *partials;
    int64_t tile_w;
    int64_t sWm, sWn;
    int N, K, m_blocks;
    int kc_lg;                   // log2 of the K chunks per pair
    int wa, wb;                  // sub-tile width (elements) of the A / B boxes
    int na_sub, nb_sub;          // boxes per chunk
    int a_cx, a_cy, b_cx, b_cy;  // box coordinate step per K chunk (x: columns, y: rows)
    uint32_t a_sub, b_sub;       // bytes per sub-tile (multiple of 1024)
    uint32_t a_pair, b_pair;     // bytes of one pair's A / B tile in a stage
    uint32_t stage_bytes;        // pps * (a_pair + b_pair)
    uint32_t pair_tx;            // bytes TMA delivers per pair chunk
    int pps;                     // pairs per stage
    int ns, nacc, nmma;
    int pf_a, pf_b;              // prefetch the A / B tiles into L2 ahead of their TMA loads
    int pf_dist;                 // how many of its own fills ahead a producer prefetches
    int hint_a, hint_b;          // L2 policy of the A / B tile loads: 0 none, 1 evict first, 2 evict last
    long long wait_limit;        // SM cycles a role waits on one barrier phase before it aborts the CTA
    int withhold_fill;           // failure-detection test: the producers skip this stage fill (-1: none)
    // windows (tc_window_kernel): the pairs of 2^wb consecutive output keys
    // accumulate into one buffer of 2^wb slots; consecutive pairs with the
    // same A tuple load its tile once
    int win_bits;
    const uint8_t *slot;         // [P] slot of each pair in its window
    const uint8_t *arun;         // [P] low nibble: pairs back to the one that loads this pair's A tile;
                                 //     high nibble (for that loader): pairs after it sharing the tile
    const uint32_t *wmask;       // [S] slots present in each window segment
    const int64_t *wbase;        // [S] output row of each window segment's first present slot
    int share_cap;               // a loaded A tile serves at most this many consecutive pairs
    uint32_t tmem_cols;
    uint32_t idesc;
    // descriptor templates (stage 0, slot 0, k step 0) and per-step offsets in
    // 16-byte units: off(kk, mb) = (kk >> lg) * sub16 + (kk & mask) * k16 + mb * mb16
    uint64_t a_desc0, b_desc0;   // start address field left 0; the kernel adds the smem base
    int a_lg, a_mask, a_sub16, a_k16, a_mb16;
    int b_lg, b_mask, b_sub16, b_k16;
    uint32_t *status;
};

// ------------------------------------------------------------- PTX wrappers

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// try_wait with a suspend-time hint: the thread sleeps in hardware until the
// phase completes or about `hint_ns` pass, instead of spinning (spinning
// warps would flood the shared-memory pipe every other role depends on).
__device__ __forceinline__ bool mbar_try_sleep(uint32_t bar, uint32_t parity, uint32_t hint_ns) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(hint_ns)
        : "memory");
    return ok != 0;
}

// Bounded wait for the phase of `parity` to complete.  Gives up when another
// role of the CTA has aborted, or after `limit` SM cycles (kWaitLimitCycles
// unless the context set a shorter limit; then raises the abort and the
// device status).  Returns false when it gave up.  Lanes of one
// warp may decide differently at the limit, so callers combine the result
// with __all_sync before any warp-collective instruction.
__device__ __noinline__ bool mbar_wait_slow(uint32_t bar, uint32_t parity, volatile uint32_t *abort_flag,
                                            uint32_t *status, long long limit) {
    const long long t0 = clock64();
    for (;;) {
        if (mbar_try_sleep(bar, parity, 100000u)) return true;
        if (*abort_flag) return false;
        if (clock64() - t0 > limit) {
            *abort_flag = 1;
            atomicOr(status, kStTimeout);
            return false;
        }
    }
}

__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile uint32_t *abort_flag,
                                          uint32_t *status, long long limit) {
    return mbar_try(bar, parity) || mbar_wait_slow(bar, parity, abort_flag, status, limit);
}

// Bounded wait used while draining after an abort (ignores the abort flag).
__device__ __noinline__ void mbar_drain(uint32_t bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!mbar_try_sleep(bar, parity, 100000u))
        if (clock64() - t0 > kWaitLimitCycles) return;
}

__device__ __forceinline__ bool elect_one() {
    uint32_t pred;
    asm volatile(
        "{\n\t.reg .b32 r;\n\t.reg .pred p;\n\t"
        "elect.sync r|p, 0xffffffff;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(pred));
    return pred != 0;
}

__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, int x, int y, int z, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
        "[%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar)
        : "memory");
}

// The same copy with an L2 eviction policy (from createpolicy).
__device__ __forceinline__ void tma_load_3d_hint(uint32_t dst, const CUtensorMap *map, int x, int y, int z,
                                                 uint32_t bar, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, "
        "{%2, %3, %4}], [%5], %6;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar), "l"(policy)
        : "memory");
}

// L2 policies: lines a copy brings in are evicted before (first) or after
// (last) lines of normal priority.
__device__ __forceinline__ uint64_t policy_of(int hint) {
    uint64_t p = 0;
    if (hint == 1)
        asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    else
        asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// Hint that a box of the tensor will be loaded soon: fetched into L2 only,
// no shared memory, no completion to track.
__device__ __forceinline__ void tma_prefetch_3d(const CUtensorMap *map, int x, int y, int z) {
    asm volatile("cp.async.bulk.prefetch.tensor.3d.L2.global.tile [%0, {%1, %2, %3}];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(x), "r"(y), "r"(z)
                 : "memory");
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float *v) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// A role's position in the ring: fill number f, its stage and the parity of
// its lap.  A role that owns the stages role, role + step, ... (< ns) moves
// to its next own fill without a division.
struct StageCursor {
    int f;
    uint32_t st, ph;
    __device__ __forceinline__ void start(int role) {
        f = role;
        st = (uint32_t)role;
        ph = 0;
    }
    __device__ __forceinline__ void next(int role, int step, uint32_t ns) {
        const uint32_t nx = st + (uint32_t)step;
        if (nx < ns) {
            f += step;
            st = nx;
        } else {
            f += (int)(ns - st) + role;
            st = (uint32_t)role;
            ph ^= 1u;
        }
    }
};

__device__ __forceinline__ int64_t find_seg(const int64_t *seg_start, int64_t S, int64_t p) {
    int64_t a = 0, b = S;
    while (a < b) {
        int64_t mid = (a + b) >> 1;
        if (seg_start[mid] <= p) a = mid + 1; else b = mid;
    }
    return a - 1;
}

__device__ __forceinline__ float epilogue(float x, int epi, float scale) {
    x *= scale;
    if (epi == UCL_EPI_RELU) x = fmaxf(x, 0.0f);
    return x;
}

// ------------------------------------------------------------------ kernel

__device__ __forceinline__ void tmem_st16_zero(uint32_t taddr) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %1, %1, %1, %1, %1, %1, %1, %1, %1, %1, %1, %1, %1, %1, "
        "%1};" ::"r"(taddr),
        "r"(0u)
        : "memory");
}

template <int KSTEPS>
__global__ void __launch_bounds__(kTcThreads, 1)
    tc_contract_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                       const TcArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const uint32_t sbase = smem_u32(smem);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + (size_t)a.ns * a.stage_bytes);
    const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8u * a.ns, accf0 = empty0 + 8u * a.ns,
                   acce0 = accf0 + 8u * a.nacc, done_bar = acce0 + 8u * a.nacc;
    uint32_t *misc = reinterpret_cast<uint32_t *>(bars + 2 * a.ns + 2 * a.nacc + 1);
    // misc[0] TMEM base, [1] abort flag, [2 + w] stage fills MMA warp w has walked past,
    // [4 + w] stages filled by producer w
    volatile uint32_t *abort_flag = misc + 1;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nmma = a.nmma;
    const uint32_t acc_cols = (uint32_t)(a.N * a.m_blocks), buf_cols = acc_cols * (uint32_t)nmma;

    if (threadIdx.x == 0) {
        for (int i = 0; i < a.ns; ++i) {
            mbar_init(full0 + 8u * i, 1);
            mbar_init(empty0 + 8u * i, 1);
        }
        for (int i = 0; i < a.nacc; ++i) {
            mbar_init(accf0 + 8u * i, (uint32_t)nmma);
            mbar_init(acce0 + 8u * i, 4);
        }
        mbar_init(done_bar, (uint32_t)nmma);
        for (int i = 1; i < 16; ++i) misc[i] = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == kProducers) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(misc)),
                     "r"(a.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = misc[0];
    if (warp >= kProducers + kMmaWarps) {
        // accumulators start at zero: every MMA accumulates, and the epilogue
        // re-zeroes a buffer after draining it
        const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
        for (uint32_t c = 0; c < a.tmem_cols; c += 16) tmem_st16_zero(tmem + lane_base + c);
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    const int unit = blockIdx.x;
    const int64_t pb = a.units.begin(unit), pe = a.units.begin(unit + 1);
    const int64_t s_first = pe > pb ? find_seg(a.seg_start, a.S, pb) : 0;
    const int64_t s_last = pe > pb ? find_seg(a.seg_start, a.S, pe - 1) : -1;

    if (warp < kProducers) {
        // ------------------------------------------------------ producers
        // Producer warp w fills the stages of fill number w, w + kProducers,
        // ...: lane j loads the tile indices of the stage's pair j (prefetched
        // one own stage ahead), lane 0 waits for the slot and posts the
        // expected bytes, then lane j issues the TMA copies of pair j.
        const int n = (int)(pe - pb) << a.kc_lg, pps = a.pps;
        const int nfills = (n + pps - 1) / pps;
        const int kmask = (1 << a.kc_lg) - 1;
        uint32_t mine = 0;
        const uint64_t pol_a = a.hint_a ? policy_of(a.hint_a) : 0ull, pol_b = a.hint_b ? policy_of(a.hint_b) : 0ull;
        // raw index loads two own fills ahead, checked only when used, so a
        // fill never waits on the latency of its own index loads
        auto load_idx = [&](int f, uint32_t &ia, uint32_t &ib) {
            ia = 0;
            ib = 0;
            const int v = f * pps + lane;
            const int64_t p = pb + (v >> a.kc_lg);
            if (f < nfills && lane < pps && v < n) {
                ia = a.pa[p];
                ib = a.pb[p];
            }
        };
        uint32_t ia, ib, ia1, ib1;
        load_idx(warp, ia, ib);
        load_idx(warp + kProducers, ia1, ib1);
        // L2 prefetch of streamed tiles (whole pairs only): at its fill f a
        // producer prefetches the pairs of fill f + pf_dist * kProducers, with
        // indices loaded one own fill earlier (out-of-range indices are skipped)
        const bool pf = (a.pf_a | a.pf_b) && a.kc_lg == 0;
        const int pf_ahead = a.pf_dist * kProducers;
        uint32_t qa = 0xFFFFFFFFu, qb = 0xFFFFFFFFu;
        auto load_pf = [&](int f2) {
            qa = 0xFFFFFFFFu;
            qb = 0xFFFFFFFFu;
            const int v = f2 * pps + lane;
            if (f2 < nfills && lane < pps && v < n) {
                qa = a.pa[pb + v];
                qb = a.pb[pb + v];
            }
        };
        if (pf) load_pf(warp + pf_ahead);
        uint32_t st = (uint32_t)(warp % a.ns), ph = (uint32_t)((warp / a.ns) & 1);
        for (int f = warp; f < nfills; f += kProducers) {
            uint32_t ia2, ib2;
            load_idx(f + 2 * kProducers, ia2, ib2);
            if (pf) {
                if (a.pf_b && (int64_t)qb < a.nB)
                    for (int q = 0; q < a.nb_sub; ++q) tma_prefetch_3d(&tmB, q * a.wb, 0, (int)qb);
                if (a.pf_a && (int64_t)qa < a.nA)
                    for (int q = 0; q < a.na_sub; ++q) tma_prefetch_3d(&tmA, q * a.wa, 0, (int)qa);
                load_pf(f + pf_ahead + kProducers);
            }
            if ((int64_t)ia >= a.nA || (int64_t)ib >= a.nB) {
                atomicOr(a.status, kStBadIndex);
                ia = 0;
                ib = 0;
            }
            if (f == a.withhold_fill) {
                // failure-detection test: this fill is neither posted nor
                // copied, so the waits of its consumers run out
                ++mine;
                ia = ia1;
                ib = ib1;
                ia1 = ia2;
                ib1 = ib2;
                st += kProducers;
                if (st >= (uint32_t)a.ns) {
                    st -= (uint32_t)a.ns;
                    ph ^= 1u;
                }
                continue;
            }
            const int np = n - f * pps < pps ? n - f * pps : pps;
            uint32_t okw = 1;
            if (lane == 0) {
                okw = mbar_wait(empty0 + 8u * st, ph ^ 1u, abort_flag, a.status, a.wait_limit) ? 1u : 0u;
                if (okw) mbar_arrive_tx(full0 + 8u * st, (uint32_t)np * a.pair_tx);
            }
            if (!__shfl_sync(0xffffffffu, okw, 0)) break;
            if (lane < np) {
                const uint32_t fb = full0 + 8u * st;
                const uint32_t sa = sbase + st * a.stage_bytes + (uint32_t)lane * a.a_pair;
                const uint32_t sb = sbase + st * a.stage_bytes + (uint32_t)a.pps * a.a_pair + (uint32_t)lane * a.b_pair;
                const int c = (f * pps + lane) & kmask;   // K chunk
                for (int q = 0; q < a.na_sub; ++q) {
                    if (a.hint_a)
                        tma_load_3d_hint(sa + q * a.a_sub, &tmA, q * a.wa + c * a.a_cx, c * a.a_cy, (int)ia, fb, pol_a);
                    else
                        tma_load_3d(sa + q * a.a_sub, &tmA, q * a.wa + c * a.a_cx, c * a.a_cy, (int)ia, fb);
                }
                for (int q = 0; q < a.nb_sub; ++q) {
                    if (a.hint_b)
                        tma_load_3d_hint(sb + q * a.b_sub, &tmB, q * a.wb + c * a.b_cx, c * a.b_cy, (int)ib, fb, pol_b);
                    else
                        tma_load_3d(sb + q * a.b_sub, &tmB, q * a.wb + c * a.b_cx, c * a.b_cy, (int)ib, fb);
                }
            }
            __syncwarp();
            ++mine;
            ia = ia1;
            ib = ib1;
            ia1 = ia2;
            ib1 = ib2;
            st += kProducers;
            if (st >= (uint32_t)a.ns) {
                st -= (uint32_t)a.ns;
                ph ^= 1u;
            }
        }
        if (lane == 0) misc[4 + warp] = mine;
    } else if (warp < kProducers + kMmaWarps) {
        // ------------------------------------------------------------ MMA
        // MMA warp w consumes the stages of fill number w, w + nmma, ... and
        // accumulates into its own half of each TMEM accumulator buffer, so
        // that one warp's bookkeeping overlaps the other's MMAs.  Every warp
        // walks all stages and segments to keep the buffer ring in step.
        // Loops are warp-uniform; descriptors are formed in uniform code and
        // one elected lane issues.
        const int w = warp - kProducers;
        if (w < nmma) {
            uint32_t aoff[KSTEPS], boff[KSTEPS];
#pragma unroll
            for (int kk = 0; kk < KSTEPS; ++kk) {
                aoff[kk] = (uint32_t)((kk >> a.a_lg) * a.a_sub16 + (kk & a.a_mask) * a.a_k16);
                boff[kk] = (uint32_t)((kk >> a.b_lg) * a.b_sub16 + (kk & a.b_mask) * a.b_k16);
            }
            const uint64_t adesc0 = a.a_desc0 + (sbase >> 4);
            const uint64_t bdesc0 = a.b_desc0 + ((sbase + (uint32_t)a.pps * a.a_pair) >> 4);
            const uint32_t stage16 = a.stage_bytes >> 4, apair16 = a.a_pair >> 4, bpair16 = a.b_pair >> 4;
            const uint32_t mb16 = (uint32_t)a.a_mb16, ncol = (uint32_t)a.N, idesc = a.idesc;
            const bool two_m = a.m_blocks > 1;
            // positions count (pair, K chunk) steps, kc per pair
            const int n = (int)(pe - pb) << a.kc_lg, pps = a.pps;
            uint32_t b = 0, aph = 0, dcol = tmem;
            int64_t s = s_first;
            int seg_end = n > 0 ? (int)((a.seg_start[s + 1] < pe ? a.seg_start[s + 1] : pe) - pb) << a.kc_lg : 0;
            bool fresh = true, ok = true;
            // Segment events: before the warp's first MMA into a segment it waits
            // for the accumulator buffer (open); at the segment's end it commits
            // the buffer to the epilogue (close).  Both warps open and close every
            // segment, in order, also segments whose pairs all lie in the other
            // warp's stages.
            auto open_seg = [&]() -> bool {
                if (!__all_sync(0xffffffffu, mbar_wait(acce0 + 8u * b, aph ^ 1u, abort_flag, a.status, a.wait_limit))) return false;
                tc_fence_after();
                dcol = tmem + b * buf_cols + (uint32_t)w * acc_cols;
                fresh = false;
                return true;
            };
            auto close_seg = [&](int pos) {
                if (elect_one()) mma_commit(accf0 + 8u * b);
                __syncwarp();
                if (++b == (uint32_t)a.nacc) {
                    b = 0;
                    aph ^= 1u;
                }
                ++s;
                if (pos < n) seg_end = (int)((a.seg_start[s + 1] < pe ? a.seg_start[s + 1] : pe) - pb) << a.kc_lg;
                fresh = true;
            };
            uint32_t st = (uint32_t)(w % a.ns), ph = (uint32_t)((w / a.ns) & 1);
            int f = w;
            for (; f * pps < n; f += nmma) {
                const int start = f * pps;
                const int np = n - start < pps ? n - start : pps;
                // segments that end inside the other warp's stages before this one
                while (seg_end <= start) {
                    if (fresh && !open_seg()) {
                        ok = false;
                        break;
                    }
                    close_seg(seg_end);
                }
                if (!ok) break;
                if (!__all_sync(0xffffffffu, mbar_wait(full0 + 8u * st, ph, abort_flag, a.status, a.wait_limit))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                uint64_t ad = adesc0 + st * stage16, bd = bdesc0 + st * stage16;
                if (!fresh && start + np <= seg_end) {
                    // the whole stage accumulates into the open buffer
                    const uint64_t ad1 = ad + apair16, bd1 = bd + bpair16;
                    const uint64_t ad2 = ad1 + apair16, bd2 = bd1 + bpair16;
                    const uint64_t ad3 = ad2 + apair16, bd3 = bd2 + bpair16;
                    if (elect_one()) {
#pragma unroll
                        for (int kk = 0; kk < KSTEPS; ++kk) {
                            mma_bf16(dcol, ad + aoff[kk], bd + boff[kk], idesc, 1u);
                            if (two_m) mma_bf16(dcol + ncol, ad + aoff[kk] + mb16, bd + boff[kk], idesc, 1u);
                        }
                        if (np > 1) {
#pragma unroll
                            for (int kk = 0; kk < KSTEPS; ++kk) {
                                mma_bf16(dcol, ad1 + aoff[kk], bd1 + boff[kk], idesc, 1u);
                                if (two_m) mma_bf16(dcol + ncol, ad1 + aoff[kk] + mb16, bd1 + boff[kk], idesc, 1u);
                            }
                        }
                        if (np > 2) {
#pragma unroll
                            for (int kk = 0; kk < KSTEPS; ++kk) {
                                mma_bf16(dcol, ad2 + aoff[kk], bd2 + boff[kk], idesc, 1u);
                                if (two_m) mma_bf16(dcol + ncol, ad2 + aoff[kk] + mb16, bd2 + boff[kk], idesc, 1u);
                            }
                        }
                        if (np > 3) {
#pragma unroll
                            for (int kk = 0; kk < KSTEPS; ++kk) {
                                mma_bf16(dcol, ad3 + aoff[kk], bd3 + boff[kk], idesc, 1u);
                                if (two_m) mma_bf16(dcol + ncol, ad3 + aoff[kk] + mb16, bd3 + boff[kk], idesc, 1u);
                            }
                        }
                        mma_commit(empty0 + 8u * st);
                    }
                    __syncwarp();
                } else {
                    // segment boundaries inside the stage: pair by pair
                    for (int jj = 0; jj < np; ++jj) {
                        if (fresh && !open_seg()) {
                            ok = false;
                            break;
                        }
                        if (elect_one()) {
#pragma unroll
                            for (int kk = 0; kk < KSTEPS; ++kk) {
                                mma_bf16(dcol, ad + aoff[kk], bd + boff[kk], idesc, 1u);
                                if (two_m) mma_bf16(dcol + ncol, ad + aoff[kk] + mb16, bd + boff[kk], idesc, 1u);
                            }
                        }
                        __syncwarp();
                        ad += apair16;
                        bd += bpair16;
                        if (start + jj + 1 == seg_end) close_seg(start + jj + 1);
                    }
                    if (!ok) break;
                    if (elect_one()) mma_commit(empty0 + 8u * st);
                    __syncwarp();
                }
                // a fast-path stage may end exactly at the segment's end
                if (!fresh && start + np == seg_end) close_seg(seg_end);
                st += (uint32_t)nmma;
                if (st >= (uint32_t)a.ns) {
                    st -= (uint32_t)a.ns;
                    ph ^= 1u;
                }
            }
            // segments that end after this warp's last stage
            while (ok && s <= s_last) {
                if (fresh && !open_seg()) {
                    ok = false;
                    break;
                }
                close_seg(seg_end);
            }
            if (lane == 0) misc[2 + w] = ok ? 0xFFFFFFFFu : (uint32_t)f;
        }
    } else {
        // ------------------------------------------------------- epilogue
        const int q = warp & 3;   // TMEM lane quadrant this warp may access
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        uint32_t b = 0, ph = 0;
        for (int64_t s = s_first; s <= s_last; ++s) {
            const int64_t ss = a.seg_start[s], se = a.seg_start[s + 1];
            if (!__all_sync(0xffffffffu, mbar_wait(accf0 + 8u * b, ph, abort_flag, a.status, a.wait_limit))) break;
            tc_fence_after();
            const int kind = (ss >= pb && se <= pe) ? 0 : (ss < pb ? 1 : 2);
            float *part = a.partials + ((int64_t)unit * 2 + (kind == 1 ? 0 : 1)) * a.tile_w;
            const uint32_t bcol = tmem + lane_base + b * buf_cols;
            for (int mb = 0; mb < a.m_blocks; ++mb) {
                const int64_t m = (int64_t)mb * 128 + q * 32 + lane;
                for (int c = 0; c < a.N / 16; ++c) {
                    float v[16];
                    const uint32_t col = (uint32_t)(mb * a.N + c * 16);
                    tmem_ld16(bcol + col, v);
                    if (nmma > 1) {
                        float v2[16];
                        tmem_ld16(bcol + acc_cols + col, v2);
#pragma unroll
                        for (int jj = 0; jj < 16; ++jj) v[jj] += v2[jj];
                    }
                    const int64_t base_off = m * a.sWm + (int64_t)c * 16 * a.sWn;
                    if (a.sWn == 1) {
                        // N contiguous in the output: this lane's 16 values are
                        // one 64-byte (fp32) or 32-byte (bf16) run
                        if (kind == 0) {
#pragma unroll
                            for (int jj = 0; jj < 16; ++jj) v[jj] = epilogue(v[jj], a.epi, a.scale);
                        }
                        if (kind == 0 && a.dout == UCL_BF16) {
                            uint32_t h[8];
#pragma unroll
                            for (int jj = 0; jj < 8; ++jj) {
                                __nv_bfloat162 t = __floats2bfloat162_rn(v[2 * jj], v[2 * jj + 1]);
                                h[jj] = *reinterpret_cast<uint32_t *>(&t);
                            }
                            uint4 *o = reinterpret_cast<uint4 *>(reinterpret_cast<__nv_bfloat16 *>(a.out) +
                                                                 s * a.tile_w + base_off);
                            o[0] = make_uint4(h[0], h[1], h[2], h[3]);
                            o[1] = make_uint4(h[4], h[5], h[6], h[7]);
                        } else {
                            float *dst = kind == 0 ? reinterpret_cast<float *>(a.out) + s * a.tile_w + base_off
                                                   : part + base_off;
                            float4 *o = reinterpret_cast<float4 *>(dst);
#pragma unroll
                            for (int jj = 0; jj < 4; ++jj)
                                o[jj] = make_float4(v[4 * jj], v[4 * jj + 1], v[4 * jj + 2], v[4 * jj + 3]);
                        }
                    } else if (kind == 0) {
                        if (a.dout == UCL_BF16) {
                            __nv_bfloat16 *o = reinterpret_cast<__nv_bfloat16 *>(a.out) + s * a.tile_w + base_off;
#pragma unroll
                            for (int jj = 0; jj < 16; ++jj) o[jj * a.sWn] = __float2bfloat16_rn(epilogue(v[jj], a.epi, a.scale));
                        } else {
                            float *o = reinterpret_cast<float *>(a.out) + s * a.tile_w + base_off;
#pragma unroll
                            for (int jj = 0; jj < 16; ++jj) o[jj * a.sWn] = epilogue(v[jj], a.epi, a.scale);
                        }
                    } else {
                        float *o = part + base_off;
#pragma unroll
                        for (int jj = 0; jj < 16; ++jj) o[jj * a.sWn] = v[jj];
                    }
                }
            }
            for (uint32_t c = 0; c < buf_cols; c += 16) tmem_st16_zero(bcol + c);
            asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(acce0 + 8u * b);
            if (++b == (uint32_t)a.nacc) {
                b = 0;
                ph ^= 1u;
            }
        }
    }

    // ---------------------------------------------------------- teardown
    __syncthreads();
    if (*abort_flag) {
        if (warp < kProducers && lane == 0) {
            // copies still in flight write into this CTA's shared memory: wait for
            // every stage this producer filled that its MMA warp did not consume
            for (uint32_t k = 0; k < misc[4 + warp]; ++k) {
                const uint32_t it = (uint32_t)warp + k * kProducers;   // fills this producer issued
                if ((int)it == a.withhold_fill) continue;   // never copied: nothing in flight
                if (it >= misc[2 + it % (uint32_t)nmma]) mbar_drain(full0 + 8u * (it % a.ns), (it / a.ns) & 1u);
            }
        }
        if (warp >= kProducers && warp < kProducers + nmma && lane == 0) {
            mma_commit(done_bar);   // tracks every MMA this thread issued
            mbar_drain(done_bar, 0);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == kProducers) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(a.tmem_cols)
                     : "memory");
    }
}

// Windowed variant.  The pair list is ordered by (output key >> wb, A tuple
// order), so the pairs of a window of 2^wb consecutive output keys are
// contiguous and those of one A tuple within it consecutive.  A window's
// accumulator buffer holds 2^wb slots (slot q at columns q * acc_cols); a
// pair accumulates into its own key's slot.  A run of consecutive pairs with
// the same A tuple loads the A tile once (into the stage of its first pair,
// the loader) and its other pairs read it from there; that stage is released
// only after the run's last pair.  Runs are cut every share_cap pairs (in
// pair-list position) and at unit starts, so that no stage is held longer
// than the ring allows.  One MMA warp; segments are window segments; the
// epilogue writes each present slot to its output row (wbase + rank of the
// slot in the window's mask), or all slots to the unit's partials.
template <int KSTEPS>
__global__ void __launch_bounds__(kTcThreads, 1)
    tc_window_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     const TcArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const uint32_t sbase = smem_u32(smem);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + (size_t)a.ns * a.stage_bytes);
    const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8u * a.ns, accf0 = empty0 + 8u * a.ns,
                   acce0 = accf0 + 8u * a.nacc, done_bar = acce0 + 8u * a.nacc;
    uint32_t *misc = reinterpret_cast<uint32_t *>(bars + 2 * a.ns + 2 * a.nacc + 1);
    // misc[0] TMEM base, [1] abort flag, [2] stage fills the MMA warp has
    // walked past, [4 + w] stages filled by producer w; then per stage four
    // pair words (slot | A source stage << 8 | A source pair << 16) and the
    // fill after which the stage is released
    volatile uint32_t *abort_flag = misc + 1;
    volatile uint32_t *pinfo = misc + 16;
    volatile int32_t *prel = reinterpret_cast<volatile int32_t *>(misc + 16 + 4 * kMaxStages);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int W = 1 << a.win_bits;
    const uint32_t acc_cols = (uint32_t)(a.N * a.m_blocks), buf_cols = acc_cols * (uint32_t)W;

    if (threadIdx.x == 0) {
        for (int i = 0; i < a.ns; ++i) {
            mbar_init(full0 + 8u * i, 1);
            mbar_init(empty0 + 8u * i, 1);
        }
        for (int i = 0; i < a.nacc; ++i) {
            mbar_init(accf0 + 8u * i, 1);
            mbar_init(acce0 + 8u * i, 4);
        }
        mbar_init(done_bar, 1);
        for (int i = 1; i < 16; ++i) misc[i] = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == kProducers) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(misc)),
                     "r"(a.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = misc[0];
    if (warp >= kProducers + kMmaWarps) {
        const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
        for (uint32_t c = 0; c < a.tmem_cols; c += 16) tmem_st16_zero(tmem + lane_base + c);
        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    const int unit = blockIdx.x;
    const int64_t pb = a.units.begin(unit), pe = a.units.begin(unit + 1);
    const int64_t s_first = pe > pb ? find_seg(a.seg_start, a.S, pb) : 0;
    const int64_t s_last = pe > pb ? find_seg(a.seg_start, a.S, pe - 1) : -1;
    const uint32_t a_tx = a.pair_tx - (uint32_t)(a.N * a.K * 2), b_tx = (uint32_t)(a.N * a.K * 2);

    if (warp < kProducers) {
        // ------------------------------------------------------ producers
        // Producer w fills the stages s with s mod kProducers == w, in fill
        // order (so each empty-barrier wait is for the release of that
        // stage's previous fill, although held stages are released out of
        // fill order); lane j takes pair j of the fill.  Each pair's A source
        // comes from arun: its loader is the pair arun's low nibble back, or
        // the unit's first pair if that is later.
        const int n = (int)(pe - pb), pps = a.pps;
        const int nfills = (n + pps - 1) / pps;
        const uint64_t pol_a = a.hint_a ? policy_of(a.hint_a) : 0ull, pol_b = a.hint_b ? policy_of(a.hint_b) : 0ull;
        uint32_t mine = 0;
        const uint32_t ns_u = (uint32_t)a.ns;
        // per-pair words loaded two own fills ahead (as in the plain kernel),
        // so that a fill never waits on the latency of its own index loads
        struct PairWords {
            uint32_t ia, ib, q, r;
        };
        auto load_words = [&](int f2) {
            PairWords w{0u, 0u, 0u, 0u};
            const int v = f2 * pps + lane;
            if (f2 < nfills && lane < pps && v < n) {
                const int64_t p = pb + v;
                w.ia = a.pa[p];
                w.ib = a.pb[p];
                w.q = a.slot[p];
                w.r = a.arun[p];
            }
            return w;
        };
        StageCursor c0, c1, c2;   // this fill and the next two own fills
        c0.start(warp);
        c1 = c0;
        c1.next(warp, kProducers, ns_u);
        c2 = c1;
        c2.next(warp, kProducers, ns_u);
        PairWords w0 = load_words(c0.f), w1 = load_words(c1.f);
        for (; c0.f < nfills; c0 = c1, c1 = c2, c2.next(warp, kProducers, ns_u)) {
            const int f = c0.f;
            const uint32_t st = c0.st, ph = c0.ph;
            const PairWords w2 = load_words(c2.f);
            const PairWords cur = w0;
            w0 = w1;
            w1 = w2;
            if (f == a.withhold_fill) {
                // failure-detection test: this fill is neither posted nor copied
                ++mine;
                continue;
            }
            const int np = n - f * pps < pps ? n - f * pps : pps;
            uint32_t ia = 0, ib = 0, info = 0;
            int rel = f;
            bool load = false;
            if (lane < np) {
                const int64_t p = pb + (int64_t)f * pps + lane;
                ia = cur.ia;
                ib = cur.ib;
                const uint32_t q = cur.q;
                const uint32_t r = cur.r;
                int64_t loader = p - (int64_t)(r & 15u);
                if (loader < pb) loader = pb;
                load = loader == p;
                if ((int64_t)ia >= a.nA || (int64_t)ib >= a.nB) {
                    atomicOr(a.status, kStBadIndex);
                    ia = 0;
                    ib = 0;
                }
                const int64_t src = loader - pb;
                const uint32_t sst = (uint32_t)((src / pps) % a.ns), sj = (uint32_t)(src % pps);
                info = q | (sst << 8) | (sj << 16);
                if (load) {
                    // the last pair reading this tile: the run's last sharer
                    // (counted from the run's own loader), at most the unit's end
                    const int64_t gl = p - (int64_t)(r & 15u);
                    const uint32_t rg = gl == p ? r : a.arun[gl];
                    int64_t last = gl + (int64_t)(rg >> 4);
                    if (last > pe - 1) last = pe - 1;
                    if (last < p) last = p;
                    rel = (int)((last - pb) / pps);
                }
            }
            // the stage is released after the latest fill any of its A tiles serves
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const int r2 = __shfl_xor_sync(0xffffffffu, rel, o);
                rel = r2 > rel ? r2 : rel;
            }
            const uint32_t lmask = __ballot_sync(0xffffffffu, load);
            const uint32_t tx = (uint32_t)__popc(lmask) * a_tx + (uint32_t)np * b_tx;
            uint32_t inf[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) inf[j] = __shfl_sync(0xffffffffu, info, j);
            uint32_t okw = 1;
            if (lane == 0) {
                okw = mbar_wait(empty0 + 8u * st, ph ^ 1u, abort_flag, a.status, a.wait_limit) ? 1u : 0u;
                if (okw) {
                    for (int j = 0; j < np; ++j) pinfo[st * 4 + j] = inf[j];
                    prel[st] = rel;
                    mbar_arrive_tx(full0 + 8u * st, tx);
                }
            }
            if (!__shfl_sync(0xffffffffu, okw, 0)) break;
            if (lane < np) {
                const uint32_t fb = full0 + 8u * st;
                const uint32_t sa = sbase + st * a.stage_bytes + (uint32_t)lane * a.a_pair;
                const uint32_t sb = sbase + st * a.stage_bytes + (uint32_t)a.pps * a.a_pair + (uint32_t)lane * a.b_pair;
                if (load)
                    for (int q = 0; q < a.na_sub; ++q) {
                        if (a.hint_a)
                            tma_load_3d_hint(sa + q * a.a_sub, &tmA, q * a.wa, 0, (int)ia, fb, pol_a);
                        else
                            tma_load_3d(sa + q * a.a_sub, &tmA, q * a.wa, 0, (int)ia, fb);
                    }
                for (int q = 0; q < a.nb_sub; ++q) {
                    if (a.hint_b)
                        tma_load_3d_hint(sb + q * a.b_sub, &tmB, q * a.wb, 0, (int)ib, fb, pol_b);
                    else
                        tma_load_3d(sb + q * a.b_sub, &tmB, q * a.wb, 0, (int)ib, fb);
                }
            }
            __syncwarp();
            ++mine;
        }
        if (lane == 0) misc[4 + warp] = mine;
    } else if (warp == kProducers) {
        // ------------------------------------------------------------ MMA
        // Fills in order; per pair its slot's columns and its A source from
        // the pair words; a stage's empty barrier is committed after the last
        // fill whose pairs read an A tile in it.
        uint32_t aoff[KSTEPS], boff[KSTEPS];
#pragma unroll
        for (int kk = 0; kk < KSTEPS; ++kk) {
            aoff[kk] = (uint32_t)((kk >> a.a_lg) * a.a_sub16 + (kk & a.a_mask) * a.a_k16);
            boff[kk] = (uint32_t)((kk >> a.b_lg) * a.b_sub16 + (kk & a.b_mask) * a.b_k16);
        }
        const uint64_t adesc0 = a.a_desc0 + (sbase >> 4);
        const uint64_t bdesc0 = a.b_desc0 + ((sbase + (uint32_t)a.pps * a.a_pair) >> 4);
        const uint32_t stage16 = a.stage_bytes >> 4, apair16 = a.a_pair >> 4, bpair16 = a.b_pair >> 4;
        const uint32_t mb16 = (uint32_t)a.a_mb16, ncol = (uint32_t)a.N, idesc = a.idesc;
        const bool two_m = a.m_blocks > 1;
        const int n = (int)(pe - pb), pps = a.pps;
        uint32_t b = 0, aph = 0, dcol = tmem;
        int64_t s = s_first;
        int seg_end = n > 0 ? (int)((a.seg_start[s + 1] < pe ? a.seg_start[s + 1] : pe) - pb) : 0;
        bool fresh = true, ok = true;
        int pend[kMaxStages];
#pragma unroll
        for (int i = 0; i < kMaxStages; ++i) pend[i] = -1;
        auto open_seg = [&]() -> bool {
            if (!__all_sync(0xffffffffu, mbar_wait(acce0 + 8u * b, aph ^ 1u, abort_flag, a.status, a.wait_limit)))
                return false;
            tc_fence_after();
            dcol = tmem + b * buf_cols;
            fresh = false;
            return true;
        };
        auto close_seg = [&](int pos) {
            if (elect_one()) mma_commit(accf0 + 8u * b);
            __syncwarp();
            if (++b == (uint32_t)a.nacc) {
                b = 0;
                aph ^= 1u;
            }
            ++s;
            if (pos < n) seg_end = (int)((a.seg_start[s + 1] < pe ? a.seg_start[s + 1] : pe) - pb);
            fresh = true;
        };
        uint32_t st = 0, ph = 0, pmask = 0;   // pmask: stages whose release waits for a later fill
        int f = 0;
        for (; f * pps < n; ++f) {
            const int start = f * pps;
            const int np = n - start < pps ? n - start : pps;
            if (!__all_sync(0xffffffffu, mbar_wait(full0 + 8u * st, ph, abort_flag, a.status, a.wait_limit))) {
                ok = false;
                break;
            }
            tc_fence_after();
            uint32_t info[4];
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) info[jj] = jj < np ? pinfo[st * 4 + jj] : 0u;
            const int rel_st = prel[st];
            const uint64_t bd0 = bdesc0 + st * stage16;
            if (!fresh && start + np <= seg_end) {
                // the whole fill accumulates into the open window: one
                // elected region issues every pair and, unless a later pair
                // still reads an A tile here, releases the stage
                if (elect_one()) {
                    for (int jj = 0; jj < np; ++jj) {
                        const uint32_t d = dcol + (info[jj] & 0xFFu) * acc_cols;
                        const uint64_t ad = adesc0 + ((info[jj] >> 8) & 0xFFu) * stage16 +
                                            ((info[jj] >> 16) & 0xFFu) * apair16;
                        const uint64_t bd = bd0 + (uint32_t)jj * bpair16;
#pragma unroll
                        for (int kk = 0; kk < KSTEPS; ++kk) {
                            mma_bf16(d, ad + aoff[kk], bd + boff[kk], idesc, 1u);
                            if (two_m) mma_bf16(d + ncol, ad + aoff[kk] + mb16, bd + boff[kk], idesc, 1u);
                        }
                    }
                    if (rel_st == f) mma_commit(empty0 + 8u * st);
                }
                __syncwarp();
                if (start + np == seg_end) close_seg(seg_end);
            } else {
                // window boundaries inside the fill: pair by pair
                for (int jj = 0; jj < np; ++jj) {
                    if (fresh && !open_seg()) {
                        ok = false;
                        break;
                    }
                    const uint32_t d = dcol + (info[jj] & 0xFFu) * acc_cols;
                    const uint64_t ad = adesc0 + ((info[jj] >> 8) & 0xFFu) * stage16 +
                                        ((info[jj] >> 16) & 0xFFu) * apair16;
                    const uint64_t bd = bd0 + (uint32_t)jj * bpair16;
                    if (elect_one()) {
#pragma unroll
                        for (int kk = 0; kk < KSTEPS; ++kk) {
                            mma_bf16(d, ad + aoff[kk], bd + boff[kk], idesc, 1u);
                            if (two_m) mma_bf16(d + ncol, ad + aoff[kk] + mb16, bd + boff[kk], idesc, 1u);
                        }
                    }
                    __syncwarp();
                    if (start + jj + 1 == seg_end) close_seg(start + jj + 1);
                }
                if (!ok) break;
                if (rel_st == f) {
                    if (elect_one()) mma_commit(empty0 + 8u * st);
                    __syncwarp();
                }
            }
            if (rel_st != f) {
                // a later pair reads an A tile loaded here: release after that fill
#pragma unroll
                for (int i = 0; i < kMaxStages; ++i)   // constant indices: pend stays in registers
                    if (i == (int)st) pend[i] = rel_st;
                pmask |= 1u << st;
            }
            if (pmask) {
#pragma unroll
                for (int i = 0; i < kMaxStages; ++i)
                    if (((pmask >> i) & 1u) && pend[i] == f) {
                        if (elect_one()) mma_commit(empty0 + 8u * i);
                        __syncwarp();
                        pmask &= ~(1u << i);
                    }
            }
            if (++st == (uint32_t)a.ns) {
                st = 0;
                ph ^= 1u;
            }
        }
        // segments that end after the last stage (none unless a wait gave up)
        while (ok && s <= s_last) {
            if (fresh && !open_seg()) {
                ok = false;
                break;
            }
            close_seg(seg_end);
        }
        if (lane == 0) misc[2] = ok ? 0xFFFFFFFFu : (uint32_t)f;
    } else if (warp >= kProducers + kMmaWarps) {
        // ------------------------------------------------------- epilogue
        const int q4 = warp & 3;
        const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
        uint32_t b = 0, ph = 0;
        for (int64_t s = s_first; s <= s_last; ++s) {
            const int64_t ss = a.seg_start[s], se = a.seg_start[s + 1];
            if (!__all_sync(0xffffffffu, mbar_wait(accf0 + 8u * b, ph, abort_flag, a.status, a.wait_limit))) break;
            tc_fence_after();
            const int kind = (ss >= pb && se <= pe) ? 0 : (ss < pb ? 1 : 2);
            const uint32_t mask = a.wmask[s];
            const int64_t base = a.wbase[s];
            float *part = a.partials + ((int64_t)unit * 2 + (kind == 1 ? 0 : 1)) * (int64_t)W * a.tile_w;
            for (int q = 0; q < W; ++q) {
                if (!((mask >> q) & 1u)) continue;   // nothing accumulated there; nobody reads it
                const int64_t row = base + __popc(mask & ((1u << q) - 1u));
                const uint32_t bcol = tmem + lane_base + b * buf_cols + (uint32_t)q * acc_cols;
                for (int mb = 0; mb < a.m_blocks; ++mb) {
                    const int64_t m = (int64_t)mb * 128 + q4 * 32 + lane;
                    for (int c = 0; c < a.N / 16; ++c) {
                        float v[16];
                        tmem_ld16(bcol + (uint32_t)(mb * a.N + c * 16), v);
                        const int64_t off = m * a.sWm + (int64_t)c * 16 * a.sWn;
                        if (kind == 0) {
#pragma unroll
                            for (int jj = 0; jj < 16; ++jj) v[jj] = epilogue(v[jj], a.epi, a.scale);
                        }
                        if (kind == 0 && a.dout == UCL_BF16) {
                            __nv_bfloat16 *o = reinterpret_cast<__nv_bfloat16 *>(a.out) + row * a.tile_w + off;
                            if (a.sWn == 1) {
                                uint32_t h[8];
#pragma unroll
                                for (int jj = 0; jj < 8; ++jj) {
                                    __nv_bfloat162 t = __floats2bfloat162_rn(v[2 * jj], v[2 * jj + 1]);
                                    h[jj] = *reinterpret_cast<uint32_t *>(&t);
                                }
                                uint4 *o4 = reinterpret_cast<uint4 *>(o);
                                o4[0] = make_uint4(h[0], h[1], h[2], h[3]);
                                o4[1] = make_uint4(h[4], h[5], h[6], h[7]);
                            } else {
#pragma unroll
                                for (int jj = 0; jj < 16; ++jj) o[jj * a.sWn] = __float2bfloat16_rn(v[jj]);
                            }
                        } else {
                            float *o = kind == 0 ? reinterpret_cast<float *>(a.out) + row * a.tile_w + off
                                                 : part + (int64_t)q * a.tile_w + off;
                            if (a.sWn == 1) {
                                float4 *o4 = reinterpret_cast<float4 *>(o);
#pragma unroll
                                for (int jj = 0; jj < 4; ++jj)
                                    o4[jj] = make_float4(v[4 * jj], v[4 * jj + 1], v[4 * jj + 2], v[4 * jj + 3]);
                            } else {
#pragma unroll
                                for (int jj = 0; jj < 16; ++jj) o[jj * a.sWn] = v[jj];
                            }
                        }
                    }
                }
            }
            for (uint32_t c = 0; c < buf_cols; c += 16) tmem_st16_zero(tmem + lane_base + b * buf_cols + c);
            asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(acce0 + 8u * b);
            if (++b == (uint32_t)a.nacc) {
                b = 0;
                ph ^= 1u;
            }
        }
    }

    // ---------------------------------------------------------- teardown
    __syncthreads();
    if (*abort_flag) {
        if (warp < kProducers && lane == 0) {
            // (the fills of this producer's stages, in fill order)
            for (uint32_t it = 0, k = 0; k < misc[4 + warp]; ++it) {
                if ((int)((it % (uint32_t)a.ns) % (uint32_t)kProducers) != warp) continue;
                ++k;
                if ((int)it == a.withhold_fill) continue;   // never copied: nothing in flight
                if (it >= misc[2]) mbar_drain(full0 + 8u * (it % a.ns), (it / a.ns) & 1u);
            }
        }
        if (warp == kProducers && lane == 0) {
            mma_commit(done_bar);
            mbar_drain(done_bar, 0);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == kProducers) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(a.tmem_cols)
                     : "memory");
    }
}

// ------------------------------------------------------------------- host

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
        else
            cudaGetLastError();
    });
    return fn;
}

// Operand geometry: the tile is [trows][tcols] row-major.  One stage holds a
// K chunk of it, [rows][cols] (all rows and a column range for K-major tiles,
// a row range for MN-major ones), fetched as cols / w boxes of {w, rows},
// each landing in its own swizzled sub-tile.
struct Operand {
    int trows, tcols, rows, cols, w, nsub;
    int cx, cy;   // box coordinate step per chunk
    uint32_t sub_bytes;
};

bool operand_geometry(int trows, int tcols, bool kmajor, int kc, Operand *op, std::string *why) {
    op->trows = trows;
    op->tcols = tcols;
    op->rows = kmajor ? trows : trows / kc;
    op->cols = kmajor ? tcols / kc : tcols;
    op->cx = kmajor ? op->cols : 0;
    op->cy = kmajor ? 0 : op->rows;
    const int rows = op->rows, cols = op->cols;
    if (rows < 16 || rows > 256 || rows % 16) {
        *why = "tile rows must be a multiple of 16 up to 256";
        return false;
    }
    if (!(cols == 16 || cols == 32 || (cols % 64 == 0 && cols <= 256))) {
        *why = "tile row length must be 16, 32 or a multiple of 64 elements";
        return false;
    }
    op->w = cols < 64 ? cols : 64;
    op->nsub = cols / op->w;
    uint32_t b = (uint32_t)rows * op->w * 2;
    op->sub_bytes = (b + 1023u) & ~1023u;
    return true;
}

struct TcGeometry {
    Operand A, B;
    uint32_t a_pair, b_pair, stage_bytes, pair_tx, smem_bytes, tmem_cols;
    int pps, ns, nacc, nmma, kc;
};

// Ring of stages: whole pairs (kc = 1) when at least four stages of one pair
// fit, else the fewest K chunks per pair that leave four.  With whole pairs, a
// stage holds pps pairs (1..4): the largest pps that keeps a stage within
// 72 KB and leaves at least four stages.
bool geometry(const TcPlan &tp, TcGeometry *g, std::string *why, int pps_override = 0, int ns_force = 0,
              int mma_force = 0) {
    const uint32_t bar_bytes = kBarBytes;
    const uint32_t avail = kSmemLimit - 1024 - bar_bytes;
    bool found = false;
    for (int kc = 1; kc <= 16 && tp.K / kc >= 16 && tp.K % kc == 0; kc *= 2) {
        // A: K-major tiles are [M][K], MN-major [K][M]; same for B with N
        if (!operand_geometry(tp.a_kmajor ? tp.M : tp.K, tp.a_kmajor ? tp.K : tp.M, tp.a_kmajor, kc, &g->A, why))
            continue;
        if (!operand_geometry(tp.b_kmajor ? tp.N : tp.K, tp.b_kmajor ? tp.K : tp.N, tp.b_kmajor, kc, &g->B, why))
            continue;
        g->a_pair = g->A.sub_bytes * g->A.nsub;
        g->b_pair = g->B.sub_bytes * g->B.nsub;
        if (avail / (g->a_pair + g->b_pair) >= 4) {
            g->kc = kc;
            found = true;
            break;
        }
    }
    if (!found) {
        if (why->empty()) *why = "tiles too large for four shared-memory stages";
        return false;
    }
    const int Kc = tp.K / g->kc;
    g->pair_tx = (uint32_t)(tp.M * Kc * 2 + tp.N * Kc * 2);
    const uint32_t per_pair = g->a_pair + g->b_pair;
    int pps = 1;
    if (g->kc == 1) {
        for (int c = 4; c >= 2; --c) {
            const uint32_t k = avail / (c * per_pair);
            if (c * per_pair <= 72u * 1024u && (k < (uint32_t)kMaxStages ? k : (uint32_t)kMaxStages) / 2 * 2 >= 4) {
                pps = c;
                break;
            }
        }
        if (pps_override > 0) pps = pps_override;
    }
    g->pps = pps;
    g->stage_bytes = pps * per_pair;
    int ns = (int)(avail / g->stage_bytes);
    if (ns > kMaxStages) ns = kMaxStages;
    if (ns < 2) {
        *why = "tiles too large for two shared-memory stages";
        return false;
    }
    const int acc_cols = tp.N * tp.m_blocks;
    // Two MMA warps (each with its own half accumulator) when two buffers of
    // two halves fit TMEM and the stage count is even.  MMA warp w takes the
    // stage fills w, w + 2, ...; the previous fill of a stage must belong to
    // the same warp, or a warp could wait on a stage's full barrier while the
    // other warp's older fill of that stage is still pending and the parity
    // test would pass a phase early.  An even ring guarantees it.  One MMA
    // warp consumes in order and is safe with any ring size.  The producers
    // take alternate fills too, and the same two cases keep their
    // empty-barrier waits exact: with an even ring every fill of a stage
    // comes from one producer, and one MMA warp releases stages in fill
    // order.  (Two MMA warps on an odd ring would release stages out of
    // order while consecutive fills of a stage come from different
    // producers, so a producer could pass a stage's empty barrier two phases
    // early.  Stage-owned producers fix that, but split an odd ring unevenly
    // between them and measured slower.)
    const bool two_fit = 512 / (2 * acc_cols) >= 2;
    if (ns_force > 0) {
        // a stage count chosen by the caller: two MMA warps only on an even ring
        if (ns > ns_force) ns = ns_force;
        g->nmma = two_fit && ns % 2 == 0 ? 2 : 1;
    } else if (two_fit && ns >= 5 && (ns & 1) && tp.m_blocks * (tp.K / g->kc) / 16 >= 8) {
        // an odd ring one stage deeper with one MMA warp: with at least eight
        // MMAs per pair one warp keeps up, and the extra stage hides more of
        // the copy latency (two-layer GNN message passing: 5 stages 51 ms
        // against 4 stages and two MMA warps 54 ms)
        g->nmma = 1;
    } else if (two_fit && ns >= 4) {
        ns &= ~1;
        g->nmma = 2;
    } else if (two_fit && ns == 2) {
        g->nmma = 2;
    } else {
        g->nmma = 1;
    }
    if (mma_force == 1) g->nmma = 1;   // caller's choice: one MMA warp (any ring)
    g->ns = ns;
    const int buf = acc_cols * g->nmma;
    g->nacc = 512 / buf < kMaxAcc ? 512 / buf : kMaxAcc;
    if (g->nacc < 1) {
        *why = "accumulator does not fit TMEM";
        return false;
    }
    uint32_t need = (uint32_t)(g->nacc * buf), cols = 32;
    while (cols < need) cols <<= 1;
    g->tmem_cols = cols;
    g->smem_bytes = 1024 + ns * g->stage_bytes + bar_bytes;
    return true;
}

// Shared-memory matrix descriptor of tcgen05 with the start address left 0:
// leading / stride byte offsets, fixed version 1 (bits 46-47), swizzle mode
// (bits 61-63: 2 = 128B, 4 = 64B, 6 = 32B).
uint64_t desc_template(const Operand &op, bool kmajor) {
    const uint64_t sbo = 8ull * op.w * 2;   // next group of 8 rows
    const uint64_t lbo = kmajor ? 16 : op.sub_bytes;   // MN-major: next swizzle atom along M / N
    const uint64_t layout = op.w == 64 ? 2 : (op.w == 32 ? 4 : 6);
    return ((lbo >> 4) << 16) | ((sbo >> 4) << 32) | (1ull << 46) | (layout << 61);
}

// Offsets (16-byte units) of K step kk: K-major tiles advance 32 bytes inside
// a swizzle row and jump to the next box every w/16 steps; MN-major tiles
// advance 16 rows.
void kstep_offsets(const Operand &op, bool kmajor, int *lg, int *mask, int *sub16, int *k16) {
    if (kmajor) {
        const int steps = op.w / 16;   // 1, 2 or 4
        *lg = steps == 4 ? 2 : (steps == 2 ? 1 : 0);
        *mask = steps - 1;
        *sub16 = (int)(op.sub_bytes >> 4);
        *k16 = 2;
    } else {
        *lg = 16;   // kk < 16: never reaches the next box
        *mask = 0xFFFF;
        *sub16 = 0;
        *k16 = 2 * op.w;   // 16 rows of w * 2 bytes
    }
}

bool make_map(CUtensorMap *m, const ucl_rel *R, const Operand &op, std::string *why) {
    auto enc = encode_fn();
    if (!enc) {
        *why = "cuTensorMapEncodeTiled unavailable";
        return false;
    }
    cuuint64_t dims[3] = {(cuuint64_t)op.tcols, (cuuint64_t)op.trows, (cuuint64_t)R->n};
    cuuint64_t strides[2] = {(cuuint64_t)op.tcols * 2, (cuuint64_t)op.trows * op.tcols * 2};
    cuuint32_t box[3] = {(cuuint32_t)op.w, (cuuint32_t)op.rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUtensorMapSwizzle swz = op.w == 64 ? CU_TENSOR_MAP_SWIZZLE_128B
                                        : (op.w == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B);
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, R->tiles, dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        *why = "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")";
        return false;
    }
    return true;
}

// Geometry of the windowed kernel: whole pairs, one MMA warp (any ring
// size), buffers of 2^win_bits accumulator slots, and the longest run of
// pairs one loaded A tile may serve: a stage is then held at most ns - 2
// fills past its own, so the producers never wait on a stage that a pair
// still to be filled needs.
bool window_geometry(const TcPlan &tp, int win_bits, TcGeometry *g, int *cap, std::string *why) {
    if (!geometry(tp, g, why)) return false;
    if (g->kc != 1) {
        *why = "windows need whole pairs per stage";
        return false;
    }
    int ns = (int)((kSmemLimit - 1024 - kBarBytes) / g->stage_bytes);
    if (ns > kMaxStages) ns = kMaxStages;
    if (ns < 3) {
        *why = "windows need at least three stages";
        return false;
    }
    g->ns = ns;
    g->nmma = 1;
    const int buf = tp.N * tp.m_blocks << win_bits;
    g->nacc = 512 / buf < kMaxAcc ? 512 / buf : kMaxAcc;
    if (g->nacc < 1) {
        *why = "window accumulators do not fit TMEM";
        return false;
    }
    uint32_t need = (uint32_t)(g->nacc * buf), cols = 32;
    while (cols < need) cols <<= 1;
    g->tmem_cols = cols;
    g->smem_bytes = 1024 + ns * g->stage_bytes + kBarBytes;
    int c = (ns - 2) * g->pps + 1;
    *cap = c < 1 ? 1 : (c > 15 ? 15 : c);
    if (const char *e = getenv("UCL_WINDOW_SHARE"))   // measurement: 0 turns A-tile sharing off
        if (atoi(e) == 0) *cap = 1;
    return true;
}

}  // namespace

int tc_window_cap(const TcPlan &tp, int win_bits) {
    TcGeometry g;
    std::string why;
    int cap = 0;
    return window_geometry(tp, win_bits, &g, &cap, &why) ? cap : 0;
}

bool tc_supported(const TcPlan &tp, const ContractArgs &a, std::string *why) {
    TcGeometry g;
    if (!geometry(tp, &g, why)) return false;
    const void *pa = tp.a_is_u ? a.U : a.V, *pb = tp.a_is_u ? a.V : a.U;
    if ((reinterpret_cast<uintptr_t>(pa) | reinterpret_cast<uintptr_t>(pb)) & 15) {
        *why = "tile arrays not 16-byte aligned";
        return false;
    }
    if (!encode_fn()) {
        *why = "cuTensorMapEncodeTiled unavailable";
        return false;
    }
    return true;
}

int tc_units(ucl_ctx *ctx, const TcPlan &, int64_t P) { return (int)(P < ctx->sm_count ? P : ctx->sm_count); }

ucl_status launch_contract_tc(ucl_ctx *ctx, const ContractArgs &a, const TcPlan &tp, const ucl_rel *ra,
                              const ucl_rel *rb) {
    TcGeometry g;
    std::string why;
    int cap = 0;
    if (a.win_bits > 0) {
        if (!window_geometry(tp, a.win_bits, &g, &cap, &why)) return fail(ctx, UCL_ERR_UNSUPPORTED, "tcgen05 path: " + why);
        if (cap != a.share_cap) return fail(ctx, UCL_ERR_UNSUPPORTED, "tcgen05 path: run cap disagrees with the key stage");
    } else if (!geometry(tp, &g, &why, 0, ctx->tune_tc_stages, ctx->tune_tc_mma)) {
        return fail(ctx, UCL_ERR_UNSUPPORTED, "tcgen05 path: " + why);
    }
    CUtensorMap mA, mB;
    if (!make_map(&mA, ra, g.A, &why) || !make_map(&mB, rb, g.B, &why))
        return fail(ctx, UCL_ERR_CUDA, "tcgen05 path: " + why);
    TcArgs k{};
    k.pa = tp.a_is_u ? a.pu : a.pv;
    k.pb = tp.a_is_u ? a.pv : a.pu;
    k.nA = ra->n;
    k.nB = rb->n;
    k.seg_start = a.seg_start;
    k.S = a.S;
    k.units = a.units;
    k.out = a.out;
    k.dout = a.dout;
    k.epi = a.epi;
    k.scale = a.scale;
    k.partials = a.partials;
    k.tile_w = a.tile_w;
    k.sWm = tp.sWm;
    k.sWn = tp.sWn;
    k.N = tp.N;
    k.K = tp.K;
    k.m_blocks = tp.m_blocks;
    k.kc_lg = g.kc == 1 ? 0 : (g.kc == 2 ? 1 : (g.kc == 4 ? 2 : (g.kc == 8 ? 3 : 4)));
    k.a_cx = g.A.cx;
    k.a_cy = g.A.cy;
    k.b_cx = g.B.cx;
    k.b_cy = g.B.cy;
    k.wa = g.A.w;
    k.wb = g.B.w;
    k.na_sub = g.A.nsub;
    k.nb_sub = g.B.nsub;
    k.a_sub = g.A.sub_bytes;
    k.b_sub = g.B.sub_bytes;
    k.a_pair = g.a_pair;
    k.b_pair = g.b_pair;
    k.stage_bytes = g.stage_bytes;
    k.pair_tx = g.pair_tx;
    k.pps = g.pps;
    k.ns = g.ns;
    k.nacc = g.nacc;
    k.nmma = g.nmma;
    // Prefetch into L2 the tiles of a streamed operand -- one too large to stay
    // in L2 (more than a quarter of it) whose tiles are each joined about once
    // (at least half as many tuples as pairs) -- when the other operand does
    // stay in L2.  Its tiles then come from HBM while the other's hit L2, and
    // a prefetch two own fills (four stages) ahead hides that latency without
    // shared memory (message passing: 0.618 -> 0.596 ms).  When both operands
    // stream (the 256-wide embeddings of the two-layer GNN) it gains nothing,
    // and prefetching a large reused operand evicts more than it saves.
    {
        int l2 = 0;
        if (cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, ctx->device) != cudaSuccess) {
            cudaGetLastError();
            l2 = 0;
        }
        const double big = l2 > 0 ? l2 / 4.0 : 32.0 * (1 << 20);
        // a banded launch covers one band: about 1 / bands of each input's tuples
        const double band = a.bands > 1 ? (double)a.bands : 1.0;
        const double na = ra->n / band, nb = rb->n / band;
        const double bytes_a = na * tp.M * tp.K * 2, bytes_b = nb * tp.N * tp.K * 2;
        const double P = (double)a.units.P;
        k.pf_a = g.kc == 1 && bytes_a > big && 2 * na >= P && bytes_b <= big;
        k.pf_b = g.kc == 1 && bytes_b > big && 2 * nb >= P && bytes_a <= big;
        if (ctx->tune_tc_prefetch >= 0) {
            // caller's choice: prefetch whichever operand is streamed (or none)
            const bool on = ctx->tune_tc_prefetch > 0 && g.kc == 1;
            k.pf_a = on && bytes_a > big && 2 * na >= P;
            k.pf_b = on && bytes_b > big && 2 * nb >= P;
        }
        k.pf_dist = 2;
        // L2 eviction hints: a streamed operand (each tuple joined about once,
        // larger than a quarter of L2) is evicted first, so that the reused
        // operand (joined at least four times per tuple) stays; that one is
        // evicted last
        k.hint_a = k.hint_b = 0;
        if (a.l2_hints) {
            const bool stream_a = bytes_a > big && 2 * na >= P, stream_b = bytes_b > big && 2 * nb >= P;
            if (stream_a && !stream_b) {
                k.hint_a = 1;
                if (P >= 4 * nb) k.hint_b = 2;
            } else if (stream_b && !stream_a) {
                k.hint_b = 1;
                if (P >= 4 * na) k.hint_a = 2;
            }
        }
    }
    k.tmem_cols = g.tmem_cols;
    // instruction descriptor, kind::f16: D fp32 (bits 4-5), A and B bf16 (7-9, 10-12),
    // A / B major (15, 16: 1 = MN-major), N >> 3 (17-22), M >> 4 (24-28), M = 128 per MMA
    k.idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(tp.a_kmajor ? 0 : 1) << 15) |
              ((uint32_t)(tp.b_kmajor ? 0 : 1) << 16) | ((uint32_t)(tp.N >> 3) << 17) | ((128u >> 4) << 24);
    k.a_desc0 = desc_template(g.A, tp.a_kmajor);
    k.b_desc0 = desc_template(g.B, tp.b_kmajor);
    kstep_offsets(g.A, tp.a_kmajor, &k.a_lg, &k.a_mask, &k.a_sub16, &k.a_k16);
    kstep_offsets(g.B, tp.b_kmajor, &k.b_lg, &k.b_mask, &k.b_sub16, &k.b_k16);
    // second M block: 128 rows further (K-major) or 128 / w swizzle atoms further (MN-major)
    k.a_mb16 = tp.a_kmajor ? (int)((128u * g.A.w * 2) >> 4) : (int)((128 / g.A.w) * (g.A.sub_bytes >> 4));
    k.status = ctx->d_status + 2;
    k.wait_limit = ctx->wait_limit_cycles > 0 ? ctx->wait_limit_cycles : kWaitLimitCycles;
    k.withhold_fill = ctx->withhold_fill;
    ctx->withhold_fill = -1;   // one launch only
    k.win_bits = a.win_bits;
    k.slot = a.slot;
    k.arun = a.arun;
    k.wmask = a.wmask;
    k.wbase = a.wbase;
    k.share_cap = cap;
    void (*kern)(const CUtensorMap, const CUtensorMap, const TcArgs) = nullptr;
    const bool win = a.win_bits > 0;
    switch (tp.K / g.kc / 16) {
        case 1: kern = win ? tc_window_kernel<1> : tc_contract_kernel<1>; break;
        case 2: kern = win ? tc_window_kernel<2> : tc_contract_kernel<2>; break;
        case 4: kern = win ? tc_window_kernel<4> : tc_contract_kernel<4>; break;
        case 8: kern = win ? tc_window_kernel<8> : tc_contract_kernel<8>; break;
        case 16: kern = win ? tc_window_kernel<16> : tc_contract_kernel<16>; break;
        default: return fail(ctx, UCL_ERR_UNSUPPORTED, "tcgen05 path: K must be 16, 32, 64, 128 or 256");
    }
    ucl_status st = cuda_check(
        ctx, cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)g.smem_bytes),
        "cudaFuncSetAttribute");
    if (st) return st;
    kern<<<a.units.G, kTcThreads, g.smem_bytes, ctx->stream>>>(mA, mB, k);
    ctx->launches++;
    return cuda_check(ctx, cudaGetLastError(), "tcgen05 kernel launch");
}

}  // namespace ucl
