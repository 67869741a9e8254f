// contract_tc3.cu -- tcgen05 contraction of a three-way star join of the
// MTTKRP shape, with the group-by sum fused into its epilogue:
//
//     W[i][r] = sum over joined triples (t, e, f) of one output key of
//               sum_{j,k} T_t[i][j][k] * E_e[j][r] * F_f[k][r]
//
// (paper Sec. 5's template with three relations; T sparse, E and F dense
// factor tiles).  Per triple the k contraction is a GEMM on the tensor
// cores and the j contraction a Hadamard product with E done by the epilogue
// warps:
//
//     P[r][(i, j)] = sum_k F[k][r] * T[(i, j)][k]          (tcgen05.mma)
//     W[i][r]     += sum_j E[j][r] * P[r][(i, j)]           (epilogue FMAs)
//
// With r = 64 rows the MMA would be M = 64; instead the two halves of i are
// stacked on the M axis: M row (x, r), x = i / 8, and two MMAs per triple
// whose A operands are F^T placed in block x of an otherwise zero 128-row
// matrix (the zero blocks sit around each F slot in shared memory, written
// once).  D then holds P[x*64 + r][(i mod 8, j)] in 128 TMEM lanes x 128
// columns, so each epilogue thread owns one (x, r) row and reduces over j in
// registers, without shuffles.
//
// Consecutive triples of one output key that share the E tuple (the pair
// list is ordered by output key, then by the first join's key) accumulate in
// the same TMEM buffer, so the epilogue runs once per such group, not per
// triple.
//
//   warp 0      TMA producer: T tile (16 x 256 rows, 32B swizzle) and F tile
//               (64 x 16 rows, 128B swizzle) of each triple into a ring of
//               stages of `pps` triples;
//   warp 6      group warp: per stage, which triples open a group, close one
//               or end an output key; for each group opening there it waits
//               until the epilogue has released the group's accumulator
//               buffer and requests the group's E tile by TMA into that
//               buffer's E slot; for each group closing there it posts to the
//               epilogue whether the group ends its output key; then it posts
//               the stage's plan;
//   warp 1      MMA issuer (owns TMEM): one thread issues two tcgen05.mma per
//               triple into the group's accumulator buffer, following the
//               plan, and commits a group's buffer after its last triple;
//   warps 2-5   epilogue: per group, load E's 16 values for its r, drain the
//               group's accumulator and fold it into 8 fp32 registers; at the
//               end of an output key, store the output tile (or a partial for
//               the fixup kernel when the key straddles two work units).
//
// Keeping the group bookkeeping (buffer waits, E requests) out of both the
// producer and the issuing thread lets the copies run a full ring ahead and
// leaves the issuing thread only stage waits, MMAs and commits.  The
// epilogue never searches the pair list nor waits on a global load.

// Every mbarrier wait is bounded; on expiry the CTA raises kStTimeout, all
// roles leave their loops, in-flight copies and MMAs are drained (bounded),
// TMEM is freed and the kernel returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "internal.cuh"

namespace ucl {

namespace {

constexpr int kThreads3 = 32 * 7;            // producer, MMA, 4 epilogue warps, group warp
constexpr long long kWait3 = 2500000000ll;   // ~1.2 s at 2.07 GHz
constexpr int kPps3 = 4;                     // triples per stage
constexpr int kStages3 = 4;
constexpr int kAcc3 = 4;                     // TMEM accumulator buffers of 128 columns
constexpr uint32_t kTBytes = 256 * 16 * 2;   // T tile: 256 rows (i, j) x 16 k, bf16
constexpr uint32_t kFBytes = 16 * 64 * 2;    // F tile: 16 rows k x 64 r, bf16
// stage: pps T tiles, then Z F0 Z F1 Z ... F(pps-1) Z (Z = zero block of kFBytes)
constexpr uint32_t kFRegion = (2 * kPps3 + 1) * kFBytes;
constexpr uint32_t kStageBytes = kPps3 * kTBytes + kFRegion;
constexpr uint32_t kEBytes = 16 * 64 * 2;    // E tile: 16 j x 64 r, bf16, one slot per accumulator buffer
// barriers: full, empty (per stage); accf, acce, ef, infoc (per buffer); done
constexpr uint32_t kBarBytes =
    8 * (3 * kStages3 + 4 * kAcc3 + 1) + 64 + 8 * kAcc3 + 4 * kStages3 * (kPps3 + 1);
constexpr uint32_t kSmem3 = 1024 + kStages3 * kStageBytes + kAcc3 * kEBytes + kBarBytes;
static_assert(kStageBytes % 1024 == 0, "stages must keep 1024-byte alignment");
static_assert(kSmem3 <= 227 * 1024, "shared memory budget");

struct Tc3Args {
    const uint32_t *idx_t, *idx_e, *idx_f;   // [P] T, E, F tuple of each triple
    int64_t nT, nE, nF;
    int64_t sEj, sEr;               // E tile strides of j and r
    const int64_t *seg_start;
    int64_t S;
    Units units;
    void *out;
    int dout, epi;
    float scale;
    float *partials;
    int64_t tile_w, sWi, sWr;
    uint32_t idesc;
    uint64_t a_desc0, b_desc0;      // start address field 0
    int t_mn;                       // T tiles [k][(i, j)]: four 64-column boxes of 16 rows (else one box of 256 rows)
    uint32_t *status;
};

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

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

// Bounded wait (see the binary kernel): false when another role aborted or
// the limit passed (then this thread raises the abort and kStTimeout).
__device__ __noinline__ bool wait3(uint32_t bar, uint32_t parity, volatile uint32_t *abort_flag, uint32_t *status) {
    const long long t0 = clock64();
    for (;;) {
        if (mbar_try_sleep(bar, parity, 100000u)) return true;
        if (*abort_flag) return false;
        if (clock64() - t0 > kWait3) {
            *abort_flag = 1;
            atomicOr(status, kStTimeout);
            return false;
        }
    }
}

__device__ __forceinline__ bool try3(uint32_t bar, uint32_t parity) {
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

// Bounded wait with an inline first attempt.
__device__ __forceinline__ bool wait3f(uint32_t bar, uint32_t parity, volatile uint32_t *abort_flag,
                                       uint32_t *status) {
    return try3(bar, parity) || wait3(bar, parity, abort_flag, status);
}

__device__ __noinline__ void drain3(uint32_t bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!mbar_try_sleep(bar, parity, 100000u))
        if (clock64() - t0 > kWait3) return;
}

__device__ __forceinline__ void arrive_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void tma3d(uint32_t dst, const CUtensorMap *map, int z, uint32_t bar, int x = 0) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
        "[%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(0), "r"(z), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void mma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}

__device__ __forceinline__ void commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 128 consecutive TMEM columns of this thread's lane, one load; the wait sits
// in the same asm statement, so no use of the outputs is scheduled before it.
__device__ __forceinline__ void tmem_ld128(uint32_t taddr, uint32_t *r) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x128.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63, %64, %65, %66, %67, %68, %69, %70, %71, %72, %73, %74, %75, %76, %77, %78, %79, %80, %81, %82, %83, %84, %85, %86, %87, %88, %89, %90, %91, %92, %93, %94, %95, %96, %97, %98, %99, %100, %101, %102, %103, %104, %105, %106, %107, %108, %109, %110, %111, %112, %113, %114, %115, %116, %117, %118, %119, %120, %121, %122, %123, %124, %125, %126, %127}, [%128];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63]), "=r"(r[64]), "=r"(r[65]), "=r"(r[66]), "=r"(r[67]), "=r"(r[68]), "=r"(r[69]), "=r"(r[70]), "=r"(r[71]), "=r"(r[72]), "=r"(r[73]), "=r"(r[74]), "=r"(r[75]), "=r"(r[76]), "=r"(r[77]), "=r"(r[78]), "=r"(r[79]), "=r"(r[80]), "=r"(r[81]), "=r"(r[82]), "=r"(r[83]), "=r"(r[84]), "=r"(r[85]), "=r"(r[86]), "=r"(r[87]), "=r"(r[88]), "=r"(r[89]), "=r"(r[90]), "=r"(r[91]), "=r"(r[92]), "=r"(r[93]), "=r"(r[94]), "=r"(r[95]), "=r"(r[96]), "=r"(r[97]), "=r"(r[98]), "=r"(r[99]), "=r"(r[100]), "=r"(r[101]), "=r"(r[102]), "=r"(r[103]), "=r"(r[104]), "=r"(r[105]), "=r"(r[106]), "=r"(r[107]), "=r"(r[108]), "=r"(r[109]), "=r"(r[110]), "=r"(r[111]), "=r"(r[112]), "=r"(r[113]), "=r"(r[114]), "=r"(r[115]), "=r"(r[116]), "=r"(r[117]), "=r"(r[118]), "=r"(r[119]), "=r"(r[120]), "=r"(r[121]), "=r"(r[122]), "=r"(r[123]), "=r"(r[124]), "=r"(r[125]), "=r"(r[126]), "=r"(r[127])
        : "r"(taddr)
        : "memory");
}

__device__ __forceinline__ int64_t seg_of(const int64_t *seg_start, int64_t S, int64_t p) {
    int64_t a = 0, b = S;
    while (a < b) {
        int64_t mid = (a + b) >> 1;
        if (seg_start[mid] <= p) a = mid + 1; else b = mid;
    }
    return a - 1;
}

__device__ __forceinline__ float epi3(float x, int epi, float scale) {
    x *= scale;
    if (epi == UCL_EPI_RELU) x = fmaxf(x, 0.0f);
    return x;
}

__global__ void __launch_bounds__(kThreads3, 1)
    tc3_contract_kernel(const __grid_constant__ CUtensorMap tmT, const __grid_constant__ CUtensorMap tmF,
                        const __grid_constant__ CUtensorMap tmE, const Tc3Args a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const uint32_t sbase = smem_u32(smem);
    // E slot of buffer b: the group's E tile, fetched by TMA when the group
    // warp opens the group (ef[b]), read by the epilogue before it frees the buffer
    const __nv_bfloat16 *eslots = reinterpret_cast<const __nv_bfloat16 *>(smem + (size_t)kStages3 * kStageBytes);
    const uint32_t eslot0 = sbase + kStages3 * kStageBytes;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + (size_t)kStages3 * kStageBytes + kAcc3 * kEBytes);
    const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8u * kStages3, accf0 = empty0 + 8u * kStages3,
                   acce0 = accf0 + 8u * kAcc3, done_bar = acce0 + 8u * kAcc3, ef0 = done_bar + 8u,
                   infoc0 = ef0 + 8u * kAcc3, planned0 = infoc0 + 8u * kAcc3;
    uint32_t *misc = reinterpret_cast<uint32_t *>(bars + 3 * kStages3 + 4 * kAcc3 + 1);
    // misc[0] TMEM base, [1] abort flag, [2] stage fills the MMA warp consumed,
    // [3] stage fills the producer issued, [4] E tiles requested, [5] E tiles
    // the epilogue received
    volatile uint32_t *abort_flag = misc + 1;
    // per accumulator buffer: [2b + 1] 1 if the group ends its output key
    // (posted at close through infoc[b])
    volatile uint32_t *info = misc + 16;
    // per stage: a word whose bit j marks triple j as opening a group, bit
    // 8 + j its group as ending the output key and bit 16 + j its group as
    // closing after it (written by the group warp before planned[st])
    volatile uint32_t *plan = info + 2 * kAcc3;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // zero blocks around the F slots: written once, read by every MMA
    for (int st = 0; st < kStages3; ++st)
        for (int z = 0; z <= kPps3; ++z) {
            uint4 *blk = reinterpret_cast<uint4 *>(smem + st * kStageBytes + kPps3 * kTBytes + 2 * z * kFBytes);
            for (int i = threadIdx.x; i < (int)(kFBytes / 16); i += kThreads3) blk[i] = make_uint4(0, 0, 0, 0);
        }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages3; ++i) {
            mbar_init(full0 + 8u * i, 1);
            mbar_init(empty0 + 8u * i, 1);
        }
        for (int i = 0; i < kAcc3; ++i) {
            mbar_init(accf0 + 8u * i, 1);
            mbar_init(acce0 + 8u * i, 4);
        }
        mbar_init(done_bar, 1);
        for (int i = 0; i < kAcc3; ++i) {
            mbar_init(ef0 + 8u * i, 1);
            mbar_init(infoc0 + 8u * i, 1);
        }
        for (int i = 0; i < kStages3; ++i) mbar_init(planned0 + 8u * i, 1);
        for (int i = 1; i < 16; ++i) misc[i] = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(misc)),
                     "r"(512)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem = misc[0];

    const int unit = blockIdx.x;
    const int64_t pb = a.units.begin(unit), pe = a.units.begin(unit + 1);
    const int n = (int)(pe - pb);
    const int64_t s_first = n > 0 ? seg_of(a.seg_start, a.S, pb) : 0;

    if (warp == 0) {
        // ------------------------------------------------------- producer
        // Copies only: lane j < pps handles triple j of each stage (indices
        // loaded one stage ahead, checked when used) and issues its T and F
        // copies.  The group
        // plan of a stage is posted separately by the group warp.
        const int nfills = (n + kPps3 - 1) / kPps3;
        auto load_idx = [&](int f, uint32_t &it, uint32_t &iff) {
            it = 0;
            iff = 0;
            const int64_t p = pb + (int64_t)f * kPps3 + lane;
            if (f < nfills && lane < kPps3 && p < pe) {
                it = a.idx_t[p];
                iff = a.idx_f[p];
            }
        };
        uint32_t it, iff;
        load_idx(0, it, iff);
        uint32_t st = 0, ph = 0, mine = 0;
        for (int f = 0; f < nfills; ++f) {
            uint32_t nit, niff;
            load_idx(f + 1, nit, niff);
            // indices are checked when used, a stage after their load, so the
            // next stage's loads stay in flight meanwhile
            if ((int64_t)it >= a.nT || (int64_t)iff >= a.nF) {
                atomicOr(a.status, kStBadIndex);
                it = 0;
                iff = 0;
            }
            const int start = f * kPps3;
            const int np = n - start < kPps3 ? n - start : kPps3;
            uint32_t okw = 1;
            if (lane == 0) {
                okw = wait3f(empty0 + 8u * st, ph ^ 1u, abort_flag, a.status) ? 1u : 0u;
                if (okw) arrive_tx(full0 + 8u * st, (uint32_t)np * (kTBytes + kFBytes));
            }
            if (!__shfl_sync(0xffffffffu, okw, 0)) break;
            if (lane < np) {
                const uint32_t fb = full0 + 8u * st, s0 = sbase + st * kStageBytes;
                if (a.t_mn) {
                    // [k][(i, j)]: 16 rows of 512 bytes as four 128-byte-wide
                    // boxes, each its own 2 KB 128B-swizzled sub-tile
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        tma3d(s0 + (uint32_t)lane * kTBytes + (uint32_t)q * (kTBytes / 4), &tmT, (int)it, fb, 64 * q);
                } else {
                    tma3d(s0 + (uint32_t)lane * kTBytes, &tmT, (int)it, fb);
                }
                tma3d(s0 + kPps3 * kTBytes + (2u * lane + 1u) * kFBytes, &tmF, (int)iff, fb);
            }
            __syncwarp();
            ++mine;
            it = nit;
            iff = niff;
            if (++st == (uint32_t)kStages3) {
                st = 0;
                ph ^= 1u;
            }
        }
        if (lane == 0) misc[3] = mine;
    } else if (warp == 6) {
        // ---------------------------------------------------- group warp
        // For each stage, in order: which triples open a group (the E tuple
        // changes, or a segment starts), close one, end an output key; for
        // each group opening there, wait until the epilogue has released the
        // group's accumulator buffer and request its E tile; then post the
        // plan (planned[st]).  It waits for the stage's previous fill to be
        // consumed (empty) so that the plan word is free.  No wait here can
        // deadlock: a stage holds at most four triples, so the group whose
        // buffer a new group reuses (four groups back) closed in an earlier,
        // already planned stage.
        const int nfills = (n + kPps3 - 1) / kPps3;
        auto load_e = [&](int f) -> uint32_t {
            const int64_t p = pb + (int64_t)f * kPps3 + lane;
            return (f < nfills && lane < kPps3 && p < pe) ? a.idx_e[p] : 0u;
        };
        // E tuples of this stage and the next (loaded a stage earlier, so that
        // the next stage's first one is read without waiting on a load)
        uint32_t ie = load_e(0), nie = load_e(1);
        uint32_t st = 0, ph = 0, e_last = 0, gb = 0, gph = 0, opened = 0, cb = 0;
        int64_t s = s_first;
        int seg_end = n > 0 ? (int)((a.seg_start[s + 1] < pe ? a.seg_start[s + 1] : pe) - pb) : 0;
        for (int f = 0; f < nfills; ++f) {
            const uint32_t nnie = load_e(f + 2);
            const int start = f * kPps3;
            const int np = n - start < kPps3 ? n - start : kPps3;
            // segment starts inside this stage (uniform; rare)
            uint32_t brk = 0;
            while (seg_end < start + np) {
                brk |= 1u << (seg_end - start);
                ++s;
                seg_end = (int)((a.seg_start[s + 1] < pe ? a.seg_start[s + 1] : pe) - pb);
            }
            // a segment (or the unit) ends right after this stage's last triple
            const bool ends_after = seg_end == start + np;
            const uint32_t eup = __shfl_up_sync(0xffffffffu, ie, 1);
            const uint32_t eprev = lane == 0 ? e_last : eup;
            const bool newg = lane < np && (start + lane == 0 || ie != eprev || ((brk >> lane) & 1u));
            const uint32_t gmask = __ballot_sync(0xffffffffu, newg) & 0xFu;
            e_last = __shfl_sync(0xffffffffu, ie, np - 1);
            const uint32_t e_next = __shfl_sync(0xffffffffu, nie, 0);
            // close flags: triple j ends its group when triple j + 1 opens one;
            // the last triple when the next stage's first does (or the unit ends)
            const uint32_t below = (1u << (np - 1)) - 1u;
            const bool last_unit = start + np == n;
            const bool next_new = last_unit || ends_after || e_next != e_last;
            const uint32_t cmask = ((gmask >> 1) & below) | ((next_new ? 1u : 0u) << (np - 1));
            const uint32_t emask = ((brk >> 1) & below) | ((last_unit || ends_after ? 1u : 0u) << (np - 1));
            uint32_t e4[kPps3];
#pragma unroll
            for (int j = 0; j < kPps3; ++j) e4[j] = __shfl_sync(0xffffffffu, ie, j);
            uint32_t okw = 1;
            if (lane == 0) {
                okw = wait3f(empty0 + 8u * st, ph ^ 1u, abort_flag, a.status) ? 1u : 0u;
                for (int j = 0; j < np && okw; ++j) {
                    if ((gmask >> j) & 1u) {
                        if (!wait3f(acce0 + 8u * gb, gph ^ 1u, abort_flag, a.status)) {
                            okw = 0;
                            break;
                        }
                        uint32_t ei = e4[j];
                        if ((int64_t)ei >= a.nE) {
                            atomicOr(a.status, kStBadIndex);
                            ei = 0;
                        }
                        arrive_tx(ef0 + 8u * gb, kEBytes);
                        tma3d(eslot0 + gb * kEBytes, &tmE, (int)ei, ef0 + 8u * gb);
                        ++opened;
                        if (++gb == (uint32_t)kAcc3) {
                            gb = 0;
                            gph ^= 1u;
                        }
                    }
                    if ((cmask >> j) & 1u) {
                        // the group ends after triple j: tell the epilogue
                        // whether it also ends its output key
                        info[2 * cb + 1] = (emask >> j) & 1u;
                        arrive(infoc0 + 8u * cb);
                        if (++cb == (uint32_t)kAcc3) cb = 0;
                    }
                }
                if (okw) {
                    plan[st * (kPps3 + 1) + kPps3] = gmask | (emask << 8) | (cmask << 16);
                    arrive(planned0 + 8u * st);
                }
            }
            if (!__shfl_sync(0xffffffffu, okw, 0)) break;
            ie = nie;
            nie = nnie;
            if (++st == (uint32_t)kStages3) {
                st = 0;
                ph ^= 1u;
            }
        }
        if (lane == 0) misc[4] = opened;
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA
        // One thread issues everything, following the group warp's plan: a
        // group accumulates into one TMEM buffer (its first MMA overwrites);
        // after its last triple the thread commits the buffer to the
        // epilogue (the group warp has already posted whether the group ends
        // its output key).
        if (lane == 0) {
            const uint64_t adesc = a.a_desc0, bdesc = a.b_desc0;
            const uint32_t idesc = a.idesc;
            uint32_t b = 0, dcol = tmem, st = 0, ph = 0, consumed = 0;
            bool ok = true;
            for (int start = 0; start < n; start += kPps3) {
                const int np = n - start < kPps3 ? n - start : kPps3;
                if (!wait3f(full0 + 8u * st, ph, abort_flag, a.status) ||
                    !wait3f(planned0 + 8u * st, ph, abort_flag, a.status)) {
                    ok = false;
                    break;
                }
                fence_after();
                const uint32_t flags = plan[st * (kPps3 + 1) + kPps3];
                const uint32_t s0 = sbase + st * kStageBytes;
                const uint64_t bd0 = bdesc + (s0 >> 4), ad0 = adesc + ((s0 + kPps3 * kTBytes + kFBytes) >> 4);
                for (int jj = 0; jj < np; ++jj) {
                    const bool newgrp = (flags >> jj) & 1u;
                    if (newgrp) dcol = tmem + b * 128u;
                    // F slot jj at (2 jj + 1) blocks; T slot jj at jj tiles
                    const uint64_t ad = ad0 + (uint64_t)(jj * (2 * kFBytes >> 4));
                    const uint64_t bd = bd0 + (uint64_t)(jj * (kTBytes >> 4));
                    // x = 0: F^T in M rows 0-63 (zeros below), i in 0..7
                    mma(dcol, ad, bd, idesc, newgrp ? 0u : 1u);
                    // x = 1: F^T in M rows 64-127 (zeros above), i in 8..15
                    mma(dcol, ad - (kFBytes >> 4), bd + ((kTBytes / 2) >> 4), idesc, 1u);
                    if ((flags >> (16 + jj)) & 1u) {
                        commit(accf0 + 8u * b);
                        if (++b == (uint32_t)kAcc3) b = 0;
                    }
                }
                commit(empty0 + 8u * st);
                ++consumed;
                if (++st == (uint32_t)kStages3) {
                    st = 0;
                    ph ^= 1u;
                }
            }
            misc[2] = ok ? 0xFFFFFFFFu : consumed;
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------- epilogue
        const int q = warp & 3;   // TMEM lane quadrant of this warp
        const int l = q * 32 + lane, x = l >> 6, r = l & 63;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        float acc[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = 0.0f;
        uint32_t b = 0, ph = 0, got_e = 0;
        int64_t s = s_first;
        const int64_t s_last = n > 0 ? seg_of(a.seg_start, a.S, pe - 1) : s_first - 1;
        while (s <= s_last) {
            // the group's E tile was requested by the group warp when it opened the group
            if (!__all_sync(0xffffffffu, wait3f(ef0 + 8u * b, ph, abort_flag, a.status))) break;
            ++got_e;
            float ef[16];
            const __nv_bfloat16 *ep = eslots + b * (kEBytes / 2) + r * a.sEr;
#pragma unroll
            for (int j = 0; j < 16; ++j) ef[j] = __bfloat162float(ep[j * a.sEj]);
            if (!__all_sync(0xffffffffu, wait3f(infoc0 + 8u * b, ph, abort_flag, a.status))) break;
            const uint32_t ends = info[2 * b + 1];
            if (!__all_sync(0xffffffffu, wait3f(accf0 + 8u * b, ph, abort_flag, a.status))) break;
            fence_after();
            uint32_t v[128];
            const uint32_t bcol = tmem + lane_base + b * 128u;
            tmem_ld128(bcol, v);
            fence_before();
            __syncwarp();
            if (lane == 0) arrive(acce0 + 8u * b);
            if (++b == (uint32_t)kAcc3) {
                b = 0;
                ph ^= 1u;
            }
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 16; ++j) acc[i] = fmaf(ef[j], __uint_as_float(v[i * 16 + j]), acc[i]);
            if (ends) {
                const int64_t ss = a.seg_start[s], se = a.seg_start[s + 1];
                const int kind = (ss >= pb && se <= pe) ? 0 : (ss < pb ? 1 : 2);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int64_t o = (int64_t)(x * 8 + i) * a.sWi + (int64_t)r * a.sWr;
                    if (kind == 0) {
                        const float y = epi3(acc[i], a.epi, a.scale);
                        if (a.dout == UCL_BF16)
                            reinterpret_cast<__nv_bfloat16 *>(a.out)[s * a.tile_w + o] = __float2bfloat16_rn(y);
                        else
                            reinterpret_cast<float *>(a.out)[s * a.tile_w + o] = y;
                    } else {
                        a.partials[((int64_t)unit * 2 + (kind == 1 ? 0 : 1)) * a.tile_w + o] = acc[i];
                    }
                    acc[i] = 0.0f;
                }
                ++s;
            }
        }
        if (warp == 2 && lane == 0) misc[5] = got_e;
    }

    // ---------------------------------------------------------- teardown
    __syncthreads();
    if (*abort_flag) {
        if (warp == 0 && lane == 0) {
            // copies still in flight land in this CTA's shared memory: wait for
            // every fill the MMA warp did not consume
            const uint32_t done = misc[2];
            for (uint32_t k = done; k < misc[3]; ++k) drain3(full0 + 8u * (k % kStages3), (k / kStages3) & 1u);
            // E tiles requested for groups the epilogue did not reach
            for (uint32_t k = misc[5]; k < misc[4]; ++k) drain3(ef0 + 8u * (k % kAcc3), (k / kAcc3) & 1u);
        }
        if (warp == 1 && lane == 0) {
            commit(done_bar);   // tracks every MMA this thread issued
            drain3(done_bar, 0);
        }
    }
    fence_before();
    __syncthreads();
    if (warp == 1) {
        fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512) : "memory");
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encode3() {
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

// 3-D map over an array of [rows][cols] bf16 tiles, one box per tile.
bool map3(CUtensorMap *m, const void *base, int64_t n, int cols, int rows, CUtensorMapSwizzle swz, std::string *why,
          int box_cols = 0) {
    auto enc = encode3();
    if (!enc) {
        *why = "cuTensorMapEncodeTiled unavailable";
        return false;
    }
    cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)rows, (cuuint64_t)n};
    cuuint64_t strides[2] = {(cuuint64_t)cols * 2, (cuuint64_t)rows * cols * 2};
    cuuint32_t box[3] = {(cuuint32_t)(box_cols ? box_cols : cols), (cuuint32_t)rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        *why = "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")";
        return false;
    }
    return true;
}

}  // namespace

int tc3_units(ucl_ctx *ctx, int64_t P) { return (int)(P < ctx->sm_count ? P : ctx->sm_count); }

ucl_status launch_contract_tc3(ucl_ctx *ctx, const ContractArgs &a, const Tc3Plan &tp, const ucl_rel *const *in) {
    const ucl_rel *T = in[tp.t], *E = in[tp.e], *F = in[tp.f];
    const uint32_t *idx[3] = {a.pu, a.pv, a.px};
    std::string why;
    if ((reinterpret_cast<uintptr_t>(T->tiles) | reinterpret_cast<uintptr_t>(F->tiles)) & 15)
        return fail(ctx, UCL_ERR_UNSUPPORTED, "tcgen05 path: tile arrays not 16-byte aligned");
    if (reinterpret_cast<uintptr_t>(E->tiles) & 15)
        return fail(ctx, UCL_ERR_UNSUPPORTED, "tcgen05 path: tile arrays not 16-byte aligned");
    CUtensorMap mT, mF, mE;
    // E is copied as stored (no swizzle): [shape0][shape1]
    const bool tmn = tp.t_mn;
    if (!(tmn ? map3(&mT, T->tiles, T->n, 256, 16, CU_TENSOR_MAP_SWIZZLE_128B, &why, 64)
              : map3(&mT, T->tiles, T->n, 16, 256, CU_TENSOR_MAP_SWIZZLE_32B, &why)) ||
        !map3(&mF, F->tiles, F->n, 64, 16, CU_TENSOR_MAP_SWIZZLE_128B, &why) ||
        !map3(&mE, E->tiles, E->n, (int)E->shape[1], (int)E->shape[0], CU_TENSOR_MAP_SWIZZLE_NONE, &why))
        return fail(ctx, UCL_ERR_CUDA, "tcgen05 path: " + why);
    Tc3Args k{};
    k.idx_t = idx[tp.t];
    k.idx_e = idx[tp.e];
    k.idx_f = idx[tp.f];
    k.nT = T->n;
    k.nE = E->n;
    k.nF = F->n;
    k.sEj = tp.sEj;
    k.sEr = tp.sEr;
    k.seg_start = a.seg_start;
    k.S = a.S;
    k.units = a.units;
    k.out = a.out;
    k.dout = a.dout;
    k.epi = a.epi;
    k.scale = a.scale;
    k.partials = a.partials;
    k.tile_w = a.tile_w;
    k.sWi = tp.sWi;
    k.sWr = tp.sWr;
    // kind::f16, D fp32, A and B bf16, A MN-major (F tile rows run over k,
    // r contiguous), B K-major (T rows (i, j), k contiguous) or, for T laid out
    // [k][(i, j)], MN-major; N = 128, M = 128
    k.t_mn = tmn ? 1 : 0;
    k.idesc = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) | ((tmn ? 1u : 0u) << 16) | ((128u >> 3) << 17) |
              ((128u >> 4) << 24);
    // A: 128B swizzle, next 64-row M atom one F block further (LBO), next 8
    // k rows 1024 bytes further (SBO).  B, K-major: 32B swizzle, 8 rows of
    // 32 bytes per core matrix group (SBO 256).  B, MN-major: 128B swizzle,
    // next 64-column N atom one 2 KB box further (LBO), next 8 k rows 1024
    // bytes further (SBO); the second half of (i, j) starts two boxes (4 KB)
    // in, the same offset as the K-major layout's row 128.
    k.a_desc0 = ((uint64_t)(kFBytes >> 4) << 16) | ((uint64_t)(1024 >> 4) << 32) | (1ull << 46) | (2ull << 61);
    k.b_desc0 = tmn ? (((uint64_t)((kTBytes / 4) >> 4) << 16) | ((uint64_t)(1024 >> 4) << 32) | (1ull << 46) |
                       (2ull << 61))
                    : (((uint64_t)(16 >> 4) << 16) | ((uint64_t)(256 >> 4) << 32) | (1ull << 46) | (6ull << 61));
    k.status = ctx->d_status + 2;
    ucl_status st = cuda_check(
        ctx, cudaFuncSetAttribute(tc3_contract_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem3),
        "cudaFuncSetAttribute");
    if (st) return st;
    tc3_contract_kernel<<<a.units.G, kThreads3, kSmem3, ctx->stream>>>(mT, mF, mE, k);
    ctx->launches++;
    return cuda_check(ctx, cudaGetLastError(), "tcgen05 kernel launch");
}

}  // namespace ucl
