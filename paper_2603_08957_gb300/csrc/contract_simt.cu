// contract_simt.cu -- the FFMA tile contraction with the segmented group-by
// sum fused into it, and the fixup of output keys whose pairs straddle two
// work units.
//
// The pair list is ordered by output key, so the SUM ... GROUP BY up(W) of
// the TR-SQL template (paper Sec. 5) is a segmented sum over consecutive
// pairs.  The pair list is cut into G contiguous units of equal pair count,
// one CTA each.  A segment that lies inside one unit is summed and written by
// that CTA (epilogue applied); a segment that crosses unit boundaries leaves
// one fp32 partial per unit it touches, and the fixup kernel adds those
// partials in unit order.  Summation order is therefore fixed: results are
// deterministic.
//
// This kernel is the general path: any label classes (batch labels, labels
// summed inside one operand, rank-0 tiles, unary EinSums, fp32 or bf16
// operands).  Accumulation is fp32 FFMA -- never TF32.  It also evaluates the
// extended EinSum of Sec. 3 (aggregate MAX / MIN / SUM of map(comb(u, v))),
// in a separate instantiation so that the plain sum of products keeps its
// FFMA inner loop; partials of split segments are folded with the same
// aggregate.
#include <algorithm>

#include "internal.cuh"

namespace ucl {

namespace {

constexpr int kSimtThreads = 256;
constexpr int kMaxTab = 2048;   // contracted-index offset table kept in shared memory

template <typename T>
__device__ __forceinline__ float ld(const T *p);
template <>
__device__ __forceinline__ float ld<float>(const float *p) { return __ldg(p); }
template <>
__device__ __forceinline__ float ld<__nv_bfloat16>(const __nv_bfloat16 *p) { return __bfloat162float(*p); }

__device__ __forceinline__ float epilogue(float x, int epi, float scale) {
    x *= scale;
    if (epi == UCL_EPI_RELU) x = fmaxf(x, 0.0f);
    return x;
}

// ---- extended EinSum: term = map(comb(u, v)) (map(u) when unary), folded by agg
__device__ __forceinline__ float sem_map(int map, float p) {
    switch (map) {
        case UCL_MAP_RELU: return fmaxf(p, 0.0f);
        case UCL_MAP_EXP: return expf(p);
        case UCL_MAP_SQUARE: return p * p;
        default: return p;
    }
}

__device__ __forceinline__ float sem_term(int comb, int map, float u, float v) {
    float p;
    switch (comb) {
        case UCL_COMB_ADD: p = u + v; break;
        case UCL_COMB_SUB: p = u - v; break;
        case UCL_COMB_DIV: p = u / v; break;
        default: p = u * v; break;
    }
    return sem_map(map, p);
}

__device__ __forceinline__ float sem_fold(int agg, float acc, float p) {
    switch (agg) {
        case UCL_AGG_MAX: return fmaxf(acc, p);
        case UCL_AGG_MIN: return fminf(acc, p);
        default: return acc + p;
    }
}

__device__ __forceinline__ float sem_identity(int agg) {
    return agg == UCL_AGG_MAX ? -INFINITY : (agg == UCL_AGG_MIN ? INFINITY : 0.0f);
}

__device__ __forceinline__ void store_out(void *out, ucl_dtype dt, int64_t idx, float x) {
    if (dt == UCL_BF16)
        reinterpret_cast<__nv_bfloat16 *>(out)[idx] = __float2bfloat16_rn(x);
    else
        reinterpret_cast<float *>(out)[idx] = x;
}

// Segment containing pair p: last s with seg_start[s] <= p.
__device__ __forceinline__ int64_t find_seg(const int64_t *seg_start, int64_t S, int64_t p) {
    int64_t a = 0, b = S;
    while (a < b) {
        int64_t mid = (a + b) >> 1;
        if (seg_start[mid] <= p) a = mid + 1; else b = mid;
    }
    return a - 1;
}

// Wide tiles with a real contraction: the whole CTA takes one segment at a
// time, threads over output elements, pairs and contracted indices in order.
template <typename TU, typename TV, bool EXT>
__global__ void __launch_bounds__(kSimtThreads, 4) simt_wide_kernel(ContractArgs a, LowerPlan lp,
                                                                   uint32_t *status) {
    __shared__ int s_cu[kMaxTab];
    __shared__ int s_cv[kMaxTab];
    const bool tab = lp.n_c <= kMaxTab;
    if (tab) {
        for (int64_t c = threadIdx.x; c < lp.n_c; c += blockDim.x) {
            int64_t rem = c;
            int ou = 0, ov = 0;
            for (int q = lp.nc - 1; q >= 0; --q) {
                int idx = (int)(rem % lp.c_ext[q]);
                rem /= lp.c_ext[q];
                ou += idx * lp.c_su[q];
                ov += idx * lp.c_sv[q];
            }
            s_cu[c] = ou;
            s_cv[c] = ov;
        }
    }
    __syncthreads();

    const TU *U = reinterpret_cast<const TU *>(a.U);
    const TV *V = reinterpret_cast<const TV *>(a.V);
    const int unit = blockIdx.x;
    const int64_t pb = a.units.begin(unit), pe = a.units.begin(unit + 1);
    uint32_t bad = 0;
    for (int64_t s = find_seg(a.seg_start, a.S, pb); s < a.S; ++s) {
        const int64_t ss = a.seg_start[s], se = a.seg_start[s + 1];
        if (ss >= pe) break;
        const int64_t p0 = ss > pb ? ss : pb, p1 = se < pe ? se : pe;
        const int kind = (ss >= pb && se <= pe) ? 0 : (ss < pb ? 1 : 2);
        for (int64_t w = threadIdx.x; w < a.tile_w; w += blockDim.x) {
            int64_t rem = w;
            int ou = 0, ov = 0;
            for (int q = lp.nw - 1; q >= 0; --q) {
                int idx = (int)(rem % lp.w_ext[q]);
                rem /= lp.w_ext[q];
                ou += idx * lp.w_su[q];
                ov += idx * lp.w_sv[q];
            }
            float acc = EXT ? sem_identity(a.agg) : 0.0f;
            for (int64_t p = p0; p < p1; ++p) {
                const uint32_t iu = a.pu[p], iv = a.pv[p];
                if (iu >= a.nU || (V && iv >= a.nV)) {
                    bad = kStBadIndex;
                    continue;
                }
                const TU *up = U + (int64_t)iu * lp.tile_u + ou;
                if (V) {
                    const TV *vp = V + (int64_t)iv * lp.tile_v + ov;
                    if (EXT && tab) {
                        for (int64_t c = 0; c < lp.n_c; ++c)
                            acc = sem_fold(a.agg, acc, sem_term(a.comb, a.map, ld<TU>(up + s_cu[c]), ld<TV>(vp + s_cv[c])));
                    } else if (tab) {
                        for (int64_t c = 0; c < lp.n_c; ++c) acc = fmaf(ld<TU>(up + s_cu[c]), ld<TV>(vp + s_cv[c]), acc);
                    } else {
                        for (int64_t c = 0; c < lp.n_c; ++c) {
                            int64_t rem2 = c;
                            int cu = 0, cv = 0;
                            for (int q = lp.nc - 1; q >= 0; --q) {
                                int idx = (int)(rem2 % lp.c_ext[q]);
                                rem2 /= lp.c_ext[q];
                                cu += idx * lp.c_su[q];
                                cv += idx * lp.c_sv[q];
                            }
                            acc = EXT ? sem_fold(a.agg, acc, sem_term(a.comb, a.map, ld<TU>(up + cu), ld<TV>(vp + cv)))
                                      : fmaf(ld<TU>(up + cu), ld<TV>(vp + cv), acc);
                        }
                    }
                } else {
                    if (tab) {
                        for (int64_t c = 0; c < lp.n_c; ++c) {
                            const float x = ld<TU>(up + s_cu[c]);
                            acc = EXT ? sem_fold(a.agg, acc, sem_map(a.map, x)) : acc + x;
                        }
                    } else {
                        for (int64_t c = 0; c < lp.n_c; ++c) {
                            int64_t rem2 = c;
                            int cu = 0;
                            for (int q = lp.nc - 1; q >= 0; --q) {
                                int idx = (int)(rem2 % lp.c_ext[q]);
                                rem2 /= lp.c_ext[q];
                                cu += idx * lp.c_su[q];
                            }
                            const float x = ld<TU>(up + cu);
                            acc = EXT ? sem_fold(a.agg, acc, sem_map(a.map, x)) : acc + x;
                        }
                    }
                }
            }
            if (kind == 0)
                store_out(a.out, a.dout, s * a.tile_w + w, epilogue(acc, a.epi, a.scale));
            else
                a.partials[((int64_t)unit * 2 + (kind == 1 ? 0 : 1)) * a.tile_w + w] = acc;
        }
    }
    if (bad) atomicOr(status, bad);
}

// Fold of one joined pair's terms for output element (ou, ov) over this
// lane's share of the contracted index range (c = c0, c0 + R, ...).
template <typename TU, typename TV, bool EXT>
__device__ __forceinline__ float pair_terms(const ContractArgs &a, const LowerPlan &lp, const int *s_cu,
                                            const int *s_cv, bool tab, const TU *up, const TV *vp, int64_t c0,
                                            int R, float acc) {
    for (int64_t c = c0; c < lp.n_c; c += R) {
        int cu, cv = 0;
        if (tab) {
            cu = s_cu[c];
            if (vp) cv = s_cv[c];
        } else {
            int64_t rem2 = c;
            cu = 0;
            for (int q = lp.nc - 1; q >= 0; --q) {
                int idx = (int)(rem2 % lp.c_ext[q]);
                rem2 /= lp.c_ext[q];
                cu += idx * lp.c_su[q];
                cv += idx * lp.c_sv[q];
            }
        }
        const float u = ld<TU>(up + cu);
        if (vp) {
            const float v = ld<TV>(vp + cv);
            acc = EXT ? sem_fold(a.agg, acc, sem_term(a.comb, a.map, u, v)) : fmaf(u, v, acc);
        } else {
            acc = EXT ? sem_fold(a.agg, acc, sem_map(a.map, u)) : acc + u;
        }
    }
    return acc;
}

// Narrow tiles, or one term per pair: teams of T warps (T = 1, 2, 4 or 8,
// from the tile width) take the unit's segments in turn, so that every warp
// stays busy.  Within a team, lanes_w lanes (a power of two, at most the tile
// width) take output elements w; when the tile is narrower than a warp the
// R = 32 / lanes_w lanes sharing an element split the contracted index range
// and their terms are folded by a fixed shuffle tree.  Pairs are visited in
// order, four index pairs loaded ahead.
template <typename TU, typename TV, bool EXT>
__global__ void __launch_bounds__(kSimtThreads, 3) simt_team_kernel(ContractArgs a, LowerPlan lp, int team_warps,
                                                                   uint32_t *status) {
    __shared__ int s_cu[kMaxTab];
    __shared__ int s_cv[kMaxTab];
    const bool tab = lp.n_c <= kMaxTab;
    if (tab) {
        for (int64_t c = threadIdx.x; c < lp.n_c; c += blockDim.x) {
            int64_t rem = c;
            int ou = 0, ov = 0;
            for (int q = lp.nc - 1; q >= 0; --q) {
                int idx = (int)(rem % lp.c_ext[q]);
                rem /= lp.c_ext[q];
                ou += idx * lp.c_su[q];
                ov += idx * lp.c_sv[q];
            }
            s_cu[c] = ou;
            s_cv[c] = ov;
        }
    }
    __syncthreads();

    const TU *U = reinterpret_cast<const TU *>(a.U);
    const TV *V = reinterpret_cast<const TV *>(a.V);
    const int T = team_warps;
    const int nteams = (int)(blockDim.x >> 5) / T;
    const int team = (int)(threadIdx.x >> 5) / T;
    const int tsize = 32 * T;
    const int tl = (int)threadIdx.x - team * tsize;
    int lanes_w = tsize;
    while (lanes_w > 1 && lanes_w > a.tile_w) lanes_w >>= 1;
    const int R = tsize / lanes_w;            // > 1 only when T = 1
    const int wl = tl % lanes_w, rl = tl / lanes_w;
    const float ident = EXT ? sem_identity(a.agg) : 0.0f;
    const int unit = blockIdx.x;
    const int64_t pb = a.units.begin(unit), pe = a.units.begin(unit + 1);
    uint32_t bad = 0;
    for (int64_t s = find_seg(a.seg_start, a.S, pb) + team; s < a.S; s += nteams) {
        const int64_t ss = a.seg_start[s], se = a.seg_start[s + 1];
        if (ss >= pe) break;
        const int64_t p0 = ss > pb ? ss : pb, p1 = se < pe ? se : pe;
        const int kind = (ss >= pb && se <= pe) ? 0 : (ss < pb ? 1 : 2);
        for (int64_t w0 = 0; w0 < a.tile_w; w0 += lanes_w) {
            const int64_t w = w0 + wl;
            const bool act = w < a.tile_w;
            int ou = 0, ov = 0;
            if (act) {
                int64_t rem = w;
                for (int q = lp.nw - 1; q >= 0; --q) {
                    int idx = (int)(rem % lp.w_ext[q]);
                    rem /= lp.w_ext[q];
                    ou += idx * lp.w_su[q];
                    ov += idx * lp.w_sv[q];
                }
            }
            float acc = ident;
            if (act) {
                int64_t p = p0;
                for (; p + 4 <= p1; p += 4) {
                    uint32_t iu[4], iv[4];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        iu[j] = a.pu[p + j];
                        iv[j] = V ? a.pv[p + j] : 0u;
                    }
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        if (iu[j] >= a.nU || (V && iv[j] >= a.nV)) {
                            bad = kStBadIndex;
                            continue;
                        }
                        acc = pair_terms<TU, TV, EXT>(a, lp, s_cu, s_cv, tab, U + (int64_t)iu[j] * lp.tile_u + ou,
                                                      V ? V + (int64_t)iv[j] * lp.tile_v + ov : nullptr, rl, R, acc);
                    }
                }
                for (; p < p1; ++p) {
                    const uint32_t iu = a.pu[p], iv = V ? a.pv[p] : 0u;
                    if (iu >= a.nU || (V && iv >= a.nV)) {
                        bad = kStBadIndex;
                        continue;
                    }
                    acc = pair_terms<TU, TV, EXT>(a, lp, s_cu, s_cv, tab, U + (int64_t)iu * lp.tile_u + ou,
                                                  V ? V + (int64_t)iv * lp.tile_v + ov : nullptr, rl, R, acc);
                }
            }
            if (R > 1) {
                // lanes sharing w differ in the bits at and above lanes_w (T = 1: one warp)
                for (int o = lanes_w; o < 32; o <<= 1) {
                    const float x = __shfl_xor_sync(0xffffffffu, acc, o);
                    acc = EXT ? sem_fold(a.agg, acc, x) : acc + x;
                }
            }
            if (act && rl == 0) {
                if (kind == 0)
                    store_out(a.out, a.dout, s * a.tile_w + w, epilogue(acc, a.epi, a.scale));
                else
                    a.partials[((int64_t)unit * 2 + (kind == 1 ? 0 : 1)) * a.tile_w + w] = acc;
            }
        }
    }
    if (bad) atomicOr(status, bad);
}

__device__ __forceinline__ float ld_any(const void *base, int64_t i, bool bf16) {
    return bf16 ? __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(base)[i])
                : __ldg(reinterpret_cast<const float *>(base) + i);
}

// Three-way EinSum (a star join such as MTTKRP): the product of the three
// tiles' entries summed over the contracted lower labels.  Operand dtypes are
// read at run time; the partial/fixup protocol is the binary kernel's.
__global__ void __launch_bounds__(kSimtThreads, 1) simt_contract3_kernel(ContractArgs a, LowerPlan lp,
                                                                      uint32_t *status) {
    __shared__ int s_c[3][kMaxTab];
    const bool tab = lp.n_c <= kMaxTab;
    const bool bu = a.du == UCL_BF16, bv = a.dv == UCL_BF16, bx = a.dx == UCL_BF16;
    if (tab) {
        for (int64_t c = threadIdx.x; c < lp.n_c; c += blockDim.x) {
            int64_t rem = c;
            int ou = 0, ov = 0, ox = 0;
            for (int q = lp.nc - 1; q >= 0; --q) {
                int idx = (int)(rem % lp.c_ext[q]);
                rem /= lp.c_ext[q];
                ou += idx * lp.c_su[q];
                ov += idx * lp.c_sv[q];
                ox += idx * lp.c_sx[q];
            }
            s_c[0][c] = ou;
            s_c[1][c] = ov;
            s_c[2][c] = ox;
        }
    }
    __syncthreads();
    const int unit = blockIdx.x;
    const int64_t pb = a.units.begin(unit), pe = a.units.begin(unit + 1);
    uint32_t bad = 0;
    for (int64_t s = find_seg(a.seg_start, a.S, pb); s < a.S; ++s) {
        const int64_t ss = a.seg_start[s], se = a.seg_start[s + 1];
        if (ss >= pe) break;
        const int64_t p0 = ss > pb ? ss : pb, p1 = se < pe ? se : pe;
        const int kind = (ss >= pb && se <= pe) ? 0 : (ss < pb ? 1 : 2);
        for (int64_t w = threadIdx.x; w < a.tile_w; w += blockDim.x) {
            int64_t rem = w;
            int64_t ou = 0, ov = 0, ox = 0;
            for (int q = lp.nw - 1; q >= 0; --q) {
                int idx = (int)(rem % lp.w_ext[q]);
                rem /= lp.w_ext[q];
                ou += idx * lp.w_su[q];
                ov += idx * lp.w_sv[q];
                ox += idx * lp.w_sx[q];
            }
            float acc = 0.0f;
            for (int64_t p = p0; p < p1; ++p) {
                const uint32_t iu = a.pu[p], iv = a.pv[p], ix = a.px[p];
                if (iu >= a.nU || iv >= a.nV || ix >= a.nX) {
                    bad = kStBadIndex;
                    continue;
                }
                const int64_t bu0 = (int64_t)iu * lp.tile_u + ou, bv0 = (int64_t)iv * lp.tile_v + ov,
                              bx0 = (int64_t)ix * lp.tile_x + ox;
                for (int64_t c = 0; c < lp.n_c; ++c) {
                    int cu, cv, cx;
                    if (tab) {
                        cu = s_c[0][c];
                        cv = s_c[1][c];
                        cx = s_c[2][c];
                    } else {
                        int64_t rem2 = c;
                        cu = cv = cx = 0;
                        for (int q = lp.nc - 1; q >= 0; --q) {
                            int idx = (int)(rem2 % lp.c_ext[q]);
                            rem2 /= lp.c_ext[q];
                            cu += idx * lp.c_su[q];
                            cv += idx * lp.c_sv[q];
                            cx += idx * lp.c_sx[q];
                        }
                    }
                    acc = fmaf(ld_any(a.U, bu0 + cu, bu) * ld_any(a.V, bv0 + cv, bv), ld_any(a.X, bx0 + cx, bx), acc);
                }
            }
            if (kind == 0)
                store_out(a.out, a.dout, s * a.tile_w + w, epilogue(acc, a.epi, a.scale));
            else
                a.partials[((int64_t)unit * 2 + (kind == 1 ? 0 : 1)) * a.tile_w + w] = acc;
        }
    }
    if (bad) atomicOr(status, bad);
}

// Boundary c (between units c-1 and c) owns the segment that crosses it if
// that segment starts inside unit c-1; it sums the segment's partials in unit
// order and writes the output tile.
__global__ void __launch_bounds__(kSimtThreads) fixup_kernel(ContractArgs a) {
    const int c = blockIdx.x + 1;
    const int64_t p = a.units.begin(c);
    if (p >= a.units.base + a.units.P) return;
    const int64_t s = find_seg(a.seg_start, a.S, p);
    const int64_t ss = a.seg_start[s], se = a.seg_start[s + 1];
    if (ss >= p || ss < a.units.begin(c - 1)) return;
    // units c .. u_end - 1 hold the segment's continuation partials (slot 0)
    int u_end = c;
    while (u_end < a.units.G && a.units.begin(u_end) < se) ++u_end;
    if (a.fixup_bytes && threadIdx.x == 0) {
        // partials of units c - 1 .. u_end - 1 read, one output tile written
        const int osz = a.dout == UCL_BF16 ? 2 : 4;
        atomicAdd(a.fixup_bytes, (unsigned long long)(a.tile_w * (4 * (u_end - c + 1) + osz)));
    }
    // kU elements per thread per round, all loads of a partial issued before
    // any is used, so a round costs one memory latency per partial rather
    // than one per element; the fold order (units in order) is unchanged
    constexpr int kU = 8;
    const float *__restrict__ first = a.partials + ((int64_t)(c - 1) * 2 + 1) * a.tile_w;
    const int64_t step = blockDim.x;
    for (int64_t w0 = threadIdx.x; w0 < a.tile_w; w0 += step * kU) {
        float acc[kU];
#pragma unroll
        for (int q = 0; q < kU; ++q) {
            const int64_t w = w0 + q * step;
            acc[q] = w < a.tile_w ? __ldg(first + w) : 0.0f;
        }
        for (int u = c; u < u_end; ++u) {
            const float *__restrict__ pp = a.partials + (int64_t)u * 2 * a.tile_w;
            float v[kU];
#pragma unroll
            for (int q = 0; q < kU; ++q) {
                const int64_t w = w0 + q * step;
                v[q] = w < a.tile_w ? __ldg(pp + w) : 0.0f;
            }
#pragma unroll
            for (int q = 0; q < kU; ++q) acc[q] = sem_fold(a.agg, acc[q], v[q]);
        }
#pragma unroll
        for (int q = 0; q < kU; ++q) {
            const int64_t w = w0 + q * step;
            if (w < a.tile_w) store_out(a.out, a.dout, s * a.tile_w + w, epilogue(acc[q], a.epi, a.scale));
        }
    }
}

// Windowed fixup (the windowed tcgen05 kernel's partials): boundary c owns
// the window segment that crosses it if that segment starts inside unit
// c - 1; for each present slot it sums the slot's partials in unit order and
// writes the slot's output row.  Partials: [unit][2][2^win_bits][tile_w].
__global__ void __launch_bounds__(kSimtThreads) fixup_window_kernel(ContractArgs a) {
    const int c = blockIdx.x + 1;
    const int64_t p = a.units.begin(c);
    if (p >= a.units.base + a.units.P) return;
    const int64_t s = find_seg(a.seg_start, a.S, p);
    const int64_t ss = a.seg_start[s], se = a.seg_start[s + 1];
    if (ss >= p || ss < a.units.begin(c - 1)) return;
    int u_end = c;
    while (u_end < a.units.G && a.units.begin(u_end) < se) ++u_end;
    const int W = 1 << a.win_bits;
    const uint32_t mask = a.wmask[s];
    const int64_t base = a.wbase[s];
    if (a.fixup_bytes && threadIdx.x == 0) {
        const int osz = a.dout == UCL_BF16 ? 2 : 4;
        atomicAdd(a.fixup_bytes,
                  (unsigned long long)(__popc(mask) * a.tile_w * (4 * (u_end - c + 1) + osz)));
    }
    for (int q = 0; q < W; ++q) {
        if (!((mask >> q) & 1u)) continue;
        const int64_t row = base + __popc(mask & ((1u << q) - 1u));
        const float *__restrict__ first = a.partials + (((int64_t)(c - 1) * 2 + 1) * W + q) * a.tile_w;
        for (int64_t w = threadIdx.x; w < a.tile_w; w += blockDim.x) {
            float acc = __ldg(first + w);
            for (int u = c; u < u_end; ++u) acc += __ldg(a.partials + (((int64_t)u * 2) * W + q) * a.tile_w + w);
            store_out(a.out, a.dout, row * a.tile_w + w, epilogue(acc, a.epi, a.scale));
        }
    }
}

// Band sum: output key f is the sum, in band order, of its band partials
// part[order[r]] for r in [fstart[f], fstart[f + 1]) (fp32 tiles), then the
// epilogue and the output cast.  One CTA per output tile at a time; two
// 16-byte loads per thread and row in flight.
__global__ void __launch_bounds__(kSimtThreads) band_sum_kernel(const float *__restrict__ part,
                                                                const uint64_t *__restrict__ order,
                                                                const int64_t *__restrict__ fstart, int64_t S,
                                                                int64_t tile_w, void *out, int dout, int epi,
                                                                float scale, unsigned long long *bytes) {
    const bool vec = (tile_w & 3) == 0;
    const int osz = dout == UCL_BF16 ? 2 : 4;
    for (int64_t f = blockIdx.x; f < S; f += gridDim.x) {
        const int64_t r0 = fstart[f], r1 = fstart[f + 1];
        if (bytes && threadIdx.x == 0) atomicAdd(bytes, (unsigned long long)(tile_w * (4 * (r1 - r0) + osz)));
        if (vec) {
            const int64_t step = (int64_t)blockDim.x * 4;
            for (int64_t e0 = (int64_t)threadIdx.x * 4; e0 < tile_w; e0 += 2 * step) {
                const int64_t e1 = e0 + step;
                const bool two = e1 < tile_w;
                float4 a0 = make_float4(0.f, 0.f, 0.f, 0.f), a1 = a0;
                for (int64_t r = r0; r < r1; ++r) {
                    const float *row = part + (int64_t)order[r] * tile_w;
                    const float4 v0 = __ldg(reinterpret_cast<const float4 *>(row + e0));
                    const float4 v1 = two ? __ldg(reinterpret_cast<const float4 *>(row + e1)) : a1;
                    a0.x += v0.x; a0.y += v0.y; a0.z += v0.z; a0.w += v0.w;
                    if (two) { a1.x += v1.x; a1.y += v1.y; a1.z += v1.z; a1.w += v1.w; }
                }
                for (int h = 0; h < (two ? 2 : 1); ++h) {
                    const float4 a = h ? a1 : a0;
                    const int64_t e = h ? e1 : e0;
                    const float x0 = epilogue(a.x, epi, scale), x1 = epilogue(a.y, epi, scale),
                                x2 = epilogue(a.z, epi, scale), x3 = epilogue(a.w, epi, scale);
                    if (dout == UCL_BF16) {
                        __nv_bfloat162 lo = __floats2bfloat162_rn(x0, x1), hi = __floats2bfloat162_rn(x2, x3);
                        uint2 w;
                        w.x = *reinterpret_cast<uint32_t *>(&lo);
                        w.y = *reinterpret_cast<uint32_t *>(&hi);
                        *reinterpret_cast<uint2 *>(reinterpret_cast<__nv_bfloat16 *>(out) + f * tile_w + e) = w;
                    } else {
                        *reinterpret_cast<float4 *>(reinterpret_cast<float *>(out) + f * tile_w + e) =
                            make_float4(x0, x1, x2, x3);
                    }
                }
            }
        } else {
            for (int64_t e = threadIdx.x; e < tile_w; e += blockDim.x) {
                float acc = 0.0f;
                for (int64_t r = r0; r < r1; ++r) acc += __ldg(part + (int64_t)order[r] * tile_w + e);
                store_out(out, (ucl_dtype)dout, f * tile_w + e, epilogue(acc, epi, scale));
            }
        }
    }
}

}  // namespace

void launch_band_sum(ucl_ctx *ctx, const float *part, const uint64_t *order, const int64_t *fstart, int64_t S,
                     int64_t tile_w, void *out, ucl_dtype dout, int epi, float scale, unsigned long long *bytes) {
    if (S <= 0) return;
    const int64_t grid = std::min<int64_t>(S, (int64_t)ctx->sm_count * 8);
    band_sum_kernel<<<(int)grid, kSimtThreads, 0, ctx->stream>>>(part, order, fstart, S, tile_w, out, (int)dout, epi,
                                                                  scale, bytes);
    ctx->launches++;
}

void launch_contract_simt(ucl_ctx *ctx, const ContractArgs &a, const LowerPlan &lp) {
    const int G = a.units.G;
    if (G <= 0) return;
    if (a.X) {
        simt_contract3_kernel<<<G, kSimtThreads, 0, ctx->stream>>>(a, lp, ctx->d_status + 2);
        ctx->launches++;
        return;
    }
    const bool ext = a.agg != UCL_AGG_SUM || a.map != UCL_MAP_IDENT || (a.V && a.comb != UCL_COMB_MUL);
    // wide tiles with a real contraction: one segment per CTA at a time;
    // otherwise warp teams (one warp per 32 output elements, up to the CTA)
    const bool wide = a.tile_w >= kSimtThreads && lp.n_c >= 8;
    int team = 1;
    while (team < kSimtThreads / 32 && (int64_t)team * 64 <= a.tile_w) team <<= 1;
#define UCL_SIMT(TU, TV)                                                                                         \
    (wide ? (ext ? simt_wide_kernel<TU, TV, true><<<G, kSimtThreads, 0, ctx->stream>>>(a, lp, ctx->d_status + 2)   \
                 : simt_wide_kernel<TU, TV, false><<<G, kSimtThreads, 0, ctx->stream>>>(a, lp, ctx->d_status + 2)) \
          : (ext ? simt_team_kernel<TU, TV, true><<<G, kSimtThreads, 0, ctx->stream>>>(a, lp, team,                \
                                                                                      ctx->d_status + 2)           \
                 : simt_team_kernel<TU, TV, false><<<G, kSimtThreads, 0, ctx->stream>>>(a, lp, team,               \
                                                                                       ctx->d_status + 2)))
    if (a.du == UCL_F32 && (!a.V || a.dv == UCL_F32))
        UCL_SIMT(float, float);
    else if (a.du == UCL_F32)
        UCL_SIMT(float, __nv_bfloat16);
    else if (!a.V || a.dv == UCL_BF16)
        UCL_SIMT(__nv_bfloat16, __nv_bfloat16);
    else
        UCL_SIMT(__nv_bfloat16, float);
#undef UCL_SIMT
    ctx->launches++;
}

void launch_fixup_window(ucl_ctx *ctx, const ContractArgs &a) {
    if (a.units.G <= 1) return;
    fixup_window_kernel<<<a.units.G - 1, kSimtThreads, 0, ctx->stream>>>(a);
    ctx->launches++;
}

void launch_fixup(ucl_ctx *ctx, const ContractArgs &a) {
    if (a.units.G <= 1) return;
    fixup_kernel<<<a.units.G - 1, kSimtThreads, 0, ctx->stream>>>(a);
    ctx->launches++;
}

}  // namespace ucl
