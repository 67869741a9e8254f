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
// operands).  Accumulation is fp32 FFMA -- never TF32.
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

template <typename TU, typename TV>
__global__ void __launch_bounds__(kSimtThreads) simt_contract_kernel(ContractArgs a, LowerPlan lp,
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
            float acc = 0.0f;
            for (int64_t p = p0; p < p1; ++p) {
                const uint32_t iu = a.pu[p], iv = a.pv[p];
                if (iu >= a.nU || (V && iv >= a.nV)) {
                    bad = kStBadIndex;
                    continue;
                }
                const TU *up = U + (int64_t)iu * lp.tile_u + ou;
                if (V) {
                    const TV *vp = V + (int64_t)iv * lp.tile_v + ov;
                    if (tab) {
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
                            acc = fmaf(ld<TU>(up + cu), ld<TV>(vp + cv), acc);
                        }
                    }
                } else {
                    if (tab) {
                        for (int64_t c = 0; c < lp.n_c; ++c) acc += ld<TU>(up + s_cu[c]);
                    } else {
                        for (int64_t c = 0; c < lp.n_c; ++c) {
                            int64_t rem2 = c;
                            int cu = 0;
                            for (int q = lp.nc - 1; q >= 0; --q) {
                                int idx = (int)(rem2 % lp.c_ext[q]);
                                rem2 /= lp.c_ext[q];
                                cu += idx * lp.c_su[q];
                            }
                            acc += ld<TU>(up + cu);
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

__device__ __forceinline__ float ld_any(const void *base, int64_t i, bool bf16) {
    return bf16 ? __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(base)[i])
                : __ldg(reinterpret_cast<const float *>(base) + i);
}

// Three-way EinSum (a star join such as MTTKRP): the product of the three
// tiles' entries summed over the contracted lower labels.  Operand dtypes are
// read at run time; the partial/fixup protocol is the binary kernel's.
__global__ void __launch_bounds__(kSimtThreads) simt_contract3_kernel(ContractArgs a, LowerPlan lp,
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
    if (p >= a.units.P) return;
    const int64_t s = find_seg(a.seg_start, a.S, p);
    const int64_t ss = a.seg_start[s], se = a.seg_start[s + 1];
    if (ss >= p || ss < a.units.begin(c - 1)) return;
    // units c .. u_end - 1 hold the segment's continuation partials (slot 0)
    int u_end = c;
    while (u_end < a.units.G && a.units.begin(u_end) < se) ++u_end;
    const float *first = a.partials + ((int64_t)(c - 1) * 2 + 1) * a.tile_w;
    for (int64_t w = threadIdx.x; w < a.tile_w; w += blockDim.x) {
        float acc = first[w];
        for (int u = c; u < u_end; ++u) acc += a.partials[((int64_t)u * 2) * a.tile_w + w];
        store_out(a.out, a.dout, s * a.tile_w + w, epilogue(acc, a.epi, a.scale));
    }
}

}  // namespace

void launch_contract_simt(ucl_ctx *ctx, const ContractArgs &a, const LowerPlan &lp) {
    const int G = a.units.G;
    if (G <= 0) return;
    if (a.X) {
        simt_contract3_kernel<<<G, kSimtThreads, 0, ctx->stream>>>(a, lp, ctx->d_status + 2);
        ctx->launches++;
        return;
    }
    if (a.du == UCL_F32 && (!a.V || a.dv == UCL_F32))
        simt_contract_kernel<float, float><<<G, kSimtThreads, 0, ctx->stream>>>(a, lp, ctx->d_status + 2);
    else if (a.du == UCL_F32)
        simt_contract_kernel<float, __nv_bfloat16><<<G, kSimtThreads, 0, ctx->stream>>>(a, lp, ctx->d_status + 2);
    else if (!a.V || a.dv == UCL_BF16)
        simt_contract_kernel<__nv_bfloat16, __nv_bfloat16><<<G, kSimtThreads, 0, ctx->stream>>>(a, lp, ctx->d_status + 2);
    else
        simt_contract_kernel<__nv_bfloat16, float><<<G, kSimtThreads, 0, ctx->stream>>>(a, lp, ctx->d_status + 2);
    ctx->launches++;
}

void launch_fixup(ucl_ctx *ctx, const ContractArgs &a) {
    if (a.units.G <= 1) return;
    fixup_kernel<<<a.units.G - 1, kSimtThreads, 0, ctx->stream>>>(a);
    ctx->launches++;
}

}  // namespace ucl
