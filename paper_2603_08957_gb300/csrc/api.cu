// api.cu -- the C ABI (include/ucl.h): spec parsing and validation, plan
// building, relation management and the stage schedule of one UCL EinSum.
//
// Stage schedule of ucl_einsum (paper Sec. 5, Eq. eqn-TRA):
//   0  pack keys -> radix sort both inputs by join key (skipped for inputs
//      already sorted by it) -> per-U-tuple matching range in V -> scan;
//      host sync #1 reads the pair count
//   1  expand pairs (u, v, packed output key) -> stable radix sort by output
//      key -> segment heads -> scan; host sync #2 reads the segment count
//   2  allocate the output relation; segment starts + output keys; tile
//      contraction with the group-by sum fused into its epilogue
//   3  fixup of segments split across work units
#include <algorithm>
#include <cstdlib>
#include <cstdio>
#include <new>

#include "internal.cuh"

using namespace ucl;

namespace {

struct Oom {};

// ------------------------------------------------------------------ spec

struct Label {
    char c;
    bool upper;
    int64_t ext = 0;
    int pos[4] = {-1, -1, -1, -1};   // key column / tile dim in input k (k < 3), output at [3]
};

struct Spec {
    int n_in = 0;
    std::string op[3];
    std::string out;
    std::vector<Label> labs;
    int find(char c) const {
        for (size_t i = 0; i < labs.size(); ++i)
            if (labs[i].c == c) return (int)i;
        return -1;
    }
    const std::string &operand(int k) const { return k == 3 ? out : op[k]; }
};

bool is_alpha(char c) { return (c >= 'a' && c <= 'z') || (c >= 'A' && c <= 'Z'); }
bool is_upper(char c) { return c >= 'A' && c <= 'Z'; }

ucl_status parse_spec(ucl_ctx *ctx, const char *text, int n_in, Spec &s) {
    if (!text) return fail(ctx, UCL_ERR_ARG, "spec is NULL");
    if (n_in < 1 || n_in > 3) return fail(ctx, UCL_ERR_ARG, "n_in must be 1, 2 or 3");
    std::string t(text);
    size_t arrow = t.find("->");
    if (arrow == std::string::npos) return fail(ctx, UCL_ERR_SPEC, "spec has no '->'");
    std::string lhs = t.substr(0, arrow);
    s.out = t.substr(arrow + 2);
    int k = 0;
    for (char c : lhs) {
        if (c == ',') {
            if (++k >= 3) return fail(ctx, UCL_ERR_SPEC, "too many operands");
        } else if (is_alpha(c)) {
            s.op[k] += c;
        } else {
            return fail(ctx, UCL_ERR_SPEC, std::string("bad character in spec: ") + c);
        }
    }
    if (k + 1 != n_in) return fail(ctx, UCL_ERR_SPEC, "operand count does not match n_in");
    s.n_in = n_in;
    for (char c : s.out)
        if (!is_alpha(c)) return fail(ctx, UCL_ERR_SPEC, std::string("bad character in output: ") + c);
    for (int i = 0; i <= n_in; ++i) {
        const std::string &o = i < n_in ? s.op[i] : s.out;
        if ((int)o.size() > kMaxCols) return fail(ctx, UCL_ERR_UNSUPPORTED, "operand has more than 15 labels");
        for (size_t a = 0; a < o.size(); ++a)
            for (size_t b = a + 1; b < o.size(); ++b)
                if (o[a] == o[b]) return fail(ctx, UCL_ERR_SPEC, std::string("label repeated in one operand: ") + o[a]);
    }
    for (int i = 0; i < n_in; ++i)
        for (char c : s.op[i])
            if (s.find(c) < 0) {
                Label L;
                L.c = c;
                L.upper = is_upper(c);
                s.labs.push_back(L);
            }
    for (char c : s.out)
        if (s.find(c) < 0) return fail(ctx, UCL_ERR_SPEC, std::string("output label not in any input: ") + c);
    for (int i = 0; i <= n_in; ++i) {
        const std::string &o = i < n_in ? s.op[i] : s.out;
        int cu = 0, cl = 0;
        for (char c : o) {
            Label &L = s.labs[s.find(c)];
            L.pos[i < n_in ? i : 3] = L.upper ? cu++ : cl++;
        }
    }
    if ((int)s.labs.size() > kMaxLow + kMaxCols) return fail(ctx, UCL_ERR_UNSUPPORTED, "too many labels");
    return UCL_OK;
}

// Arity and extents of the inputs against the spec (Sec. 3: one bound per label).
ucl_status bind_extents(ucl_ctx *ctx, Spec &s, ucl_rel *const *in) {
    for (int k = 0; k < s.n_in; ++k) {
        const ucl_rel *R = in[k];
        if (!R) return fail(ctx, UCL_ERR_ARG, "input relation is NULL");
        if (R->ctx != ctx) return fail(ctx, UCL_ERR_ARG, "input relation belongs to another context");
        int nu = 0, nl = 0;
        for (char c : s.op[k]) (is_upper(c) ? nu : nl)++;
        if (R->u != nu || R->r != nl)
            return fail(ctx, UCL_ERR_SHAPE, "operand " + std::to_string(k) + " '" + s.op[k] +
                                                "' does not match the relation's key/tile arity");
        for (Label &L : s.labs) {
            int p = L.pos[k];
            if (p < 0) continue;
            int64_t e = L.upper ? R->bounds[p] : R->shape[p];
            if (L.ext == 0) L.ext = e;
            else if (L.ext != e)
                return fail(ctx, UCL_ERR_SHAPE, std::string("label '") + L.c + "' has two different extents");
        }
    }
    return UCL_OK;
}

// Row-major stride of lower label L inside operand k's tile (0 if absent).
int64_t tile_stride(const Spec &s, int k, const Label &L) {
    int p = L.pos[k];
    if (p < 0) return 0;
    int64_t st = 1;
    const std::string &o = s.operand(k);
    for (int a = (int)o.size() - 1; a >= 0; --a) {
        const Label &M = s.labs[s.find(o[a])];
        if (M.upper) continue;
        if (M.pos[k] == p) break;
        st *= M.ext;
    }
    return st;
}

struct KeyPlan {
    // join order: (ord[0] JOIN ord[1]) JOIN ord[2]; inputs in spec order for
    // one or two inputs
    int ord[3] = {0, 1, 2};
    std::vector<int> join;   // label ids of the first join's attributes, ord[0]'s order
    int join_bits = 0;
    KeyPack join_u{}, join_v{};   // packers of the first join key for ord[0], ord[1]
    // three inputs: the attributes ord[2] shares with ord[0] or ord[1], in
    // ord[2]'s column order, each supplied by ord[0] if it has it, else ord[1]
    std::vector<int> join2;
    int join2_bits = 0;
    KeyPack join2_a{}, join2_b{}, join2_c{};
    KeyPack out_k[3]{};      // output-key bit fields each input supplies (spec order)
    int out_bits = 0;
    KeyUnpack unpack{};
    int64_t out_bounds[kMaxCols] = {};
    int uw = 0;
    bool ident_u = false, ident_v = false, ident_c = false;   // input already ordered by its join key
};

// An input whose keys are sorted and whose leading key columns are the join
// attributes, in order, is already grouped by join key.
bool leading_cols(const Spec &s, const ucl_rel *R, int k, const std::vector<int> &labs) {
    if (labs.empty()) return true;
    if (!R->sorted) return false;
    for (size_t q = 0; q < labs.size(); ++q)
        if (s.labs[labs[q]].pos[k] != (int)q) return false;
    return true;
}

int shared_bits(const Spec &s, int a, int b) {
    int t = 0;
    for (const Label &L : s.labs)
        if (L.upper && L.pos[a] >= 0 && L.pos[b] >= 0) t += bit_width(L.ext);
    return t;
}

ucl_status plan_keys(ucl_ctx *ctx, const Spec &s, ucl_rel *const *in, KeyPlan &kp) {
    const int n = s.n_in;
    if (n == 3) {
        // join first the two inputs that share the most key bits (a pair that
        // shares none would be a cross product)
        const int pairs[3][3] = {{0, 1, 2}, {0, 2, 1}, {1, 2, 0}};
        int best = 0, bb = -1;
        for (int q = 0; q < 3; ++q) {
            int b = shared_bits(s, pairs[q][0], pairs[q][1]);
            if (b > bb) { bb = b; best = q; }
        }
        for (int q = 0; q < 3; ++q) kp.ord[q] = pairs[best][q];
    }
    // output key: W's upper labels, first most significant
    std::vector<int> wl;
    for (char c : s.out) {
        int L = s.find(c);
        if (s.labs[L].upper) wl.push_back(L);
    }
    kp.uw = (int)wl.size();
    int total = 0;
    for (int L : wl) total += bit_width(s.labs[L].ext);
    if (total > 64) return fail(ctx, UCL_ERR_UNSUPPORTED, "output key needs more than 64 bits");
    kp.out_bits = total;
    kp.unpack.uw = kp.uw;
    int shift = total;
    for (int q = 0; q < kp.uw; ++q) {
        const Label &L = s.labs[wl[q]];
        int b = bit_width(L.ext);
        shift -= b;
        kp.unpack.shift[q] = shift;
        kp.unpack.bits[q] = b;
        kp.out_bounds[q] = L.ext;
        // supplier: the first input in join order that has the label
        for (int j = 0; j < n; ++j) {
            const int k = kp.ord[j];
            if (L.pos[k] >= 0) {
                kp.out_k[k].f[kp.out_k[k].nf++] = KeyField{L.pos[k], shift, b};
                break;
            }
        }
    }
    if (n < 2) return UCL_OK;
    const int ka = kp.ord[0], kb = kp.ord[1];
    // first join: upper labels of both inputs, in ord[0]'s order
    for (char c : s.op[ka]) {
        int L = s.find(c);
        if (s.labs[L].upper && s.labs[L].pos[kb] >= 0) kp.join.push_back(L);
    }
    total = 0;
    for (int L : kp.join) total += bit_width(s.labs[L].ext);
    if (total > 64) return fail(ctx, UCL_ERR_UNSUPPORTED, "join key needs more than 64 bits");
    kp.join_bits = total;
    shift = total;
    for (int L : kp.join) {
        int b = bit_width(s.labs[L].ext);
        shift -= b;
        kp.join_u.f[kp.join_u.nf++] = KeyField{s.labs[L].pos[ka], shift, b};
        kp.join_v.f[kp.join_v.nf++] = KeyField{s.labs[L].pos[kb], shift, b};
    }
    kp.ident_u = leading_cols(s, in[ka], ka, kp.join);
    kp.ident_v = leading_cols(s, in[kb], kb, kp.join);
    if (n < 3) return UCL_OK;
    const int kc = kp.ord[2];
    for (char c : s.op[kc]) {
        int L = s.find(c);
        if (s.labs[L].upper && (s.labs[L].pos[ka] >= 0 || s.labs[L].pos[kb] >= 0)) kp.join2.push_back(L);
    }
    total = 0;
    for (int L : kp.join2) total += bit_width(s.labs[L].ext);
    if (total > 64) return fail(ctx, UCL_ERR_UNSUPPORTED, "join key needs more than 64 bits");
    kp.join2_bits = total;
    shift = total;
    for (int L : kp.join2) {
        const Label &M = s.labs[L];
        int b = bit_width(M.ext);
        shift -= b;
        kp.join2_c.f[kp.join2_c.nf++] = KeyField{M.pos[kc], shift, b};
        if (M.pos[ka] >= 0)
            kp.join2_a.f[kp.join2_a.nf++] = KeyField{M.pos[ka], shift, b};
        else
            kp.join2_b.f[kp.join2_b.nf++] = KeyField{M.pos[kb], shift, b};
    }
    kp.ident_c = leading_cols(s, in[kc], kc, kp.join2);
    return UCL_OK;
}

ucl_status plan_lower(ucl_ctx *ctx, const Spec &s, ucl_rel *const *in, LowerPlan &lp) {
    memset(&lp, 0, sizeof(lp));
    lp.tile_u = in[0]->tile;
    lp.tile_v = s.n_in > 1 ? in[1]->tile : 1;
    lp.tile_x = s.n_in > 2 ? in[2]->tile : 1;
    lp.tile_w = 1;
    for (char c : s.out) {
        const Label &L = s.labs[s.find(c)];
        if (L.upper) continue;
        lp.w_ext[lp.nw] = (int)L.ext;
        lp.w_su[lp.nw] = (int)tile_stride(s, 0, L);
        lp.w_sv[lp.nw] = s.n_in > 1 ? (int)tile_stride(s, 1, L) : 0;
        lp.w_sx[lp.nw] = s.n_in > 2 ? (int)tile_stride(s, 2, L) : 0;
        lp.tile_w *= L.ext;
        lp.nw++;
    }
    lp.n_c = 1;
    for (const Label &L : s.labs) {
        if (L.upper || L.pos[3] >= 0) continue;
        if (lp.nc >= kMaxLow) return fail(ctx, UCL_ERR_UNSUPPORTED, "too many contracted labels");
        lp.c_ext[lp.nc] = (int)L.ext;
        lp.c_su[lp.nc] = (int)tile_stride(s, 0, L);
        lp.c_sv[lp.nc] = s.n_in > 1 ? (int)tile_stride(s, 1, L) : 0;
        lp.c_sx[lp.nc] = s.n_in > 2 ? (int)tile_stride(s, 2, L) : 0;
        lp.n_c *= L.ext;
        lp.nc++;
    }
    if (lp.tile_w >= (1ll << 31) || lp.tile_u >= (1ll << 31) || lp.tile_v >= (1ll << 31) ||
        lp.tile_x >= (1ll << 31))
        return fail(ctx, UCL_ERR_UNSUPPORTED, "tile has 2^31 or more elements");
    return UCL_OK;
}

// tcgen05 shape: exactly one M label (lower, in A and W), one N label (lower,
// in B and W) and one K label (lower, in A and B), nothing else lower; both
// operands bf16.  The operand giving the larger M-side extent becomes A.
bool plan_tc(const Spec &s, ucl_rel *const *in, TcPlan &tp, std::string *why) {
    memset(&tp, 0, sizeof(tp));
    if (s.n_in != 2) { *why = "not a binary EinSum"; return false; }
    if (in[0]->dtype != UCL_BF16 || in[1]->dtype != UCL_BF16) { *why = "operands are not bf16"; return false; }
    int mu = -1, nv = -1, kk = -1;
    for (size_t i = 0; i < s.labs.size(); ++i) {
        const Label &L = s.labs[i];
        if (L.upper) continue;
        bool a = L.pos[0] >= 0, b = L.pos[1] >= 0, w = L.pos[3] >= 0;
        if (a && !b && w) { if (mu >= 0) { *why = "several labels of U's output side"; return false; } mu = (int)i; }
        else if (!a && b && w) { if (nv >= 0) { *why = "several labels of V's output side"; return false; } nv = (int)i; }
        else if (a && b && !w) { if (kk >= 0) { *why = "several contracted labels"; return false; } kk = (int)i; }
        else { *why = "batch or single-operand lower labels"; return false; }
    }
    if (mu < 0 || nv < 0 || kk < 0) { *why = "tile kernel is not a GEMM"; return false; }
    const Label &Lu = s.labs[mu], &Lv = s.labs[nv], &Lk = s.labs[kk];
    // A gets the side with an extent of 128 or 256; prefer U on ties
    auto m_ok = [](int64_t e) { return e == 128 || e == 256; };
    auto n_ok = [](int64_t e) { return e >= 16 && e <= 256 && e % 16 == 0; };
    if (m_ok(Lu.ext) && n_ok(Lv.ext)) tp.a_is_u = 1;
    else if (m_ok(Lv.ext) && n_ok(Lu.ext)) tp.a_is_u = 0;
    else { *why = "M/N extents do not fit tcgen05 (M 128|256, N 16..256 step 16)"; return false; }
    if (Lk.ext != 16 && Lk.ext != 32 && Lk.ext != 64 && Lk.ext != 128 && Lk.ext != 256) {
        *why = "K extent must be 16, 32, 64, 128 or 256";
        return false;
    }
    const int ka = tp.a_is_u ? 0 : 1, kb = 1 - ka;
    const Label &LM = tp.a_is_u ? Lu : Lv, &LN = tp.a_is_u ? Lv : Lu;
    tp.M = (int)LM.ext;
    tp.N = (int)LN.ext;
    tp.K = (int)Lk.ext;
    tp.m_blocks = tp.M / 128;
    // K-major when K is the fastest tile dim of the operand
    tp.a_kmajor = Lk.pos[ka] > LM.pos[ka];
    tp.b_kmajor = Lk.pos[kb] > LN.pos[kb];
    tp.sWm = tile_stride(s, 3, LM);
    tp.sWn = tile_stride(s, 3, LN);
    return true;
}

// Three inputs of the MTTKRP shape: T with lower labels (i, e, f) or
// (f, i, e) in that tile order, factor E with e and r, factor F with f and r laid out [f][r],
// output with i and r; no other lower label; extents i = e = f = 16,
// r = 64; all bf16.  E is the factor of the first join when T is in it (its
// tuple changes least often along the pair list).
bool plan_tc3(const Spec &s, ucl_rel *const *in, const KeyPlan &kp, Tc3Plan &tp, std::string *why) {
    memset(&tp, 0, sizeof(tp));
    if (s.n_in != 3) { *why = "not a three-input EinSum"; return false; }
    for (int k = 0; k < 3; ++k)
        if (in[k]->dtype != UCL_BF16) { *why = "operands are not bf16"; return false; }
    tp.t = -1;
    for (int k = 0; k < 3; ++k)
        if (in[k]->r == 3) tp.t = k;
    if (tp.t < 0 || in[(tp.t + 1) % 3]->r != 2 || in[(tp.t + 2) % 3]->r != 2) {
        *why = "not one 3-d tile and two 2-d factor tiles";
        return false;
    }
    const int t = tp.t;
    // the label at each T tile position; the factor holding each
    int lab[3] = {-1, -1, -1};
    for (size_t i = 0; i < s.labs.size(); ++i)
        if (!s.labs[i].upper && s.labs[i].pos[t] >= 0) lab[s.labs[i].pos[t]] = (int)i;
    // T laid out [i][e][f] (f fastest: a K-major MMA operand with 32-byte
    // rows) or [f][i][e] ((i, e) contiguous: an MN-major operand with
    // 128-byte rows); i is the output label
    tp.t_mn = s.labs[lab[0]].pos[3] < 0 && s.labs[lab[1]].pos[3] >= 0;
    const int li = tp.t_mn ? lab[1] : lab[0], le = tp.t_mn ? lab[2] : lab[1], lf = tp.t_mn ? lab[0] : lab[2];
    const Label &Li = s.labs[li], &Le = s.labs[le], &Lf = s.labs[lf];
    int fe = -1, ff = -1;
    for (int k = 0; k < 3; ++k) {
        if (k == t) continue;
        if (Le.pos[k] >= 0) fe = k;
        if (Lf.pos[k] >= 0) ff = k;
    }
    if (Li.pos[3] < 0 || Le.pos[3] >= 0 || Lf.pos[3] >= 0 || fe < 0 || ff < 0 || fe == ff ||
        Li.pos[fe] >= 0 || Li.pos[ff] >= 0 || Le.pos[ff] >= 0 || Lf.pos[fe] >= 0) {
        *why = "tile kernel is not MTTKRP-shaped";
        return false;
    }
    int rl = -1;
    for (size_t i = 0; i < s.labs.size(); ++i) {
        const Label &L = s.labs[i];
        if (L.upper || (int)i == lab[0] || (int)i == lab[1] || (int)i == lab[2]) continue;
        if (rl >= 0 || L.pos[fe] < 0 || L.pos[ff] < 0 || L.pos[3] < 0) {
            *why = "tile kernel is not MTTKRP-shaped";
            return false;
        }
        rl = (int)i;
    }
    if (rl < 0) { *why = "no rank label"; return false; }
    const Label &Lr = s.labs[rl];
    if (Li.ext != 16 || Le.ext != 16 || Lf.ext != 16 || Lr.ext != 64) {
        *why = "extents must be i = j = k = 16, r = 64";
        return false;
    }
    if (Lf.pos[ff] != 0 || Lr.pos[ff] != 1) { *why = "F tile must be laid out [k][r]"; return false; }
    (void)kp;
    tp.e = fe;
    tp.f = ff;
    tp.sEj = tile_stride(s, fe, Le);
    tp.sEr = tile_stride(s, fe, Lr);
    tp.sWi = tile_stride(s, 3, Li);
    tp.sWr = tile_stride(s, 3, Lr);
    return true;
}

// --------------------------------------------------------------- helpers

size_t dsize(ucl_dtype d) { return d == UCL_BF16 ? 2 : 4; }

// Banding of the contracted label.  When U (the operand whose tuples each
// join many V tuples) is larger than L2, the contraction re-reads U's tiles
// from HBM: the pairs of one output key visit the whole range of the join
// label, and all CTAs together sweep all of U at every moment.  Cutting the
// leading join label into B ranges (bands) whose share of U fits L2, and
// contracting band after band, keeps U's working set in L2.  Each band sums
// into fp32 partials keyed (band, output key), and a band sum adds them in
// band order.  The EinSum computed is unchanged: the band is an extra upper
// label of the partial output, derived from the join label and summed out
// again (the Sec. 5 template applied twice, with part of the contracted label
// promoted in between).  The band field is packed above the output key, from
// the top bits of U's join label.
struct BandPlan {
    int B = 1, bits = 0;
};

constexpr int kMaxBands = 16;   // 2 (B + 1) band ranges are read in one sizing sync
constexpr int64_t kSegUnitPairs = 16384;   // pair lists up to this size are cut at segment boundaries

BandPlan plan_bands(ucl_ctx *ctx, const Spec &s, ucl_rel *const *in, KeyPlan &kp, bool tc_ok) {
    BandPlan bp;
    if (s.n_in != 2 || !tc_ok || kp.join.empty() || ctx->tune_bands == 0 || ctx->tune_bands == 1) return bp;
    const Label &L = s.labs[kp.join[0]];
    const int ku = kp.ord[0];
    if (L.pos[3] >= 0 || kp.out_k[ku].nf >= kMaxCols) return bp;   // the join label is kept in the output
    const ucl_rel *U = in[ku], *V = in[kp.ord[1]];
    const double ubytes = (double)U->n * (double)U->tile * (double)dsize(U->dtype);
    const int jb = bit_width(L.ext);
    int B = 1;
    if (ctx->tune_bands > 1) {
        B = std::min(ctx->tune_bands, kMaxBands);
    } else {
        // bands of at most twice the L2 size: with the streamed operand's
        // loads marked evict-first, the reused operand's band then mostly
        // hits L2 (more bands add (band, key) partials for little gain)
        const double l2 = ctx->l2_bytes > 0 ? (double)ctx->l2_bytes : 126e6;
        if (!(ubytes > 2 * l2 && V->n >= 4 * U->n)) return bp;
        while (B < kMaxBands && ubytes / B > 2 * l2) B *= 2;
    }
    int bits = 0;
    while ((1 << bits) < B) ++bits;
    if (bits > jb) bits = jb;
    if (bits == 0 || kp.out_bits + bits > 64) return bp;
    bp.B = 1 << bits;
    bp.bits = bits;
    kp.out_k[ku].f[kp.out_k[ku].nf++] = KeyField{L.pos[ku], kp.out_bits, bits, jb - bits};
    return bp;
}

// Windows of output keys for the windowed tcgen05 kernel: the pairs of 2^wb
// consecutive output keys accumulate in one TMEM buffer of 2^wb slots, so
// that the pairs of one A tuple within a window load its tile once.  It pays
// when A's tuples are each joined many times and A's tile is at least B's;
// windows of as many keys as two buffers hold.  Returns wb (0: none) and the
// kernel's run cap.
int plan_windows(ucl_ctx *ctx, const Spec &s, ucl_rel *const *in, const KeyPlan &kp, const TcPlan &tp, bool tc_ok,
                 int *cap) {
    *cap = 0;
    if (s.n_in != 2 || !tc_ok || ctx->tune_window == 0) return 0;
    const ucl_rel *RA = tp.a_is_u ? in[0] : in[1], *RB = tp.a_is_u ? in[1] : in[0];
    if ((reinterpret_cast<uintptr_t>(RA->tiles) | reinterpret_cast<uintptr_t>(RB->tiles)) & 15) return 0;
    int wb = 0;
    if (ctx->tune_window > 0) {
        wb = ctx->tune_window;
    } else {
        // not chosen automatically: measured slower than the plain kernel
        // on the message-passing shapes (see the design notes)
        (void)RB;
        return 0;
    }
    if (wb < 1 || wb > 5 || wb > kp.out_bits) return 0;
    const int c = tc_window_cap(tp, wb);
    if (c < 1) return 0;
    *cap = c;
    return wb;
}

// Take the next workspace arena in turn.  The stream in use first waits until
// main has finished the call that used it last; a grown arena is merged into
// one block.
int arena_begin(ucl_ctx *ctx) {
    const int a = ctx->arena_next;
    ctx->arena_next = (a + 1) % ucl_ctx::kArenas;
    ctx->arena = &ctx->arenas[a];
    if (ctx->stream != ctx->main) cudaStreamWaitEvent(ctx->stream, ctx->arena_done[a], 0);
    Arena &A = *ctx->arena;
    if (A.blocks.size() > 1) {
        size_t total = A.total();
        for (auto &b : A.blocks) ctx_free(ctx, b.ptr, b.size);
        A.blocks.clear();
        char *p = (char *)ctx_alloc(ctx, total);
        if (p) A.blocks.push_back({p, total});
    }
    A.used = 0;
    return a;
}

// Events of a timed call: [0] key stage start, [1] after the join count,
// [2] after the segments (key stream), [3] before the contraction, [4] after
// it, [5] after the fixup (main).  Stage s spans events kStageFrom[s] ..
// kStageFrom[s] + 1.
constexpr int kCallEvents = 6;
constexpr int kStageFrom[UCL_NSTAGES] = {0, 1, 3, 4};

void record(ucl_ctx *ctx, int i) {
    if (ctx->cur_ev) cudaEventRecord(ctx->cur_ev[i], ctx->stream);
}

// Claim the events of one timed call (grows the pool on demand).
ucl_status begin_timed_call(ucl_ctx *ctx) {
    ctx->cur_ev = nullptr;
    if (!ctx->timing) return UCL_OK;
    const size_t per = kCallEvents, need = per * (ctx->ev_calls + 1);
    while (ctx->ev_pool.size() < need) {
        cudaEvent_t e;
        ucl_status st = cuda_check(ctx, cudaEventCreate(&e), "cudaEventCreate");
        if (st) return st;
        ctx->ev_pool.push_back(e);
    }
    ctx->cur_ev = &ctx->ev_pool[per * ctx->ev_calls];
    ctx->ev_calls++;
    return UCL_OK;
}

// Read n int64 device scalars after draining the stream in use.  Word 1 of
// the device status holds validation flags (returned in *flags, cleared);
// word 2 holds error bits raised by earlier main-stream kernels of this
// context, sticky until a read on main reports and clears them (a key-stream
// read reports them if already set but leaves the word to main, whose kernels
// may still be writing it).
ucl_status sync_read(ucl_ctx *ctx, const int64_t *dev, int n, int64_t *host, uint32_t *flags = nullptr) {
    cudaError_t e = cudaSuccess;
    if (n > ucl_ctx::kPinnedRead) return fail(ctx, UCL_ERR_ARG, "too many values for one sizing sync");
    if (n > 0) e = cudaMemcpyAsync(ctx->h_pinned, dev, sizeof(int64_t) * n, cudaMemcpyDeviceToHost, ctx->stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(ctx->h_pinned + ucl_ctx::kPinnedRead, ctx->d_status, 4 * sizeof(uint32_t), cudaMemcpyDeviceToHost,
                            ctx->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(ctx->stream);
    if (e != cudaSuccess) return cuda_check(ctx, e, "stream sync");
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_check(ctx, e, "kernel launch");
    for (int i = 0; i < n; ++i) host[i] = ctx->h_pinned[i];
    uint32_t words[4];
    memcpy(words, ctx->h_pinned + ucl_ctx::kPinnedRead, sizeof(words));
    if (flags) *flags = words[1];
    const bool on_main = ctx->stream == ctx->main;
    if (words[1]) cudaMemsetAsync(ctx->d_status + 1, 0, sizeof(uint32_t), ctx->stream);
    if (words[2] && on_main) cudaMemsetAsync(ctx->d_status + 2, 0, sizeof(uint32_t), ctx->stream);
    if (words[2] & kStTimeout) return fail(ctx, UCL_ERR_TIMEOUT, "a device-side wait timed out");
    if (words[2] & kStBadIndex) return fail(ctx, UCL_ERR_CUDA, "a device-side bounds check failed");
    return UCL_OK;
}

// Key stage of ucl_einsum on the key stream; back to main with main ordered
// after everything the key stream did so far.
void to_key_stream(ucl_ctx *ctx) { ctx->stream = ctx->kstream; }
void to_main(ucl_ctx *ctx) {
    if (ctx->stream == ctx->main) return;
    cudaEventRecord(ctx->ev_order, ctx->kstream);
    cudaStreamWaitEvent(ctx->main, ctx->ev_order, 0);
    ctx->stream = ctx->main;
}

// Relation keys became valid at this point of main.
void keys_ready(ucl_ctx *ctx, ucl_rel *R) {
    if (!R->ev_keys && cudaEventCreateWithFlags(&R->ev_keys, cudaEventDisableTiming) != cudaSuccess) {
        cudaGetLastError();
        R->ev_keys = nullptr;
        return;
    }
    cudaEventRecord(R->ev_keys, ctx->main);
}

// The stream in use waits until a relation's keys are valid (main order when
// it has no event).
void wait_keys(ucl_ctx *ctx, const ucl_rel *R) {
    if (ctx->stream == ctx->main) return;
    if (R->ev_keys) cudaStreamWaitEvent(ctx->stream, R->ev_keys, 0);
    else order_after_main(ctx);
}

struct Fail {
    ucl_status st;
};

// Throw on error so that the stage schedule can bail out from any depth.
void check(ucl_status st) {
    if (st != UCL_OK) throw Fail{st};
}

ucl_rel *new_rel(ucl_ctx *ctx) {
    ucl_rel *r = new (std::nothrow) ucl_rel();
    if (r) {
        r->ctx = ctx;
        ctx->live_rels++;
    }
    return r;
}

KeyPack full_pack(const ucl_rel *R, int *bits) {
    KeyPack kp{};
    int total = 0;
    for (int c = 0; c < R->u; ++c) total += bit_width(R->bounds[c]);
    *bits = total;
    int shift = total;
    for (int c = 0; c < R->u; ++c) {
        int b = bit_width(R->bounds[c]);
        shift -= b;
        kp.f[kp.nf++] = KeyField{c, shift, b};
    }
    return kp;
}

}  // namespace

// =================================================================== ucl::

namespace ucl {

int bit_width(int64_t bound) {
    int b = 0;
    while (b < 63 && ((int64_t)1 << b) < bound) ++b;
    return b;
}

ucl_status fail(ucl_ctx *ctx, ucl_status st, const std::string &msg) {
    if (ctx) ctx->err = msg;
    return st;
}

ucl_status cuda_check(ucl_ctx *ctx, cudaError_t e, const char *what) {
    if (e == cudaSuccess) return UCL_OK;
    cudaGetLastError();
    return fail(ctx, UCL_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

void order_after_main(ucl_ctx *ctx) {
    if (ctx->stream == ctx->main) return;
    cudaEventRecord(ctx->ev_order, ctx->main);
    cudaStreamWaitEvent(ctx->stream, ctx->ev_order, 0);
}

// Device memory comes and goes in main's order (the allocator hooks' stream,
// or the stream-ordered pool on main).  A block handed out while the key
// stream is in use may have been freed on main with main's readers still
// queued: the key stream is ordered after main first.
void *ctx_alloc(ucl_ctx *ctx, size_t bytes) {
    if (bytes == 0) bytes = 256;
    bytes = (bytes + 255) & ~(size_t)255;
    void *p = nullptr;
    if (ctx->alloc) {
        p = ctx->alloc(bytes, ctx->user);
    } else if (cudaMallocAsync(&p, bytes, ctx->main) != cudaSuccess) {
        cudaGetLastError();
        p = nullptr;
    }
    if (p) order_after_main(ctx);
    return p;
}

void ctx_free(ucl_ctx *ctx, void *p, size_t bytes) {
    if (!p) return;
    bytes = (bytes + 255) & ~(size_t)255;
    if (ctx->free_fn) ctx->free_fn(p, bytes, ctx->user);
    else cudaFreeAsync(p, ctx->main);
}

void *ws_get(ucl_ctx *ctx, size_t bytes) {
    Arena &A = *ctx->arena;
    bytes = (bytes + 255) & ~(size_t)255;
    if (bytes == 0) bytes = 256;
    if (A.blocks.empty() || A.used + bytes > A.blocks.back().size) {
        size_t want = std::max(bytes, std::max((size_t)(1 << 22), A.total()));
        char *p = (char *)ctx_alloc(ctx, want);
        if (!p) throw Oom();
        A.blocks.push_back({p, want});
        A.used = 0;
    }
    char *p = A.blocks.back().ptr + A.used;
    A.used += bytes;
    return p;
}

}  // namespace ucl

// ===================================================================== ABI

extern "C" {

const char *ucl_status_str(ucl_status st) {
    switch (st) {
        case UCL_OK: return "UCL_OK";
        case UCL_ERR_ARG: return "UCL_ERR_ARG";
        case UCL_ERR_SPEC: return "UCL_ERR_SPEC";
        case UCL_ERR_SHAPE: return "UCL_ERR_SHAPE";
        case UCL_ERR_DUP_KEY: return "UCL_ERR_DUP_KEY";
        case UCL_ERR_KEY_RANGE: return "UCL_ERR_KEY_RANGE";
        case UCL_ERR_OOM: return "UCL_ERR_OOM";
        case UCL_ERR_CUDA: return "UCL_ERR_CUDA";
        case UCL_ERR_UNSUPPORTED: return "UCL_ERR_UNSUPPORTED";
        case UCL_ERR_TIMEOUT: return "UCL_ERR_TIMEOUT";
    }
    return "UCL_ERR_UNKNOWN";
}

const char *ucl_last_error(const ucl_ctx *ctx) { return ctx ? ctx->err.c_str() : "NULL context"; }

ucl_status ucl_ctx_create(int device, void *stream, ucl_alloc_fn alloc, ucl_free_fn free_fn, void *user,
                          ucl_ctx **out) {
    if (!out) return UCL_ERR_ARG;
    *out = nullptr;
    if ((alloc == nullptr) != (free_fn == nullptr)) return UCL_ERR_ARG;
    ucl_ctx *ctx = new (std::nothrow) ucl_ctx();
    if (!ctx) return UCL_ERR_OOM;
    ctx->device = device;
    ctx->stream = ctx->main = (cudaStream_t)stream;
    ctx->alloc = alloc;
    ctx->free_fn = free_fn;
    ctx->user = user;
    ucl_status st = cuda_check(ctx, cudaSetDevice(device), "cudaSetDevice");
    if (!st) st = cuda_check(ctx, cudaDeviceGetAttribute(&ctx->sm_count, cudaDevAttrMultiProcessorCount, device),
                             "device attribute");
    if (!st && !alloc) {
        // default allocator: keep freed blocks in the device's pool across syncs
        cudaMemPool_t pool;
        st = cuda_check(ctx, cudaDeviceGetDefaultMemPool(&pool, device), "cudaDeviceGetDefaultMemPool");
        uint64_t keep = ~0ull;
        if (!st) st = cuda_check(ctx, cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep),
                                 "cudaMemPoolSetAttribute");
    }
    if (!st && cudaDeviceGetAttribute(&ctx->l2_bytes, cudaDevAttrL2CacheSize, device) != cudaSuccess) {
        cudaGetLastError();
        ctx->l2_bytes = 0;
    }
    if (const char *e = getenv("UCL_BANDS")) ctx->tune_bands = atoi(e);
    if (const char *e = getenv("UCL_L2_HINTS")) ctx->tune_hints = atoi(e);
    if (const char *e = getenv("UCL_TC_STAGES")) ctx->tune_tc_stages = atoi(e);
    if (const char *e = getenv("UCL_SEG_UNITS")) ctx->tune_seg_units = atoi(e);
    if (const char *e = getenv("UCL_TC_MMA")) ctx->tune_tc_mma = atoi(e);
    if (const char *e = getenv("UCL_TC_PREFETCH")) ctx->tune_tc_prefetch = atoi(e);
    if (const char *e = getenv("UCL_WINDOW")) ctx->tune_window = atoi(e);
    if (!st) st = cuda_check(ctx, cudaMalloc(&ctx->d_status, 256), "cudaMalloc status");
    if (!st) st = cuda_check(ctx, cudaMemset(ctx->d_status, 0, 256), "cudaMemset status");
    if (!st) st = cuda_check(ctx, cudaMallocHost(&ctx->h_pinned, ucl_ctx::kPinnedWords * sizeof(int64_t)), "cudaMallocHost");
    if (!st) st = cuda_check(ctx, cudaStreamCreateWithFlags(&ctx->kstream, cudaStreamNonBlocking), "cudaStreamCreate");
    if (!st) st = cuda_check(ctx, cudaEventCreateWithFlags(&ctx->ev_order, cudaEventDisableTiming), "cudaEventCreate");
    if (!st) st = cuda_check(ctx, cudaStreamCreateWithFlags(&ctx->cstream, cudaStreamNonBlocking), "cudaStreamCreate");
    if (!st) st = cuda_check(ctx, cudaEventCreateWithFlags(&ctx->ev_copy0, cudaEventDisableTiming), "cudaEventCreate");
    if (!st) st = cuda_check(ctx, cudaEventCreateWithFlags(&ctx->ev_copy1, cudaEventDisableTiming), "cudaEventCreate");
    for (int i = 0; i < ucl_ctx::kArenas && !st; ++i)
        st = cuda_check(ctx, cudaEventCreateWithFlags(&ctx->arena_done[i], cudaEventDisableTiming), "cudaEventCreate");
    if (st) {
        if (ctx->d_status) cudaFree(ctx->d_status);
        if (ctx->h_pinned) cudaFreeHost(ctx->h_pinned);
        if (ctx->kstream) cudaStreamDestroy(ctx->kstream);
        if (ctx->ev_order) cudaEventDestroy(ctx->ev_order);
        if (ctx->cstream) cudaStreamDestroy(ctx->cstream);
        if (ctx->ev_copy0) cudaEventDestroy(ctx->ev_copy0);
        if (ctx->ev_copy1) cudaEventDestroy(ctx->ev_copy1);
        for (cudaEvent_t e : ctx->arena_done)
            if (e) cudaEventDestroy(e);
        delete ctx;
        return st;
    }
    *out = ctx;
    return UCL_OK;
}

ucl_status ucl_ctx_destroy(ucl_ctx *ctx) {
    if (!ctx) return UCL_ERR_ARG;
    if (ctx->live_rels) return fail(ctx, UCL_ERR_ARG, "relations still alive on this context");
    cudaStreamSynchronize(ctx->kstream);
    cudaStreamSynchronize(ctx->main);
    ctx->stream = ctx->main;
    for (Arena &A : ctx->arenas)
        for (auto &b : A.blocks) ctx_free(ctx, b.ptr, b.size);
    cudaStreamSynchronize(ctx->main);
    cudaFree(ctx->d_status);
    cudaFreeHost(ctx->h_pinned);
    cudaStreamDestroy(ctx->kstream);
    cudaStreamSynchronize(ctx->cstream);
    cudaStreamDestroy(ctx->cstream);
    cudaEventDestroy(ctx->ev_order);
    cudaEventDestroy(ctx->ev_copy0);
    cudaEventDestroy(ctx->ev_copy1);
    for (cudaEvent_t e : ctx->arena_done) cudaEventDestroy(e);
    for (cudaEvent_t e : ctx->ev_pool) cudaEventDestroy(e);
    delete ctx;
    return UCL_OK;
}

ucl_status ucl_ctx_set_timing(ucl_ctx *ctx, int enable) {
    if (!ctx) return UCL_ERR_ARG;
    ctx->timing = enable ? 1 : 0;
    return UCL_OK;
}

ucl_status ucl_ctx_synchronize(ucl_ctx *ctx) {
    if (!ctx) return UCL_ERR_ARG;
    cudaSetDevice(ctx->device);
    cudaError_t e = cudaStreamSynchronize(ctx->kstream);
    if (e != cudaSuccess) return cuda_check(ctx, e, "stream sync");
    ctx->stream = ctx->main;
    return sync_read(ctx, nullptr, 0, nullptr);
}

ucl_status ucl_get_last_stats(ucl_ctx *ctx, ucl_stats *out) {
    if (!ctx || !out) return UCL_ERR_ARG;
    if (ctx->last.timed && ctx->cur_ev) {
        cudaError_t e = cudaEventSynchronize(ctx->cur_ev[kCallEvents - 1]);
        if (e != cudaSuccess) return cuda_check(ctx, e, "event sync");
        for (int i = 0; i < UCL_NSTAGES; ++i)
            cudaEventElapsedTime(&ctx->last.stage_ms[i], ctx->cur_ev[kStageFrom[i]], ctx->cur_ev[kStageFrom[i] + 1]);
    }
    *out = ctx->last;
    return UCL_OK;
}

ucl_status ucl_ctx_timings(ucl_ctx *ctx, float *ms, int max_calls, int *n_calls, int reset) {
    if (!ctx || (max_calls > 0 && !ms)) return UCL_ERR_ARG;
    const int per = kCallEvents;
    if (n_calls) *n_calls = ctx->ev_calls;
    if (ctx->ev_calls > 0 && max_calls > 0) {
        cudaError_t e = cudaEventSynchronize(ctx->ev_pool[(size_t)per * ctx->ev_calls - 1]);
        if (e != cudaSuccess) return cuda_check(ctx, e, "event sync");
        for (int c = 0; c < ctx->ev_calls && c < max_calls; ++c)
            for (int i = 0; i < UCL_NSTAGES; ++i)
                cudaEventElapsedTime(&ms[c * UCL_NSTAGES + i], ctx->ev_pool[(size_t)per * c + kStageFrom[i]],
                                     ctx->ev_pool[(size_t)per * c + kStageFrom[i] + 1]);
    }
    if (reset) {
        ctx->ev_calls = 0;
        ctx->cur_ev = nullptr;
        ctx->last.timed = 0;
    }
    return UCL_OK;
}

ucl_status ucl_ctx_set_wait_limit(ucl_ctx *ctx, int64_t cycles) {
    if (!ctx || cycles < 0) return fail(ctx, UCL_ERR_ARG, "bad wait limit");
    ctx->wait_limit_cycles = cycles;
    return UCL_OK;
}

ucl_status ucl_ctx_withhold_stage(ucl_ctx *ctx, int fill) {
    if (!ctx || fill < -1) return fail(ctx, UCL_ERR_ARG, "bad stage fill");
    ctx->withhold_fill = fill;
    return UCL_OK;
}

ucl_status ucl_ctx_fixup_bytes(ucl_ctx *ctx, int64_t *bytes, int reset) {
    if (!ctx || !bytes) return fail(ctx, UCL_ERR_ARG, "NULL context or output");
    cudaSetDevice(ctx->device);
    unsigned long long *d = reinterpret_cast<unsigned long long *>(ctx->d_status + ucl_ctx::kFixupCounterWord);
    unsigned long long h = 0;
    cudaError_t e = cudaMemcpyAsync(&h, d, sizeof(h), cudaMemcpyDeviceToHost, ctx->main);
    if (e == cudaSuccess) e = cudaStreamSynchronize(ctx->main);
    if (e == cudaSuccess && reset) e = cudaMemsetAsync(d, 0, sizeof(h), ctx->main);
    if (e != cudaSuccess) return cuda_check(ctx, e, "fixup byte counter");
    *bytes = (int64_t)h;
    return UCL_OK;
}

ucl_status ucl_relation_create(ucl_ctx *ctx, int64_t n, int u, const int32_t *keys, const int64_t *key_bounds,
                               int r, const int64_t *tile_shape, ucl_dtype dtype, const void *tiles, ucl_mem mem,
                               ucl_rel **out) {
    if (!out) return fail(ctx, UCL_ERR_ARG, "out is NULL");
    *out = nullptr;
    if (!ctx) return UCL_ERR_ARG;
    if (n < 0 || u < 0 || u > kMaxCols || r < 0 || r > kMaxCols) return fail(ctx, UCL_ERR_ARG, "bad n, u or r");
    if (dtype != UCL_BF16 && dtype != UCL_F32) return fail(ctx, UCL_ERR_ARG, "bad dtype");
    if (mem != UCL_MEM_DEVICE_BORROW && mem != UCL_MEM_DEVICE_COPY && mem != UCL_MEM_HOST_COPY)
        return fail(ctx, UCL_ERR_ARG, "bad mem");
    if ((u > 0 && !key_bounds) || (r > 0 && !tile_shape)) return fail(ctx, UCL_ERR_ARG, "bounds/shape is NULL");
    if (n > 0 && ((u > 0 && !keys) || !tiles)) return fail(ctx, UCL_ERR_ARG, "keys/tiles is NULL");
    if (n >= (1ll << 32) - 1) return fail(ctx, UCL_ERR_UNSUPPORTED, "2^32 or more tuples");
    cudaSetDevice(ctx->device);
    ucl_rel tmp;
    tmp.ctx = ctx;
    tmp.n = n;
    tmp.u = u;
    tmp.r = r;
    tmp.dtype = dtype;
    for (int c = 0; c < u; ++c) {
        if (key_bounds[c] < 1 || key_bounds[c] > (1ll << 31)) return fail(ctx, UCL_ERR_ARG, "key bound out of [1, 2^31]");
        tmp.bounds[c] = key_bounds[c];
    }
    tmp.tile = 1;
    for (int q = 0; q < r; ++q) {
        if (tile_shape[q] < 1) return fail(ctx, UCL_ERR_SHAPE, "tile extent < 1");
        tmp.shape[q] = tile_shape[q];
        tmp.tile *= tile_shape[q];
        if (tmp.tile >= (1ll << 31)) return fail(ctx, UCL_ERR_UNSUPPORTED, "tile has 2^31 or more elements");
    }
    KeyPack fp = full_pack(&tmp, &tmp.key_bits);
    if (tmp.key_bits > 64) return fail(ctx, UCL_ERR_UNSUPPORTED, "key columns need more than 64 bits");
    if (u == 0 && n > 1) return fail(ctx, UCL_ERR_DUP_KEY, "more than one tuple in a key-less relation");

    size_t kbytes = (size_t)n * u * sizeof(int32_t), tbytes = (size_t)n * tmp.tile * dsize(dtype);
    size_t koff = (tbytes + 255) & ~(size_t)255;
    bool copying = false;   // a tile copy is in flight on the copy stream
    if (mem == UCL_MEM_DEVICE_BORROW) {
        tmp.keys = const_cast<int32_t *>(keys);
        tmp.tiles = const_cast<void *>(tiles);
    } else if (n > 0) {
        tmp.own_bytes = koff + kbytes;
        tmp.own_block = ctx_alloc(ctx, tmp.own_bytes);
        if (!tmp.own_block) return fail(ctx, UCL_ERR_OOM, "allocation of relation storage failed");
        tmp.tiles = tmp.own_block;
        tmp.keys = (int32_t *)((char *)tmp.own_block + koff);
        cudaMemcpyKind kind = mem == UCL_MEM_HOST_COPY ? cudaMemcpyHostToDevice : cudaMemcpyDeviceToDevice;
        // The tile copy goes on the copy stream, ordered after main's earlier
        // work (the block may be one main freed a moment ago), so that the key
        // copy and validation below run on main while it is in flight.  Main
        // is ordered after the copy before this call returns.
        cudaError_t e = cudaEventRecord(ctx->ev_copy0, ctx->stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(ctx->cstream, ctx->ev_copy0, 0);
        if (e == cudaSuccess) e = cudaMemcpyAsync(tmp.tiles, tiles, tbytes, kind, ctx->cstream);
        if (e == cudaSuccess) e = cudaEventRecord(ctx->ev_copy1, ctx->cstream);
        if (e == cudaSuccess) copying = true;
        if (e == cudaSuccess && kbytes) e = cudaMemcpyAsync(tmp.keys, keys, kbytes, kind, ctx->stream);
        if (e != cudaSuccess) {
            if (copying) cudaStreamWaitEvent(ctx->stream, ctx->ev_copy1, 0);
            ctx_free(ctx, tmp.own_block, tmp.own_bytes);
            return cuda_check(ctx, e, "copy of relation storage");
        }
    }
    tmp.sorted = 1;
    ucl_status st = UCL_OK;
    ucl_rel *R = nullptr;
    if (n > 0 && u > 0) {
        const int arena = arena_begin(ctx);
        try {
            uint64_t *packed = (uint64_t *)ws_get(ctx, sizeof(uint64_t) * n);
            launch_check_keys(ctx, tmp.keys, u, n, tmp.bounds, fp, packed);
            uint32_t flags = 0;
            st = sync_read(ctx, nullptr, 0, nullptr, &flags);
            if (!st && (flags & kStKeyRange)) st = fail(ctx, UCL_ERR_KEY_RANGE, "key outside [0, bound)");
            if (!st && (flags & kStUnsorted)) {
                tmp.sorted = 0;
                uint64_t *alt = (uint64_t *)ws_get(ctx, sizeof(uint64_t) * n);
                int which = radix_sort(ctx, packed, nullptr, alt, nullptr, n, tmp.key_bits);
                launch_check_dups(ctx, which ? alt : packed, n);
                st = sync_read(ctx, nullptr, 0, nullptr, &flags);
                if (!st && (flags & kStDupKey)) st = fail(ctx, UCL_ERR_DUP_KEY, "duplicate key");
            }
        } catch (Oom &) {
            st = fail(ctx, UCL_ERR_OOM, "workspace allocation failed");
        }
        cudaEventRecord(ctx->arena_done[arena], ctx->main);
    }
    if (!st && !(R = new_rel(ctx))) st = fail(ctx, UCL_ERR_OOM, "host allocation failed");
    if (st) {
        if (copying) cudaStreamWaitEvent(ctx->stream, ctx->ev_copy1, 0);
        if (tmp.own_block) ctx_free(ctx, tmp.own_block, tmp.own_bytes);
        return st;
    }
    *R = tmp;
    // keys are valid here: the key stream may start on them while the tile
    // copy is still in flight; main (contractions, frees) waits for the copy
    keys_ready(ctx, R);
    if (copying) {
        cudaStreamWaitEvent(ctx->stream, ctx->ev_copy1, 0);
        // host memory may be reused as soon as this call returns
        if (mem == UCL_MEM_HOST_COPY) {
            cudaError_t e = cudaEventSynchronize(ctx->ev_copy1);
            if (e != cudaSuccess) {
                ucl_relation_destroy(R);
                return cuda_check(ctx, e, "copy of relation storage");
            }
        }
    }
    *out = R;
    ctx->err.clear();
    return UCL_OK;
}

ucl_status ucl_relation_destroy(ucl_rel *rel) {
    if (!rel) return UCL_ERR_ARG;
    ucl_ctx *ctx = rel->ctx;
    if (rel->own_block) ctx_free(ctx, rel->own_block, rel->own_bytes);
    if (rel->ev_keys) cudaEventDestroy(rel->ev_keys);
    ctx->live_rels--;
    delete rel;
    return UCL_OK;
}

ucl_status ucl_relation_info(const ucl_rel *rel, int64_t *n, int *u, int *r, int64_t *key_bounds,
                             int64_t *tile_shape, ucl_dtype *dtype) {
    if (!rel) return UCL_ERR_ARG;
    if (n) *n = rel->n;
    if (u) *u = rel->u;
    if (r) *r = rel->r;
    if (key_bounds) for (int c = 0; c < rel->u; ++c) key_bounds[c] = rel->bounds[c];
    if (tile_shape) for (int q = 0; q < rel->r; ++q) tile_shape[q] = rel->shape[q];
    if (dtype) *dtype = rel->dtype;
    return UCL_OK;
}

ucl_status ucl_relation_data(const ucl_rel *rel, const int32_t **keys, const void **tiles) {
    if (!rel) return UCL_ERR_ARG;
    if (keys) *keys = rel->keys;
    if (tiles) *tiles = rel->tiles;
    return UCL_OK;
}

ucl_status ucl_relation_download(const ucl_rel *rel, int32_t *keys_host, void *tiles_host) {
    if (!rel) return UCL_ERR_ARG;
    ucl_ctx *ctx = rel->ctx;
    cudaSetDevice(ctx->device);
    cudaError_t e = cudaSuccess;
    if (keys_host && rel->n * rel->u > 0)
        e = cudaMemcpyAsync(keys_host, rel->keys, sizeof(int32_t) * rel->n * rel->u, cudaMemcpyDeviceToHost,
                            ctx->stream);
    if (e == cudaSuccess && tiles_host && rel->n > 0)
        e = cudaMemcpyAsync(tiles_host, rel->tiles, dsize(rel->dtype) * rel->n * rel->tile, cudaMemcpyDeviceToHost,
                            ctx->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(ctx->stream);
    return cuda_check(ctx, e, "download");
}

ucl_status ucl_einsum(ucl_ctx *ctx, const char *spec_text, int n_in, ucl_rel *const *in, const ucl_einsum_opts *opts,
                      ucl_rel **out) {
    if (!out) return fail(ctx, UCL_ERR_ARG, "out is NULL");
    *out = nullptr;
    if (!ctx || !in) return fail(ctx, UCL_ERR_ARG, "NULL context or inputs");
    ucl_einsum_opts o{UCL_F32, UCL_EPI_NONE, 1.0f, UCL_PATH_AUTO, UCL_AGG_SUM, UCL_COMB_MUL, UCL_MAP_IDENT};
    if (opts) o = *opts;
    if ((o.out_dtype != UCL_BF16 && o.out_dtype != UCL_F32) || (o.epi != UCL_EPI_NONE && o.epi != UCL_EPI_RELU) ||
        o.path < UCL_PATH_AUTO || o.path > UCL_PATH_TC || o.agg < UCL_AGG_SUM || o.agg > UCL_AGG_MIN ||
        o.comb < UCL_COMB_MUL || o.comb > UCL_COMB_DIV || o.map < UCL_MAP_IDENT || o.map > UCL_MAP_SQUARE)
        return fail(ctx, UCL_ERR_ARG, "bad options");
    // the extended EinSum (anything but a sum of products) runs on the FFMA path
    const bool extended = o.agg != UCL_AGG_SUM || o.map != UCL_MAP_IDENT || (n_in > 1 && o.comb != UCL_COMB_MUL);
    if (extended && n_in == 3) return fail(ctx, UCL_ERR_UNSUPPORTED, "three inputs take the sum of products only");
    if (extended && o.path == UCL_PATH_TC)
        return fail(ctx, UCL_ERR_UNSUPPORTED, "tcgen05 path: the sum of products only");
    Spec s;
    ucl_status st = parse_spec(ctx, spec_text, n_in, s);
    if (st) return st;
    if ((st = bind_extents(ctx, s, in))) return st;
    KeyPlan kp;
    if ((st = plan_keys(ctx, s, in, kp))) return st;
    LowerPlan lp;
    if ((st = plan_lower(ctx, s, in, lp))) return st;
    TcPlan tp;
    Tc3Plan tp3;
    std::string why;
    const bool tc_ok = !extended && (n_in == 3 ? plan_tc3(s, in, kp, tp3, &why) : plan_tc(s, in, tp, &why));
    if (o.path == UCL_PATH_TC && !tc_ok) return fail(ctx, UCL_ERR_UNSUPPORTED, "tcgen05 path: " + why);
    const BandPlan bp = plan_bands(ctx, s, in, kp, tc_ok && o.path != UCL_PATH_SIMT);
    int win_cap = 0;
    const int wb = n_in == 2 ? plan_windows(ctx, s, in, kp, tp, tc_ok && o.path != UCL_PATH_SIMT, &win_cap) : 0;
    const bool banded = bp.B > 1;
    const int sort_bits = kp.out_bits + bp.bits;
    cudaSetDevice(ctx->device);

    const ucl_rel *U = in[0];
    const ucl_rel *V = n_in > 1 ? in[1] : nullptr;
    const ucl_rel *X = n_in > 2 ? in[2] : nullptr;
    const int64_t nU = U->n, nV = V ? V->n : 1, nX = X ? X->n : 1;
    // join order: A = ord[0], B = ord[1], C = ord[2] (spec order for < 3 inputs)
    const ucl_rel *A = in[kp.ord[0]], *B = n_in > 1 ? in[kp.ord[1]] : nullptr, *C = n_in > 2 ? in[kp.ord[2]] : nullptr;
    const int64_t nA = A->n, nB = B ? B->n : 1, nC = C ? C->n : 1;
    ucl_stats stats{};
    ctx->launches = 0;
    ucl_rel *R = nullptr;
    if ((st = begin_timed_call(ctx))) return st;
    // The key stage (stages 0 and 1 and the segment pass) runs on the key
    // stream, so that it overlaps the contraction of the previous call still
    // queued on main; the output relation, the contraction and the fixup are
    // on main.
    to_key_stream(ctx);
    const int arena = arena_begin(ctx);
    for (int k = 0; k < n_in; ++k) wait_keys(ctx, in[k]);
    try {
        record(ctx, 0);
        // [0] pair count, [1] segment count, [2] triple count or, banded,
        // [2, 2 + B] band starts and [3 + B, 3 + 2B] their segment indices,
        // [39] banded: output key count
        int64_t *d_scal = (int64_t *)ws_get(ctx, 40 * sizeof(int64_t));
        // ---------------------------------------------------------- stage 0
        // pack keys; sort each side of a join by its join key unless it is
        // already grouped; count the joined pairs (for three inputs: the
        // pairs of the first join, then the triples)
        int64_t P = 0, P1 = 0;
        // small binary EinSums: the whole key stage in one CTA and one sync;
        // more pairs than it holds fall through to the general path
        bool small = false;
        int64_t *sm_seg = nullptr;
        int32_t *sm_keys = nullptr;
        uint32_t *sm_pu = nullptr, *sm_pv = nullptr;
        int64_t sm_S = 0;
        if (n_in == 2 && !banded && wb == 0 && small_join_fits(nA, nB)) {
            sm_seg = (int64_t *)ws_get(ctx, 8 * (kSmallPairs + 1));
            sm_keys = (int32_t *)ws_get(ctx, 4 * (size_t)kSmallPairs * (kp.uw > 0 ? kp.uw : 1));
            sm_pu = (uint32_t *)ws_get(ctx, 4 * kSmallPairs);
            sm_pv = (uint32_t *)ws_get(ctx, 4 * kSmallPairs);
            launch_small_join(ctx, A->keys, A->u, nA, B->keys, B->u, nB, kp.join_u, kp.join_v, kp.out_k[kp.ord[0]],
                              kp.out_k[kp.ord[1]], kp.unpack, !kp.join.empty(), d_scal, sm_seg, sm_keys, sm_pu,
                              sm_pv);
            int64_t h[2] = {0, 0};
            check(sync_read(ctx, d_scal, 2, h));
            if (h[0] <= kSmallPairs) {
                small = true;
                P = h[0];
                sm_S = h[1];
            }
        }
        uint64_t *koA = nullptr, *koB = nullptr, *koC = nullptr;
        uint64_t *permA = nullptr, *permB = nullptr, *permC = nullptr;
        int64_t *off = nullptr, *off2 = nullptr;
        uint32_t *lo = nullptr, *lo2 = nullptr;
        uint64_t *pk1 = nullptr, *pv1 = nullptr;
        auto sort_by = [&](uint64_t *&jk, int64_t cnt, int bits, uint64_t *&perm) {
            uint64_t *vals = (uint64_t *)ws_get(ctx, 8 * cnt), *ka = (uint64_t *)ws_get(ctx, 8 * cnt),
                     *va = (uint64_t *)ws_get(ctx, 8 * cnt);
            launch_iota(ctx, vals, cnt);
            if (radix_sort(ctx, jk, vals, ka, va, cnt, bits)) { jk = ka; perm = va; } else perm = vals;
        };
        auto sync_count = [&](int64_t *dev) {
            int64_t h = 0;
            check(sync_read(ctx, dev, 1, &h));
            if (h >= (1ll << 31)) check(fail(ctx, UCL_ERR_UNSUPPORTED, "more than 2^31-1 joined pairs"));
            return h;
        };
        if (small) {
            record(ctx, 1);
        } else if (nA > 0 && nB > 0 && nC > 0) {
            koA = (uint64_t *)ws_get(ctx, 8 * nA);
            uint64_t *jkA = B ? (uint64_t *)ws_get(ctx, 8 * nA) : nullptr;
            launch_pack(ctx, A->keys, A->u, nA, kp.join_u, jkA, kp.out_k[kp.ord[0]], koA);
            if (!B) {
                record(ctx, 1);
                P = nA;
            } else {
                koB = (uint64_t *)ws_get(ctx, 8 * nB);
                uint64_t *jkB = (uint64_t *)ws_get(ctx, 8 * nB);
                launch_pack(ctx, B->keys, B->u, nB, kp.join_v, jkB, kp.out_k[kp.ord[1]], koB);
                const bool join = !kp.join.empty();
                if (join && !kp.ident_u) sort_by(jkA, nA, kp.join_bits, permA);
                if (join && !kp.ident_v) sort_by(jkB, nB, kp.join_bits, permB);
                int64_t *cnt = (int64_t *)ws_get(ctx, 8 * nA);
                lo = (uint32_t *)ws_get(ctx, 4 * nA);
                off = (int64_t *)ws_get(ctx, 8 * nA);
                launch_join_count(ctx, join ? jkA : nullptr, nA, join ? jkB : nullptr, nB, cnt, lo);
                scan_i64(ctx, cnt, off, nA, d_scal);
                if (!C) {
                    record(ctx, 1);
                    P = sync_count(d_scal);
                } else if ((P1 = sync_count(d_scal)) > 0) {
                    // second join: each pair's key on the attributes C shares
                    pk1 = (uint64_t *)ws_get(ctx, 8 * P1);
                    pv1 = (uint64_t *)ws_get(ctx, 8 * P1);
                    launch_expand(ctx, off, nA, lo, permA, permB, koA, koB, P1, pk1, pv1);
                    koC = (uint64_t *)ws_get(ctx, 8 * nC);
                    uint64_t *jkC = (uint64_t *)ws_get(ctx, 8 * nC);
                    launch_pack(ctx, C->keys, C->u, nC, kp.join2_c, jkC, kp.out_k[kp.ord[2]], koC);
                    const bool join2 = !kp.join2.empty();
                    uint64_t *jkP = nullptr;
                    if (join2) {
                        uint64_t *ja = nullptr, *jb = nullptr;
                        if (kp.join2_a.nf) {
                            ja = (uint64_t *)ws_get(ctx, 8 * nA);
                            launch_pack(ctx, A->keys, A->u, nA, kp.join2_a, ja, KeyPack{}, nullptr);
                        }
                        if (kp.join2_b.nf) {
                            jb = (uint64_t *)ws_get(ctx, 8 * nB);
                            launch_pack(ctx, B->keys, B->u, nB, kp.join2_b, jb, KeyPack{}, nullptr);
                        }
                        jkP = (uint64_t *)ws_get(ctx, 8 * P1);
                        launch_pair_keys(ctx, pv1, P1, ja, jb, jkP);
                        if (!kp.ident_c) sort_by(jkC, nC, kp.join2_bits, permC);
                    }
                    int64_t *cnt2 = (int64_t *)ws_get(ctx, 8 * P1);
                    lo2 = (uint32_t *)ws_get(ctx, 4 * P1);
                    off2 = (int64_t *)ws_get(ctx, 8 * P1);
                    launch_join_count(ctx, jkP, P1, join2 ? jkC : nullptr, nC, cnt2, lo2);
                    scan_i64(ctx, cnt2, off2, P1, d_scal + 2);
                    record(ctx, 1);
                    P = sync_count(d_scal + 2);
                } else {
                    record(ctx, 1);
                }
            }
        } else {
            record(ctx, 1);
        }

        // ---------------------------------------------------------- stage 1
        int64_t S = 0;
        int64_t band_start[kMaxBands + 1] = {}, band_seg[kMaxBands + 1] = {};
        int64_t *flag = nullptr;
        uint64_t *pk = nullptr, *pv = nullptr;
        int64_t *seg_excl = nullptr;
        if (P > 0 && !small) {
            pk = (uint64_t *)ws_get(ctx, 8 * P);
            pv = (uint64_t *)ws_get(ctx, 8 * P);
            uint64_t *pk2 = (uint64_t *)ws_get(ctx, 8 * P), *pv2 = (uint64_t *)ws_get(ctx, 8 * P);
            if (C)
                launch_expand3(ctx, off2, P1, lo2, permC, pk1, koC, P, pk, pv);
            else if (B)
                launch_expand(ctx, off, nA, lo, permA, permB, koA, koB, P, pk, pv);
            else
                launch_unary_pairs(ctx, koA, P, pk, pv);
            // Pairs are expanded in A's row order (each A row's partners
            // contiguous).  When A is visited in its own ascending key order
            // and alone supplies the output key, as its leading key columns,
            // the pairs are already in output-key order: the stable sort
            // would leave them as they are, so it is skipped.
            // (pairs in output-key order are also in window order; sharing
            // of A tiles only needs equal A tuples to be adjacent to pay)
            bool presorted = A->sorted && permA == nullptr && !banded;
            for (int k = 1; k < n_in && presorted; ++k) presorted = kp.out_k[kp.ord[k]].nf == 0;
            for (int q = 0; q < kp.out_k[kp.ord[0]].nf && presorted; ++q)
                presorted = kp.out_k[kp.ord[0]].f[q].col == q;
            // windows: sort by (band, output key >> wb) only, keeping the
            // expansion order (A tuple order) inside a window
            if (!presorted && radix_sort(ctx, pk, pv, pk2, pv2, P, sort_bits - wb, wb)) { pk = pk2; pv = pv2; }
            flag = (int64_t *)ws_get(ctx, 8 * P);
            seg_excl = (int64_t *)ws_get(ctx, 8 * P);
            launch_heads(ctx, pk, P, flag, wb);
            scan_i64(ctx, flag, seg_excl, P, d_scal + 1);
            if (banded)
                launch_band_ranges(ctx, pk, P, seg_excl, d_scal + 1, kp.out_bits, bp.B, d_scal + 2, d_scal + 3 + bp.B);
            int64_t h[1 + 2 * (kMaxBands + 1)];
            check(sync_read(ctx, d_scal + 1, banded ? 1 + 2 * (bp.B + 1) : 1, h));
            S = h[0];
            for (int b = 0; banded && b <= bp.B; ++b) {
                band_start[b] = h[1 + b];
                band_seg[b] = h[2 + bp.B + b];
            }
        }

        // ------------------------------------------------------ segments
        // one pass over the sorted pairs: each segment's output key (into
        // the workspace; copied into the output relation on main) and
        // start, and each pair's input rows
        int64_t *seg_start = nullptr;
        uint32_t *pu = nullptr, *pvi = nullptr, *pxi = nullptr;
        int32_t *okeys = nullptr;
        if (small) {
            S = sm_S;
            seg_start = sm_seg;
            pu = sm_pu;
            pvi = sm_pv;
            okeys = sm_keys;
        } else if (P > 0) {
            seg_start = (int64_t *)ws_get(ctx, 8 * (S + 1));
            pu = (uint32_t *)ws_get(ctx, 4 * P);
            pvi = (uint32_t *)ws_get(ctx, 4 * P);
            pxi = X ? (uint32_t *)ws_get(ctx, 4 * P) : nullptr;
            okeys = (int32_t *)ws_get(ctx, 4 * (size_t)S * kp.uw);
            if (X) {
                uint32_t *const idx[3] = {pu, pvi, pxi};
                launch_segments3(ctx, pk, pv, pv1, seg_excl, P, S, kp.unpack, kp.ord, okeys, seg_start, idx);
            } else {
                launch_segments(ctx, pk, pv, seg_excl, P, S, kp.unpack, okeys, seg_start, pu, pvi, wb);
            }
        }
        // banded: the S (band, output key) segments hold fp32 partials; sort
        // them by (output key, band) and find the output keys
        // windows: per pair its slot and A-tile run, per window segment its
        // present slots and first row; rows are the (band and) output keys
        // present, in key order
        const int64_t Sseg = S;   // pair segments (windows when wb > 0)
        uint8_t *wslot = nullptr, *warun = nullptr;
        uint32_t *wmask = nullptr;
        int64_t *wbase = nullptr;
        uint64_t *rowkey = nullptr;
        int64_t rows = S;
        if (wb > 0 && P > 0) {
            wslot = (uint8_t *)ws_get(ctx, (size_t)P);
            warun = (uint8_t *)ws_get(ctx, (size_t)P);
            wmask = (uint32_t *)ws_get(ctx, 4 * (size_t)Sseg);
            int64_t *wcnt = (int64_t *)ws_get(ctx, 8 * (size_t)Sseg);
            wbase = (int64_t *)ws_get(ctx, 8 * (size_t)Sseg);
            check(cuda_check(ctx, cudaMemsetAsync(wmask, 0, 4 * (size_t)Sseg, ctx->stream), "memset"));
            launch_win_slots(ctx, pk, P, wb, flag, seg_excl, wslot, wmask);
            launch_win_count(ctx, wmask, Sseg, wcnt);
            scan_i64(ctx, wcnt, wbase, Sseg, d_scal + 38);
            launch_arun(ctx, tp.a_is_u ? pu : pvi, P, win_cap, warun);
            check(sync_read(ctx, d_scal + 38, 1, &rows));
            rowkey = (uint64_t *)ws_get(ctx, 8 * (size_t)rows);
            launch_win_rows(ctx, pk, seg_start, Sseg, wmask, wbase, wb, rowkey);
            if (!banded) {
                S = rows;
                okeys = (int32_t *)ws_get(ctx, 4 * (size_t)S * kp.uw);
                launch_unpack_keys(ctx, rowkey, S, kp.unpack, okeys);
            }
        }
        const int64_t Sp = rows;   // rows the contraction writes (band partials when banded)
        uint64_t *band_order = nullptr;
        int64_t *fstart = nullptr;
        if (banded && P > 0) {
            uint64_t *sk = (uint64_t *)ws_get(ctx, 8 * Sp), *sv = (uint64_t *)ws_get(ctx, 8 * Sp),
                     *sk2 = (uint64_t *)ws_get(ctx, 8 * Sp), *sv2 = (uint64_t *)ws_get(ctx, 8 * Sp);
            if (wb > 0)
                launch_band_keys(ctx, rowkey, nullptr, Sp, kp.out_bits, bp.bits, sk, sv);
            else
                launch_band_keys(ctx, pk, seg_start, Sp, kp.out_bits, bp.bits, sk, sv);
            if (radix_sort(ctx, sk, sv, sk2, sv2, Sp, sort_bits)) {
                sk = sk2;
                sv = sv2;
            }
            int64_t *flag2 = (int64_t *)ws_get(ctx, 8 * Sp), *excl2 = (int64_t *)ws_get(ctx, 8 * Sp);
            launch_heads(ctx, sk, Sp, flag2, bp.bits);
            scan_i64(ctx, flag2, excl2, Sp, d_scal + 39);
            int64_t hs = 0;
            check(sync_read(ctx, d_scal + 39, 1, &hs));
            S = hs;
            okeys = (int32_t *)ws_get(ctx, 4 * (size_t)S * kp.uw);
            fstart = (int64_t *)ws_get(ctx, 8 * (S + 1));
            launch_band_outputs(ctx, sk, excl2, Sp, S, bp.bits, kp.unpack, okeys, fstart);
            band_order = sv;
        }
        record(ctx, 2);
        to_main(ctx);

        // output relation: keys ascending by construction
        R = new_rel(ctx);
        if (!R) check(fail(ctx, UCL_ERR_OOM, "host allocation failed"));
        R->n = S;
        R->u = kp.uw;
        R->r = lp.nw;
        for (int q = 0; q < kp.uw; ++q) R->bounds[q] = kp.out_bounds[q];
        for (int q = 0; q < lp.nw; ++q) R->shape[q] = lp.w_ext[q];
        R->dtype = o.out_dtype;
        R->tile = lp.tile_w;
        R->sorted = 1;
        R->key_bits = kp.out_bits;
        if (S > 0) {
            size_t tbytes = (size_t)S * lp.tile_w * dsize(o.out_dtype);
            size_t koff = (tbytes + 255) & ~(size_t)255;
            R->own_bytes = koff + (size_t)S * kp.uw * 4;
            R->own_block = ctx_alloc(ctx, R->own_bytes);
            if (!R->own_block) throw Oom();
            R->tiles = R->own_block;
            R->keys = (int32_t *)((char *)R->own_block + koff);
            if (kp.uw > 0)
                check(cuda_check(ctx, cudaMemcpyAsync(R->keys, okeys, (size_t)S * kp.uw * 4,
                                                      cudaMemcpyDeviceToDevice, ctx->main), "copy of output keys"));
        }
        keys_ready(ctx, R);

        // ------------------------------------------------------ stage 2, 3
        record(ctx, 3);
        int path = UCL_PATH_SIMT;
        if (P > 0) {
            ContractArgs a{};
            a.U = U->tiles;
            a.V = V ? V->tiles : nullptr;
            a.X = X ? X->tiles : nullptr;
            a.du = U->dtype;
            a.dv = V ? V->dtype : U->dtype;
            a.dx = X ? X->dtype : U->dtype;
            a.nU = nU;
            a.nV = V ? nV : 0;
            a.nX = X ? nX : 0;
            a.pu = pu;
            a.pv = pvi;
            a.px = pxi;
            a.seg_start = seg_start;
            a.S = Sseg;
            a.out = R->tiles;
            a.dout = o.out_dtype;
            a.epi = o.epi;
            a.scale = o.scale;
            a.agg = o.agg;
            a.comb = o.comb;
            a.map = o.map;
            a.tile_w = lp.tile_w;
            a.fixup_bytes = reinterpret_cast<unsigned long long *>(ctx->d_status + ucl_ctx::kFixupCounterWord);
            bool use_tc = tc_ok && o.path != UCL_PATH_SIMT;
            if (use_tc && n_in < 3) {
                std::string why2;
                if (!tc_supported(tp, a, &why2)) {
                    if (o.path == UCL_PATH_TC) check(fail(ctx, UCL_ERR_UNSUPPORTED, "tcgen05 path: " + why2));
                    use_tc = false;
                }
            }
            if (wb > 0 && !use_tc) check(fail(ctx, UCL_ERR_UNSUPPORTED, "windowed pair list without the tcgen05 path"));
            int G = use_tc ? (n_in == 3 ? tc3_units(ctx, P) : tc_units(ctx, tp, P))
                           : (int)std::min<int64_t>(P, (int64_t)ctx->sm_count * 4);
            // On the tcgen05 path, small pair lists and lists of one pair per
            // segment are cut at segment boundaries (at most one unit per
            // segment): no segment needs a partial or the fixup launch, and a
            // unit's pairs stream through its pipeline either way.  The FFMA
            // kernels walk a unit's pairs one after another, so they keep the
            // even split (more, shorter units), as do banded and windowed
            // launches.
            const bool seg_units = use_tc && ctx->tune_seg_units != 0 && !banded && wb == 0 && Sseg > 0 &&
                                   (P <= kSegUnitPairs || P == Sseg);
            if (seg_units && G > Sseg) G = (int)Sseg;
            a.units.P = P;
            a.units.G = G;
            a.units.base = 0;
            a.units.seg = seg_units ? seg_start : nullptr;
            a.units.S = Sseg;
            a.bands = bp.B;
            a.l2_hints = ctx->tune_hints;
            stats.n_units = G;
            a.win_bits = wb;
            a.slot = wslot;
            a.arun = warun;
            a.wmask = wmask;
            a.wbase = wbase;
            a.share_cap = win_cap;
            a.partials = (float *)ws_get(ctx, sizeof(float) * 2 * (size_t)G * ((size_t)1 << wb) * lp.tile_w);
            auto contract = [&](const ContractArgs &c) {
                if (use_tc && n_in == 3) {
                    check(launch_contract_tc3(ctx, c, tp3, in));
                    path = UCL_PATH_TC;
                } else if (use_tc) {
                    const ucl_rel *ra = tp.a_is_u ? U : V, *rb = tp.a_is_u ? V : U;
                    check(launch_contract_tc(ctx, c, tp, ra, rb));
                    path = UCL_PATH_TC;
                } else {
                    launch_contract_simt(ctx, c, lp);
                }
            };
            if (!banded) {
                contract(a);
                record(ctx, 4);
                if (wb > 0)
                    launch_fixup_window(ctx, a);
                else if (!seg_units)
                    launch_fixup(ctx, a);
                record(ctx, 5);
            } else {
                // band after band into fp32 partials keyed (band, output
                // key), each band cut into its own G units; then the band sum
                const size_t pbytes = sizeof(float) * (size_t)Sp * lp.tile_w;
                float *part = (float *)ctx_alloc(ctx, pbytes);
                if (!part) throw Oom();
                for (int b = 0; b < bp.B; ++b) {
                    const int64_t Pb = band_start[b + 1] - band_start[b];
                    if (Pb <= 0) continue;
                    ContractArgs c = a;
                    c.seg_start = seg_start + band_seg[b];
                    c.S = band_seg[b + 1] - band_seg[b];
                    c.units.P = Pb;
                    c.units.seg = nullptr;
                    c.units.G = use_tc ? tc_units(ctx, tp, Pb) : (int)std::min<int64_t>(Pb, (int64_t)ctx->sm_count * 4);
                    c.units.base = band_start[b];
                    c.out = wb > 0 ? part : part + (size_t)band_seg[b] * lp.tile_w;
                    if (wb > 0) {
                        c.wmask = wmask + band_seg[b];
                        c.wbase = wbase + band_seg[b];
                    }
                    c.dout = UCL_F32;
                    c.epi = UCL_EPI_NONE;
                    c.scale = 1.0f;
                    contract(c);
                    if (wb > 0) launch_fixup_window(ctx, c); else launch_fixup(ctx, c);
                }
                record(ctx, 4);
                launch_band_sum(ctx, part, band_order, fstart, S, lp.tile_w, R->tiles, o.out_dtype, o.epi, o.scale,
                                a.fixup_bytes);
                record(ctx, 5);
                ctx_free(ctx, part, pbytes);
            }
        } else {
            record(ctx, 4);
            record(ctx, 5);
        }
        check(cuda_check(ctx, cudaGetLastError(), "kernel launch"));

        stats.n_pairs = P;
        stats.n_segments = S;
        stats.n_bands = bp.B;
        stats.n_band_segments = Sp;
        stats.flops = 2.0 * (double)P * (double)lp.tile_w * (double)lp.n_c;
        stats.bytes_contract = (double)nU * U->tile * dsize(U->dtype) +
                               (V ? (double)nV * V->tile * dsize(V->dtype) : 0.0) +
                               (X ? (double)nX * X->tile * dsize(X->dtype) : 0.0) +
                               (double)S * lp.tile_w * dsize(o.out_dtype) + 4.0 * n_in * (double)P;
        stats.path = path;
        stats.launches = ctx->launches;
        stats.timed = ctx->cur_ev != nullptr;
        ctx->last = stats;
        *out = R;
        R = nullptr;
        ctx->err.clear();
    } catch (Oom &) {
        st = fail(ctx, UCL_ERR_OOM, "device allocation failed");
    } catch (Fail &f) {
        st = f.st;
    }
    to_main(ctx);
    cudaEventRecord(ctx->arena_done[arena], ctx->main);
    if (R) ucl_relation_destroy(R);
    return st;
}

ucl_status ucl_repartition(ucl_ctx *ctx, const char *spec_text, const ucl_rel *in, ucl_rel **out) {
    if (!out) return fail(ctx, UCL_ERR_ARG, "out is NULL");
    *out = nullptr;
    if (!ctx || !in || !spec_text) return fail(ctx, UCL_ERR_ARG, "NULL context, relation or spec");
    if (in->ctx != ctx) return fail(ctx, UCL_ERR_ARG, "relation belongs to another context");
    // ------------------------------------------------------------ plan
    const std::string t(spec_text);
    const size_t arrow = t.find("->");
    if (arrow == std::string::npos) return fail(ctx, UCL_ERR_SPEC, "spec has no '->'");
    const std::string lhs = t.substr(0, arrow), rhs = t.substr(arrow + 2);
    auto lower = [](char c) { return (char)(c >= 'A' && c <= 'Z' ? c - 'A' + 'a' : c); };
    // labels are named by their input-side letter; the output side is either
    // "<keys>|<tile dims>" (input letters as written) or the input letters
    // with their case changed to the new class (compared without case)
    const size_t bar = rhs.find('|');
    const bool explicit_form = bar != std::string::npos;
    const std::string rhs_letters = explicit_form ? rhs.substr(0, bar) + rhs.substr(bar + 1) : rhs;
    for (size_t a = 0; a < lhs.size(); ++a) {
        if (!is_alpha(lhs[a])) return fail(ctx, UCL_ERR_SPEC, "labels must be letters");
        for (size_t b = a + 1; b < lhs.size(); ++b)
            if (lhs[a] == lhs[b] || (!explicit_form && lower(lhs[a]) == lower(lhs[b])))
                return fail(ctx, UCL_ERR_SPEC,
                            "a label appears twice on the input side (without '|' letters compare without case)");
    }
    for (char c : rhs_letters)
        if (!is_alpha(c)) return fail(ctx, UCL_ERR_SPEC, "labels must be letters");
    if (lhs.size() != rhs_letters.size()) return fail(ctx, UCL_ERR_SPEC, "both sides must hold the same labels");
    struct RL {
        char name;
        bool in_up, out_up;
        int in_pos, out_pos;
        int64_t ext;
    };
    std::vector<RL> labs;
    int iu = 0, il = 0;
    for (char c : lhs) {
        RL L{c, is_upper(c), false, is_upper(c) ? iu++ : il++, -1, 0};
        labs.push_back(L);
    }
    if (iu != in->u || il != in->r)
        return fail(ctx, UCL_ERR_SHAPE, "input side does not match the relation's key/tile arity");
    int ou = 0, ol = 0;
    for (size_t q = 0; q < rhs_letters.size(); ++q) {
        const char c = rhs_letters[q];
        RL *L = nullptr;
        for (RL &M : labs)
            if (explicit_form ? M.name == c : lower(M.name) == lower(c)) L = &M;
        if (!L || L->out_pos >= 0) return fail(ctx, UCL_ERR_SPEC, "both sides must hold the same labels");
        L->out_up = explicit_form ? q < bar : is_upper(c);
        L->out_pos = L->out_up ? ou++ : ol++;
    }
    for (RL &L : labs) L.ext = L.in_up ? in->bounds[L.in_pos] : in->shape[L.in_pos];
    auto by_out = [&](bool up) {
        std::vector<const RL *> v(up ? ou : ol);
        for (const RL &L : labs)
            if (L.out_up == up) v[L.out_pos] = &L;
        return v;
    };
    const std::vector<const RL *> oup = by_out(true), olow = by_out(false);
    int64_t tile_out = 1, np = 1;
    for (const RL *L : olow) tile_out *= L->ext;
    for (const RL *L : oup)
        if (!L->in_up) np *= L->ext;
    if (tile_out >= (1ll << 31) || np >= (1ll << 31)) return fail(ctx, UCL_ERR_UNSUPPORTED, "output tile too large");
    // output key packing (output order) and the kept-key packing (kept labels, output order)
    KeyUnpack un{};
    un.uw = ou;
    int total = 0;
    for (const RL *L : oup) total += bit_width(L->ext);
    if (total > 64) return fail(ctx, UCL_ERR_UNSUPPORTED, "output key needs more than 64 bits");
    RepartKeys rk{};
    rk.uw = ou;
    rk.np = np;
    KeyPack kpack{};
    int kbits_total = 0;
    for (const RL *L : oup)
        if (L->in_up) kbits_total += bit_width(L->ext);
    {
        int sh = total, ksh = kbits_total;
        int64_t pdiv = np;
        for (int q = 0; q < ou; ++q) {
            const RL &L = *oup[q];
            const int b = bit_width(L.ext);
            sh -= b;
            un.shift[q] = sh;
            un.bits[q] = b;
            rk.osh[q] = sh;
            rk.promoted[q] = !L.in_up;
            if (L.in_up) {
                ksh -= b;
                rk.ksh[q] = ksh;
                rk.kbits[q] = b;
                kpack.f[kpack.nf++] = KeyField{L.in_pos, ksh, b};
            } else {
                pdiv /= L.ext;
                rk.pdiv[q] = pdiv;
                rk.pext[q] = L.ext;
            }
        }
    }
    // element routing
    RepartCopy pc{};
    pc.r = in->r;
    pc.u = in->u;
    pc.tile_in = in->tile;
    pc.tile_out = tile_out;
    pc.np = np;
    auto out_stride = [&](const RL &L) {
        int64_t st = 1;
        for (int q = ol - 1; q > L.out_pos; --q) st *= olow[q]->ext;
        return st;
    };
    for (const RL &L : labs) {
        if (L.in_up) {
            pc.kstride[L.in_pos] = L.out_up ? 0 : out_stride(L);
        } else {
            pc.ext[L.in_pos] = L.ext;
            pc.ostride[L.in_pos] = L.out_up ? 0 : out_stride(L);
            if (L.out_up) pc.pstride[L.in_pos] = rk.pdiv[L.out_pos];
        }
    }
    // kept labels lead the output key, in the input's leading columns' order?
    bool kept_first = true, kept_leading = true;
    {
        bool seen_promoted = false;
        int kq = 0;
        for (const RL *L : oup) {
            if (!L->in_up) seen_promoted = true;
            else {
                if (seen_promoted) kept_first = false;
                if (L->in_pos != kq) kept_leading = false;
                ++kq;
            }
        }
    }
    cudaSetDevice(ctx->device);
    ucl_stats stats{};
    ctx->launches = 0;
    ucl_rel *R = nullptr;
    ucl_status st;
    if ((st = begin_timed_call(ctx))) return st;
    const int arena = arena_begin(ctx);
    try {
        record(ctx, 0);
        int64_t *d_scal = (int64_t *)ws_get(ctx, 8 * sizeof(int64_t));
        const int64_t n = in->n;
        // distinct kept keys and each tuple's rank among them
        int64_t kd = 0;
        uint32_t *rank = nullptr;
        uint64_t *dk = nullptr;
        if (n > 0) {
            rank = (uint32_t *)ws_get(ctx, 4 * n);
            if (kpack.nf == 0) {
                kd = 1;
                check(cuda_check(ctx, cudaMemsetAsync(rank, 0, 4 * n, ctx->stream), "cudaMemsetAsync"));
                record(ctx, 1);
            } else {
                uint64_t *kk = (uint64_t *)ws_get(ctx, 8 * n), *perm = nullptr;
                launch_pack(ctx, in->keys, in->u, n, kpack, kk, KeyPack{}, nullptr);
                if (!(in->sorted && kept_leading)) {
                    uint64_t *vals = (uint64_t *)ws_get(ctx, 8 * n), *ka = (uint64_t *)ws_get(ctx, 8 * n),
                             *va = (uint64_t *)ws_get(ctx, 8 * n);
                    launch_iota(ctx, vals, n);
                    if (radix_sort(ctx, kk, vals, ka, va, n, kbits_total)) { kk = ka; perm = va; } else perm = vals;
                }
                int64_t *flag = (int64_t *)ws_get(ctx, 8 * n), *excl = (int64_t *)ws_get(ctx, 8 * n);
                launch_heads(ctx, kk, n, flag);
                scan_i64(ctx, flag, excl, n, d_scal);
                dk = (uint64_t *)ws_get(ctx, 8 * n);
                launch_kept_rank(ctx, kk, flag, excl, perm, n, rank, dk);
                record(ctx, 1);
                check(sync_read(ctx, d_scal, 1, &kd));
            }
        } else {
            record(ctx, 1);
        }
        const int64_t n_out = kd * np;
        if (n_out >= (1ll << 31)) check(fail(ctx, UCL_ERR_UNSUPPORTED, "more than 2^31-1 output tuples"));
        R = new_rel(ctx);
        if (!R) check(fail(ctx, UCL_ERR_OOM, "host allocation failed"));
        R->n = n_out;
        R->u = ou;
        R->r = ol;
        for (int q = 0; q < ou; ++q) R->bounds[q] = oup[q]->ext;
        for (int q = 0; q < ol; ++q) R->shape[q] = olow[q]->ext;
        R->dtype = in->dtype;
        R->tile = tile_out;
        R->sorted = 1;
        R->key_bits = total;
        const size_t es = dsize(in->dtype);
        if (n_out > 0) {
            size_t tbytes = (size_t)n_out * tile_out * es;
            size_t koff = (tbytes + 255) & ~(size_t)255;
            R->own_bytes = koff + (size_t)n_out * ou * 4 + 4;
            R->own_block = ctx_alloc(ctx, R->own_bytes);
            if (!R->own_block) throw Oom();
            R->tiles = R->own_block;
            R->keys = (int32_t *)((char *)R->own_block + koff);
            // output keys; slot order is key order when the kept labels lead
            uint64_t *okey = (uint64_t *)ws_get(ctx, 8 * n_out);
            uint32_t *pos = nullptr;
            if (kept_first) {
                launch_out_keys(ctx, dk, n_out, rk, okey, nullptr);
                launch_out_place(ctx, okey, nullptr, n_out, un, nullptr, R->keys);
            } else {
                uint64_t *iota = (uint64_t *)ws_get(ctx, 8 * n_out), *ka = (uint64_t *)ws_get(ctx, 8 * n_out),
                         *va = (uint64_t *)ws_get(ctx, 8 * n_out);
                launch_out_keys(ctx, dk, n_out, rk, okey, iota);
                if (radix_sort(ctx, okey, iota, ka, va, n_out, total)) { okey = ka; iota = va; }
                pos = (uint32_t *)ws_get(ctx, 4 * n_out);
                launch_out_place(ctx, okey, iota, n_out, un, pos, R->keys);
            }
            record(ctx, 2);
            record(ctx, 3);
            // every input element to its place; positions no element maps to
            // exist only when labels are stacked, and are zero
            bool stacked = false;
            for (const RL &L : labs) stacked |= L.in_up && !L.out_up;
            if (stacked)
                check(cuda_check(ctx, cudaMemsetAsync(R->tiles, 0, tbytes, ctx->stream), "cudaMemsetAsync"));
            launch_repart_scatter(ctx, in->tiles, in->dtype, in->keys, rank, pos, n, pc, R->tiles);
            record(ctx, 4);
        } else {
            record(ctx, 2);
            record(ctx, 3);
            record(ctx, 4);
        }
        record(ctx, 5);
        keys_ready(ctx, R);
        check(cuda_check(ctx, cudaGetLastError(), "kernel launch"));
        stats.n_pairs = n;
        stats.n_segments = n_out;
        stats.flops = 0.0;
        stats.bytes_contract = (double)n * in->tile * es + (double)n_out * tile_out * es + 4.0 * n * in->u +
                               4.0 * n_out * ou;
        stats.path = UCL_PATH_SIMT;
        stats.launches = ctx->launches;
        stats.timed = ctx->cur_ev != nullptr;
        ctx->last = stats;
        *out = R;
        R = nullptr;
        ctx->err.clear();
        st = UCL_OK;
    } catch (Oom &) {
        st = fail(ctx, UCL_ERR_OOM, "device allocation failed");
    } catch (Fail &f) {
        st = f.st;
    }
    cudaEventRecord(ctx->arena_done[arena], ctx->main);
    if (R) ucl_relation_destroy(R);
    return st;
}

ucl_status ucl_relation_stats(ucl_ctx *ctx, const ucl_rel *rel, int64_t *nnz, int64_t *distinct) {
    if (!ctx || !rel) return fail(ctx, UCL_ERR_ARG, "NULL context or relation");
    if (rel->ctx != ctx) return fail(ctx, UCL_ERR_ARG, "relation belongs to another context");
    cudaSetDevice(ctx->device);
    StatsGeom g;
    stats_geometry(rel, g);
    const int nc = rel->u + rel->r;
    ucl_status st = UCL_OK;
    const int arena = arena_begin(ctx);
    try {
        int64_t *d = (int64_t *)ws_get(ctx, sizeof(int64_t) * (1 + nc));
        uint32_t *bits = (uint32_t *)ws_get(ctx, sizeof(uint32_t) * (size_t)std::max<int64_t>(g.words, 1));
        check(cuda_check(ctx, cudaMemsetAsync(d, 0, sizeof(int64_t) * (1 + nc), ctx->stream), "cudaMemsetAsync"));
        if (g.words > 0)
            check(cuda_check(ctx, cudaMemsetAsync(bits, 0, sizeof(uint32_t) * g.words, ctx->stream),
                             "cudaMemsetAsync"));
        launch_relation_stats(ctx, rel, g, bits, reinterpret_cast<unsigned long long *>(d), nullptr);
        launch_popc(ctx, bits, g, d + 1);
        int64_t h[1 + 2 * kMaxCols];
        check(sync_read(ctx, d, 1 + nc, h));
        if (nnz) *nnz = h[0];
        if (distinct)
            for (int c = 0; c < nc; ++c) distinct[c] = h[1 + c];
        ctx->err.clear();
    } catch (Oom &) {
        st = fail(ctx, UCL_ERR_OOM, "device allocation failed");
    } catch (Fail &f) {
        st = f.st;
    }
    cudaEventRecord(ctx->arena_done[arena], ctx->main);
    return st;
}

ucl_status ucl_drop_zero_tiles(ucl_ctx *ctx, const ucl_rel *in, ucl_rel **out) {
    if (!out) return fail(ctx, UCL_ERR_ARG, "out is NULL");
    *out = nullptr;
    if (!ctx || !in) return fail(ctx, UCL_ERR_ARG, "NULL context or relation");
    if (in->ctx != ctx) return fail(ctx, UCL_ERR_ARG, "relation belongs to another context");
    cudaSetDevice(ctx->device);
    ucl_status st = UCL_OK;
    ucl_rel *R = nullptr;
    const int arena = arena_begin(ctx);
    try {
        const int64_t n = in->n;
        int64_t m = 0;
        int64_t *flag = nullptr, *excl = nullptr;
        if (n > 0) {
            int64_t *d_total = (int64_t *)ws_get(ctx, sizeof(int64_t));
            flag = (int64_t *)ws_get(ctx, sizeof(int64_t) * n);
            excl = (int64_t *)ws_get(ctx, sizeof(int64_t) * n);
            check(cuda_check(ctx, cudaMemsetAsync(flag, 0, sizeof(int64_t) * n, ctx->stream), "cudaMemsetAsync"));
            StatsGeom g;
            stats_geometry(in, g);
            g.smem_dims = 0;
            launch_relation_stats(ctx, in, g, nullptr, nullptr, flag);
            scan_i64(ctx, flag, excl, n, d_total);
            check(sync_read(ctx, d_total, 1, &m));
        }
        R = new_rel(ctx);
        if (!R) check(fail(ctx, UCL_ERR_OOM, "host allocation failed"));
        R->n = m;
        R->u = in->u;
        R->r = in->r;
        for (int c = 0; c < in->u; ++c) R->bounds[c] = in->bounds[c];
        for (int q = 0; q < in->r; ++q) R->shape[q] = in->shape[q];
        R->dtype = in->dtype;
        R->tile = in->tile;
        R->sorted = in->sorted;
        R->key_bits = in->key_bits;
        if (m > 0) {
            const size_t tbytes = (size_t)m * in->tile * dsize(in->dtype);
            const size_t koff = (tbytes + 255) & ~(size_t)255;
            R->own_bytes = koff + (size_t)m * in->u * 4;
            R->own_block = ctx_alloc(ctx, R->own_bytes);
            if (!R->own_block) throw Oom();
            R->tiles = R->own_block;
            R->keys = (int32_t *)((char *)R->own_block + koff);
            launch_compact(ctx, in, flag, excl, R->tiles, R->keys);
        }
        check(cuda_check(ctx, cudaGetLastError(), "kernel launch"));
        keys_ready(ctx, R);
        *out = R;
        R = nullptr;
        ctx->err.clear();
    } catch (Oom &) {
        st = fail(ctx, UCL_ERR_OOM, "device allocation failed");
    } catch (Fail &f) {
        st = f.st;
    }
    cudaEventRecord(ctx->arena_done[arena], ctx->main);
    if (R) ucl_relation_destroy(R);
    return st;
}

}  // extern "C"
