// k_enum.cu -- exact ES(k) (Sec. 2.1) by exhaustive search, rows with n <= 32.
//
// Every size-k subset A of the row's keys is covered -- either evaluated, or
// excluded together with a whole group of subsets by a rigorous bound -- and
// the one of smallest es(A) is reported (exact ties: smallest colex rank).
// Instead of O(k d) work per subset, the walk below spends a few fp32
// instructions per subset it visits, and on the measured rows the bounds
// exclude most subsets without visiting them; the walk counts the nodes,
// subsets (leaves) and fp32 operations it spends (fw_best_subset_read_stats).
//
// (1) With u_j = p_j (v_j - mu), Lemma 2.1 gives es(A)^2 = Q(A) / P(A)^2,
//     Q(A) = ||sum_{j in A} u_j||^2, P(A) = sum_{j in A} p_j.  With
//     t = es(A0)^2 for the top-k set A0, the subsets that can beat or tie A0
//     are exactly those with val(A) = Q(A) - t P(A)^2 <= 0, a quadratic form
//     in the membership indicator.
// (2) Two exact ways to write val: the "direct" form over the keys of A
//     (entries G'_xy = u_x.u_y - t p_x p_y), and the "difference" form over
//     S = A xor A0 (keys removed from A0 carry sign -1; val(empty) = 0; linear
//     term l_x = 2 s_x (g0.u_x - t P0 p_x) with g0 = sum_{A0} u_j).  In fp32
//     each has a rigorous error bound kappa * (sum of a_x over the keys it
//     touches)^2 (a_x >= |u_x| + sqrt(t) p_x bounds every entry); the bound is
//     itself a quadratic form and is folded into the entries, so "computed
//     value <= 0" is a necessary condition for val <= 0.  For each removal set
//     R of A0 the walk uses the form with the smaller bound: the difference
//     form while the removed keys are light, the direct form once heavy keys
//     are removed (where the difference form would cancel large terms).
// (3) Meet in the middle: R ranges over all subsets of A0 (phase 1, values
//     from scratch); the added keys split into an outer set H' (depth-first,
//     phase 2) and an inner set L of EM keys whose enumeration is fully
//     unrolled over register-resident entries (template recursion).
// Subsets that pass the test (typically 1-8 per row) are re-scored exactly in
// double-float and the minimum taken.  Rows whose candidates overflow the
// buffer (degenerate rows, e.g. all v_j equal) go to an exhaustive fp64 path
// written in the difference form.
#include "fw_internal.h"

namespace fw {
namespace {

constexpr int EM = 12;    // inner key set size
constexpr int ECAP = 32;  // candidate masks per row
constexpr int FBS = 64;   // chunks (blocks) per row on the exhaustive path
constexpr int MAXD = 24;  // depth bound of the phase-2 walk
constexpr int PERM = 48;  // local index space per row: NS <= EM + 32

__host__ __device__ constexpr int tri(int a, int b, int n) { return a * n - a * (a - 1) / 2 + (b - a); }

struct EnumArgs {
    RowsDev R;
    const int32_t *k;
    uint64_t *best_rank;
    float *best_gap;
    int32_t *best_idx;
    int k_max;
    float *topk_gap;
    int32_t *row_status;
    uint32_t *cand;       // [rows][ECAP] original-key masks
    int32_t *cand_count;  // [rows]
    int32_t *fb_list;     // [rows]
    int32_t *fb_count;    // [1]
    double *fb_e;         // [rows][FBS] best es^2 of each chunk of an exhaustive row
    unsigned long long *fb_r;  // [rows][FBS] its colex rank
    float *slots;         // [rows][stride] walk tables
    uint8_t *perms;       // [rows][PERM] local key order
    float2 *kg;           // [rows] kappa, |g0| (rounded up)
    int stride;           // floats per row slot (odd)
    unsigned long long *stats;  // [4] walk counters: inner enumerations, their leaves,
                                // their fp32 operations, nodes / classes skipped by a bound
};

// Per-row slot (floats).  Local key order: L (EM inner keys, padded), A0 (k),
// H' (nHp outer added keys).  Entries "folded" have the error-bound term
// kappa a_x a_y subtracted; G' = u.u - t p p^T; l = difference-form linear term.
//   [0, EM)        Gd  : folded direct-form diagonal of L (+inf on padding)
//   [EM, 2EM)      lS  : extra difference-form diagonal of L (l_j - 4 kappa g0n a_j)
//   [2EM, 3EM)     aL  : a_j of L
//   [3EM, 3EM+EM^2) G2 : 2 x folded off-diagonal of L x L (square, zero diagonal)
//   A0 rows (k x RA, RA = EM + k + nHp + 2): raw G'(x, L) | G'(x, A0) | G'(x, H') | a_x | l_x
//   H' rows (nHp x RH, RH = EM + nHp + 2): folded G'(y, L) | HH (2 x folded off-diagonal,
//                                          folded diagonal) | l_y - 4 kappa g0n a_y | a_y
//   inner bound (npref(k) + 1): prefix sums of the ascending G2 entries x < y of L
//                               (pref[m] = sum of the m smallest), then sum |G2|
//   root bound (nprefr(k) + 1): the same over every pair of keys that can be
//                               added back (L and H'), then the sum of their |pair terms|
constexpr int OFF_A = 3 * EM + EM * EM;
__host__ __device__ constexpr int cmax_inner(int k) { return k < EM ? k : EM; }
__host__ __device__ constexpr int npref(int k) { return cmax_inner(k) * (cmax_inner(k) - 1) / 2 + 1; }
__host__ __device__ constexpr int nprefr(int k) { return k * (k - 1) / 2 + 1; }
__host__ __device__ constexpr int off_pref(int k, int nHp)
{
    return OFF_A + k * (EM + k + nHp + 2) + nHp * (EM + nHp + 2);
}
__host__ __device__ constexpr int off_prefr(int k, int nHp) { return off_pref(k, nHp) + npref(k) + 1; }
__host__ __device__ constexpr int slot_floats(int k, int nHp) { return off_prefr(k, nHp) + nprefr(k) + 1; }

// Ascending sort of 16 registers: Batcher's odd-even merge network (63
// compare-exchanges, indices fixed at compile time).
__device__ __forceinline__ void sort16(float (&x)[16])
{
#pragma unroll
    for (int p = 1; p < 16; p <<= 1)
#pragma unroll
        for (int kk = p; kk >= 1; kk >>= 1)
#pragma unroll
            for (int j = kk % p; j + kk < 16; j += 2 * kk)
#pragma unroll
                for (int i = 0; i < kk; ++i) {
                    if (i + j + kk >= 16) break;
                    if ((i + j) / (2 * p) == (i + j + kk) / (2 * p)) {
                        const float a = x[i + j], b = x[i + j + kk];
                        x[i + j] = fminf(a, b);
                        x[i + j + kk] = fmaxf(a, b);
                    }
                }
}

// Relative slack of the inner bound: covers the rounding of the bound and of
// the inner walk's chains (at most 1 + 12 + 66 additions) twice over.
constexpr float kInnerSlack = 1.52587890625e-5f;  // 2^-16

// Relative slack of the bound over every set that adds back r keys: twice the
// longest chain such a set's value goes through (q, r linear terms, r(r-1)/2
// pair terms and the walk's own adds), in units of 2^-24.
__device__ __forceinline__ float root_slack(int r) { return (float)(2 * (r * (r + 1) / 2 + r + 32)) * 5.9604645e-8f; }

struct Walk {
    const float *slot;
    const uint8_t *perm;  // local index -> original key
    int k, nL, nHp;
    int half;             // which of the row's two lanes: takes every other R of each size class
    uint32_t sync_mask;   // lanes that walk rows of identical (n, k); 0 when they differ
    float kappa, g0n;
    uint32_t *cand;
    int32_t *ccount;
    unsigned long long *stats;
};

// Leaves (C(EM, c)) and fp32 add/min operations of one inner<c> enumeration
// (the dfs below: one add per visited key, the running sums of the remaining
// keys at every internal node, one min per leaf, three to merge the minima).
__host__ __device__ constexpr unsigned long long dfs_ops(int C, int E)
{
    return (C >= 1 && E <= EM - C)
               ? 1ull + (C == 1 ? 1ull : (unsigned long long)(EM - E - 1) + dfs_ops(C - 1, E + 1)) + dfs_ops(C, E + 1)
               : 0ull;
}
__host__ __device__ constexpr unsigned long long dfs_leaves(int C, int E)
{
    return (C >= 1 && E <= EM - C) ? (C == 1 ? 1ull : dfs_leaves(C - 1, E + 1)) + dfs_leaves(C, E + 1) : 0ull;
}
struct InnerCost {
    unsigned long long leaves[EM + 1], ops[EM + 1];
};
constexpr InnerCost make_inner_cost()
{
    InnerCost t{};
    for (int c = 0; c <= EM; ++c) {
        t.leaves[c] = c == 0 ? 1ull : dfs_leaves(c, 0);
        t.ops[c] = c == 0 ? 0ull : dfs_ops(c, 0) + 3ull;
    }
    return t;
}
static __constant__ InnerCost c_inner_cost = make_inner_cost();

// ---- slow path: list every inner set C (size c) of a node whose folded value is <= 0
__device__ __noinline__ void collect(const Walk W, uint32_t keep0, uint32_t hmask, const float *w, float q, int c)
{
    const float *G2 = W.slot + 3 * EM;
    uint32_t amask = keep0;
    for (uint32_t m = hmask; m; m &= m - 1) amask |= 1u << W.perm[EM + W.k + __ffs(m) - 1];
    uint32_t cm = c == 0 ? 0u : (1u << c) - 1u;
    const uint32_t lim = 1u << W.nL;
    for (;;) {
        float v = q;
        for (uint32_t a = cm; a; a &= a - 1) {
            const int j = __ffs(a) - 1;
            v += w[j];
            for (uint32_t b2 = a & (a - 1); b2; b2 &= b2 - 1) v += G2[j * EM + __ffs(b2) - 1];
        }
        if (v <= 0.f) {
            uint32_t m = amask;
            for (uint32_t a = cm; a; a &= a - 1) m |= 1u << W.perm[__ffs(a) - 1];
            const int sl = atomicAdd(W.ccount, 1);
            if (sl < ECAP) W.cand[sl] = m;
        }
        if (c == 0) break;
        const uint32_t lo = cm & (0u - cm);  // next subset of the same size (Gosper's rule)
        const uint32_t rr = cm + lo;
        cm = (((rr ^ cm) >> 2) / lo) | rr;
        if (cm >= lim) break;
    }
}

// ---- inner enumeration over the size-C subsets of {E..EM-1}, fully unrolled.
// r[j] = diagonal + 2 h_j + 2 sum_{i chosen} G2_ij for the keys still available.
template <int C, int E>
__device__ __forceinline__ void dfs(const float (&r)[EM], float val, const float (&G2)[EM][EM], float (&mn)[4])
{
    if constexpr (C >= 1 && E <= EM - C) {
        const float v = val + r[E];
        if constexpr (C == 1) {
            mn[E & 3] = fminf(mn[E & 3], v);
        } else {
            float rr[EM];
#pragma unroll
            for (int j = E + 1; j < EM; ++j) rr[j] = r[j] + G2[E][j];
            dfs<C - 1, E + 1>(rr, v, G2, mn);
        }
        dfs<C, E + 1>(r, val, G2, mn);
    }
}

template <int C>
__device__ __forceinline__ float inner(const float (&w)[EM], float q, const float (&G2)[EM][EM])
{
    if constexpr (C == 0) {
        return q;
    } else {
        float mn[4] = {INFINITY, INFINITY, INFINITY, INFINITY};
        dfs<C, 0>(w, q, G2, mn);
        return fminf(fminf(mn[0], mn[1]), fminf(mn[2], mn[3]));
    }
}

__device__ __forceinline__ float inner_dispatch(int c, const float (&w)[EM], float q, const float (&G2)[EM][EM])
{
    switch (c) {
    case 0: return inner<0>(w, q, G2);
    case 1: return inner<1>(w, q, G2);
    case 2: return inner<2>(w, q, G2);
    case 3: return inner<3>(w, q, G2);
    case 4: return inner<4>(w, q, G2);
    case 5: return inner<5>(w, q, G2);
    case 6: return inner<6>(w, q, G2);
    case 7: return inner<7>(w, q, G2);
    case 8: return inner<8>(w, q, G2);
    case 9: return inner<9>(w, q, G2);
    case 10: return inner<10>(w, q, G2);
    case 11: return inner<11>(w, q, G2);
    case 12: return inner<12>(w, q, G2);
    default: return INFINITY;
    }
}

// The whole walk of one row (one lane).  Compiled once; every kernel
// instantiation calls it.
__device__ __noinline__ void walk_row(const Walk W)
{
    const float kap = W.kappa, g0n = W.g0n;
    const int k = W.k, nL = W.nL, nHp = W.nHp;
    const int RA = EM + k + nHp + 2, RH = EM + nHp + 2;
    const float *SA = W.slot + OFF_A;
    const float *SH = SA + k * RA;
    const float *PF = W.slot + off_pref(k, nHp);  // inner-bound prefix sums, then sum |G2|
    const float g2abs = PF[npref(k)];
    const float *PR = W.slot + off_prefr(k, nHp);  // root-bound prefix sums, then sum |pair terms|
    const float pabs = PR[nprefr(k)];
    float Gd[EM], lS[EM], aL[EM], G2[EM][EM];
#pragma unroll
    for (int x = 0; x < EM; ++x) {
        Gd[x] = W.slot[x];
        lS[x] = W.slot[EM + x];
        aL[x] = W.slot[2 * EM + x];
#pragma unroll
        for (int y = x + 1; y < EM; ++y) G2[x][y] = W.slot[3 * EM + x * EM + y];
    }
    float base[MAXD];  // per H' key: sum over the phase-1 outer keys of the folded E(x, y)
    float hst[MAXD][EM];
    float qst[MAXD];
    int path[MAXD];
    const uint32_t nR = 1u << k;
    unsigned long long n_inner = 0, n_leaf = 0, n_ops = 0, n_skip = 0;
    // Removal sets R of A0 by size class; the row's two lanes take alternate
    // members of the same class at the same time, so they run the same code.
    for (int r = 0; r <= k; ++r) {
        if (r > nL + nHp) break;  // cannot add back r keys
        uint32_t R = r == 0 ? 0u : (1u << r) - 1u;
        bool valid = true;
        auto next_same_size = [&](uint32_t x) -> uint32_t {  // Gosper's rule
            if (x == 0u) return nR;
            const uint32_t lo = x & (0u - x);
            const uint32_t ri = x + lo;
            return (((ri ^ x) >> 2) / lo) | ri;
        };
        if (W.half) {
            R = next_same_size(R);
            valid = R < nR;
        }
        while (valid) {
        // choose the form with the smaller error bound
        float sR = 0.f, sK = 0.f;
        for (int x = 0; x < k; ++x) {
            const float ax = SA[x * RA + RA - 2];
            if ((R >> x) & 1u) sR += ax;
            else sK += ax;
        }
        const bool sform = sR * (4.f * g0n + sR) <= sK * sK;
        const uint32_t O = sform ? R : (~R & (nR - 1u));  // outer keys of A0 in this form
        const float sgn = sform ? -1.f : 1.f;            // their sign
        // phase 1: h (inner keys), q, base (H' keys) from scratch, fixed trip counts
        float h[EM];
#pragma unroll
        for (int j = 0; j < EM; ++j) h[j] = 0.f;
        float q = 0.f;
        for (int y = 0; y < nHp; ++y) base[y] = 0.f;
        for (int x = 0; x < k; ++x) {
            const float on = ((O >> x) & 1u) ? 1.f : 0.f;
            const float *row = SA + x * RA;
            const float ax = row[RA - 2], kax = kap * ax;
            const float so = sgn * on, ko = kax * on;
#pragma unroll
            for (int j = 0; j < EM; ++j) h[j] += fmaf(so, row[j], -ko * aL[j]);
            float dq = row[EM + x] - kax * ax;
            if (sform) dq += row[RA - 1] - 4.f * kax * g0n;
            for (int x2 = 0; x2 < x; ++x2) {
                const float on2 = ((O >> x2) & 1u) ? 2.f : 0.f;
                dq += on2 * (row[EM + x2] - kax * SA[x2 * RA + RA - 2]);  // sign^2 = +1
            }
            q += on * dq;
            for (int y = 0; y < nHp; ++y) base[y] += fmaf(so, row[EM + k + y], -ko * SH[y * RH + RH - 1]);
        }
        uint32_t keep0 = 0u;  // original-key mask of the kept part of A0
        for (int x = 0; x < k; ++x)
            if (!((R >> x) & 1u)) keep0 |= 1u << W.perm[EM + x];
        float GdS[EM];
#pragma unroll
        for (int j = 0; j < EM; ++j) GdS[j] = sform ? Gd[j] + lS[j] : Gd[j];
        // Every set that adds back r keys from L and H' has value q + (its r
        // linear terms) + (its r(r-1)/2 pair terms).  The m-th smallest linear
        // term of L u H' is at least min(m-th smallest over L, least over H'),
        // and the pair terms are at least the smallest ones of the row; when
        // that bound is positive beyond rounding, no subset of this R passes.
        bool skip_r = false;
        if (r >= 2) {
            float ws[16];
            float aw = 0.f;
#pragma unroll
            for (int j = 0; j < EM; ++j) {
                ws[j] = fmaf(2.f, h[j], GdS[j]);
                aw += ws[j] < INFINITY ? fabsf(ws[j]) : 0.f;
            }
#pragma unroll
            for (int j = EM; j < 16; ++j) ws[j] = INFINITY;
            sort16(ws);
            float hmin = INFINITY;
            for (int y = 0; y < nHp; ++y) {
                const float *hr = SH + y * RH;
                float lin = hr[EM + y] + 2.f * base[y];
                if (sform) lin += hr[RH - 2];
                hmin = fminf(hmin, lin);
                aw += fabsf(lin);
            }
            float sl = 0.f;
#pragma unroll
            for (int m = 0; m < 16; ++m) sl += m < r ? fminf(ws[m], hmin) : 0.f;
            for (int m = 16; m < r; ++m) sl += hmin;
            const float lb = q + sl + PR[r * (r - 1) / 2];
            skip_r = lb > root_slack(r) * (fabsf(q) + aw + pabs);
        }
        if (skip_r) {
            ++n_skip;
            R = next_same_size(R);
            if (R < nR) R = next_same_size(R);
            valid = R < nR;
            continue;
        }
        // phase 2: depth-first over I subset of H' with |I| <= r
        int depth = 0, e = 0;
        uint32_t imask = 0u;  // local H' bits
        for (;;) {
            const int c = r - depth;  // inner keys still to add
            if (c >= 0 && c <= nL) {
                float w[EM];
#pragma unroll
                for (int j = 0; j < EM; ++j) w[j] = fmaf(2.f, h[j], GdS[j]);
                // Every size-c set C of L has value q + sum_C w + sum_{pairs of C} G2
                // >= q + (c smallest w) + (c(c-1)/2 smallest G2): when that bound is
                // positive beyond rounding, no set of this node can pass the test.
                bool skip = false;
                if (c >= 3) {
                    float ws[16];
                    float aw = 0.f;
#pragma unroll
                    for (int j = 0; j < EM; ++j) {
                        ws[j] = w[j];
                        aw += w[j] < INFINITY ? fabsf(w[j]) : 0.f;
                    }
#pragma unroll
                    for (int j = EM; j < 16; ++j) ws[j] = INFINITY;
                    sort16(ws);
                    float sw = 0.f;
#pragma unroll
                    for (int j = 0; j < EM; ++j) sw += j < c ? ws[j] : 0.f;
                    const float lb = q + sw + PF[c * (c - 1) / 2];
                    skip = lb > kInnerSlack * (fabsf(q) + aw + g2abs);
                }
                if (!skip) {
                    ++n_inner;
                    n_leaf += c_inner_cost.leaves[c];
                    n_ops += c_inner_cost.ops[c];
                    const float mval = inner_dispatch(c, w, q, G2);
                    if (mval <= 0.f) collect(W, keep0, imask, w, q, c);
                } else {
                    ++n_skip;
                }
            }
            if (!(depth < r && e < nHp && depth < MAXD)) {
                bool done = true;  // back up to the next sibling
                while (depth > 0) {
                    --depth;
                    const int pe = path[depth];
                    imask &= ~(1u << pe);
#pragma unroll
                    for (int j = 0; j < EM; ++j) h[j] = hst[depth][j];
                    q = qst[depth];
                    e = pe + 1;
                    if (e < nHp) {
                        done = false;
                        break;
                    }
                }
                if (done) break;
            }
            // descend into key e of H'
#pragma unroll
            for (int j = 0; j < EM; ++j) hst[depth][j] = h[j];
            qst[depth] = q;
            path[depth] = e;
            const float *hrow = SH + e * RH;
#pragma unroll
            for (int j = 0; j < EM; ++j) h[j] += hrow[j];
            float dq = hrow[EM + e] + 2.f * base[e];
            if (sform) dq += hrow[RH - 2];
            for (int t = 0; t < depth; ++t) dq += hrow[EM + path[t]];
            q += dq;
            imask |= 1u << e;
            ++depth;
            ++e;
        }
        R = next_same_size(R);
        if (R < nR) R = next_same_size(R);
        valid = R < nR;
        }
        // The two halves may differ by one member in this class; meet again
        // before the next one.  Every lane in sync_mask walks the same (n, k),
        // hence runs this loop the same number of times.
        if (W.sync_mask) __syncwarp(W.sync_mask);
    }
    atomicAdd(W.stats + 0, n_inner);
    atomicAdd(W.stats + 1, n_leaf);
    atomicAdd(W.stats + 2, n_ops);
    atomicAdd(W.stats + 3, n_skip);
}

// Write one Gram entry (or a_x / l_x) into the walk tables of a row slot.
// Tables are described in the slot layout comment above.
struct SlotGeom {
    float *slot;
    int k, nL, nHp, RA, RH, offH;
    float kap, g0n;
};
__device__ __forceinline__ void put_entry(const SlotGeom &S, int la, int lb, float g, float aa, float ab)
{
    // row la, column lb (la != lb), g = G'_ab
    const int eA = EM, eH = EM + S.k;
    if (la < eA) {
        if (lb < eA) S.slot[3 * EM + la * EM + lb] = 2.f * (g - S.kap * aa * ab);
    } else if (la < eH) {
        S.slot[OFF_A + (la - eA) * S.RA + lb] = g;
    } else {
        float *hr = S.slot + S.offH + (la - eH) * S.RH;
        if (lb < eA) hr[lb] = g - S.kap * aa * ab;
        else if (lb >= eH) hr[EM + (lb - eH)] = 2.f * (g - S.kap * aa * ab);
    }
}
__device__ __forceinline__ void put_diag(const SlotGeom &S, int l, float g, float a)
{
    const int eA = EM, eH = EM + S.k;
    if (l < eA) {
        S.slot[l] = g - S.kap * a * a;
        S.slot[2 * EM + l] = a;
    } else if (l < eH) {
        S.slot[OFF_A + (l - eA) * S.RA + l] = g;
        S.slot[OFF_A + (l - eA) * S.RA + S.RA - 2] = a;
    } else {
        float *hr = S.slot + S.offH + (l - eH) * S.RH;
        hr[EM + (l - eH)] = g - S.kap * a * a;
        hr[S.RH - 1] = a;
    }
}
__device__ __forceinline__ void put_linear(const SlotGeom &S, int l, float lin, float a)
{
    const int eA = EM, eH = EM + S.k;
    if (l < eA) S.slot[EM + l] = lin - 4.f * S.kap * S.g0n * a;
    else if (l < eH) S.slot[OFF_A + (l - eA) * S.RA + S.RA - 1] = lin;
    else S.slot[S.offH + (l - eH) * S.RH + S.RH - 2] = lin - 4.f * S.kap * S.g0n * a;
}

// pref[m] = sum of the m smallest of vals[0, E) for m <= need, then
// pref[need + 1] = sum |vals| (E <= 512).  Each lane holds its entries
// lane + 32 u in registers; every round the warp takes the smallest unused one
// (equal values: any of them, the sums do not depend on it).
__device__ __forceinline__ void smallest_prefix(const float *vals, int E, int need, float *pref, int lane)
{
    float x[16];
    float ab = 0.f;
#pragma unroll
    for (int u = 0; u < 16; ++u) {
        const int e = lane + 32 * u;
        x[u] = e < E ? vals[e] : INFINITY;
        ab += e < E ? fabsf(x[u]) : 0.f;
    }
    ab = warp_sum(ab);
    float run = 0.f;
    if (lane == 0) pref[0] = 0.f;
    for (int m = 0; m < need; ++m) {
        float bv = INFINITY;
        int bu = 0;
#pragma unroll
        for (int u = 0; u < 16; ++u)
            if (x[u] < bv) {
                bv = x[u];
                bu = u;
            }
        float wv = bv;
        int wl = lane;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(FW_FULL, wv, o);
            const int ol = __shfl_xor_sync(FW_FULL, wl, o);
            if (ov < wv || (ov == wv && ol < wl)) {
                wv = ov;
                wl = ol;
            }
        }
        if (lane == wl)
#pragma unroll
            for (int u = 0; u < 16; ++u)
                if (u == bu) x[u] = INFINITY;
        run += wv < INFINITY ? wv : 0.f;
        if (lane == 0) pref[m + 1] = run;
    }
    if (lane == 0) pref[need + 1] = ab;
}

constexpr int ERW = 16;  // rows per warp (two lanes per row)
constexpr int MAXT = 3;         // Gram tiles (2 x 4 products) per lane: 33 rows need at most 96
constexpr int PPL = 8 * MAXT;   // Gram product slots per lane

// ---- the search in three kernels.  k_enum_prep: one warp per row builds the
// row's walk tables (slot, key order, kappa and |g0|) in shared memory and
// writes them out; k_enum_walk: one warp = ERW rows, two lanes per row split
// its removal sets; k_enum_rescore: one warp per row re-scores the row's
// candidates exactly and lists the rows left to the exhaustive path.
constexpr int PREP_W = 4;  // warps (rows) per block of k_enum_prep
constexpr int RS_W = 8;    // warps (rows) per block of k_enum_rescore

// per-warp shared memory of k_enum_prep (floats): slot, staged values, a_x,
// p (double), key order and its inverse; a multiple of 4
__host__ __device__ constexpr int prep_floats(int stride, int ust)
{
    return ((stride + 1) / 2 * 2 + ust + 32 + 64 + (PERM + 32) / 4 + 3) / 4 * 4;
}
constexpr int RCB = 8;     // candidates re-scored per pass over the values
// per-warp shared memory of k_enum_rescore (floats): the staged values
__host__ __device__ constexpr int rescore_floats(int ust) { return (ust + 3) / 4 * 4; }

template <int DPL, typename VT>
__global__ void __launch_bounds__(32 * PREP_W, 4) k_enum_prep(const EnumArgs a)
{
    extern __shared__ float smem[];
    constexpr int d = DPL * 32;
    constexpr int DCH = d < 64 ? d : 64;  // dimensions staged at a time
    constexpr int TCH = DCH / 32;         // per-lane dims in one chunk
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    const int ust_floats = (((a.R.max_n + 1) * (DCH + 1)) + 1) & ~1;
    float *slot = smem + (size_t)wib * prep_floats(a.stride, ust_floats);  // [stride]
    float *Ust = slot + (a.stride + 1) / 2 * 2;                             // [max_n+1][DCH+1]
    float *aX = Ust + ust_floats;                                            // [32]
    float *pfl = aX + 32;                                                    // [32] p (rounded)
    uint8_t *perms = reinterpret_cast<uint8_t *>(aX + 96);                   // [PERM]
    uint8_t *inv = perms + PERM;                                             // [32]
    const int64_t row = (int64_t)blockIdx.x * PREP_W + wib;
    if (row >= a.R.rows) return;
    const int64_t g = row / a.R.R;
    const int64_t ri = row - g * a.R.R;
    const int n = a.R.n[g];
    const int k = a.k[row];
    int status = FW_OK;
    if (n < 1 || n > a.R.max_n || n > 32 || k < 1 || k > n || k > a.k_max) status = FW_ERR_INVALID_ARG;
    const float *lg = a.R.logits + a.R.logit_off[g] + ri * (status == FW_OK ? n : 0);
    const float l = (status == FW_OK && lane < n) ? lg[lane] : -INFINITY;
    if (status == FW_OK && __any_sync(FW_FULL, lane < n && !isfinite(l))) status = FW_ERR_NONFINITE;
    if (status != FW_OK) {
        if (lane == 0) {
            if (a.row_status) a.row_status[row] = status;
            a.cand_count[row] = -1;
            a.best_gap[row] = __int_as_float(0x7fc00000);
            a.best_rank[row] = ~0ull;
            if (a.topk_gap) a.topk_gap[row] = __int_as_float(0x7fc00000);
        }
        for (int t = lane; t < a.k_max; t += 32) a.best_idx[row * a.k_max + t] = -1;
        return;
    }
    const VT *V = reinterpret_cast<const VT *>(a.R.v) + a.R.v_off[g];
    const float M = warp_max(l);
    double p = lane < n ? exp((double)l - (double)M) : 0.0;
    p = p / warp_sum_d(p);
    int rank = 0;
    for (int s2 = 0; s2 < n; ++s2) {
        const float ls = __shfl_sync(FW_FULL, l, s2);
        rank += (ls > l) || (ls == l && s2 < lane);
    }
    const bool inA0 = lane < n && rank < k;
    const uint32_t A0 = __ballot_sync(FW_FULL, inA0);
    const df pd = df_from_double(p);
    // local key order: L = first nL keys outside A0, then A0, then H'
    const int nL = min(EM, n - k);
    const int nHp = n - k - nL;
    uint8_t *perm = perms;
    if (lane < n) {
        const uint32_t below = (1u << lane) - 1u;
        const int bo = __popc(~A0 & below);
        const int bi = __popc(A0 & below);
        const int loc = inA0 ? EM + bi : (bo < nL ? bo : EM + k + (bo - nL));
        perm[loc] = (uint8_t)lane;
        inv[lane] = (uint8_t)loc;
        pfl[lane] = (float)p;
    }
    SlotGeom S;
    S.slot = slot;
    S.k = k;
    S.nL = nL;
    S.nHp = nHp;
    S.RA = EM + k + nHp + 2;
    S.RH = EM + nHp + 2;
    S.offH = OFF_A + k * S.RA;
    const int tot = slot_floats(k, nHp);
    for (int i = lane; i < tot; i += 32) S.slot[i] = (i >= nL && i < EM) ? INFINITY : 0.f;
    // Gram entries over the n keys plus g0 (index n), staged DCH dimensions at a
    // time.  The upper triangle is cut into tiles of 2 rows x 4 columns (lane
    // takes tiles lane, lane + 32, ...); a tile reads 6 staged values per
    // dimension for its 8 products, and each product is four interleaved
    // partial sums per chunk.  Slot i = 8 * tile + 4 * (x - x0) + (y - y0);
    // px_ = -1 marks slots outside the triangle (and |g0|^2, known exactly).
    const int R1 = n + 1, nby = (R1 + 3) / 4;
    int tx0[MAXT], ty0[MAXT];
    int px_[PPL], py_[PPL];
    float acc[PPL];
#pragma unroll
    for (int tl = 0; tl < MAXT; ++tl) {
        int tid_ = lane + 32 * tl, bx = 0;
        bool ok = true;
        for (;;) {  // rows 2bx, 2bx+1 hold tiles by = bx/2 .. nby-1
            if (2 * bx >= R1) {
                ok = false;
                break;
            }
            const int cnt = nby - bx / 2;
            if (tid_ < cnt) break;
            tid_ -= cnt;
            ++bx;
        }
        tx0[tl] = ok ? 2 * bx : -1;
        ty0[tl] = ok ? 4 * (bx / 2 + tid_) : -1;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int x = tx0[tl] + (e >> 2), y = ty0[tl] + (e & 3);
            const bool in = ok && x <= y && y < R1 && x < n;
            px_[8 * tl + e] = in ? x : -1;
            py_[8 * tl + e] = y;
            acc[8 * tl + e] = 0.f;
        }
    }
    df g0[DPL];
#pragma unroll
    for (int t = 0; t < DPL; ++t) g0[t] = df_zero();
#pragma unroll
    for (int ch = 0; ch < DPL / TCH; ++ch) {
        __syncwarp();
        // the chunk's values of all n keys into Ust (loads issued back to back)
        stage_value_cols<DCH>(V, n, d, ch * DCH, Ust, lane);
        __syncwarp();
        // mu over the chunk's columns (j ascending, double-float), then
        // u_j = p_j (v_j - mu) in place
        df mu[TCH];
#pragma unroll
        for (int tt = 0; tt < TCH; ++tt) mu[tt] = df_zero();
        for (int j = 0; j < n; ++j) {
            const df pj = shfl_df(pd, j);
#pragma unroll
            for (int tt = 0; tt < TCH; ++tt)
                mu[tt] = df_add(mu[tt], df_mul_f(pj, Ust[j * (DCH + 1) + lane + 32 * tt]));
        }
        for (int j = 0; j < n; ++j) {
            const df pj = shfl_df(pd, j);
            const bool in = (A0 >> j) & 1u;
#pragma unroll
            for (int tt = 0; tt < TCH; ++tt) {
                const int t = ch * TCH + tt;
                float *cell = Ust + j * (DCH + 1) + lane + 32 * tt;
                const df u = df_mul(pj, df_rsub_f(*cell, mu[tt]));
                *cell = u.hi;
                if (in) g0[t] = df_add(g0[t], u);
            }
        }
#pragma unroll
        for (int tt = 0; tt < TCH; ++tt) Ust[n * (DCH + 1) + lane + 32 * tt] = g0[ch * TCH + tt].hi;
        __syncwarp();
#pragma unroll
        for (int tl = 0; tl < MAXT; ++tl) {
            if (tx0[tl] < 0) continue;
            const float *ux[2], *uy[4];
#pragma unroll
            for (int e = 0; e < 2; ++e) ux[e] = Ust + min(tx0[tl] + e, n) * (DCH + 1);
#pragma unroll
            for (int e = 0; e < 4; ++e) uy[e] = Ust + min(ty0[tl] + e, n) * (DCH + 1);
            float sp[8][4];
#pragma unroll
            for (int e = 0; e < 8; ++e)
#pragma unroll
                for (int c4 = 0; c4 < 4; ++c4) sp[e][c4] = 0.f;
            for (int c = 0; c < DCH; c += 4) {
#pragma unroll
                for (int c4 = 0; c4 < 4; ++c4) {
                    const float a0 = ux[0][c + c4], a1 = ux[1][c + c4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float b = uy[e][c + c4];
                        sp[e][c4] = fmaf(a0, b, sp[e][c4]);
                        sp[4 + e][c4] = fmaf(a1, b, sp[4 + e][c4]);
                    }
                }
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[8 * tl + e] += (sp[e][0] + sp[e][1]) + (sp[e][2] + sp[e][3]);
        }
    }
    df nrm = df_zero();
#pragma unroll
    for (int t = 0; t < DPL; ++t) nrm = df_add(nrm, df_mul(g0[t], g0[t]));
    nrm = warp_sum_df(nrm);
    const double P0 = warp_sum_d(inA0 ? p : 0.0);
    const double g0n2 = fmax(df_to_double(nrm), 0.0);
    const double t = g0n2 / (P0 * P0);  // es(A0)^2
    const double sqt = sqrt(t);
    if (lane == 0 && a.topk_gap) a.topk_gap[row] = (float)sqt;
    // kappa: 2.2x the per-subset error bound of an fp32 evaluation of either form
    const int Lc = k * (k + 1) / 2 + 2 * n + 16;
    S.kap = (float)(2.2 * ((double)d * 0.25 + Lc + 16) * 5.9604644775390625e-8);
    S.g0n = (float)sqrt(g0n2) * 1.0001f;
    // a_x = |u_x| + sqrt(t) p_x (rounded up) from the diagonal entries
#pragma unroll
    for (int i = 0; i < PPL; ++i)
        if (px_[i] >= 0 && px_[i] == py_[i] && px_[i] < n)
            aX[px_[i]] = sqrtf(fmaxf(acc[i], 0.f)) * 1.0001f + ((float)sqt * pfl[px_[i]]) * 1.0001f;
    __syncwarp();
    // scatter the folded entries into the walk tables
    const float tf = (float)t, P0f = (float)P0;
#pragma unroll
    for (int i = 0; i < PPL; ++i) {
        const int x = px_[i], y = py_[i];
        if (x < 0 || x == n) continue;
        // G' = u.u - t p p^T in fp32 (a few ulps of a_x a_y, inside kappa's slack)
        const float tpx = tf * pfl[x];
        if (y == n) {
            const float sx = ((A0 >> x) & 1u) ? -2.f : 2.f;
            put_linear(S, inv[x], sx * fmaf(-tpx, P0f, acc[i]), aX[x]);
        } else {
            const float gp = fmaf(-tpx, pfl[y], acc[i]);
            if (x == y) {
                put_diag(S, inv[x], gp, aX[x]);
            } else {
                put_entry(S, inv[x], inv[y], gp, aX[x], aX[y]);
                put_entry(S, inv[y], inv[x], gp, aX[y], aX[x]);
            }
        }
    }
    __syncwarp();
    // Bounds of the walk: the pair terms of the inner set L (G2, x < y) and of
    // every two keys that can be added back (L x L, H' x H' from HH, H' x L as
    // twice the folded G'(y, L)); for each list the prefix sums of its
    // smallest terms (pref[m] = sum of the m smallest) and the sum of |terms|.
    // The warp takes the smallest remaining term round by round.
    {
        const int nLL = EM * (EM - 1) / 2, nHH = nHp * (nHp - 1) / 2, E = nLL + nHH + EM * nHp;
        float *vals = Ust;
        float *PF = S.slot + off_pref(k, nHp), *PR = S.slot + off_prefr(k, nHp);
        if (E <= ust_floats && E <= 512) {
            for (int e = lane; e < E; e += 32) {
                float v;
                if (e < nLL) {
                    int x = 0, rem = e;
                    while (rem >= EM - 1 - x) {
                        rem -= EM - 1 - x;
                        ++x;
                    }
                    v = S.slot[3 * EM + x * EM + x + 1 + rem];
                } else if (e < nLL + nHH) {
                    int x = 0, rem = e - nLL;
                    while (rem >= nHp - 1 - x) {
                        rem -= nHp - 1 - x;
                        ++x;
                    }
                    v = S.slot[S.offH + x * S.RH + EM + x + 1 + rem];
                } else {
                    const int f = e - nLL - nHH, y = f / EM, j = f - y * EM;
                    v = 2.f * S.slot[S.offH + y * S.RH + j];
                }
                vals[e] = v;
            }
            __syncwarp();
            // pass 0: the first nLL entries (L x L) for the inner bound; pass 1: all E
            for (int pass = 0; pass < 2; ++pass) {
                const int En = pass == 0 ? nLL : E;
                const int need = (pass == 0 ? npref(k) : nprefr(k)) - 1;
                smallest_prefix(vals, En, need, pass == 0 ? PF : PR, lane);
            }
        } else if (lane == 0) {  // (cannot happen for n <= 32; the bounds then never prune)
            for (int m = 0; m < npref(k); ++m) PF[m] = -INFINITY;
            PF[npref(k)] = 0.f;
            for (int m = 0; m < nprefr(k); ++m) PR[m] = -INFINITY;
            PR[nprefr(k)] = 0.f;
        }
        __syncwarp();
    }
    // the tables out: slot, key order, kappa and |g0|
    for (int i = lane; i < tot; i += 32) a.slots[row * a.stride + i] = S.slot[i];
    if (lane < PERM / 4)
        reinterpret_cast<uint32_t *>(a.perms + row * PERM)[lane] = reinterpret_cast<const uint32_t *>(perm)[lane];
    if (lane == 0) {
        a.kg[row] = make_float2(S.kap, S.g0n);
        a.cand_count[row] = k <= 31 ? 0 : ECAP + 1;  // k = 32: the exhaustive path
        if (a.row_status) a.row_status[row] = FW_OK;
    }
}

__global__ void __launch_bounds__(32, 1) k_enum_walk(const EnumArgs a)
{
    extern __shared__ float smem[];
    const int lane = threadIdx.x;
    float *slots = smem;                                                   // [ERW][stride]
    uint8_t *perms = reinterpret_cast<uint8_t *>(smem + ERW * a.stride);   // [ERW][PERM]
    const int64_t row0 = (int64_t)blockIdx.x * ERW;
    const int nrow = (int)min((int64_t)ERW, a.R.rows - row0);
    {
        // ERW * stride is a multiple of 4 floats, so every block's tables start 16-byte aligned
        const float *src = a.slots + row0 * a.stride;
        const int tot = nrow * a.stride, nv = tot / 4;
        for (int i = lane; i < nv; i += 32)
            reinterpret_cast<float4 *>(slots)[i] = reinterpret_cast<const float4 *>(src)[i];
        for (int i = 4 * nv + lane; i < tot; i += 32) slots[i] = src[i];
        const int pv = nrow * PERM / 16;
        for (int i = lane; i < pv; i += 32)
            reinterpret_cast<uint4 *>(perms)[i] = reinterpret_cast<const uint4 *>(a.perms + row0 * PERM)[i];
    }
    __syncwarp();
    const int rr = lane & (ERW - 1);
    const int64_t row = row0 + rr;
    Walk my;
    const bool my_walk = rr < nrow && a.cand_count[row] == 0;
    if (my_walk) {
        const int n = a.R.n[row / a.R.R];
        my.k = a.k[row];
        my.nL = min(EM, n - my.k);
        my.nHp = n - my.k - my.nL;
        my.slot = slots + rr * a.stride;
        my.perm = perms + rr * PERM;
        my.half = lane / ERW;
        const float2 kg = a.kg[row];
        my.kappa = kg.x;
        my.g0n = kg.y;
        my.cand = a.cand + row * ECAP;
        my.ccount = a.cand_count + row;
        my.stats = a.stats;
    }
    {
        const uint32_t wmask = __ballot_sync(FW_FULL, my_walk);
        const int key = my_walk ? (my.k << 8) | (my.nL << 16) | my.nHp : -1;
        const int key0 = __shfl_sync(FW_FULL, key, wmask ? __ffs(wmask) - 1 : 0);
        const bool same = __all_sync(FW_FULL, !my_walk || key == key0);
        my.sync_mask = same ? wmask : 0u;
    }
    if (my_walk) walk_row(my);
}

template <int DPL, typename VT>
__global__ void __launch_bounds__(32 * RS_W) k_enum_rescore(const EnumArgs a)
{
    extern __shared__ float smem[];
    constexpr int d = DPL * 32;
    constexpr int DCH = d < 64 ? d : 64;
    constexpr int TCH = DCH / 32;
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    const int ust_floats = (((a.R.max_n + 1) * (DCH + 1)) + 1) & ~1;
    float *Ust = smem + (size_t)wib * rescore_floats(ust_floats);  // [max_n+1][DCH+1]
    const int64_t row = (int64_t)blockIdx.x * RS_W + wib;
    if (row >= a.R.rows) return;
    const int cc = a.cand_count[row];
    if (cc < 0) return;  // invalid row, outputs already written
    if (cc > ECAP || cc == 0) {
        if (lane == 0) a.fb_list[atomicAdd(a.fb_count, 1)] = (int)row;
        return;
    }
    const int64_t g = row / a.R.R;
    const int64_t ri = row - g * a.R.R;
    const int n = a.R.n[g];
    const int k = a.k[row];
    const VT *V = reinterpret_cast<const VT *>(a.R.v) + a.R.v_off[g];
    const float *lg = a.R.logits + a.R.logit_off[g] + ri * n;
    const float l = lane < n ? lg[lane] : -INFINITY;
    const float M = warp_max(l);
    double p = lane < n ? exp((double)l - (double)M) : 0.0;
    p = p / warp_sum_d(p);
    const df pd = df_from_double(p);
    // candidates in groups of RCB; per 64-column chunk: stage the values, mu over
    // the chunk, and each candidate's g over the chunk, whose squares add into a
    // per-lane partial (same order of operations as one pass over all columns)
    double best = INFINITY;
    uint64_t brank = ~0ull;
    uint32_t bmask = 0u;
    for (int c0 = 0; c0 < cc; c0 += RCB) {
        uint32_t cm[RCB];
        df sq[RCB];
#pragma unroll
        for (int ci = 0; ci < RCB; ++ci) {
            cm[ci] = c0 + ci < cc ? a.cand[row * ECAP + c0 + ci] : 0u;
            sq[ci] = df_zero();
        }
        for (int ch = 0; ch < DPL / TCH; ++ch) {
            __syncwarp();
            stage_value_cols<DCH>(V, n, d, ch * DCH, Ust, lane);
            __syncwarp();
            df mu[TCH];
#pragma unroll
            for (int tt = 0; tt < TCH; ++tt) mu[tt] = df_zero();
            for (int j = 0; j < n; ++j) {
                const df pj = shfl_df(pd, j);
#pragma unroll
                for (int tt = 0; tt < TCH; ++tt)
                    mu[tt] = df_add(mu[tt], df_mul_f(pj, Ust[j * (DCH + 1) + lane + 32 * tt]));
            }
#pragma unroll
            for (int ci = 0; ci < RCB; ++ci) {
                df gv[TCH];
#pragma unroll
                for (int tt = 0; tt < TCH; ++tt) gv[tt] = df_zero();
                for (uint32_t mm = cm[ci]; mm; mm &= mm - 1) {
                    const int j = __ffs(mm) - 1;
                    const df pj = shfl_df(pd, j);
#pragma unroll
                    for (int tt = 0; tt < TCH; ++tt)
                        gv[tt] = df_add(gv[tt], df_mul(pj, df_rsub_f(Ust[j * (DCH + 1) + lane + 32 * tt], mu[tt])));
                }
#pragma unroll
                for (int tt = 0; tt < TCH; ++tt) sq[ci] = df_add(sq[ci], df_mul(gv[tt], gv[tt]));
            }
        }
#pragma unroll
        for (int ci = 0; ci < RCB; ++ci) {
            if (c0 + ci >= cc) break;
            const uint32_t m = cm[ci];
            const df s3 = warp_sum_df(sq[ci]);
            const double P = warp_sum_d(((m >> lane) & 1u) ? p : 0.0);
            const double e = fmax(df_to_double(s3), 0.0) / (P * P);
            const uint64_t rk = colex_rank_mask(m);
            if (e < best || (e == best && rk < brank)) {
                best = e;
                brank = rk;
                bmask = m;
            }
        }
    }
    if (lane == 0) {
        a.best_gap[row] = (float)sqrt(best);
        a.best_rank[row] = brank;
    }
    const bool mine = (bmask >> lane) & 1u;
    const int pos = __popc(bmask & ((1u << lane) - 1u));
    if (mine) a.best_idx[row * a.k_max + pos] = lane;
    for (int t = k + lane; t < a.k_max; t += 32) a.best_idx[row * a.k_max + t] = -1;
}

// ---- exhaustive path: FBS blocks per listed row, every C(n,k) subset in colex
// order, each evaluated in the difference form around the top-k set
// (es^2 = t + val / P^2) so that heavy keys kept in A0 never cancel.  A first
// pass screens every subset in fp32 with a rigorous error bound; the second
// evaluates in fp64 only those whose lower bound reaches the chunk's smallest
// upper bound.
template <int DPL, typename VT>
__global__ void __launch_bounds__(256) k_enum_exhaustive(const EnumArgs a)
{
    constexpr int d = DPL * 32;
    __shared__ double Gs[33][34];
    __shared__ double Ms[32][33];
    __shared__ float Mf[32][33];  // Ms in fp32, off-diagonal entries doubled
    __shared__ double ps[32];
    __shared__ float pf[32];
    __shared__ float ured_f[256];
    __shared__ double ured_e[256];
    __shared__ unsigned long long ured_r[256];
    __shared__ double s_t, s_P0;
    __shared__ uint32_t s_A0;
    extern __shared__ float dyn[];
    float *Ush = dyn;                 // [33][d+1]
    float *Usl = dyn + 33 * (d + 1);  // [33][d]
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int cnt = *a.fb_count;
    for (int item = blockIdx.x; item < cnt * FBS; item += gridDim.x) {
        const int li = item / FBS, chunk = item % FBS;
        const int64_t row = a.fb_list[li];
        const int64_t g = row / a.R.R;
        const int64_t ri = row - g * a.R.R;
        const int n = a.R.n[g];
        const int k = a.k[row];
        const VT *V = reinterpret_cast<const VT *>(a.R.v) + a.R.v_off[g];
        const float *lg = a.R.logits + a.R.logit_off[g] + ri * n;
        if (wid == 0) {
            const float l = lane < n ? lg[lane] : -INFINITY;
            const float M = warp_max(l);
            double p = lane < n ? exp((double)l - (double)M) : 0.0;
            p = p / warp_sum_d(p);
            ps[lane] = p;
            int rank = 0;
            for (int s = 0; s < n; ++s) {
                const float ls = __shfl_sync(FW_FULL, l, s);
                rank += (ls > l) || (ls == l && s < lane);
            }
            const uint32_t A0 = __ballot_sync(FW_FULL, lane < n && rank < k);
            const df pd = df_from_double(p);
            df mu[DPL], g0[DPL];
#pragma unroll
            for (int t = 0; t < DPL; ++t) mu[t] = g0[t] = df_zero();
            for (int j = 0; j < n; ++j) {
                const df pj = shfl_df(pd, j);
#pragma unroll
                for (int t = 0; t < DPL; ++t)
                    mu[t] = df_add(mu[t], df_mul_f(pj, load_v(V, (int64_t)j * d + lane + 32 * t)));
            }
            for (int j = 0; j < n; ++j) {
                const df pj = shfl_df(pd, j);
#pragma unroll
                for (int t = 0; t < DPL; ++t) {
                    const int c = lane + 32 * t;
                    const df u = df_mul(pj, df_rsub_f(load_v(V, (int64_t)j * d + c), mu[t]));
                    Ush[j * (d + 1) + c] = u.hi;
                    Usl[j * d + c] = u.lo;
                    if ((A0 >> j) & 1u) g0[t] = df_add(g0[t], u);
                }
            }
            df nrm = df_zero();
#pragma unroll
            for (int t = 0; t < DPL; ++t) {
                const int c = lane + 32 * t;
                Ush[n * (d + 1) + c] = g0[t].hi;
                Usl[n * d + c] = g0[t].lo;
                nrm = df_add(nrm, df_mul(g0[t], g0[t]));
            }
            nrm = warp_sum_df(nrm);
            const double P0 = warp_sum_d(((A0 >> lane) & 1u) ? p : 0.0);
            if (lane == 0) {
                s_P0 = P0;
                s_t = fmax(df_to_double(nrm), 0.0) / (P0 * P0);
                s_A0 = A0;
            }
        }
        __syncthreads();
        // Gram entries G_xy = u_x . u_y (row n: g0) in double-float, four
        // interleaved partial sums per product
        for (int q = tid; q < (n + 1) * (n + 1); q += blockDim.x) {
            const int x = q / (n + 1), y = q % (n + 1);
            if (y < x) continue;
            df s4[4] = {df_zero(), df_zero(), df_zero(), df_zero()};
            for (int c = 0; c < d; c += 4) {
#pragma unroll
                for (int c4 = 0; c4 < 4; ++c4) {
                    const df ux = {Ush[x * (d + 1) + c + c4], Usl[x * d + c + c4]};
                    const df uy = {Ush[y * (d + 1) + c + c4], Usl[y * d + c + c4]};
                    s4[c4] = df_add(s4[c4], df_mul(ux, uy));
                }
            }
            const double s = df_to_double(df_add(df_add(s4[0], s4[1]), df_add(s4[2], s4[3])));
            Gs[x][y] = s;
            Gs[y][x] = s;
        }
        __syncthreads();
        const double t = s_t, P0 = s_P0;
        const uint32_t A0 = s_A0;
        for (int q = tid; q < n * n; q += blockDim.x) {  // x <= y, mirrored (exactly symmetric)
            const int x = q / n, y = q % n;
            if (y < x) continue;
            const double sx = ((A0 >> x) & 1u) ? -1.0 : 1.0, sy = ((A0 >> y) & 1u) ? -1.0 : 1.0;
            double m = sx * sy * (Gs[x][y] - t * ps[x] * ps[y]);
            if (x == y) m += 2.0 * sx * (Gs[x][n] - t * P0 * ps[x]);
            Ms[x][y] = Ms[y][x] = m;
            Mf[x][y] = Mf[y][x] = (float)(x == y ? m : 2.0 * m);
            if (y == x) pf[x] = (float)ps[x];
        }
        __syncthreads();
        const uint64_t total = binom64(n, k);
        const uint64_t cper = (total + FBS - 1) / FBS;  // this block's share of the colex ranks
        const uint64_t clo = cper * chunk;
        const uint64_t chi = clo + cper < total ? clo + cper : total;
        const uint64_t span = chi > clo ? chi - clo : 0;
        const uint64_t per = (span + blockDim.x - 1) / blockDim.x;
        const uint64_t lo = clo + per * tid;
        const uint64_t hi = lo + per < chi ? lo + per : chi;
        // colex unranking, successor and mask of a k-combination
        auto unrank = [&](uint64_t r, int *cmb) {
            int top = n - 1;
            for (int i = k; i >= 1; --i) {  // largest c with C(c, i) <= r
                int c = i - 1;
                while (c + 1 <= top && binom64(c + 1, i) <= r) ++c;
                r -= binom64(c, i);
                cmb[i - 1] = c;
                top = c - 1;
            }
        };
        auto succ = [&](int *cmb) {
            int i = 0;
            while (i < k - 1 && cmb[i] + 1 == cmb[i + 1]) ++i;
            ++cmb[i];
            for (int q2 = 0; q2 < i; ++q2) cmb[q2] = q2;
        };
        // fp32 value of es^2 in the difference form with a rigorous bound on
        // its error: the fp32 entries are the fp64 ones rounded (relative error
        // u), a sum over N terms in any order adds at most N u times the sum of
        // their magnitudes, P(A) sums k positive terms, and the reciprocal,
        // products and the final sum add a few u more (plus the denormal floor
        // per term)
        const float tf = (float)t;
        auto bound = [&](float val, float ab, float P, float N, float &elo, float &ehi) {
            if (!(P > 1e-17f)) {
                elo = -INFINITY;
                ehi = INFINITY;
                return;
            }
            const float u = 5.9604645e-8f;
            const float inv = __frcp_rn(P * P);
            const float e = tf + val * inv;
            const float err = 1.05f * inv * ((N + 2.f) * u * ab + fabsf(val) * (float)(2 * k + 6) * u +
                                             (N + 2.f) * 1.4013e-45f) +
                              2.f * u * (fabsf(tf) + fabsf(e));
            if (!(fabsf(e) < INFINITY) || !(err < INFINITY)) {
                elo = -INFINITY;
                ehi = INFINITY;
                return;
            }
            elo = e - err;
            ehi = e + err;
        };
        // The chunk's ranks in colex order.  Consecutive ranks mostly differ in
        // the lowest member z only, so for each set of the other k - 1 members
        // ("rest") the part over S_r = rest xor A0 is summed once, and each z
        // adds (z not in A0) or removes (z in A0, hence in S_r) its own row:
        // val(S_r xor {z}) = val(S_r) +- (M'_zz + sum_{y in S_r, y != z} M'_zy),
        // M' = Mf (off-diagonal entries doubled).  f(mask, rank, val, sum of
        // |terms|, P, number of terms).
        auto visit = [&](auto &&f) {
            if (lo >= hi) return;
            int cmb[32];
            unrank(lo, cmb);
            uint64_t rk = lo;
            for (;;) {
                uint32_t rest = 0u;
                for (int i = 1; i < k; ++i) rest |= 1u << cmb[i];
                const uint32_t Sr = rest ^ A0;
                float vr = 0.f, ar = 0.f, Pr = 0.f;
                for (uint32_t m1 = Sr; m1; m1 &= m1 - 1) {
                    const int x = __ffs(m1) - 1;
                    for (uint32_t m2 = m1; m2; m2 &= m2 - 1) {
                        const float v = Mf[x][__ffs(m2) - 1];
                        vr += v;
                        ar += fabsf(v);
                    }
                }
                for (uint32_t m1 = rest; m1; m1 &= m1 - 1) Pr += pf[__ffs(m1) - 1];
                const int sr = __popc(Sr);
                const float Nr = (float)(sr * (sr + 1) / 2 + sr + 1);
                const int zmax = k > 1 ? cmb[1] : n;
                for (int z = cmb[0]; z < zmax; ++z) {
                    float r2 = Mf[z][z], a2 = fabsf(r2);
                    for (uint32_t m1 = Sr & ~(1u << z); m1; m1 &= m1 - 1) {
                        const float v = Mf[z][__ffs(m1) - 1];
                        r2 += v;
                        a2 += fabsf(v);
                    }
                    const float val = ((A0 >> z) & 1u) ? vr - r2 : vr + r2;
                    f(rest | (1u << z), rk, val, ar + a2, Pr + pf[z], Nr);
                    if (++rk >= hi) return;
                }
                if (k == 1) return;  // (all n ranks visited)
                cmb[0] = zmax - 1;   // the run of z is over: next rest
                succ(cmb);
            }
        };
        // pass 1: the smallest upper bound over the chunk
        float ub = INFINITY;
        visit([&](uint32_t, uint64_t, float val, float ab, float P, float N) {
            float elo, ehi;
            bound(val, ab, P, N, elo, ehi);
            ub = fminf(ub, fmaxf(ehi, 0.f));
        });
        ured_f[tid] = ub;
        __syncthreads();
        for (int s = blockDim.x / 2; s > 0; s >>= 1) {
            if (tid < s) ured_f[tid] = fminf(ured_f[tid], ured_f[tid + s]);
            __syncthreads();
        }
        ub = ured_f[0];
        // pass 2: fp64 values of the subsets that may reach that bound
        double best = INFINITY;
        unsigned long long brank = ~0ull;
        visit([&](uint32_t am, uint64_t rk, float val, float ab, float P, float N) {
            float elo, ehi;
            bound(val, ab, P, N, elo, ehi);
            if (!(elo <= ub)) return;
            const uint32_t S = am ^ A0;
            double dv = 0.0, Pd = P0;
            for (uint32_t m1 = S; m1; m1 &= m1 - 1) {
                const int x = __ffs(m1) - 1;
                Pd += ((A0 >> x) & 1u) ? -ps[x] : ps[x];
                dv += Ms[x][x];
                for (uint32_t m2 = m1 & (m1 - 1); m2; m2 &= m2 - 1) dv += 2.0 * Ms[x][__ffs(m2) - 1];
            }
            const double e = fmax(t + dv / (Pd * Pd), 0.0);
            if (e < best) {
                best = e;
                brank = rk;
            }
        });
        ured_e[tid] = best;
        ured_r[tid] = brank;
        __syncthreads();
        for (int s = blockDim.x / 2; s > 0; s >>= 1) {
            if (tid < s) {
                const double e2 = ured_e[tid + s];
                const unsigned long long r2 = ured_r[tid + s];
                if (e2 < ured_e[tid] || (e2 == ured_e[tid] && r2 < ured_r[tid])) {
                    ured_e[tid] = e2;
                    ured_r[tid] = r2;
                }
            }
            __syncthreads();
        }
        if (tid == 0) {
            a.fb_e[(int64_t)li * FBS + chunk] = ured_e[0];
            a.fb_r[(int64_t)li * FBS + chunk] = ured_r[0];
        }
        __syncthreads();
    }
}

// merge the chunks of every exhaustive row: smallest es^2, then smallest rank
__global__ void k_enum_exhaustive_merge(const EnumArgs a)
{
    const int cnt = *a.fb_count;
    for (int li = blockIdx.x * blockDim.x + threadIdx.x; li < cnt; li += gridDim.x * blockDim.x) {
        const int64_t row = a.fb_list[li];
        double be = INFINITY;
        unsigned long long br = ~0ull;
        for (int c = 0; c < FBS; ++c) {
            const double e = a.fb_e[(int64_t)li * FBS + c];
            const unsigned long long r = a.fb_r[(int64_t)li * FBS + c];
            if (e < be || (e == be && r < br)) {
                be = e;
                br = r;
            }
        }
        const int64_t g = row / a.R.R;
        const int n = a.R.n[g];
        const int k = a.k[row];
        a.best_rank[row] = br;
        a.best_gap[row] = (float)sqrt(be);
        uint64_t r = br;
        int top = n - 1;
        for (int i = k; i >= 1; --i) {
            int c = i - 1;
            while (c + 1 <= top && binom64(c + 1, i) <= r) ++c;
            r -= binom64(c, i);
            a.best_idx[row * a.k_max + (i - 1)] = c;
            top = c - 1;
        }
        for (int q2 = k; q2 < a.k_max; ++q2) a.best_idx[row * a.k_max + q2] = -1;
    }
}

}  // namespace

// floats per row slot: the largest table set over every n <= max_n, k <= k_max (odd stride)
static int enum_stride(int max_n, int k_max)
{
    int best = 1;
    for (int n = 1; n <= max_n && n <= 32; ++n)
        for (int k = 1; k <= n && k <= k_max; ++k) {
            const int nL = n - k < EM ? n - k : EM;
            const int v = slot_floats(k, n - k - nL);
            best = v > best ? v : best;
        }
    return best | 1;
}

// Slot stride of the workspace: the largest over every k <= max_n, so that it
// bounds the stride of any k_max.
static int enum_ws_stride(const RowsDev &R) { return enum_stride(R.max_n, R.max_n < 32 ? R.max_n : 32); }

size_t enum_workspace(const RowsDev &R)
{
    const size_t rows = (size_t)R.rows;
    return align256(rows * ECAP * 4) + align256(rows * 4) + align256(rows * 4) + 256 +
           2 * align256(rows * FBS * 8) + align256(rows * (size_t)enum_ws_stride(R) * 4) +
           align256(rows * PERM) + align256(rows * 8);
}

fw_status best_subset(const RowsDev &R, const int32_t *k, uint64_t *best_rank, float *best_gap, int32_t *best_idx,
                      int k_max, float *topk_gap, int32_t *row_status, void *ws, size_t ws_bytes, cudaStream_t s)
{
    if (R.rows == 0) return FW_OK;
    if (ws_bytes < enum_workspace(R)) return FW_ERR_WORKSPACE;
    char *w = (char *)ws;
    EnumArgs a;
    a.R = R;
    a.k = k;
    a.best_rank = best_rank;
    a.best_gap = best_gap;
    a.best_idx = best_idx;
    a.k_max = k_max;
    a.topk_gap = topk_gap;
    a.row_status = row_status;
    a.cand = (uint32_t *)w;
    w += align256((size_t)R.rows * ECAP * 4);
    a.cand_count = (int32_t *)w;
    w += align256((size_t)R.rows * 4);
    a.fb_list = (int32_t *)w;
    w += align256((size_t)R.rows * 4);
    a.fb_count = (int32_t *)w;
    a.stats = (unsigned long long *)(w + 64);  // the same 256-byte block, zeroed below
    w += 256;
    a.fb_e = (double *)w;
    w += align256((size_t)R.rows * FBS * 8);
    a.fb_r = (unsigned long long *)w;
    w += align256((size_t)R.rows * FBS * 8);
    a.slots = (float *)w;
    w += align256((size_t)R.rows * (size_t)enum_ws_stride(R) * 4);
    a.perms = (uint8_t *)w;
    w += align256((size_t)R.rows * PERM);
    a.kg = (float2 *)w;
    a.stride = enum_stride(R.max_n, k_max);
    FW_CUDA_CHECK(cudaMemsetAsync(a.fb_count, 0, 256, s));
    int sms = 0;
    if (device_sms(&sms) != FW_OK) return FW_ERR_CUDA;
    FW_DISPATCH(R.d, R.v_dtype, {
        constexpr int DCH = DPL * 32 < 64 ? DPL * 32 : 64;
        const int ust = (((R.max_n + 1) * (DCH + 1)) + 1) & ~1;
        const size_t smem_p = (size_t)PREP_W * prep_floats(a.stride, ust) * sizeof(float);
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_enum_prep<DPL, VT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem_p));
        FW_LAUNCH((k_enum_prep<DPL, VT>), (unsigned)((R.rows + PREP_W - 1) / PREP_W), 32 * PREP_W, smem_p, s, a);
        const size_t smem_w = (size_t)ERW * a.stride * sizeof(float) + ERW * PERM;
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_enum_walk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_w));
        FW_LAUNCH(k_enum_walk, (unsigned)((R.rows + ERW - 1) / ERW), 32, smem_w, s, a);
        const size_t smem_r = (size_t)RS_W * rescore_floats(ust) * sizeof(float);
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_enum_rescore<DPL, VT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem_r));
        FW_LAUNCH((k_enum_rescore<DPL, VT>), (unsigned)((R.rows + RS_W - 1) / RS_W), 32 * RS_W, smem_r, s, a);
        const size_t smem2 = (size_t)33 * (2 * DPL * 32 + 1) * sizeof(float);
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_enum_exhaustive<DPL, VT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem2));
        FW_LAUNCH((k_enum_exhaustive<DPL, VT>), (unsigned)sms * 4, 256, smem2, s, a);
        FW_LAUNCH(k_enum_exhaustive_merge, 8, 128, 0, s, a);
    });
    return FW_OK;
}

fw_status best_subset_stats(const RowsDev &R, const void *ws, fw_best_subset_stats *out, cudaStream_t s)
{
    const char *w = (const char *)ws;
    const int32_t *cand_count = (const int32_t *)(w + align256((size_t)R.rows * ECAP * 4));
    const char *blk = w + align256((size_t)R.rows * ECAP * 4) + 2 * align256((size_t)R.rows * 4);
    int32_t fb = 0;
    unsigned long long st[4] = {0, 0, 0, 0};
    if (cudaMemcpyAsync(&fb, blk, 4, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaMemcpyAsync(st, blk + 64, sizeof(st), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return FW_ERR_CUDA;
    int64_t cands = 0;
    int32_t buf[4096];
    for (int64_t r0 = 0; r0 < R.rows; r0 += 4096) {
        const int64_t cnt = R.rows - r0 < 4096 ? R.rows - r0 : 4096;
        if (cudaMemcpyAsync(buf, cand_count + r0, (size_t)cnt * 4, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
            cudaStreamSynchronize(s) != cudaSuccess)
            return FW_ERR_CUDA;
        for (int64_t i = 0; i < cnt; ++i)
            if (buf[i] > 0 && buf[i] <= ECAP) cands += buf[i];
    }
    out->rows_exhaustive = fb;
    out->candidates = cands;
    out->inner_nodes = st[0];
    out->inner_leaves = st[1];
    out->inner_ops = st[2];
    out->skipped = st[3];
    return FW_OK;
}

}  // namespace fw
