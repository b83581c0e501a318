// k_enum.cu -- exact ES(k) (Sec. 2.1) by exhaustive search, rows with n <= 32.
//
// Every size-k subset A of the row's keys is examined; the one of smallest
// es(A) is reported (exact ties: smallest colex rank).  Instead of O(k d)
// work per subset, the walk below spends ~4 fp32 instructions per subset:
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

constexpr int EM = 10;    // inner key set size
constexpr int ECAP = 32;  // candidate masks per row
constexpr int MAXD = 24;  // depth bound of the phase-2 walk
constexpr int PERM = 48;  // local index space per row: NS <= EM + 32

__host__ __device__ constexpr int tri(int a, int b, int n) { return a * n - a * (a - 1) / 2 + (b - a); }
__device__ __forceinline__ int tri_s(int a, int b, int n) { return a <= b ? tri(a, b, n) : tri(b, a, n); }

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
    int stride;           // floats per row slot (odd)
};

// Per-row slot (floats), local key order [L (EM, padded) | A0 (k) | H' (nHp)], NS = EM + k + nHp:
//   GP : upper triangle of G'_xy = u_x.u_y - t p_x p_y over the NS local keys
//   AA : a_x [NS];  LL : l_x [NS] (difference-form linear term, sign included)
__host__ __device__ constexpr int slot_floats(int NS) { return NS * (NS + 1) / 2 + 2 * NS; }

struct Walk {
    const float *slot;
    const uint8_t *perm;  // local index -> original key
    int k, nL, nHp, NS;
    float kappa, g0n;
    uint32_t *cand;
    int32_t *ccount;
};

__device__ __forceinline__ float GPx(const Walk &W, int x, int y) { return W.slot[tri_s(x, y, W.NS)]; }
__device__ __forceinline__ float AAx(const Walk &W, int x) { return W.slot[W.NS * (W.NS + 1) / 2 + x]; }
__device__ __forceinline__ float LLx(const Walk &W, int x) { return W.slot[W.NS * (W.NS + 1) / 2 + W.NS + x]; }

// ---- slow path: list every inner set C (size c) of a node whose folded value is <= 0
__device__ __noinline__ void collect(const Walk W, uint32_t amask_outer, const float *w, float q, int c)
{
    uint32_t cm = c == 0 ? 0u : (1u << c) - 1u;
    const uint32_t lim = 1u << W.nL;
    for (;;) {
        float v = q;
        for (uint32_t a = cm; a; a &= a - 1) {
            const int j = __ffs(a) - 1;
            v += w[j];
            for (uint32_t b2 = a & (a - 1); b2; b2 &= b2 - 1) {
                const int j2 = __ffs(b2) - 1;
                v += 2.f * (GPx(W, j, j2) - W.kappa * AAx(W, j) * AAx(W, j2));
            }
        }
        if (v <= 0.f) {
            uint32_t m = amask_outer;
            for (uint32_t a = cm; a; a &= a - 1) m |= 1u << W.perm[__ffs(a) - 1];
            const int s = *W.ccount;
            if (s < ECAP) W.cand[s] = m;
            *W.ccount = s + 1;
        }
        if (c == 0) break;
        const uint32_t lo = cm & (0u - cm);  // next subset of the same size (Gosper's rule)
        const uint32_t r = cm + lo;
        cm = (((r ^ cm) >> 2) / lo) | r;
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
    default: return INFINITY;
    }
}

// Push key e of H' onto the phase-2 path: update h, q, the added-key mask.
__device__ __forceinline__ void push_added(const Walk &W, int e, int depth, bool sform, const float (&aL)[EM],
                                           float (&h)[EM], float &q, const float *base, const int *path,
                                           uint32_t &imask)
{
    const int ly = EM + W.k + e;
    const float ay = AAx(W, ly), kay = W.kappa * ay;
#pragma unroll
    for (int j = 0; j < EM; ++j)
        if (j < W.nL) h[j] += GPx(W, ly, j) - kay * aL[j];
    float dq = GPx(W, ly, ly) - kay * ay + 2.f * base[e];
    if (sform) dq += LLx(W, ly) - 4.f * kay * W.g0n;
    for (int t = 0; t < depth; ++t) {
        const int lz = EM + W.k + path[t];
        dq += 2.f * (GPx(W, ly, lz) - kay * AAx(W, lz));
    }
    q += dq;
    imask |= 1u << W.perm[ly];
}

// The whole walk of one row (one lane).  Compiled once; every kernel
// instantiation calls it.
__device__ __noinline__ void walk_row(const Walk W)
{
    const float kap = W.kappa, g0n = W.g0n;
    const int k = W.k, nL = W.nL, nHp = W.nHp;
    const int A0b = EM, Hb = EM + k;  // local index bases
    float aL[EM], Gd[EM], lS[EM], G2[EM][EM];
#pragma unroll
    for (int x = 0; x < EM; ++x) {
        const bool real = x < nL;
        aL[x] = real ? AAx(W, x) : 0.f;
        Gd[x] = real ? GPx(W, x, x) - kap * aL[x] * aL[x] : INFINITY;
        lS[x] = real ? LLx(W, x) - 4.f * kap * g0n * aL[x] : 0.f;
#pragma unroll
        for (int y = x + 1; y < EM; ++y)
            G2[x][y] = (real && y < nL) ? 2.f * (GPx(W, x, y) - kap * aL[x] * AAx(W, y)) : 0.f;
    }
    float base[MAXD];  // per H' key: sum over the phase-1 outer keys of E(x, y)
    float hst[MAXD][EM];
    float qst[MAXD];
    int path[MAXD];
    const uint32_t nR = 1u << k;
    for (uint32_t R = 0; R < nR; ++R) {
        const int r = __popc(R);
        if (r > nL + nHp) continue;  // cannot add back r keys
        // choose the form with the smaller error bound
        float sR = 0.f, sK = 0.f;
        for (int x = 0; x < k; ++x) {
            const float ax = AAx(W, A0b + x);
            if ((R >> x) & 1u) sR += ax;
            else sK += ax;
        }
        const bool sform = sR * (4.f * g0n + sR) <= sK * sK;
        const uint32_t O = sform ? R : (~R & (nR - 1u));  // outer keys of A0 in this form
        const float sgn = sform ? -1.f : 1.f;            // their sign
        // phase 1: h (inner keys), q, base (H' keys) from scratch
        float h[EM];
#pragma unroll
        for (int j = 0; j < EM; ++j) h[j] = 0.f;
        float q = 0.f;
        for (int y = 0; y < nHp; ++y) base[y] = 0.f;
        for (uint32_t m = O; m; m &= m - 1) {
            const int x = __ffs(m) - 1, lx = A0b + x;
            const float ax = AAx(W, lx);
            const float kax = kap * ax;
#pragma unroll
            for (int j = 0; j < EM; ++j)
                if (j < nL) h[j] += sgn * GPx(W, lx, j) - kax * aL[j];
            float dq = GPx(W, lx, lx) - kax * ax;
            if (sform) dq += LLx(W, lx) - 4.f * kax * g0n;
            for (uint32_t m2 = O & ((1u << x) - 1u); m2; m2 &= m2 - 1) {
                const int ly = A0b + __ffs(m2) - 1;
                dq += 2.f * (GPx(W, lx, ly) - kax * AAx(W, ly));  // sign^2 = +1
            }
            q += dq;
            for (int y = 0; y < nHp; ++y) base[y] += sgn * GPx(W, lx, Hb + y) - kax * AAx(W, Hb + y);
        }
        uint32_t keep0 = 0u;  // original-key mask of the kept part of A0
        for (int x = 0; x < k; ++x)
            if (!((R >> x) & 1u)) keep0 |= 1u << W.perm[A0b + x];
        // phase 2: depth-first over I subset of H' with |I| <= r
        int depth = 0, e = 0;
        uint32_t imask = 0u;
        for (;;) {
            const int c = r - depth;  // inner keys still to add
            if (c >= 0 && c <= nL) {
                float w[EM];
#pragma unroll
                for (int j = 0; j < EM; ++j) w[j] = fmaf(2.f, h[j], Gd[j]) + (sform ? lS[j] : 0.f);
                const float mval = inner_dispatch(c, w, q, G2);
                if (mval <= 0.f) collect(W, keep0 | imask, w, q, c);
            }
            if (!(depth < r && e < nHp && depth < MAXD)) {
                // back up to the next sibling
                bool done = true;
                while (depth > 0) {
                    --depth;
                    const int pe = path[depth];
                    imask &= ~(1u << W.perm[Hb + pe]);
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
            push_added(W, e, depth, sform, aL, h, q, base, path, imask);
            ++depth;
            ++e;
        }
    }
}

// ---- the fast kernel: one warp = 32 rows; prologue and re-scoring are
// warp-cooperative per row, the walk is one row per lane.
template <int DPL, typename VT>
__global__ void __launch_bounds__(32, 1) k_enum(const EnumArgs a)
{
    extern __shared__ float smem[];
    constexpr int d = DPL * 32;
    const int lane = threadIdx.x;
    float *slots = smem;                                                   // [32][stride]
    float *Ust = smem + 32 * a.stride;                                     // [max_n+1][d+1] staging
    const int ust_floats = (((a.R.max_n + 1) * (d + 1)) + 1) & ~1;        // even: keeps pscr 8-byte aligned
    double *pscr = reinterpret_cast<double *>(Ust + ust_floats);           // [32] masses
    uint8_t *perms = reinterpret_cast<uint8_t *>(pscr + 32);               // [32 rows][PERM]
    uint8_t *inv = perms + 32 * PERM;                                      // [32]
    const int64_t row0 = (int64_t)blockIdx.x * 32;

    Walk my;
    bool my_walk = false;

    // ------------------------------------------------------------ prologue
    for (int rr = 0; rr < 32; ++rr) {
        const int64_t row = row0 + rr;
        if (row >= a.R.rows) break;
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
            continue;
        }
        const VT *V = reinterpret_cast<const VT *>(a.R.v) + a.R.v_off[g];
        const float M = warp_max(l);
        double p = lane < n ? exp((double)l - (double)M) : 0.0;
        p = p / warp_sum_d(p);
        int rank = 0;
        for (int s = 0; s < n; ++s) {
            const float ls = __shfl_sync(FW_FULL, l, s);
            rank += (ls > l) || (ls == l && s < lane);
        }
        const bool inA0 = lane < n && rank < k;
        const uint32_t A0 = __ballot_sync(FW_FULL, inA0);
        const df pd = df_from_double(p);
        df mu[DPL];
#pragma unroll
        for (int t = 0; t < DPL; ++t) mu[t] = df_zero();
        for (int j = 0; j < n; ++j) {
            const df pj = shfl_df(pd, j);
#pragma unroll
            for (int t = 0; t < DPL; ++t)
                mu[t] = df_add(mu[t], df_mul_f(pj, load_v(V, (int64_t)j * d + lane + 32 * t)));
        }
        // u_j staged in fp32; g0 = sum_{A0} u_j exactly (double-float), staged as row n
        df g0[DPL];
#pragma unroll
        for (int t = 0; t < DPL; ++t) g0[t] = df_zero();
        for (int j = 0; j < n; ++j) {
            const df pj = shfl_df(pd, j);
            const bool in = (A0 >> j) & 1u;
#pragma unroll
            for (int t = 0; t < DPL; ++t) {
                const int c = lane + 32 * t;
                const df u = df_mul(pj, df_rsub_f(load_v(V, (int64_t)j * d + c), mu[t]));
                Ust[j * (d + 1) + c] = u.hi;
                if (in) g0[t] = df_add(g0[t], u);
            }
        }
        df nrm = df_zero();
#pragma unroll
        for (int t = 0; t < DPL; ++t) {
            nrm = df_add(nrm, df_mul(g0[t], g0[t]));
            Ust[n * (d + 1) + lane + 32 * t] = g0[t].hi;
        }
        nrm = warp_sum_df(nrm);
        const double P0 = warp_sum_d(inA0 ? p : 0.0);
        const double g0n2 = fmax(df_to_double(nrm), 0.0);
        const double t = g0n2 / (P0 * P0);  // es(A0)^2
        const double sqt = sqrt(t);
        if (lane == 0 && a.topk_gap) a.topk_gap[row] = (float)sqrt(t);
        // local key order: L = first nL keys outside A0, then A0, then H'
        const int nL = min(EM, n - k);
        const int nHp = n - k - nL;
        const int NS = EM + k + nHp;
        uint8_t *perm = perms + rr * PERM;
        if (lane < n) {
            const uint32_t below = (1u << lane) - 1u;
            const int bo = __popc(~A0 & below & ((n == 32) ? FW_FULL : ((1u << n) - 1u)));
            const int bi = __popc(A0 & below);
            const int loc = inA0 ? EM + bi : (bo < nL ? bo : EM + k + (bo - nL));
            perm[loc] = (uint8_t)lane;
            inv[lane] = (uint8_t)loc;
            pscr[lane] = p;
        }
        float *slot = slots + (size_t)rr * a.stride;
        for (int i = lane; i < slot_floats(NS); i += 32) slot[i] = 0.f;
        __syncwarp();
        // fp32 Gram entries over the n keys plus g0 (index n), four partial sums each
        const int npr = (n + 1) * (n + 2) / 2;
        const int off_a = NS * (NS + 1) / 2, off_l = off_a + NS;
        for (int qd = lane; qd < npr; qd += 32) {
            int x = 0, rem = qd;
            while (rem >= n + 1 - x) {
                rem -= n + 1 - x;
                ++x;
            }
            const int y = x + rem;  // x <= y <= n
            if (x == n) continue;   // |g0|^2 is known exactly
            float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
            const float *ux = Ust + x * (d + 1), *uy = Ust + y * (d + 1);
#pragma unroll 4
            for (int c = 0; c < d; c += 4) {
                s0 = fmaf(ux[c], uy[c], s0);
                s1 = fmaf(ux[c + 1], uy[c + 1], s1);
                s2 = fmaf(ux[c + 2], uy[c + 2], s2);
                s3 = fmaf(ux[c + 3], uy[c + 3], s3);
            }
            const float gxy = (s0 + s1) + (s2 + s3);
            const double px = pscr[x];
            const int lx = inv[x];
            if (y < n) {
                const double py = pscr[y];
                slot[tri_s(lx, inv[y], NS)] = (float)((double)gxy - t * px * py);
                if (x == y) slot[off_a + lx] = sqrtf(fmaxf(gxy, 0.f)) * 1.0001f + (float)(sqt * px) * 1.0001f;
            } else {
                const double sx = ((A0 >> x) & 1u) ? -1.0 : 1.0;
                slot[off_l + lx] = (float)(2.0 * sx * ((double)gxy - t * P0 * px));
            }
        }
        __syncwarp();
        if (lane == rr && k <= 31) {
            // kappa: 2x the per-subset error bound of an fp32 evaluation of either form
            const int Lc = k * (k + 1) / 2 + 2 * n + 16;
            my.slot = slot;
            my.perm = perm;
            my.k = k;
            my.nL = nL;
            my.nHp = nHp;
            my.NS = NS;
            my.kappa = (float)(2.2 * ((double)d * 0.25 + Lc + 12) * 5.9604644775390625e-8);
            my.g0n = (float)sqrt(g0n2) * 1.0001f;
            my.cand = a.cand + row * ECAP;
            my.ccount = a.cand_count + row;
            my_walk = true;
        }
        if (lane == 0) {
            a.cand_count[row] = k <= 31 ? 0 : ECAP + 1;  // k = 32: the exhaustive path
            if (a.row_status) a.row_status[row] = FW_OK;
        }
        __syncwarp();
    }
    __syncwarp();

    // ------------------------------------------------------------------ walk
    if (my_walk) walk_row(my);
    __syncwarp();

    // ----------------------------------------------------- exact re-scoring
    for (int rr = 0; rr < 32; ++rr) {
        const int64_t row = row0 + rr;
        if (row >= a.R.rows) break;
        const int cc = a.cand_count[row];
        if (cc < 0) continue;  // invalid row, outputs already written
        if (cc > ECAP || cc == 0) {
            if (lane == 0) a.fb_list[atomicAdd(a.fb_count, 1)] = (int)row;
            continue;
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
        df mu[DPL];
#pragma unroll
        for (int t = 0; t < DPL; ++t) mu[t] = df_zero();
        for (int j = 0; j < n; ++j) {
            const df pj = shfl_df(pd, j);
#pragma unroll
            for (int t = 0; t < DPL; ++t)
                mu[t] = df_add(mu[t], df_mul_f(pj, load_v(V, (int64_t)j * d + lane + 32 * t)));
        }
        double best = INFINITY;
        uint64_t brank = ~0ull;
        uint32_t bmask = 0u;
        for (int ci = 0; ci < cc; ++ci) {
            const uint32_t m = a.cand[row * ECAP + ci];
            df gv[DPL];
#pragma unroll
            for (int t = 0; t < DPL; ++t) gv[t] = df_zero();
            for (uint32_t mm = m; mm; mm &= mm - 1) {
                const int j = __ffs(mm) - 1;
                const df pj = shfl_df(pd, j);
#pragma unroll
                for (int t = 0; t < DPL; ++t)
                    gv[t] = df_add(gv[t], df_mul(pj, df_rsub_f(load_v(V, (int64_t)j * d + lane + 32 * t), mu[t])));
            }
            df s = df_zero();
#pragma unroll
            for (int t = 0; t < DPL; ++t) s = df_add(s, df_mul(gv[t], gv[t]));
            s = warp_sum_df(s);
            const double P = warp_sum_d(((m >> lane) & 1u) ? p : 0.0);
            const double e = fmax(df_to_double(s), 0.0) / (P * P);
            const uint64_t rk = colex_rank_mask(m);
            if (e < best || (e == best && rk < brank)) {
                best = e;
                brank = rk;
                bmask = m;
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
}

// ---- exhaustive fp64 path: one block per listed row, every C(n,k) subset in
// colex order, each evaluated in the difference form around the top-k set
// (es^2 = t + val / P^2) so that heavy keys kept in A0 never cancel.
template <int DPL, typename VT>
__global__ void __launch_bounds__(256) k_enum_exhaustive(const EnumArgs a)
{
    constexpr int d = DPL * 32;
    __shared__ double Gs[33][34];
    __shared__ double Ms[32][33];
    __shared__ double ps[32];
    __shared__ double ured_e[256];
    __shared__ unsigned long long ured_r[256];
    __shared__ double s_t, s_P0;
    __shared__ uint32_t s_A0;
    extern __shared__ float dyn[];
    float *Ush = dyn;                 // [33][d+1]
    float *Usl = dyn + 33 * (d + 1);  // [33][d]
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int cnt = *a.fb_count;
    for (int li = blockIdx.x; li < cnt; li += gridDim.x) {
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
        for (int q = tid; q < (n + 1) * (n + 1); q += blockDim.x) {
            const int x = q / (n + 1), y = q % (n + 1);
            if (y < x) continue;
            double s = 0.0;
            for (int c = 0; c < d; ++c)
                s += ((double)Ush[x * (d + 1) + c] + (double)Usl[x * d + c]) *
                     ((double)Ush[y * (d + 1) + c] + (double)Usl[y * d + c]);
            Gs[x][y] = s;
            Gs[y][x] = s;
        }
        __syncthreads();
        const double t = s_t, P0 = s_P0;
        const uint32_t A0 = s_A0;
        for (int q = tid; q < n * n; q += blockDim.x) {
            const int x = q / n, y = q % n;
            const double sx = ((A0 >> x) & 1u) ? -1.0 : 1.0, sy = ((A0 >> y) & 1u) ? -1.0 : 1.0;
            double m = sx * sy * (Gs[x][y] - t * ps[x] * ps[y]);
            if (x == y) m += 2.0 * sx * (Gs[x][n] - t * P0 * ps[x]);
            Ms[x][y] = m;
        }
        __syncthreads();
        const uint64_t total = binom64(n, k);
        const uint64_t per = (total + blockDim.x - 1) / blockDim.x;
        const uint64_t lo = per * tid;
        const uint64_t hi = lo + per < total ? lo + per : total;
        double best = INFINITY;
        unsigned long long brank = ~0ull;
        if (lo < hi) {
            int cmb[32];
            uint64_t r = lo;
            int top = n - 1;
            for (int i = k; i >= 1; --i) {  // unrank: largest c with C(c, i) <= r
                int c = i - 1;
                while (c + 1 <= top && binom64(c + 1, i) <= r) ++c;
                r -= binom64(c, i);
                cmb[i - 1] = c;
                top = c - 1;
            }
            for (uint64_t rk = lo; rk < hi; ++rk) {
                uint32_t am = 0u;
                for (int i = 0; i < k; ++i) am |= 1u << cmb[i];
                const uint32_t S = am ^ A0;
                double val = 0.0, P = P0;
                for (uint32_t m1 = S; m1; m1 &= m1 - 1) {
                    const int x = __ffs(m1) - 1;
                    P += ((A0 >> x) & 1u) ? -ps[x] : ps[x];
                    val += Ms[x][x];
                    for (uint32_t m2 = m1 & (m1 - 1); m2; m2 &= m2 - 1) val += 2.0 * Ms[x][__ffs(m2) - 1];
                }
                const double e = fmax(t + val / (P * P), 0.0);
                if (e < best) {
                    best = e;
                    brank = rk;
                }
                int i = 0;  // colex successor
                while (i < k - 1 && cmb[i] + 1 == cmb[i + 1]) ++i;
                ++cmb[i];
                for (int q2 = 0; q2 < i; ++q2) cmb[q2] = q2;
            }
        }
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
            const unsigned long long rk = ured_r[0];
            a.best_rank[row] = rk;
            a.best_gap[row] = (float)sqrt(ured_e[0]);
            uint64_t r = rk;
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
        __syncthreads();
    }
}

}  // namespace

// NS = EM + k + nHp <= max(n, EM + k): sized from the largest n and k
static int enum_stride(int max_n, int k_max)
{
    const int kk = k_max < max_n ? k_max : max_n;
    const int NS = max_n > EM + kk ? max_n : EM + kk;
    return slot_floats(NS) | 1;
}

size_t enum_workspace(const RowsDev &R)
{
    const size_t rows = (size_t)R.rows;
    return align256(rows * ECAP * 4) + align256(rows * 4) + align256(rows * 4) + 256;
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
    a.stride = enum_stride(R.max_n, k_max);
    FW_CUDA_CHECK(cudaMemsetAsync(a.fb_count, 0, sizeof(int32_t), s));
    FW_DISPATCH(R.d, R.v_dtype, {
        const size_t smem = ((size_t)32 * a.stride + (size_t)(R.max_n + 1) * (DPL * 32 + 1) + 2) * sizeof(float) +
                            32 * sizeof(double) + 32 * PERM + 32;
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_enum<DPL, VT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        const unsigned grid = (unsigned)((R.rows + 31) / 32);
        FW_LAUNCH((k_enum<DPL, VT>), grid, 32, smem, s, a);
        const size_t smem2 = (size_t)33 * (2 * DPL * 32 + 1) * sizeof(float);
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_enum_exhaustive<DPL, VT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem2));
        FW_LAUNCH((k_enum_exhaustive<DPL, VT>), 152, 256, smem2, s, a);
    });
    return FW_OK;
}

}  // namespace fw
