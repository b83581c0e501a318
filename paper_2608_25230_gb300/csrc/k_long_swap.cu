// k_long_swap.cu -- the balancing selector (Sec. 2.1) inside the candidate set
// (Definition 2.2) for rows of any length.
//
// One persistent block walks rows.  Per row, one pass over the keys
// accumulates the band sums S_b = sum p_j v_j (band = number of budgets that
// drop key j), the band masses and every key's single-key error
// p_j ||v_j - o|| (o = the dense output given by fw_dense_and_topk_gap).  Per
// budget: the E extras are the dropped keys of largest single-key error (a
// radix select on the error's bits, ties to lower indices); the current set
// is described by
//   g = sum_{A} u_i = pbar(A) N_A - p(A) N_{A^c},  u_i = p_i w_i,  w = v - mu,
// with mu = sum_b S_b and disjoint sums, so g carries no cancellation.
//
// Scoring a swap.  With N = |g|^2 and P = p(A), exchanging kept i for pool key
// j changes es^2 by D_ij / (P^2 P'^2), P' = P + p_j - p_i, where
//   D_ij = (alpha_i + beta_j - 2 p_i p_j C_ij) P^2 - N (p_j - p_i)(2P + p_j - p_i),
//   alpha_i = p_i^2 |w_i|^2 - 2 p_i g.w_i,  beta_j = p_j^2 |w_j|^2 + 2 p_j g.w_j,
//   C_ij = w_i . w_j.
// The swap lowers es iff D_ij < 0; the round takes the pair of smallest
// D_ij / P'^2 (ties: smallest i, then j) and stops when that is not negative.
//
// Only C_ij needs a d-long product per pair, and |C_ij| <= |w_i||w_j|.  Each
// round therefore works in three steps:
//  1. one pass over the kept keys computes g.w_i exactly (so alpha_i) and a
//     lower bound of min_j D_ij / P'^2 in which C_ij is replaced by that
//     Cauchy-Schwarz bound and the pool is taken in 8 groups of consecutive
//     beta_j, each group through its least beta_j, largest p_j|w_j| and
//     extreme p_j (D is increasing in p_j - p_i for p_j - p_i > -P);
//  2. the key with the least bound is scored exactly against the whole pool,
//     which bounds the round's best score from above;
//  3. every key whose bound does not exceed that (plus a rounding allowance)
//     is scored exactly, and the best of those pairs is the round's choice.
// A key whose bound exceeds an attained score cannot hold the minimum, so the
// choice is the one that scoring every pair would make; on measured rows the
// bound leaves about 0.1-3 % of the kept keys to step 3.
#include <algorithm>

#include "fw_internal.h"

namespace fw {
namespace {

constexpr int SWT = 256;     // threads per block
constexpr int SWMAXE = kLongSwapMaxE;  // largest pool size E
constexpr int SWGRP = 8;     // pool groups in the lower bound
constexpr int QL = 4;        // lanes per kept key in the passes over kept keys
constexpr int KPI = SWT / QL;  // kept keys per block iteration

struct LSArgs {
    RowsDev R;
    const int32_t *k;
    int nb;
    const uint32_t *thr_key;
    const int32_t *thr_idx;
    const float *o;
    const float *row_max;
    const float *row_sum;
    int E, Ep, max_swaps;
    int32_t *n_swaps, *swap_out, *swap_in, *capped;
    float *refined_gap, *topk_gap;
    // per-block scratch, each [gridDim.x][max_n]
    float *ebuf;     // single-key error^2 of every key
    int32_t *kbuf;   // key at each position of the current kept list
    float *pbuf;     // its mass
    float *xbuf;     // its |w|^2
    float *lbuf;     // its lower bound of the round
    float *abuf;     // its alpha of the round
    int32_t *sbuf;   // positions left for exact scoring
};

__device__ __forceinline__ float block_sum(float v, float *red)
{
    v = warp_sum(v);
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) red[w] = v;
    __syncthreads();
    float t = 0.f;
    for (int i = 0; i < SWT / 32; ++i) t += red[i];
    __syncthreads();
    return t;
}

__device__ __forceinline__ float block_min(float v, float *red)
{
    v = warp_min(v);
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) red[w] = v;
    __syncthreads();
    float t = INFINITY;
    for (int i = 0; i < SWT / 32; ++i) t = fminf(t, red[i]);
    __syncthreads();
    return t;
}

// Eight consecutive elements of a value row as floats (p 16-byte aligned).
__device__ __forceinline__ void ld8(const uint16_t *p, float (&x)[8])
{
    const uint4 u = __ldg(reinterpret_cast<const uint4 *>(p));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int m = 0; m < 4; ++m) {
        x[2 * m] = __uint_as_float(w[m] << 16);
        x[2 * m + 1] = __uint_as_float(w[m] & 0xffff0000u);
    }
}
__device__ __forceinline__ void ld8(const float *p, float (&x)[8])
{
    const float4 a = __ldg(reinterpret_cast<const float4 *>(p));
    const float4 b = __ldg(reinterpret_cast<const float4 *>(p) + 1);
    x[0] = a.x, x[1] = a.y, x[2] = a.z, x[3] = a.w;
    x[4] = b.x, x[5] = b.y, x[6] = b.z, x[7] = b.w;
}

// D_ij / P'^2 for one pair (the fast form of the file comment).
__device__ __forceinline__ float pair_score(float alpha, float p_i, float p_j, float beta, float cij, float P,
                                           float P2, float N)
{
    const float cross = p_i * p_j * cij;
    const float delta = alpha + beta - 2.f * cross;
    const float dp = p_j - p_i;
    const float Pp = P + dp;
    const float D = delta * P2 - N * dp * (2.f * P + dp);
    return D / (Pp * Pp);
}

// The fast form divides D (a difference of terms of size ~N P^2) by P'^2, so
// its rounding grows like P^2 / P'^2; it is trusted while P'^2 >= P^2 / 16
// (error ~1e-6 N, inside the decision margins that matter).  A swap that
// removes more of the kept mass is rescored from g' = g - u_i + u_j, which keeps
// the cancellation in d-vectors.
__device__ __forceinline__ bool needs_vector(float P, float p_i, float p_j)
{
    const float Pp = P + p_j - p_i;
    return !(16.f * Pp * Pp >= P * P);
}

// Rounding allowances of the lower bound.  alpha_i and beta_j are computed once
// and shared by the bound and the exact scores, so the bound only has to cover
// the few operations that combine them (kRoundRel, about 16 ulps, of their
// magnitude), the
// rounding of the computed cross product C_ij against |w_i||w_j| (d ulps at
// most) and, where a pair may take the vector form, that form's rounding.
constexpr float kRoundRel = 1e-6f;
constexpr float kUlp = 1.2e-7f;

// The score from |g'|^2, g' = g - u_i + u_j summed by the caller.
__device__ __forceinline__ float vector_score(float gp2, float P, float p_i, float p_j, float P2, float N)
{
    const float Pp = P + p_j - p_i;
    return gp2 * (P2 / (Pp * Pp)) - N;
}

__device__ __forceinline__ bool pair_less(float s, unsigned long long k, float bs, unsigned long long bk)
{
    return s < bs || (s == bs && k < bk);
}

// Exact scores of the pairs of the kept positions in list[0, cnt) (entries
// < 0 are skipped), 4 lanes per position; folds them into the calling lane's
// best (score, (i, j) key, position, slot).  Block-uniform in cnt.
template <int DPL, typename VT>
__device__ __forceinline__ void score_positions(const int *list, int cnt, const int *kb, const float *pk,
                                                const float *ak, const float *xk, const VT *V, const float *mu,
                                                const float *g, const float *Wt, int Ep, const float *pj,
                                                const float *betaj, const float *rj, const int *idxj, int nadd,
                                                float P, float P2, float N, float sqN, float &best,
                                                unsigned long long &bkey, int &bt, int &bq)
{
    constexpr int d = DPL * 32;
    constexpr int CPL = d / QL;
    const int lane = threadIdx.x & 31, gq = threadIdx.x / QL, sub = threadIdx.x % QL;
    for (int s0 = 0; s0 < cnt; s0 += KPI) {
        const int s = s0 + gq;
        const int t0 = s < cnt ? list[s] : -1;
        const bool valid = t0 >= 0;
        const int t = valid ? t0 : 0;
        const int i = kb[t];
        const float p_i = pk[t], al = ak[t], s_i = p_i * sqrtf(xk[t]);
        const VT *vr = V + (int64_t)i * d + sub * CPL;
        const float *mur = mu + sub * CPL;
        for (int q0 = 0; q0 < Ep; q0 += 16) {
            float acc[16];
#pragma unroll
            for (int m = 0; m < 16; ++m) acc[m] = 0.f;
#pragma unroll 2
            for (int c0 = 0; c0 < CPL; c0 += 8) {
                float x[8];
                ld8(vr + c0, x);
#pragma unroll
                for (int m = 0; m < 8; ++m) {
                    const float w = x[m] - mur[c0 + m];
                    const float4 *wr = reinterpret_cast<const float4 *>(Wt + (sub * CPL + c0 + m) * Ep + q0);
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const float4 W4 = wr[u];
                        acc[4 * u] = fmaf(w, W4.x, acc[4 * u]);
                        acc[4 * u + 1] = fmaf(w, W4.y, acc[4 * u + 1]);
                        acc[4 * u + 2] = fmaf(w, W4.z, acc[4 * u + 2]);
                        acc[4 * u + 3] = fmaf(w, W4.w, acc[4 * u + 3]);
                    }
                }
            }
            // reduce-scatter over the 4 lanes: lane `sub` ends with slots q0 + 4 sub + m
            float h8[8];
#pragma unroll
            for (int m = 0; m < 8; ++m) {
                const bool up = sub & 2;
                const float send = up ? acc[m] : acc[m + 8];
                const float keep = up ? acc[m + 8] : acc[m];
                h8[m] = keep + __shfl_xor_sync(FW_FULL, send, 2);
            }
            float h4[4];
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                const bool up = sub & 1;
                const float send = up ? h8[m] : h8[m + 4];
                const float keep = up ? h8[m + 4] : h8[m];
                h4[m] = keep + __shfl_xor_sync(FW_FULL, send, 1);
            }
            uint32_t fl = 0;  // pairs left to the vector form
            if (valid) {
#pragma unroll
                for (int m = 0; m < 4; ++m) {
                    const int q = q0 + 4 * sub + m;
                    if (q < nadd) {
                        const float sc = pair_score(al, p_i, pj[q], betaj[q], h4[m], P, P2, N);
                        if (needs_vector(P, p_i, pj[q])) {
                            fl |= 1u << m;
                            continue;
                        }
                        const unsigned long long key =
                            ((unsigned long long)(uint32_t)i << 32) | (uint32_t)idxj[q];
                        if (pair_less(sc, key, best, bkey)) {
                            best = sc;
                            bkey = key;
                            bt = t;
                            bq = q;
                        }
                    }
                }
            }
            if (__any_sync(FW_FULL, fl != 0)) {
                // warp-uniform walk over the group's 16 pairs; each flagged pair is
                // summed by the 4 lanes of its group and scored by its owner lane
                for (int src = 0; src < QL; ++src) {
                    const uint32_t fs = __shfl_sync(FW_FULL, fl, (lane & ~(QL - 1)) | src);
                    for (int m = 0; m < 4; ++m) {
                        const bool need = (fs >> m) & 1u;
                        if (!__any_sync(FW_FULL, need)) continue;
                        const int q = q0 + 4 * src + m;
                        float gv = 0.f;
                        if (need) {
                            const float pq = pj[q];
                            for (int c0 = 0; c0 < CPL; c0 += 8) {
                                float x[8];
                                ld8(vr + c0, x);
#pragma unroll
                                for (int u = 0; u < 8; ++u) {
                                    const int c = sub * CPL + c0 + u;
                                    const float gp = fmaf(pq, Wt[c * Ep + q], fmaf(-p_i, x[u] - mu[c], g[c]));
                                    gv = fmaf(gp, gp, gv);
                                }
                            }
                        }
                        gv += __shfl_xor_sync(FW_FULL, gv, 1);
                        gv += __shfl_xor_sync(FW_FULL, gv, 2);
                        if (need && sub == src) {
                            const float sc = vector_score(gv, P, p_i, pj[q], P2, N);
                            const unsigned long long key =
                                ((unsigned long long)(uint32_t)i << 32) | (uint32_t)idxj[q];
                            if (pair_less(sc, key, best, bkey)) {
                                best = sc;
                                bkey = key;
                                bt = t;
                                bq = q;
                            }
                        }
                    }
                }
            }
        }
    }
}

template <int DPL, typename VT>
__global__ void __launch_bounds__(SWT, 2) k_long_swap(const LSArgs a)
{
    constexpr int d = DPL * 32;
    constexpr int CPL = d / QL;  // columns per lane of a 4-lane group
    const int Ep = a.Ep;         // pool slots, a multiple of 16
    extern __shared__ __align__(16) float sm[];
    float *S = sm;                     // [5][d] band sums of p v
    float *mu = S + 5 * d;             // [d]
    float *o = mu + d;                 // [d]   dense output given by the caller
    float *g = o + d;                  // [d]
    float *wdep = g + d;               // [d]   w of the key leaving A
    float *wtmp = wdep + d;            // [d]   w of a single key being scored / entering A
    float *Wt = wtmp + d;              // [d][Ep] pool vectors w_j, slot-major inner
    float *pj = Wt + d * Ep;           // [Ep] masses of the pool slots
    float *betaj = pj + Ep;            // [Ep]
    float *rj = betaj + Ep;            // [Ep] p_j |w_j|
    int *idxj = reinterpret_cast<int *>(rj + Ep);      // [Ep] keys in the slots
    int *ord = idxj + Ep;                               // [Ep] slots by ascending beta
    int *cand = ord + Ep;                               // [KPI] nominated positions
    float4 *grp = reinterpret_cast<float4 *>(cand + KPI);  // [SWGRP] bmin, rmax, pmin, pmax
    float *gab = reinterpret_cast<float *>(grp + SWGRP);  // [SWGRP] largest |beta| of each group
    float *red = gab + SWGRP;          // [32]
    float *mass = red + 32;            // [8]
    uint32_t *hist = reinterpret_cast<uint32_t *>(mass + 8);  // [256]
    __shared__ uint32_t s_misc[8];
    __shared__ int s_cnt, s_bt, s_bq;
    __shared__ float s_best;
    __shared__ unsigned long long s_bkey;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int gq = tid / QL, sub = tid % QL;  // 4-lane group and lane within it
    const size_t boff = (size_t)blockIdx.x * a.R.max_n;
    float *eb = a.ebuf + boff;
    int *kb = a.kbuf + boff;
    float *pk = a.pbuf + boff;
    float *xk = a.xbuf + boff;
    float *lbk = a.lbuf + boff;
    float *ak = a.abuf + boff;
    int *sl = a.sbuf + boff;
    const int nb = a.nb, MS = a.max_swaps;

    for (int64_t row = blockIdx.x; row < a.R.rows; row += gridDim.x) {
        const int64_t grp_i = row / a.R.R;
        const int64_t ri = row - grp_i * a.R.R;
        const int n = a.R.n[grp_i];
        const float *lg = a.R.logits + a.R.logit_off[grp_i] + ri * n;
        const VT *V = reinterpret_cast<const VT *>(a.R.v) + a.R.v_off[grp_i];
        const float M = a.row_max[row];
        const float Zi = 1.f / a.row_sum[row];
        uint32_t tk[4];
        int ti[4];
        for (int b = 0; b < 4; ++b) {
            tk[b] = b < nb ? a.thr_key[row * nb + b] : 0u;
            ti[b] = b < nb ? a.thr_idx[row * nb + b] : -1;
        }
        for (int i = tid; i < d; i += SWT) o[i] = a.o[row * d + i];
        for (int i = tid; i < 5 * d; i += SWT) S[i] = 0.f;
        if (tid < 8) mass[tid] = 0.f;
        __syncthreads();
        // ---- one pass: band sums, band masses, single-key errors of every key
        {
            float acc[5][DPL];
            float macc[5];
#pragma unroll
            for (int b = 0; b < 5; ++b) {
                macc[b] = 0.f;
#pragma unroll
                for (int t = 0; t < DPL; ++t) acc[b][t] = 0.f;
            }
            for (int j = wid; j < n; j += SWT / 32) {
                const float x = lg[j];
                const float p = expf(x - M) * Zi;
                const uint32_t key = order_key(x);
                int band = 0;
                for (int b = 0; b < nb; ++b) band += !(key > tk[b] || (key == tk[b] && j <= ti[b]));
                float dist = 0.f;
#pragma unroll
                for (int t = 0; t < DPL; ++t) {
                    const int c = lane + 32 * t;
                    const float v = load_v(V, (int64_t)j * d + c);
#pragma unroll
                    for (int b = 0; b < 5; ++b) acc[b][t] = fmaf(band == b ? p : 0.f, v, acc[b][t]);
                    const float w = v - o[c];
                    dist = fmaf(w, w, dist);
                }
                dist = warp_sum(dist);
#pragma unroll
                for (int b = 0; b < 5; ++b) macc[b] += band == b ? p : 0.f;
                if (lane == 0) eb[j] = p * p * dist;  // single-key error squared
            }
#pragma unroll
            for (int b = 0; b < 5; ++b) {
#pragma unroll
                for (int t = 0; t < DPL; ++t) atomicAdd(&S[b * d + lane + 32 * t], acc[b][t]);
                if (lane == 0) atomicAdd(&mass[b], macc[b]);
            }
        }
        __syncthreads();
        for (int c = tid; c < d; c += SWT) {
            float m = 0.f;
            for (int b = 0; b < 5; ++b) m += S[b * d + c];
            mu[c] = m;
        }
        __syncthreads();

        for (int b = 0; b < nb; ++b) {
            const int64_t rb = row * nb + b;
            const int kbud = a.k[rb];
            int sb = 0;
            for (int b2 = 0; b2 < nb; ++b2) {
                const int k2 = a.k[row * nb + b2];
                sb += (k2 < kbud) || (k2 == kbud && b2 < b);
            }
            if (kbud < 1 || kbud > n) {
                if (tid == 0) {
                    a.n_swaps[rb] = 0;
                    a.refined_gap[rb] = __int_as_float(0x7fc00000);
                    if (a.topk_gap) a.topk_gap[rb] = __int_as_float(0x7fc00000);
                    if (a.capped) a.capped[rb] = 0;
                }
                for (int t = tid; t < MS; t += SWT) a.swap_out[rb * MS + t] = a.swap_in[rb * MS + t] = -1;
                continue;
            }
            // g, P, N for the top-k set; kept-key list
            float P = 0.f, Pb = 0.f;
            for (int q = 0; q < 5; ++q) {
                if (q <= sb) P += mass[q];
                else Pb += mass[q];
            }
            for (int c = tid; c < d; c += SWT) {
                float NA = 0.f, NC = 0.f;
                for (int q = 0; q < 5; ++q) {
                    if (q <= sb) NA += S[q * d + c];
                    else NC += S[q * d + c];
                }
                g[c] = Pb * NA - P * NC;
            }
            if (tid == 0) s_cnt = 0;
            __syncthreads();
            const uint32_t T = tk[b];
            const int TI = ti[b];
            for (int j = tid; j < n; j += SWT) {
                const uint32_t key = order_key(lg[j]);
                if (key > T || (key == T && j <= TI)) kb[atomicAdd(&s_cnt, 1)] = j;
            }
            float gl = 0.f;
            for (int c = tid; c < d; c += SWT) gl = fmaf(g[c], g[c], gl);
            float N = block_sum(gl, red);  // contains the __syncthreads the list needs
            const int nk = s_cnt;
            if (tid == 0 && a.topk_gap) a.topk_gap[rb] = sqrtf(N) / P;
            // ---- pool extras: the E dropped keys of largest error (radix select on the bits)
            const int ndrop = n - kbud;
            const int Eeff = a.E < ndrop ? a.E : ndrop;
            int nadd = 0;
            if (Eeff > 0) {
                uint32_t prefix = 0u, pmask = 0u, rem = (uint32_t)Eeff;
                for (int pass = 0; pass < 4; ++pass) {
                    const int shift = 24 - 8 * pass;
                    for (int i = tid; i < 256; i += SWT) hist[i] = 0u;
                    __syncthreads();
                    for (int j = tid; j < n; j += SWT) {
                        const uint32_t key = order_key(lg[j]);
                        if (key > T || (key == T && j <= TI)) continue;
                        const uint32_t e = __float_as_uint(eb[j]);
                        if ((e & pmask) == prefix) atomicAdd(&hist[(e >> shift) & 255u], 1u);
                    }
                    __syncthreads();
                    if (tid == 0) {
                        uint32_t cum = 0;
                        for (int v = 255; v >= 0; --v) {
                            const uint32_t c = hist[v];
                            if (cum + c >= rem) {
                                s_misc[0] = prefix | ((uint32_t)v << shift);
                                s_misc[1] = rem - cum;
                                break;
                            }
                            cum += c;
                        }
                    }
                    __syncthreads();
                    prefix = s_misc[0];
                    rem = s_misc[1];
                    pmask |= 255u << shift;
                    __syncthreads();
                }
                // keys above the threshold, then the first `rem` equal ones in index order
                if (tid == 0) s_cnt = 0;
                __syncthreads();
                for (int j = tid; j < n; j += SWT) {
                    const uint32_t key = order_key(lg[j]);
                    if (key > T || (key == T && j <= TI)) continue;
                    if (__float_as_uint(eb[j]) > prefix) idxj[atomicAdd(&s_cnt, 1)] = j;
                }
                __syncthreads();
                uint32_t base = 0;
                const int above = s_cnt;
                for (int j0 = 0; j0 < n && base < rem; j0 += SWT) {
                    const int j = j0 + tid;
                    bool match = false;
                    if (j < n) {
                        const uint32_t key = order_key(lg[j]);
                        match = !(key > T || (key == T && j <= TI)) && __float_as_uint(eb[j]) == prefix;
                    }
                    const uint32_t bal = __ballot_sync(FW_FULL, match);
                    if (lane == 0) hist[wid] = __popc(bal);
                    __syncthreads();
                    uint32_t before = 0, total = 0;
                    for (int w = 0; w < SWT / 32; ++w) {
                        if (w < wid) before += hist[w];
                        total += hist[w];
                    }
                    if (match) {
                        const uint32_t r = base + before + __popc(bal & ((1u << lane) - 1u));
                        if (r < rem) idxj[above + r] = j;
                    }
                    __syncthreads();
                    base += total;
                }
                nadd = above + (int)rem;
                __syncthreads();
            }
            // stage the pool: w_j = v_j - mu in slots [0, nadd), zeros above
            for (int e = tid; e < d * Ep; e += SWT) {
                const int c = e / Ep, q = e - c * Ep;
                Wt[e] = q < nadd ? load_v(V, (int64_t)idxj[q] * d + c) - mu[c] : 0.f;
            }
            for (int q = tid; q < Ep; q += SWT) {
                pj[q] = q < nadd ? expf(lg[idxj[q]] - M) * Zi : 0.f;
                if (q >= nadd) idxj[q] = -1;
            }
            __syncthreads();

            int taken = 0, cap = 0;
            bool first = true;
            for (;;) {
                if (nadd == 0 || nk == 0) break;
                const float P2 = P * P, twoP = 2.f * P, sqN = sqrtf(N);
                // ---- pool terms of the round: beta_j, p_j |w_j|; slots ordered by beta
                for (int q = wid; q < nadd; q += SWT / 32) {
                    float s2 = 0.f, sg = 0.f;
                    for (int c = lane; c < d; c += 32) {
                        const float w = Wt[c * Ep + q];
                        s2 = fmaf(w, w, s2);
                        sg = fmaf(g[c], w, sg);
                    }
                    s2 = warp_sum(s2);
                    sg = warp_sum(sg);
                    const float p = pj[q];
                    if (lane == 0) {
                        betaj[q] = p * p * s2 + 2.f * p * sg;
                        rj[q] = p * sqrtf(s2);
                    }
                }
                __syncthreads();
                if (wid == 0) {
                    for (int q = lane; q < nadd; q += 32) {
                        const uint32_t kq = order_key(betaj[q]);
                        int r = 0;
                        for (int q2 = 0; q2 < nadd; ++q2) {
                            const uint32_t k2 = order_key(betaj[q2]);
                            r += (k2 < kq) || (k2 == kq && q2 < q);
                        }
                        ord[r] = q;
                    }
                    __syncwarp();
                    if (lane < SWGRP) {
                        const int lo = lane * nadd / SWGRP, hi = (lane + 1) * nadd / SWGRP;
                        float4 G = make_float4(INFINITY, 0.f, 1.f, 0.f);
                        float ba = 0.f;
                        if (hi > lo) {
                            G.x = betaj[ord[lo]];
                            G.z = INFINITY;
                            for (int r = lo; r < hi; ++r) {
                                const int q = ord[r];
                                G.x = fminf(G.x, betaj[q]);
                                G.y = fmaxf(G.y, rj[q]);
                                G.z = fminf(G.z, pj[q]);
                                G.w = fmaxf(G.w, pj[q]);
                                ba = fmaxf(ba, fabsf(betaj[q]));
                            }
                        }
                        grp[lane] = G;
                        gab[lane] = ba;
                    }
                }
                __syncthreads();
                // ---- step 1: exact g.w_i and the lower bound of every kept key; each
                // 4-lane group nominates the key of least bound among those it saw
                float lbmin = INFINITY;
                int tmin = -1;
                for (int t0 = 0; t0 < nk; t0 += KPI) {
                    const int t = t0 + gq;
                    const bool valid = t < nk;
                    const int i = kb[valid ? t : 0];
                    const VT *vr = V + (int64_t)i * d + sub * CPL;
                    const float *mur = mu + sub * CPL, *gr = g + sub * CPL;
                    float sg = 0.f, s2 = 0.f;
#pragma unroll
                    for (int c0 = 0; c0 < CPL; c0 += 8) {
                        float x[8];
                        ld8(vr + c0, x);
#pragma unroll
                        for (int m = 0; m < 8; ++m) {
                            const float w = x[m] - mur[c0 + m];
                            sg = fmaf(w, gr[c0 + m], sg);
                            if (first) s2 = fmaf(w, w, s2);
                        }
                    }
                    sg += __shfl_xor_sync(FW_FULL, sg, 1);
                    sg += __shfl_xor_sync(FW_FULL, sg, 2);
                    float p_i, x2;
                    if (first) {
                        s2 += __shfl_xor_sync(FW_FULL, s2, 1);
                        s2 += __shfl_xor_sync(FW_FULL, s2, 2);
                        p_i = expf(lg[i] - M) * Zi;
                        x2 = s2;
                        if (valid && sub == 0) {
                            pk[t] = p_i;
                            xk[t] = x2;
                        }
                    } else {
                        p_i = pk[valid ? t : 0];
                        x2 = xk[valid ? t : 0];
                    }
                    const float alpha = p_i * p_i * x2 - 2.f * p_i * sg;
                    const float s_i = p_i * sqrtf(x2);
                    float lb = INFINITY;
#pragma unroll
                    for (int gi = sub; gi < SWGRP; gi += QL) {
                        const float4 G = grp[gi];  // least beta, largest p|w|, least and largest p
                        const float dmax = G.w - p_i, dmin = G.z - p_i;
                        const float dabs = fmaxf(fabsf(dmin), fabsf(dmax));
                        const float sr = s_i * G.y;
                        const float LB = (alpha + G.x - 2.f * sr) * P2 - N * dmax * (twoP + dmax);
                        const float den = LB >= 0.f ? P + dmax : P + dmin;
                        const float dlo = P + dmin;
                        const float mag = (fabsf(alpha) + gab[gi] + 2.f * sr) * P2 + N * dabs * (twoP + dabs);
                        float allow = kRoundRel * mag + (float)d * kUlp * 2.f * sr * P2;
                        if (!(16.f * dlo * dlo >= P2)) {  // some pair may take the vector form
                            const float tv = sqN + s_i + G.y;
                            allow += kRoundRel * tv * tv * P2;
                        }
                        lb = fminf(lb, dlo > 0.f ? LB / (den * den) - allow / (dlo * dlo) : -INFINITY);
                    }
                    lb = fminf(lb, __shfl_xor_sync(FW_FULL, lb, 1));
                    lb = fminf(lb, __shfl_xor_sync(FW_FULL, lb, 2));
                    if (valid) {
                        if (sub == 0) {
                            lbk[t] = lb;
                            ak[t] = alpha;
                        }
                        if (lb < lbmin) {
                            lbmin = lb;
                            tmin = t;
                        }
                    }
                }
                first = false;
                if (sub == 0) cand[gq] = tmin;
                __syncthreads();
                // ---- step 2: exact scores of the nominated keys -> an attained score UB
                float best = INFINITY;
                unsigned long long bkey = ~0ull;
                int bt = -1, bq = -1;
                score_positions<DPL, VT>(cand, KPI, kb, pk, ak, xk, V, mu, g, Wt, Ep, pj, betaj, rj, idxj, nadd, P, P2,
                                         N, sqN, best, bkey, bt, bq);
                const float UB = block_min(best, red);
                // ---- step 3: exact scores of every key whose bound does not exceed UB.
                // A key's bound lies below every score computed for its pairs (the
                // bound carries the rounding allowance), so the keys left out hold no
                // pair scoring at or below UB, and the best pair is among those kept.
                const float thr = UB;
                if (tid == 0) s_cnt = 0;
                __syncthreads();
                for (int t0 = 0; t0 < nk; t0 += SWT) {
                    const int t = t0 + tid;
                    const bool keep = t < nk && !(lbk[t] > thr);
                    const uint32_t bal = __ballot_sync(FW_FULL, keep);
                    int basew = 0;
                    if (lane == 0 && bal) basew = atomicAdd(&s_cnt, __popc(bal));
                    basew = __shfl_sync(FW_FULL, basew, 0);
                    if (keep) sl[basew + __popc(bal & ((1u << lane) - 1u))] = t;
                }
                __syncthreads();
                const int nsv = s_cnt;
                best = INFINITY;
                bkey = ~0ull;
                bt = bq = -1;
                score_positions<DPL, VT>(sl, nsv, kb, pk, ak, xk, V, mu, g, Wt, Ep, pj, betaj, rj, idxj, nadd, P, P2, N,
                                         sqN, best, bkey, bt, bq);
                // block argmin of (score, i, j)
                if (tid == 0) {
                    s_best = INFINITY;
                    s_bkey = ~0ull;
                }
                float wb = warp_min(best);
                if (lane == 0) red[wid] = wb;
                __syncthreads();
                if (tid == 0) {
                    float m = INFINITY;
                    for (int w = 0; w < SWT / 32; ++w) m = fminf(m, red[w]);
                    s_best = m;
                }
                __syncthreads();
                if (best == s_best) atomicMin(&s_bkey, bkey);
                __syncthreads();
                if (best == s_best && bkey == s_bkey && bt >= 0) {
                    s_bt = bt;
                    s_bq = bq;
                }
                __syncthreads();
                const float bs = s_best;
                const unsigned long long bk = s_bkey;
                if (!(bs < 0.f)) break;  // no pair strictly decreases es
                if (taken >= MS) {
                    cap = 1;
                    break;
                }
                // apply: g += u_j - u_i, P += p_j - p_i; slot qj of the pool takes i
                const int bi = (int)(bk >> 32), bj = (int)(bk & 0xffffffffu);
                const int tb = s_bt, qj = s_bq;
                const float p_i = pk[tb];
                const float p_j = pj[qj];
                for (int c = tid; c < d; c += SWT) {
                    wdep[c] = load_v(V, (int64_t)bi * d + c) - mu[c];
                    wtmp[c] = Wt[c * Ep + qj];
                }
                __syncthreads();
                float gl2 = 0.f, x2n = 0.f;
                for (int c = tid; c < d; c += SWT) {
                    const float gn = g[c] + p_j * wtmp[c] - p_i * wdep[c];
                    g[c] = gn;
                    Wt[c * Ep + qj] = wdep[c];
                    gl2 = fmaf(gn, gn, gl2);
                    x2n = fmaf(wtmp[c], wtmp[c], x2n);
                }
                if (tid == 0) {
                    idxj[qj] = bi;
                    pj[qj] = p_i;
                    kb[tb] = bj;
                    pk[tb] = p_j;
                    a.swap_out[rb * MS + taken] = bi;
                    a.swap_in[rb * MS + taken] = bj;
                }
                P = P - p_i + p_j;
                N = block_sum(gl2, red);
                x2n = block_sum(x2n, red);
                if (tid == 0) xk[tb] = x2n;
                __syncthreads();
                ++taken;
            }
            if (tid == 0) {
                a.n_swaps[rb] = taken;
                a.refined_gap[rb] = sqrtf(N) / P;
                if (a.capped) a.capped[rb] = cap;
            }
            for (int t = taken + tid; t < MS; t += SWT) a.swap_out[rb * MS + t] = a.swap_in[rb * MS + t] = -1;
            __syncthreads();
        }
        __syncthreads();
    }
}

// pool slots rounded up to the 16-slot blocks of the exact scoring step
inline int pool_slots(int E) { return std::max(16, (E + 15) / 16 * 16); }

template <int DPL> size_t ls_smem(int Ep)
{
    constexpr int d = DPL * 32;
    return sizeof(float) * (10 * (size_t)d + (size_t)d * Ep + 5 * (size_t)Ep + KPI + 5 * SWGRP + 32 + 8 + 256) + 64;
}

}  // namespace

// two resident blocks per SM (the launch bounds guarantee the registers for it)
static unsigned ls_grid(const RowsDev &R) { return (unsigned)std::min<int64_t>(R.rows, 152 * 2); }

static size_t ls_array_bytes(const RowsDev &R) { return align256((size_t)ls_grid(R) * R.max_n * 4); }

size_t long_swap_workspace(const RowsDev &R, int nb, int E, int max_swaps)
{
    (void)nb, (void)E, (void)max_swaps;
    return ls_array_bytes(R) * 7;
}

fw_status long_swap(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &topk, int E, int max_swaps,
                    int32_t *n_swaps, int32_t *swap_out, int32_t *swap_in, float *refined_gap, float *topk_gap,
                    int32_t *capped, void *ws, size_t ws_bytes, cudaStream_t s)
{
    (void)ws_bytes;
    if (E > SWMAXE) return FW_ERR_UNSUPPORTED;
    LSArgs a;
    a.R = R;
    a.k = k;
    a.nb = nb;
    a.thr_key = topk.thr_key;
    a.thr_idx = topk.thr_idx;
    a.o = topk.o;
    a.row_max = topk.row_max;
    a.row_sum = topk.row_sum;
    a.E = E;
    a.Ep = pool_slots(E);
    a.max_swaps = max_swaps;
    a.n_swaps = n_swaps;
    a.swap_out = swap_out;
    a.swap_in = swap_in;
    a.capped = capped;
    a.refined_gap = refined_gap;
    a.topk_gap = topk_gap;
    const unsigned grid = ls_grid(R);
    const size_t arr = ls_array_bytes(R);
    char *w = (char *)ws;
    a.ebuf = (float *)(w + 0 * arr);
    a.kbuf = (int32_t *)(w + 1 * arr);
    a.pbuf = (float *)(w + 2 * arr);
    a.xbuf = (float *)(w + 3 * arr);
    a.lbuf = (float *)(w + 4 * arr);
    a.abuf = (float *)(w + 5 * arr);
    a.sbuf = (int32_t *)(w + 6 * arr);
    FW_DISPATCH(R.d, R.v_dtype, {
        const size_t smem = ls_smem<DPL>(a.Ep);
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_long_swap<DPL, VT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem));
        FW_LAUNCH((k_long_swap<DPL, VT>), grid, SWT, smem, s, a);
    });
    return FW_OK;
}

}  // namespace fw
