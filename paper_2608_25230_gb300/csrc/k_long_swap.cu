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
// Only C_ij needs a d-long product per pair, and it does not depend on g: a
// swap changes one kept position (the key that enters) and one pool slot (the
// key that leaves takes the entering key's slot).  So the block keeps the
// table C[slot][position] in its workspace: the first round of a budget fills
// it (a k x d by d x E product in register tiles), and every later round
// recomputes only the changed slot's column and the changed position's row.
// A round is then one pass over the kept keys -- per key the exact product
// g.w_i (so alpha_i), the new column entry, and the scan of its E stored
// entries -- with O(d + E) work per key instead of O(E d).  Four lanes share a
// key (each a quarter of the columns and of the slots); the pass is software
// pipelined (the next key's value row is in flight while the current one is
// scored).  In the scan D_ij is regrouped as A_i + B_j + p_i (h_j + k_j C_ij)
// with per-key A_i and per-slot B_j, h_j, k_j, so a pair costs three fused
// operations and one approximate division.  Each lane keeps its least score
// and the first position where it occurred; the lanes holding the block's
// least score score that position's pairs again with the same operations and
// the smallest (i, j) among the pairs at that score wins.  (Two positions of
// one lane at exactly the same fp32 score keep the first: such pairs are tied
// to ~1e-7 relative, a decision no fp32 evaluation can settle.)
#include <algorithm>
#include <climits>

#include "fw_internal.h"

namespace fw {
namespace {

constexpr int SWT = 256;     // threads per block
constexpr int SWMAXE = kLongSwapMaxE;  // largest pool size E
constexpr int TK = 2;        // kept keys per thread in the first-round product tile
constexpr int TS = 8;        // pool slots per thread in that tile (4 threads cover 32)
constexpr int QL = 4;        // lanes per kept key in the round pass
constexpr int KPI = SWT / QL;  // kept keys per block iteration of the pass
// resident blocks per SM: three for rows up to 8,192 keys (short rounds, whose
// fixed per-round costs want more blocks), two above (the registers keep the
// next key's value row, table entries and mass in flight without spilling)
constexpr int LS_BPS_SHORT = 3, LS_BPS_LONG = 2, LS_LONG_N = 8192;
inline int ls_bps(const RowsDev &R) { return R.max_n > LS_LONG_N ? LS_BPS_LONG : LS_BPS_SHORT; }

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
    // per-block cross-product table, [gridDim.x][cstride][Ep] (position-major)
    float *cbuf;
    int cstride;     // positions per block table (max_n rounded up to a multiple of 4)
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

// The fast form divides D (a difference of terms of size ~N P^2) by P'^2, so
// its rounding grows like P^2 / P'^2; it is trusted while P'^2 >= P^2 / 16.
// A swap that removes more of the kept mass is scored from g' = g - u_i + u_j,
// which keeps the cancellation in d-vectors.

// The score from |g'|^2, g' = g - u_i + u_j.
__device__ __forceinline__ float vector_score(float gp2, float P, float p_i, float p_j, float P2, float N)
{
    const float Pp = P + p_j - p_i;
    return gp2 * (P2 / (Pp * Pp)) - N;
}


// Up to 16 sixteen-byte loads of a value row, all issued before any use:
// NV vectors of 8 bf16 or 4 fp32 elements.
template <typename VT, int NV> struct RowChunk;
template <int NV> struct RowChunk<uint16_t, NV> {
    uint4 u[NV];
    __device__ __forceinline__ void load(const uint16_t *p)
    {
#pragma unroll
        for (int i = 0; i < NV; ++i) u[i] = __ldg(reinterpret_cast<const uint4 *>(p) + i);
    }
    __device__ __forceinline__ float at(int c) const  // c is a constant after unrolling
    {
        const uint4 v = u[c >> 3];
        const int e = (c >> 1) & 3;
        const uint32_t w = e == 0 ? v.x : e == 1 ? v.y : e == 2 ? v.z : v.w;
        return (c & 1) ? __uint_as_float(w & 0xffff0000u) : __uint_as_float(w << 16);
    }
};
template <int NV> struct RowChunk<float, NV> {
    float4 u[NV];
    __device__ __forceinline__ void load(const float *p)
    {
#pragma unroll
        for (int i = 0; i < NV; ++i) u[i] = __ldg(reinterpret_cast<const float4 *>(p) + i);
    }
    __device__ __forceinline__ float at(int c) const
    {
        const float4 v = u[c >> 2];
        const int e = c & 3;
        return e == 0 ? v.x : e == 1 ? v.y : e == 2 ? v.z : v.w;
    }
};

// First round of a budget: C[q][t] = w_{kb[t]} . w_q for every kept position
// t < nk and pool slot q in the 32-slot blocks below nadd.  A thread owns 2
// consecutive positions x 8 slots; the 4 threads of a group cover 32 slots.
// The sum over the d columns runs in column order, as in the later rounds.
template <int DPL, typename VT>
__device__ __forceinline__ void cross_table(const int *kb, int nk, const VT *V, const float *mu, const float *Wt,
                                            int Ep, int nadd, float *cb, int cstride)
{
    constexpr int d = DPL * 32;
    const int sub = threadIdx.x & 3, grp = threadIdx.x >> 2;
    constexpr int GROUPS = SWT / 4;
    for (int base = 0; base < nk; base += GROUPS * TK) {
        const int t0 = base + grp * TK;
        if (t0 >= nk) break;
        const VT *vr[TK];
#pragma unroll
        for (int u = 0; u < TK; ++u) vr[u] = V + (int64_t)kb[t0 + u < nk ? t0 + u : t0] * d;
        for (int q0 = 0; q0 < nadd; q0 += 32) {
            float acc[TK][TS];
#pragma unroll
            for (int u = 0; u < TK; ++u)
#pragma unroll
                for (int s = 0; s < TS; ++s) acc[u][s] = 0.f;
            const float *wq = Wt + q0 + sub * TS;
            // one 16-byte vector per position in flight ahead of the one in use
            constexpr int EPV = 16 / (int)sizeof(VT);
            RowChunk<VT, 1> cur[TK];
#pragma unroll
            for (int u = 0; u < TK; ++u) cur[u].load(vr[u]);
#pragma unroll 1
            for (int c0 = 0; c0 < d; c0 += EPV) {
                RowChunk<VT, 1> nxt[TK];
                const int cn = c0 + EPV < d ? c0 + EPV : c0;
#pragma unroll
                for (int u = 0; u < TK; ++u) nxt[u].load(vr[u] + cn);
#pragma unroll
                for (int m = 0; m < EPV; ++m) {
                    const float mc = mu[c0 + m];
                    const float4 A = *reinterpret_cast<const float4 *>(wq + (c0 + m) * Ep);
                    const float4 B = *reinterpret_cast<const float4 *>(wq + (c0 + m) * Ep + 4);
                    const float ws[TS] = {A.x, A.y, A.z, A.w, B.x, B.y, B.z, B.w};
#pragma unroll
                    for (int u = 0; u < TK; ++u) {
                        const float x = cur[u].at(m) - mc;
#pragma unroll
                        for (int s = 0; s < TS; ++s) acc[u][s] = fmaf(x, ws[s], acc[u][s]);
                    }
                }
#pragma unroll
                for (int u = 0; u < TK; ++u) cur[u] = nxt[u];
            }
            #pragma unroll
            for (int u = 0; u < TK; ++u) {
                float4 *dst = reinterpret_cast<float4 *>(cb + (size_t)(t0 + u) * Ep + q0 + sub * TS);
                __stcs(dst, make_float4(acc[u][0], acc[u][1], acc[u][2], acc[u][3]));
                __stcs(dst + 1, make_float4(acc[u][4], acc[u][5], acc[u][6], acc[u][7]));
            }
        }
    }
}

// The 16-byte vectors sub, sub + 4, ... of a value row (4 lanes per row),
// each lane's loads issued before any use.
template <int DPL, typename VT> struct LaneRow {
    static constexpr int EPV = 16 / (int)sizeof(VT);       // elements per vector
    static constexpr int NVL = DPL * 32 / EPV / QL;          // vectors per lane
    RowChunk<VT, 1> u[NVL];
    __device__ __forceinline__ void load(const VT *vr, int sub)
    {
#pragma unroll
        for (int k = 0; k < NVL; ++k) u[k].load(vr + (k * QL + sub) * EPV);
    }
};

// This lane's part of g.w and |w|^2, w = v - mu.
template <int DPL, typename VT>
__device__ __forceinline__ void lane_products(const VT *vr, const float *mu, const float *g, int sub, float &sg,
                                              float &s2)
{
    using L = LaneRow<DPL, VT>;
    L row;
    row.load(vr, sub);
    sg = 0.f;
    s2 = 0.f;
#pragma unroll
    for (int k = 0; k < L::NVL; ++k) {
        const int c0 = (k * QL + sub) * L::EPV;
#pragma unroll
        for (int e = 0; e < L::EPV; ++e) {
            const float w = row.u[k].at(e) - mu[c0 + e];
            sg = fmaf(w, g[c0 + e], sg);
            s2 = fmaf(w, w, s2);
        }
    }
}

// This lane's part of v.g and v.y from its loaded vectors.
template <int DPL, typename VT>
__device__ __forceinline__ void lane_products_v_row(const LaneRow<DPL, VT> &row, const float *g, const float *y,
                                                    int sub, float &vg, float &vy)
{
    using L = LaneRow<DPL, VT>;
    vg = 0.f;
    vy = 0.f;
#pragma unroll
    for (int k = 0; k < L::NVL; ++k) {
        const int c0 = (k * QL + sub) * L::EPV;
#pragma unroll
        for (int e = 0; e < L::EPV; e += 4) {
            const float4 g4 = *reinterpret_cast<const float4 *>(g + c0 + e);
            const float4 y4 = *reinterpret_cast<const float4 *>(y + c0 + e);
            const float gg[4] = {g4.x, g4.y, g4.z, g4.w}, yy[4] = {y4.x, y4.y, y4.z, y4.w};
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                const float v = row.u[k].at(e + h);
                vg = fmaf(v, gg[h], vg);
                vy = fmaf(v, yy[h], vy);
            }
        }
    }
}

// |g - u_i + u_j|^2 for one pair, from the value row of i and the pool column
// of j (the vector form of needs_vector's pairs).
template <int DPL, typename VT>
__device__ __forceinline__ float vector_gp2(const VT *vr, const float *mu, const float *g, const float *Wt, int Ep,
                                            int q, float p_i, float p_j)
{
    constexpr int d = DPL * 32;
    float gv = 0.f;
    for (int c0 = 0; c0 < d; c0 += 8) {
        float x[8];
        ld8(vr + c0, x);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int c = c0 + u;
            const float gp = fmaf(p_j, Wt[c * Ep + q], fmaf(-p_i, x[u] - mu[c], g[c]));
            gv = fmaf(gp, gp, gv);
        }
    }
    return gv;
}

// Score D / P'^2 of one pair in the regrouped fast form: sq = (B_j, k_j, h_j,
// p_j), Ai = A_i, Pm = P - p_i.
__device__ __forceinline__ float fast_score(float4 sq, float cij, float p_i, float Ai, float Pm)
{
    const float Pp = Pm + sq.w;
    return __fdividef(fmaf(p_i, fmaf(sq.y, cij, sq.z), Ai + sq.x), Pp * Pp);
}

template <int DPL, typename VT>
__device__ __noinline__ float vector_pair_score(const VT *vr, const float *mu, const float *g, const float *Wt, int Ep,
                                                int q, float p_i, float p_j, float P, float P2, float N)
{
    return vector_score(vector_gp2<DPL, VT>(vr, mu, g, Wt, Ep, q, p_i, p_j), P, p_i, p_j, P2, N);
}

// The fast form where P'^2 >= P^2 / 16, else the vector form.
template <int DPL, typename VT>
__device__ __forceinline__ float any_score(float4 sq, float cij, float p_i, float Ai, float Pm, float P, float P2,
                                           float N, const VT *vr, const float *mu, const float *g, const float *Wt,
                                           int Ep, int q)
{
    const float Pp = Pm + sq.w;
    if (16.f * Pp * Pp >= P2) return fast_score(sq, cij, p_i, Ai, Pm);
    return vector_pair_score<DPL, VT>(vr, mu, g, Wt, Ep, q, p_i, sq.w, P, P2, N);
}

template <int DPL, typename VT, int BPS>
__global__ void __launch_bounds__(SWT, BPS) k_long_swap(const LSArgs a)
{
    constexpr int d = DPL * 32;
    const int Ep = a.Ep;         // pool slots, a multiple of 32
    extern __shared__ __align__(16) float sm[];
    float *S = sm;                     // [5][d] band sums of p v
    float *mu = S + 5 * d;             // [d]
    float *o = mu + d;                 // [d]   dense output given by the caller
    float *g = o + d;                  // [d]
    float *wdep = g + d;               // [d]   w of the key that left A last (its pool slot's column)
    float *wtmp = wdep + d;            // [d]   w of the key that entered A last
    float *Wt = wtmp + d;              // [d][Ep] pool vectors w_j, slot-major inner
    // per-round slot terms of the regrouped score: B_j, k_j, h_j, p_j ([Ep] each)
    float *sB = Wt + d * Ep, *sK = sB + Ep, *sH = sK + Ep, *sP = sH + Ep;
    float *pj = sP + Ep;               // [Ep] masses of the pool slots
    float *betaj = pj + Ep;            // [Ep]
    int *idxj = reinterpret_cast<int *>(betaj + Ep);  // [Ep] keys in the slots
    float *red = reinterpret_cast<float *>(idxj + Ep);  // [32]
    float *mass = red + 32;            // [8]
    uint32_t *hist = reinterpret_cast<uint32_t *>(mass + 8);  // [256]
    __shared__ uint32_t s_misc[8];
    __shared__ int s_cnt, s_bt, s_bq;
    __shared__ float s_gm, s_ym, s_pmin;
    __shared__ unsigned long long s_bkey;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int gq = tid / QL, sub = tid % QL;  // key group and lane within it
    const size_t boff = (size_t)blockIdx.x * a.R.max_n;
    float *eb = a.ebuf + boff;
    int *kb = a.kbuf + boff;
    float *pk = a.pbuf + boff;
    float *xk = a.xbuf + boff;
    const int cs = a.cstride;
    float *cb = a.cbuf + (size_t)blockIdx.x * Ep * cs;  // [cs][Ep]
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
            // 16 consecutive keys per warp and step: lanes l and l + 16 find the
            // mass and band of key j0 + (l mod 16); then the warp walks the 16
            // value rows (lane = column), and the 16 partial |v_j - o|^2 are summed
            // by a transposed butterfly (lane l ends with key j0 + (l mod 16))
            constexpr int KS = 16;
            for (int j0 = wid * KS; j0 < n; j0 += (SWT / 32) * KS) {
                const int jl = j0 + (lane & (KS - 1));
                float pl = 0.f;
                int bl = 0;
                if (jl < n) {
                    const float x = lg[jl];
                    pl = expf(x - M) * Zi;
                    const uint32_t key = order_key(x);
                    for (int b = 0; b < nb; ++b) bl += !(key > tk[b] || (key == tk[b] && jl <= ti[b]));
                }
                float dd[KS];
#pragma unroll
                for (int u0 = 0; u0 < KS; u0 += 4) {
                    float v[4][DPL];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int j = j0 + u0 + u < n ? j0 + u0 + u : j0;
#pragma unroll
                        for (int t = 0; t < DPL; ++t) v[u][t] = load_v(V, (int64_t)j * d + lane + 32 * t);
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const float p = __shfl_sync(FW_FULL, pl, u0 + u);
                        const int band = __shfl_sync(FW_FULL, bl, u0 + u);
                        const bool live = j0 + u0 + u < n;
                        // band is the same for the whole warp: one accumulator set is touched
#pragma unroll
                        for (int b = 0; b < 5; ++b)
                            if (live && b == band) {
#pragma unroll
                                for (int t = 0; t < DPL; ++t) acc[b][t] = fmaf(p, v[u][t], acc[b][t]);
                                macc[b] += p;
                            }
                        float dist = 0.f;
#pragma unroll
                        for (int t = 0; t < DPL; ++t) {
                            const float w = v[u][t] - o[lane + 32 * t];
                            dist = fmaf(w, w, dist);
                        }
                        dd[u0 + u] = dist;
                    }
                }
                // transposed butterfly: the step with offset h leaves lane l the
                // keys whose bit h equals lane bit h; after h = 1 it holds key
                // l mod 16, and the last step adds the other half of the columns
#pragma unroll
                for (int h = KS / 2; h >= 1; h >>= 1) {
                    const bool up = lane & h;
#pragma unroll
                    for (int u = 0; u < h; ++u) {
                        const float send = up ? dd[u] : dd[u + h];
                        const float keep = up ? dd[u + h] : dd[u];
                        dd[u] = keep + __shfl_xor_sync(FW_FULL, send, h);
                    }
                }
                dd[0] += __shfl_xor_sync(FW_FULL, dd[0], KS);
                if (jl < n && lane < KS) eb[jl] = pl * pl * dd[0];  // single-key error squared
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
            int tprev = -1, qprev = -1;  // position that entered and slot that changed last round
            for (;;) {
                if (nadd == 0 || nk == 0) break;
                const float P2 = P * P;
                // ---- pool terms of the round: beta_j
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
                        const float beta = p * p * s2 + 2.f * p * sg;
                        betaj[q] = beta;
                        // D_ij = A_i + B_j + p_i (h_j + k_j C_ij) (the file comment's D regrouped)
                        sB[q] = beta * P2 - N * p * fmaf(2.f, P, p);
                        sK[q] = -2.f * P2 * p;
                        sH[q] = 2.f * N * p;
                        sP[q] = p;
                    }
                }
                if (wid == SWT / 32 - 1) {  // mu.g and mu.(changed slot's vector) for the folded products
                    float a1 = 0.f, a2 = 0.f;
                    for (int c = lane; c < d; c += 32) {
                        a1 = fmaf(mu[c], g[c], a1);
                        a2 = fmaf(mu[c], wdep[c], a2);
                    }
                    a1 = warp_sum(a1);
                    a2 = warp_sum(a2);
                    float pm = INFINITY;
                    for (int q = lane; q < nadd; q += 32) pm = fminf(pm, pj[q]);
                    pm = warp_min(pm);
                    if (lane == 0) {
                        s_gm = a1;
                        s_ym = a2;
                        s_pmin = pm;
                    }
                }
                // ---- cross products: the whole table in the first round, else the
                // row of the position that changed (its column entries come below)
                if (first) {
                    cross_table<DPL, VT>(kb, nk, V, mu, Wt, Ep, nadd, cb, cs);
                } else {
                    // warps split the columns, lanes take the slots of a 32-slot block
                    float *part = reinterpret_cast<float *>(hist);  // [8][32]
                    constexpr int CPW = d / (SWT / 32);
                    for (int q0 = 0; q0 < nadd; q0 += 32) {
                        const int q = q0 + lane;
                        float c2 = 0.f;
#pragma unroll 4
                        for (int c = wid * CPW; c < (wid + 1) * CPW; ++c) c2 = fmaf(wtmp[c], Wt[c * Ep + q], c2);
                        part[wid * 32 + lane] = c2;
                        __syncthreads();
                        if (wid == 0 && q < nadd) {
                            float c3 = 0.f;
                            for (int w = 0; w < SWT / 32; ++w) c3 += part[w * 32 + lane];
                            __stcs(cb + (size_t)tprev * Ep + q, c3);
                        }
                        __syncthreads();
                    }
                }
                __syncthreads();
                // ---- one pass over the kept keys: exact g.w_i, the changed slot's
                // entry, and every pair of the key from the table
                // Four lanes per kept key: lane `sub` holds the row's 16-byte
                // vectors sub, sub + 4, ... and the pool slots q0 + 4m + sub of every
                // 32-slot block.  Each lane keeps the least of its scores and the
                // position where it first occurred; the block's least score then
                // picks the lanes whose pairs are scored again.
                float lmin = INFINITY, lp = 0.f, lA = 0.f;
                int lt = -1, li = 0;
                const float gm = s_gm, ym = s_ym;
                const float pmin = s_pmin;  // least pool mass (the vector form's test)
                // the scores of key t (position) from its products; cq0: its table
                // entries of the first 32-slot block, read ahead
                auto score_key = [&](int t, int i, const VT *vr, float sg, float sn, float p_i, float x2, bool col,
                                     float (&cq0)[8]) {
                    const float alpha = p_i * p_i * x2 - 2.f * p_i * sg;
                    const float Ai = alpha * P2 + N * p_i * (2.f * P - p_i);
                    const float Pm = P - p_i;
                    // every pair of this key takes the fast form unless some pool
                    // mass leaves P' below P / 4
                    const bool fast = 16.f * (Pm + pmin) * (Pm + pmin) >= P2;
                    float kmin = INFINITY;
                    for (int q0 = 0; q0 < nadd; q0 += 32) {
                        const int qb = q0 + 8 * sub;  // this lane's 8 consecutive slots
                        float cq[8];
                        if (q0 == 0) {
#pragma unroll
                            for (int m = 0; m < 8; ++m) cq[m] = cq0[m];
                        } else {
                            const float4 *src = reinterpret_cast<const float4 *>(cb + (size_t)t * Ep + qb);
                            const float4 c0 = __ldcs(src), c1 = __ldcs(src + 1);
                            cq[0] = c0.x, cq[1] = c0.y, cq[2] = c0.z, cq[3] = c0.w;
                            cq[4] = c1.x, cq[5] = c1.y, cq[6] = c1.z, cq[7] = c1.w;
                        }
                        if (col && qprev >= qb && qprev < qb + 8) {
                            const int mm = qprev - qb;
#pragma unroll
                            for (int m = 0; m < 8; ++m)
                                if (m == mm) cq[m] = sn;
                            __stcs(cb + (size_t)t * Ep + qprev, sn);
                        }
                        const int nq = nadd - qb;  // slot qb + m exists iff m < nq
                        if (fast && nq >= 8) {
#pragma unroll
                            for (int h = 0; h < 8; h += 4) {
                                const float4 B4 = *reinterpret_cast<const float4 *>(sB + qb + h);
                                const float4 K4 = *reinterpret_cast<const float4 *>(sK + qb + h);
                                const float4 H4 = *reinterpret_cast<const float4 *>(sH + qb + h);
                                const float4 P4 = *reinterpret_cast<const float4 *>(sP + qb + h);
                                kmin = fminf(kmin, fast_score(make_float4(B4.x, K4.x, H4.x, P4.x), cq[h], p_i, Ai, Pm));
                                kmin = fminf(kmin, fast_score(make_float4(B4.y, K4.y, H4.y, P4.y), cq[h + 1], p_i, Ai, Pm));
                                kmin = fminf(kmin, fast_score(make_float4(B4.z, K4.z, H4.z, P4.z), cq[h + 2], p_i, Ai, Pm));
                                kmin = fminf(kmin, fast_score(make_float4(B4.w, K4.w, H4.w, P4.w), cq[h + 3], p_i, Ai, Pm));
                            }
                        } else {
#pragma unroll
                            for (int m = 0; m < 8; ++m)
                                if (m < nq) {
                                    const int q = qb + m;
                                    kmin = fminf(kmin, any_score<DPL, VT>(make_float4(sB[q], sK[q], sH[q], sP[q]), cq[m],
                                                                          p_i, Ai, Pm, P, P2, N, vr, mu, g, Wt, Ep, q));
                                }
                        }
                    }
                    if (kmin < lmin) {  // first position of the lane's least score
                        lmin = kmin;
                        lt = t;
                        li = i;
                        lp = p_i;
                        lA = Ai;
                    }
                };
                auto load_cq0 = [&](int t, float (&cq0)[8]) {  // slots 8 sub .. 8 sub + 7
                    const float4 *src = reinterpret_cast<const float4 *>(cb + (size_t)t * Ep + 8 * sub);
                    const float4 c0 = __ldcs(src), c1 = __ldcs(src + 1);
                    cq0[0] = c0.x, cq0[1] = c0.y, cq0[2] = c0.z, cq0[3] = c0.w;
                    cq0[4] = c1.x, cq0[5] = c1.y, cq0[6] = c1.z, cq0[7] = c1.w;
                };
                if (first) {
                    for (int t0 = 0; t0 < nk; t0 += KPI) {
                        const int t = t0 + gq;
                        const bool valid = t < nk;
                        const int ts = valid ? t : t0;
                        const int i = kb[ts];
                        const VT *vr = V + (int64_t)i * d;
                        float cq0[8];
                        load_cq0(ts, cq0);
                        float sg, sn;  // g.w_i and |w_i|^2 from w itself
                        lane_products<DPL, VT>(vr, mu, g, sub, sg, sn);
                        sg += __shfl_xor_sync(FW_FULL, sg, 1);
                        sn += __shfl_xor_sync(FW_FULL, sn, 1);
                        sg += __shfl_xor_sync(FW_FULL, sg, 2);
                        sn += __shfl_xor_sync(FW_FULL, sn, 2);
                        const float p_i = expf(lg[i] - M) * Zi;
                        if (!valid) continue;
                        if (sub == 0) {
                            pk[t] = p_i;
                            xk[t] = sn;
                        }
                        score_key(t, i, vr, sg, sn, p_i, sn, false, cq0);
                    }
                } else {
                    // software pipeline: the value row, table entries and mass of
                    // the next iteration and the kept index of the one after are in
                    // flight during this one
                    const int niter = (nk + KPI - 1) / KPI;
                    int i_cur = kb[gq < nk ? gq : nk - 1];
                    int i_next = kb[gq + KPI < nk ? gq + KPI : nk - 1];
                    LaneRow<DPL, VT> row;
                    row.load(V + (int64_t)i_cur * d, sub);
                    float cq0[8];
                    load_cq0(gq < nk ? gq : nk - 1, cq0);
                    float p_i = pk[gq < nk ? gq : nk - 1], x2 = xk[gq < nk ? gq : nk - 1];
                    for (int it = 0; it < niter; ++it) {
                        const int t = it * KPI + gq;
                        const bool valid = t < nk;
                        const int tn = t + KPI < nk ? t + KPI : nk - 1;
                        float cqn[8];
                        load_cq0(tn, cqn);
                        const float p_n = pk[tn], x2_n = xk[tn];
                        LaneRow<DPL, VT> rown;
                        rown.load(V + (int64_t)i_next * d, sub);
                        const int tnn = t + 2 * KPI;
                        const int i_nn = kb[tnn < nk ? tnn : nk - 1];
                        float sg, sn;  // v_i.g and v_i . (the changed slot's vector)
                        lane_products_v_row<DPL, VT>(row, g, wdep, sub, sg, sn);
                        sg += __shfl_xor_sync(FW_FULL, sg, 1);
                        sn += __shfl_xor_sync(FW_FULL, sn, 1);
                        sg += __shfl_xor_sync(FW_FULL, sg, 2);
                        sn += __shfl_xor_sync(FW_FULL, sn, 2);
                        if (valid)
                            score_key(t, i_cur, V + (int64_t)i_cur * d, sg - gm, sn - ym, p_i, x2, t != tprev, cq0);
                        row = rown;
                        i_cur = i_next;
                        i_next = i_nn;
#pragma unroll
                        for (int m = 0; m < 8; ++m) cq0[m] = cqn[m];
                        p_i = p_n;
                        x2 = x2_n;
                    }
                }
                first = false;
                // the block's least score
                {
                    const float wb = warp_min(lmin);
                    if (lane == 0) red[wid] = wb;
                    if (tid == 0) s_bkey = ~0ull;
                }
                __syncthreads();
                float bmin = INFINITY;
                for (int w = 0; w < SWT / 32; ++w) bmin = fminf(bmin, red[w]);
                // the lanes that attain it score their position's pairs again (the
                // same operations on the same inputs); the smallest (i, j) wins
                unsigned long long mykey = ~0ull;
                int myt = -1, myq = -1;
                if (bmin < 0.f && lt >= 0 && lmin == bmin) {
                    const float Pm = P - lp;
                    const VT *vr = V + (int64_t)li * d;
                    for (int q = 0; q < nadd; ++q) {
                        if (((q >> 3) & (QL - 1)) != sub) continue;  // this lane's slots
                        const float sc = any_score<DPL, VT>(make_float4(sB[q], sK[q], sH[q], sP[q]),
                                                            __ldcs(cb + (size_t)lt * Ep + q), lp, lA, Pm, P, P2, N,
                                                            vr, mu, g, Wt, Ep, q);
                        if (sc == bmin) {
                            const unsigned long long key = ((unsigned long long)(uint32_t)li << 32) | (uint32_t)idxj[q];
                            if (key < mykey) {
                                mykey = key;
                                myt = lt;
                                myq = q;
                            }
                        }
                    }
                    if (mykey != ~0ull) atomicMin(&s_bkey, mykey);
                }
                __syncthreads();
                if (mykey != ~0ull && mykey == s_bkey) {
                    s_bt = myt;
                    s_bq = myq;
                }
                __syncthreads();
                const float bs = s_bkey != ~0ull ? bmin : INFINITY;
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
                tprev = tb;
                qprev = qj;
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

// pool slots rounded up to the 32-slot blocks of the product tile
inline int pool_slots(int E) { return std::max(32, (E + 31) / 32 * 32); }

template <int DPL> size_t ls_smem(int Ep)
{
    constexpr int d = DPL * 32;
    return sizeof(float) * (10 * (size_t)d + (size_t)d * Ep + 7 * (size_t)Ep + 32 + 8 + 256) + 64;
}

}  // namespace

// ls_bps(R) resident blocks per SM (the launch bounds guarantee the registers
// for it); the workspace is sized by the same count, queried from the current device
static unsigned ls_grid(const RowsDev &R)
{
    int sms = 0;
    if (device_sms(&sms) != FW_OK) sms = 152;  // no device: the size query still answers
    return (unsigned)std::min<int64_t>(R.rows, (int64_t)sms * ls_bps(R));
}

static size_t ls_array_bytes(const RowsDev &R) { return align256((size_t)ls_grid(R) * R.max_n * 4); }

static int ls_cstride(const RowsDev &R) { return (R.max_n + 3) / 4 * 4; }

static size_t ls_table_bytes(const RowsDev &R, int E)
{
    return align256((size_t)ls_grid(R) * pool_slots(E) * ls_cstride(R) * 4);
}

size_t long_swap_workspace(const RowsDev &R, int nb, int E, int max_swaps)
{
    (void)nb, (void)max_swaps;
    return ls_array_bytes(R) * 4 + ls_table_bytes(R, E);
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
    a.cstride = ls_cstride(R);
    const unsigned grid = ls_grid(R);
    const size_t arr = ls_array_bytes(R);
    char *w = (char *)ws;
    a.ebuf = (float *)(w + 0 * arr);
    a.kbuf = (int32_t *)(w + 1 * arr);
    a.pbuf = (float *)(w + 2 * arr);
    a.xbuf = (float *)(w + 3 * arr);
    a.cbuf = (float *)(w + 4 * arr);
    const bool lng = ls_bps(R) == LS_BPS_LONG;
    FW_DISPATCH(R.d, R.v_dtype, {
        const size_t smem = ls_smem<DPL>(a.Ep);
        auto kern = lng ? k_long_swap<DPL, VT, LS_BPS_LONG> : k_long_swap<DPL, VT, LS_BPS_SHORT>;
        FW_CUDA_CHECK(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        FW_LAUNCH(kern, grid, SWT, smem, s, a);
    });
    return FW_OK;
}

}  // namespace fw
