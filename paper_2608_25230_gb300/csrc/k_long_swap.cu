// k_long_swap.cu -- the balancing selector (Sec. 2.1) inside the candidate set
// (Definition 2.2) for rows of any length.
//
// One persistent block walks rows.  Per row, one pass over the keys
// accumulates the band sums S_b = sum p_j v_j (band = number of budgets that
// drop key j), the band masses and every dropped key's single-key error
// p_j ||v_j - o|| (o = the dense output given by fw_dense_and_topk_gap).  Per
// budget: the E extras are the dropped keys of largest single-key error (a
// radix select on the error's bits, ties to lower indices); the current set
// is described by
//   g = sum_{A} u_i = pbar(A) N_A - p(A) N_{A^c},  u_i = p_i (v_i - mu),
// with mu = sum_b S_b and disjoint sums, so g carries no cancellation.
// Each round scores every (kept i, pool j outside A) pair without subtracting
// two rounded gaps: with N = |g|^2 and P = p(A),
//   delta = |u_i|^2 + |u_j|^2 - 2 g.u_i + 2 g.u_j - 2 u_i.u_j,
//   D_ij  = delta P^2 - N (p_j - p_i)(2P - p_i + p_j),
// es(A - i + j)^2 = es(A)^2 + D_ij / (P^2 P'^2), so the swap decreases es iff
// D_ij < 0 and the best pair minimises D_ij / P'^2 (ties: smallest i, then j).
// The cross terms u_i.u_j come from a block-wide pass over the kept keys
// against the pool vectors staged in shared memory.
#include <algorithm>

#include "fw_internal.h"

namespace fw {
namespace {

constexpr int SWT = 256;    // threads per block
constexpr int SWADD = 96;   // pool vectors outside A (E + swaps)
constexpr int SWG = 32;     // pool vectors per accumulation group

struct LSArgs {
    RowsDev R;
    const int32_t *k;
    int nb;
    const uint32_t *thr_key;
    const int32_t *thr_idx;
    const float *o;
    const float *row_max;
    const float *row_sum;
    int E, max_swaps;
    int32_t *n_swaps, *swap_out, *swap_in, *capped;
    float *refined_gap, *topk_gap;
    float *ebuf;     // [gridDim.x][max_n] single-key error^2 (or -1 for kept keys)
    int32_t *kbuf;   // [gridDim.x][max_n] kept-key list of the current set
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

template <int DPL, typename VT>
__global__ void __launch_bounds__(SWT) k_long_swap(const LSArgs a)
{
    constexpr int d = DPL * 32;
    extern __shared__ float sm[];
    float *S = sm;                     // [5][d] band sums of p v
    float *mu = S + 5 * d;             // [d]
    float *o = mu + d;                 // [d]   dense output given by the caller
    float *g = o + d;                  // [d]
    float *Wt = g + d;                 // [d][SWADD] pool vectors w_j = v_j - mu
    float *pj = Wt + d * SWADD;        // [SWADD] masses of the pool vectors
    float *betaj = pj + SWADD;         // [SWADD] |u_j|^2 + 2 g.u_j
    int *idxj = reinterpret_cast<int *>(betaj + SWADD);  // [SWADD] their keys
    float *red = reinterpret_cast<float *>(idxj + SWADD);     // [32]
    float *mass = red + 32;            // [8]
    uint32_t *hist = reinterpret_cast<uint32_t *>(mass + 8);  // [256]
    __shared__ uint32_t s_misc[8];
    __shared__ int s_cnt;
    __shared__ float s_best;
    __shared__ unsigned long long s_bkey;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    float *eb = a.ebuf + (size_t)blockIdx.x * a.R.max_n;
    int *kb = a.kbuf + (size_t)blockIdx.x * a.R.max_n;
    const int nb = a.nb, MS = a.max_swaps;

    for (int64_t row = blockIdx.x; row < a.R.rows; row += gridDim.x) {
        const int64_t grp = row / a.R.R;
        const int64_t ri = row - grp * a.R.R;
        const int n = a.R.n[grp];
        const float *lg = a.R.logits + a.R.logit_off[grp] + ri * n;
        const VT *V = reinterpret_cast<const VT *>(a.R.v) + a.R.v_off[grp];
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
            // stage pool vectors w_j = v_j - mu and their masses
            for (int e = tid; e < nadd * d; e += SWT) {
                const int q = e / d, c = e % d;
                Wt[c * SWADD + q] = load_v(V, (int64_t)idxj[q] * d + c) - mu[c];
            }
            for (int q = tid; q < nadd; q += SWT) pj[q] = expf(lg[idxj[q]] - M) * Zi;
            __syncthreads();
            int taken = 0, cap = 0;
            for (;;) {
                if (nadd == 0 || nk == 0) break;
                // beta_j = |u_j|^2 + 2 g.u_j, one warp per pool vector
                for (int q = wid; q < nadd; q += SWT / 32) {
                    float s2 = 0.f, sg = 0.f;
                    for (int c = lane; c < d; c += 32) {
                        const float w = Wt[c * SWADD + q];
                        s2 = fmaf(w, w, s2);
                        sg = fmaf(g[c], w, sg);
                    }
                    s2 = warp_sum(s2);
                    sg = warp_sum(sg);
                    const float p = pj[q];
                    if (lane == 0) betaj[q] = p * p * s2 + 2.f * p * sg;
                }
                if (tid == 0) {
                    s_best = INFINITY;
                    s_bkey = ~0ull;
                }
                __syncthreads();
                float best = INFINITY;
                unsigned long long bkey = ~0ull;
                const float P2 = P * P;
                for (int t = tid; t < nk; t += SWT) {
                    const int i = kb[t];
                    const float p_i = expf(lg[i] - M) * Zi;
                    float alpha = 0.f;  // |u_i|^2 - 2 g.u_i
                    for (int q0 = 0; q0 < nadd; q0 += SWG) {
                        float accq[SWG];
#pragma unroll
                        for (int q = 0; q < SWG; ++q) accq[q] = 0.f;
                        float dg = 0.f, w2 = 0.f;
                        for (int c = 0; c < d; ++c) {
                            const float w = load_v(V, (int64_t)i * d + c) - mu[c];
                            dg = fmaf(g[c], w, dg);
                            w2 = fmaf(w, w, w2);
#pragma unroll
                            for (int q = 0; q < SWG; ++q) accq[q] = fmaf(w, Wt[c * SWADD + q0 + q], accq[q]);
                        }
                        alpha = p_i * p_i * w2 - 2.f * p_i * dg;
#pragma unroll
                        for (int q = 0; q < SWG; ++q) {
                            const int qq = q0 + q;
                            if (qq < nadd) {
                                const float p_j = pj[qq];
                                const float cross = p_i * p_j * accq[q];
                                const float delta = alpha + betaj[qq] - 2.f * cross;
                                const float dp = p_j - p_i;
                                const float Pp = P + dp;
                                const float D = delta * P2 - N * dp * (2.f * P + dp);
                                const float sc = D / (Pp * Pp);
                                const unsigned long long key =
                                    ((unsigned long long)(uint32_t)i << 32) | (uint32_t)idxj[qq];
                                if (sc < best || (sc == best && key < bkey)) {
                                    best = sc;
                                    bkey = key;
                                }
                            }
                        }
                    }
                }
                // block argmin of (score, i, j)
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
                const float bs = s_best;
                const unsigned long long bk = s_bkey;
                if (!(bs < 0.f)) break;  // no pair strictly decreases es
                if (taken >= MS) {
                    cap = 1;
                    break;
                }
                const int bi = (int)(bk >> 32), bj = (int)(bk & 0xffffffffu);
                // apply: g += u_j - u_i, P += p_j - p_i; the pool gains i, loses j
                int qj = 0;
                for (int q = 0; q < nadd; ++q)
                    if (idxj[q] == bj) qj = q;
                const float p_i = expf(lg[bi] - M) * Zi;
                const float p_j = pj[qj];
                __syncthreads();
                for (int c = tid; c < d; c += SWT) {
                    const float wi = load_v(V, (int64_t)bi * d + c) - mu[c];
                    const float wj = Wt[c * SWADD + qj];
                    g[c] = g[c] + p_j * wj - p_i * wi;
                    Wt[c * SWADD + qj] = wi;
                }
                for (int t = tid; t < nk; t += SWT)
                    if (kb[t] == bi) kb[t] = bj;
                __syncthreads();
                if (tid == 0) {
                    idxj[qj] = bi;
                    pj[qj] = p_i;
                    a.swap_out[rb * MS + taken] = bi;
                    a.swap_in[rb * MS + taken] = bj;
                }
                P = P - p_i + p_j;
                float gl2 = 0.f;
                for (int c = tid; c < d; c += SWT) gl2 = fmaf(g[c], g[c], gl2);
                N = block_sum(gl2, red);
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

template <int DPL> constexpr size_t ls_smem()
{
    constexpr int d = DPL * 32;
    return sizeof(float) * (5 * d + 3 * d + (size_t)d * SWADD + 3 * SWADD + 32 + 8 + 256) + 64;
}

}  // namespace

static unsigned ls_grid(const RowsDev &R) { return (unsigned)std::min<int64_t>(R.rows, 152 * 2); }

size_t long_swap_workspace(const RowsDev &R, int nb, int E, int max_swaps)
{
    (void)nb, (void)E, (void)max_swaps;
    return align256((size_t)ls_grid(R) * R.max_n * 4) * 2;
}

fw_status long_swap(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &topk, int E, int max_swaps,
                    int32_t *n_swaps, int32_t *swap_out, int32_t *swap_in, float *refined_gap, float *topk_gap,
                    int32_t *capped, void *ws, size_t ws_bytes, cudaStream_t s)
{
    (void)ws_bytes;
    if (E + max_swaps > SWADD) return FW_ERR_UNSUPPORTED;
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
    a.max_swaps = max_swaps;
    a.n_swaps = n_swaps;
    a.swap_out = swap_out;
    a.swap_in = swap_in;
    a.capped = capped;
    a.refined_gap = refined_gap;
    a.topk_gap = topk_gap;
    const unsigned grid = ls_grid(R);
    a.ebuf = (float *)ws;
    a.kbuf = (int32_t *)((char *)ws + align256((size_t)grid * R.max_n * 4));
    FW_DISPATCH(R.d, R.v_dtype, {
        const size_t smem = ls_smem<DPL>();
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_long_swap<DPL, VT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem));
        FW_LAUNCH((k_long_swap<DPL, VT>), grid, SWT, smem, s, a);
    });
    return FW_OK;
}

}  // namespace fw
