// k_small.cu -- rows with at most 32 keys (the exact-search workloads).
//
// One warp per row.  Lane j owns key j for the softmax and the top-k rank;
// for vector quantities lane l owns dimensions l, l+32, ...  Masses are fp64
// (one exp per key), vector sums are double-float on the fp32 pipe, so every
// output carries ~1e-13 relative error against an fp64 evaluation of the
// definitions.
#include <algorithm>

#include "fw_internal.h"

namespace fw {
namespace {

struct SmallGapArgs {
    RowsDev R;
    const int32_t *k;
    int nb;
    fw_gap_out out;
};

// Definition 2.1 / Sec. 2.1 / Lemma 2.1 for one row and up to four budgets.
// NBM: budgets held in registers (1, or up to 4)
template <int DPL, typename VT, int NBM>
__global__ void __launch_bounds__(256) k_small_gap(const SmallGapArgs a)
{
    const int lane = threadIdx.x & 31;
    const int64_t row = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (row >= a.R.rows) return;
    const int64_t g = row / a.R.R;
    const int64_t ri = row - g * a.R.R;
    const int n = a.R.n[g];
    constexpr int d = DPL * 32;
    int32_t *st = a.out.row_status;
    if (n < 1 || n > 32) {
        if (lane == 0 && st) st[row] = FW_ERR_INVALID_ARG;
        return;
    }
    const float *lg = a.R.logits + a.R.logit_off[g] + ri * n;
    const VT *V = reinterpret_cast<const VT *>(a.R.v) + a.R.v_off[g];
    const float l = lane < n ? lg[lane] : -INFINITY;
    if (__any_sync(FW_FULL, lane < n && !isfinite(l))) {
        if (lane == 0 && st) st[row] = FW_ERR_NONFINITE;
        return;
    }
    // softmax masses (fp64)
    const float M = warp_max(l);
    double p = lane < n ? exp((double)l - (double)M) : 0.0;
    const double Z = warp_sum_d(p);
    p = p / Z;
    // rank in the order (logit desc, index asc)
    int rank = 0;
    for (int s = 0; s < n; ++s) {
        const float ls = __shfl_sync(FW_FULL, l, s);
        rank += (ls > l) || (ls == l && s < lane);
    }
    const int nb = a.nb;
    uint32_t mask[NBM];
    int status = FW_OK;
#pragma unroll
    for (int b = 0; b < NBM; ++b) {
        mask[b] = 0u;
        if (b >= nb) continue;
        const int kb = a.k[row * nb + b];
        if (kb < 1 || kb > n) {
            status = FW_ERR_INVALID_ARG;
            continue;
        }
        mask[b] = __ballot_sync(FW_FULL, lane < n && rank < kb);
        if (lane < n && rank == kb - 1) {
            if (a.out.thr_key) a.out.thr_key[row * nb + b] = order_key(l);
            if (a.out.thr_idx) a.out.thr_idx[row * nb + b] = lane;
        }
        if (a.out.kept_bits) {
            uint32_t *w = a.out.kept_bits + (row * nb + b) * (int64_t)a.out.kept_words;
            for (int t = lane; t < a.out.kept_words; t += 32) w[t] = t == 0 ? mask[b] : 0u;
        }
    }
    // dense output mu = sum_j p_j v_j
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
    // g_A = sum_{j in A} p_j (v_j - mu) for each budget (Lemma 2.1)
    df gA[NBM][DPL];
#pragma unroll
    for (int b = 0; b < NBM; ++b)
#pragma unroll
        for (int t = 0; t < DPL; ++t) gA[b][t] = df_zero();
    for (int j = 0; j < n; ++j) {
        const df pj = shfl_df(pd, j);
#pragma unroll
        for (int t = 0; t < DPL; ++t) {
            const df tj = df_mul(pj, df_rsub_f(load_v(V, (int64_t)j * d + lane + 32 * t), mu[t]));
#pragma unroll
            for (int b = 0; b < NBM; ++b)
                if ((mask[b] >> j) & 1u) gA[b][t] = df_add(gA[b][t], tj);
        }
    }
    if (a.out.o) {
#pragma unroll
        for (int t = 0; t < DPL; ++t) a.out.o[row * d + lane + 32 * t] = mu[t].hi + mu[t].lo;  // rounded once
    }
#pragma unroll
    for (int b = 0; b < NBM; ++b) {
        if (mask[b] == 0u) continue;
        const bool in = (mask[b] >> lane) & 1u;
        const double PA = warp_sum_d(in ? p : 0.0);
        const double PD = warp_sum_d(in ? 0.0 : p);
        df nrm = df_zero();
#pragma unroll
        for (int t = 0; t < DPL; ++t) nrm = df_add(nrm, df_mul(gA[b][t], gA[b][t]));
        nrm = warp_sum_df(nrm);
        const double phi = sqrt(fmax(df_to_double(nrm), 0.0));
        const int64_t rb = row * nb + b;
        if (lane == 0) {
            a.out.gap[rb] = (float)(phi / PA);
            a.out.dropped[rb] = (float)PD;
            if (a.out.phi) a.out.phi[rb] = (float)phi;
        }
        if (a.out.o_kept) {  // mu + g_A / P(A) in double-float, rounded once
            const df invP = df_from_double(1.0 / PA);
#pragma unroll
            for (int t = 0; t < DPL; ++t) {
                const df ok = df_add(mu[t], df_mul(gA[b][t], invP));
                a.out.o_kept[rb * d + lane + 32 * t] = ok.hi + ok.lo;
            }
        }
    }
    if (lane == 0) {
        if (a.out.row_max) a.out.row_max[row] = M;
        if (a.out.row_sum) a.out.row_sum[row] = (float)Z;
        if (st) st[row] = status;
    }
}

// ------------------------------------------------------------------ swap rule

struct SmallSwapArgs {
    RowsDev R;
    const int32_t *k;
    int nb;
    const uint32_t *thr_key;
    const int32_t *thr_idx;
    int E, max_swaps;
    int32_t *n_swaps, *swap_out, *swap_in, *capped;
    float *refined_gap, *topk_gap;
    int nr;  // rows of the per-warp tables
};

// shared memory per warp (floats): U [nr][d+1] (the values, then the high
// parts of u), G [nr][33]; nr = max_n rounded up to a multiple of 4
__host__ __device__ constexpr int swap_smem_floats(int nr, int d) { return nr * (d + 1) + nr * 33; }

// The balancing selector (Sec. 2.1) inside the candidate set (Definition 2.2).
// Pair scores are screened in fp32 from the Gram matrix G = U U^T of the
// centred, weighted points u_j = p_j (v_j - mu) (es(A)^2 = ||sum_A u_j||^2 /
// p(A)^2, Lemma 2.1); every pair whose fp32 score is within a rigorous error
// bound of the best one is re-scored in double-float and the decision is
// taken on those exact values.
template <int DPL, typename VT>
__global__ void __launch_bounds__(64) k_small_swap(const SmallSwapArgs a)
{
    extern __shared__ float smem[];
    constexpr int d = DPL * 32;
    const int lane = threadIdx.x & 31;
    const int wib = threadIdx.x >> 5;
    float *Uhi = smem + (size_t)wib * swap_smem_floats(a.nr, d);
    float *G = Uhi + a.nr * (d + 1);
    const int64_t row = (int64_t)blockIdx.x * (blockDim.x >> 5) + wib;
    if (row >= a.R.rows) return;
    const int64_t g = row / a.R.R;
    const int64_t ri = row - g * a.R.R;
    const int n = a.R.n[g];
    const int nb = a.nb;
    const int MS = a.max_swaps;
    auto fail_row = [&]() {
        for (int b = 0; b < nb; ++b) {
            const int64_t rb = row * nb + b;
            if (lane == 0) {
                a.n_swaps[rb] = 0;
                a.refined_gap[rb] = __int_as_float(0x7fc00000);
                if (a.topk_gap) a.topk_gap[rb] = __int_as_float(0x7fc00000);
                if (a.capped) a.capped[rb] = 0;
            }
            for (int t = lane; t < MS; t += 32) a.swap_out[rb * MS + t] = a.swap_in[rb * MS + t] = -1;
        }
    };
    if (n < 1 || n > 32) {
        fail_row();
        return;
    }
    const float *lg = a.R.logits + a.R.logit_off[g] + ri * n;
    const VT *V = reinterpret_cast<const VT *>(a.R.v) + a.R.v_off[g];
    const float l = lane < n ? lg[lane] : -INFINITY;
    if (__any_sync(FW_FULL, lane < n && !isfinite(l))) {
        fail_row();
        return;
    }
    const float M = warp_max(l);
    double p = lane < n ? exp((double)l - (double)M) : 0.0;
    p = p / warp_sum_d(p);
    const df pd = df_from_double(p);
    // the row's values into Uhi (loads issued back to back), then mu from there
    stage_value_cols<d>(V, n, d, 0, Uhi, lane);
    __syncwarp();
    df mu[DPL];
#pragma unroll
    for (int t = 0; t < DPL; ++t) mu[t] = df_zero();
    for (int j = 0; j < n; ++j) {
        const df pj = shfl_df(pd, j);
#pragma unroll
        for (int t = 0; t < DPL; ++t) mu[t] = df_add(mu[t], df_mul_f(pj, Uhi[j * (d + 1) + lane + 32 * t]));
    }
    // u_j = p_j (v_j - mu): high parts in place in Uhi (the exact re-scoring
    // recomputes the double-float value from V); ||u_j||^2, held by lane j, only
    // where a budget restricts the pool (E < n - k)
    bool need_e2 = false;
    for (int b = 0; b < nb; ++b) need_e2 |= a.E < n - a.k[row * nb + b];
    double e2 = 0.0;
    for (int j = 0; j < n; ++j) {
        const df pj = shfl_df(pd, j);
        df s = df_zero();
#pragma unroll
        for (int t = 0; t < DPL; ++t) {
            const int c = lane + 32 * t;
            const df u = df_mul(pj, df_rsub_f(Uhi[j * (d + 1) + c], mu[t]));
            Uhi[j * (d + 1) + c] = u.hi;
            if (need_e2) s = df_add(s, df_mul(u, u));
        }
        if (need_e2) {
            s = warp_sum_df(s);
            if (lane == j) e2 = df_to_double(s);
        }
    }
    __syncwarp();
    // fp32 Gram matrix, four interleaved partial sums per dot product
    const int npairs = n * (n + 1) / 2;
    for (int q = lane; q < npairs; q += 32) {
        int x = 0, rem = q;
        while (rem >= n - x) {
            rem -= n - x;
            ++x;
        }
        const int y = x + rem;
        float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
        const float *ux = Uhi + x * (d + 1), *uy = Uhi + y * (d + 1);
        for (int c = 0; c < d; c += 4) {
            s0 = fmaf(ux[c], uy[c], s0);
            s1 = fmaf(ux[c + 1], uy[c + 1], s1);
            s2 = fmaf(ux[c + 2], uy[c + 2], s2);
            s3 = fmaf(ux[c + 3], uy[c + 3], s3);
        }
        const float s = (s0 + s1) + (s2 + s3);
        G[x * 33 + y] = s;
        G[y * 33 + x] = s;
    }
    __syncwarp();
    const float unorm = lane < n ? sqrtf(fmaxf(G[lane * 33 + lane], 0.f)) : 0.f;
    const uint32_t all = n == 32 ? FW_FULL : ((1u << n) - 1u);

    for (int b = 0; b < nb; ++b) {
        const int64_t rb = row * nb + b;
        const int kb = a.k[rb];
        const uint32_t tk = a.thr_key[rb];
        const int ti = a.thr_idx[rb];
        const uint32_t key = order_key(l);
        uint32_t A = __ballot_sync(FW_FULL, lane < n && (key > tk || (key == tk && lane <= ti)));
        if (kb < 1 || kb > n || __popc(A) != kb) {
            if (lane == 0) {
                a.n_swaps[rb] = 0;
                a.refined_gap[rb] = __int_as_float(0x7fc00000);
                if (a.topk_gap) a.topk_gap[rb] = __int_as_float(0x7fc00000);
                if (a.capped) a.capped[rb] = 0;
            }
            for (int t = lane; t < MS; t += 32) a.swap_out[rb * MS + t] = a.swap_in[rb * MS + t] = -1;
            continue;
        }
        // candidate set: A plus the E dropped keys of largest single-key error
        uint32_t pool;
        if (a.E >= n - kb) {
            pool = all;
        } else {
            const bool dropped = lane < n && !((A >> lane) & 1u);
            int cnt = 0;
            for (int s = 0; s < n; ++s) {
                const double es = __shfl_sync(FW_FULL, e2, s);
                const bool ds = !((A >> s) & 1u);
                cnt += ds && (es > e2 || (es == e2 && s < lane));
            }
            pool = A | __ballot_sync(FW_FULL, dropped && cnt < a.E);
        }
        // S = sum of the k+1 largest ||u_x|| over the pool (error-bound scale)
        float S;
        {
            const bool inp = (pool >> lane) & 1u;
            int cnt = 0;
            for (int s = 0; s < n; ++s) {
                const float us = __shfl_sync(FW_FULL, unorm, s);
                cnt += ((pool >> s) & 1u) && (us > unorm || (us == unorm && s < lane));
            }
            S = warp_sum(inp && cnt <= kb ? unorm : 0.f) * 1.0001f;
        }
        // bound on the fp32 error of a screened score, times P(A - i + j)^2: the
        // Gram entries and sums (CB S^2), and 8 ulps of Q <= S^2 for the rounded
        // P(A - i + j) and its inverse square
        const float CB = 2.0f * ((float)d * 0.25f + 2.0f * (float)kb + 12.0f) * 5.9604645e-8f;
        const float CBS = (CB + 8.f * 5.9604645e-8f) * S * S;
        // u_j in double-float, recomputed from V (the expression of the pass above)
        auto u_df = [&](int j, int t) {
            return df_mul(shfl_df(pd, j), df_rsub_f(load_v(V, (int64_t)j * d + lane + 32 * t), mu[t]));
        };
        // exact state: g_A (double-float, lanes over dims), p(A), es^2
        df gA[DPL];
#pragma unroll
        for (int t = 0; t < DPL; ++t) gA[t] = df_zero();
        for (uint32_t m = A; m; m &= m - 1) {
            const int j = __ffs(m) - 1;
#pragma unroll
            for (int t = 0; t < DPL; ++t) {
                gA[t] = df_add(gA[t], u_df(j, t));
            }
        }
        double PA = warp_sum_d(((A >> lane) & 1u) ? p : 0.0);
        auto exact_es2 = [&](const df *gv, double P) {
            df s = df_zero();
#pragma unroll
            for (int t = 0; t < DPL; ++t) s = df_add(s, df_mul(gv[t], gv[t]));
            s = warp_sum_df(s);
            return fmax(df_to_double(s), 0.0) / (P * P);
        };
        double cur = exact_es2(gA, PA);
        if (a.topk_gap && lane == 0) a.topk_gap[rb] = (float)sqrt(cur);
        int taken = 0, cap = 0;
        for (;;) {
            const uint32_t add = pool & ~A;
            const int na = __popc(A), nadd = __popc(add);
            if (nadd == 0) break;
            // h_x = sum_{y in A} G_xy and Q_A = sum_{x in A} h_x, fp32
            float h = 0.f;
            if (lane < n)
                for (uint32_t m = A; m; m &= m - 1) h += G[lane * 33 + __ffs(m) - 1];
            const float QA = warp_sum(((A >> lane) & 1u) ? h : 0.f);
            // fp32 screening of every (kept i, added j) pair, lane j taking the
            // added key j: Q(A - i + j) = (Q_A - 2 h_i + G_ii) + (2 h_j + G_jj) - 2 G_ij,
            // P(A - i + j) = P(A - i) + p_j (two positive terms)
            const bool isadd = (add >> lane) & 1u;
            const float cj = lane < n ? 2.f * h + G[lane * 33 + lane] : 0.f;
            const float pjf = (float)p;
            float best_up = INFINITY;
            for (uint32_t mi = A; mi; mi &= mi - 1) {
                const int i = __ffs(mi) - 1;
                const float ci = QA - 2.f * __shfl_sync(FW_FULL, h, i) + G[i * 33 + i];
                const float Pp = (float)(PA - __shfl_sync(FW_FULL, p, i)) + pjf;
                const float inv = 1.f / (Pp * Pp);
                const float sc = (ci + cj - 2.f * G[i * 33 + (lane < n ? lane : 0)]) * inv;
                if (isadd) best_up = fminf(best_up, sc + CBS * inv);
            }
            best_up = warp_min(best_up);
            // exact re-scoring, in (i, j) order, of every pair that may be the best
            double best = INFINITY;
            int bi = -1, bj = -1;
            for (uint32_t mi = A; mi; mi &= mi - 1) {
                const int i = __ffs(mi) - 1;
                const float ci = QA - 2.f * __shfl_sync(FW_FULL, h, i) + G[i * 33 + i];
                const float Pp = (float)(PA - __shfl_sync(FW_FULL, p, i)) + pjf;
                const float inv = 1.f / (Pp * Pp);
                const float sc = (ci + cj - 2.f * G[i * 33 + (lane < n ? lane : 0)]) * inv;
                uint32_t cand = __ballot_sync(FW_FULL, isadd && sc - CBS * inv <= best_up);
                while (cand) {
                    const int j = __ffs(cand) - 1;
                    cand &= cand - 1;
                    df gn[DPL];
#pragma unroll
                    for (int t = 0; t < DPL; ++t) {
                        gn[t] = df_add(df_sub(gA[t], u_df(i, t)), u_df(j, t));
                    }
                    const double P2 = PA - __shfl_sync(FW_FULL, p, i) + __shfl_sync(FW_FULL, p, j);
                    const double e = exact_es2(gn, P2);
                    if (e < best) {
                        best = e;
                        bi = i;
                        bj = j;
                    }
                }
            }
            if (!(best < cur)) break;
            if (taken >= MS) {
                cap = 1;
                break;
            }
#pragma unroll
            for (int t = 0; t < DPL; ++t) {
                gA[t] = df_add(df_sub(gA[t], u_df(bi, t)), u_df(bj, t));
            }
            PA = PA - __shfl_sync(FW_FULL, p, bi) + __shfl_sync(FW_FULL, p, bj);
            A = (A & ~(1u << bi)) | (1u << bj);
            cur = best;
            if (lane == 0) {
                a.swap_out[rb * MS + taken] = bi;
                a.swap_in[rb * MS + taken] = bj;
            }
            ++taken;
        }
        if (lane == 0) {
            a.n_swaps[rb] = taken;
            a.refined_gap[rb] = (float)sqrt(cur);
            if (a.capped) a.capped[rb] = cap;
        }
        for (int t = lane; t < MS; t += 32)
            if (t >= taken) a.swap_out[rb * MS + t] = a.swap_in[rb * MS + t] = -1;
    }
}

}  // namespace

fw_status small_gap(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &out, cudaStream_t s)
{
    if (R.rows == 0) return FW_OK;
    const SmallGapArgs a{R, k, nb, out};
    const int warps = 8;
    const unsigned grid = (unsigned)((R.rows + warps - 1) / warps);
    if (nb == 1) {
        FW_DISPATCH(R.d, R.v_dtype, FW_LAUNCH((k_small_gap<DPL, VT, 1>), grid, warps * 32, 0, s, a));
    } else {
        FW_DISPATCH(R.d, R.v_dtype, FW_LAUNCH((k_small_gap<DPL, VT, 4>), grid, warps * 32, 0, s, a));
    }
    return FW_OK;
}

fw_status small_swap(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &topk, int E,
                     int max_swaps, int32_t *n_swaps, int32_t *swap_out, int32_t *swap_in,
                     float *refined_gap, float *topk_gap, int32_t *capped, cudaStream_t s)
{
    if (R.rows == 0) return FW_OK;
    const int nr = (std::min(R.max_n, 32) + 3) / 4 * 4;
    const SmallSwapArgs a{R, k, nb, topk.thr_key, topk.thr_idx, E, max_swaps, n_swaps, swap_out,
                          swap_in, capped, refined_gap, topk_gap, nr};
    FW_DISPATCH(R.d, R.v_dtype, {
        const int warps = DPL >= 8 ? 1 : 2;
        const size_t smem = (size_t)warps * swap_smem_floats(nr, DPL * 32) * sizeof(float);
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_small_swap<DPL, VT>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        const unsigned grid = (unsigned)((R.rows + warps - 1) / warps);
        FW_LAUNCH((k_small_swap<DPL, VT>), grid, warps * 32, smem, s, a);
    });
    return FW_OK;
}

}  // namespace fw
