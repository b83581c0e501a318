// k_audit.cu -- the deployed selectors audited in Sec. 2.3 / App. C, as
// kernels: for every row and budget s, the kept set that each rule would
// choose, scored with Definition 2.1's es(A) = ||m_A - mu|| (to be set against
// the top-mass set and ES_pool).  The rules, with App. C's settings:
//   StreamingLLM  the first min(4, s/2) positions (sinks) and the last
//                 s - sinks positions (recency);
//   H2O           the last s/2 positions and, among the others, the
//                 s - s/2 of largest mass accumulated over the group's rows
//                 (the KV head's query rows that share the cache);
//   SnapKV        window w = max(1, min(32, s/2)): the last w positions and,
//                 among the others, the s - w of largest pooled vote, the vote
//                 of a key being its mass summed over the group's last w rows,
//                 pooled by a maximum over 7 neighbouring positions (clipped
//                 to the candidates);
//   Quest         pages of P = max(2, s/4) consecutive keys; the floor(s/P)
//                 pages of largest maximum logit (Quest ranks pages by an
//                 upper bound on that maximum; with the row's logits at hand
//                 the bound is the maximum itself);
//   Quest-16      the same with pages of 16 keys (s >= 16).
// Equal scores keep lower positions (pages) first, as everywhere in the
// library.
//
//   k_aud_mass    accumulated masses and window votes of every group (a thread
//                 per key walks the group's rows; compensated sums);
//   k_aud_select  per group and budget the H2O and SnapKV sets (CTA-wide
//                 radix top-m), written as bit masks;
//   k_aud_row     per row: the Quest page maxima and sets, then one warp per
//                 (rule, budget) gathers its members' p_j v_j and forms es.
#include <algorithm>

#include "fw_internal.h"

namespace fw {
namespace {

constexpr int AM_T = 256;   // k_aud_mass threads
constexpr int AS_T = 512;   // k_aud_select threads
constexpr int AR_T = 256;   // k_aud_row threads (8 warps)
constexpr int A_NBMAX = 4;
constexpr int NSEL = FW_NUM_SELECTORS;

struct AudArgs {
    RowsDev R;
    int nb;
    int s[A_NBMAX];
    const float *M, *Z, *o;  // [rows], [rows], [rows][d] from the gap call
    float *G;                // ws [groups][max_n] accumulated mass
    float *vote;             // ws [groups][nb][max_n] window votes
    uint32_t *gbits;         // ws [groups][nb][2][words] H2O and SnapKV sets
    int words;
    float *es;               // [rows][NSEL][nb]
    uint32_t *bits;          // [rows][NSEL][nb][words] or null
};

__device__ __forceinline__ int snap_w(int s) { return max(1, min(32, s / 2)); }
__device__ __forceinline__ int quest_p(int q, int s) { return q == 0 ? max(2, s / 4) : 16; }

// ---------------------------------------------------------------- masses
__global__ void __launch_bounds__(AM_T) k_aud_mass(AudArgs a)
{
    __shared__ float sM[AM_T], sZ[AM_T];
    const int tid = threadIdx.x;
    const int Rg = a.R.R;
    for (int64_t g = blockIdx.y; g < a.R.num_groups; g += gridDim.y) {
        const int n = a.R.n[g];
        const float *lg = a.R.logits + a.R.logit_off[g];
        int wfirst[A_NBMAX];  // first row of each budget's window
#pragma unroll
        for (int b = 0; b < A_NBMAX; ++b) wfirst[b] = b < a.nb ? max(0, Rg - snap_w(a.s[b])) : Rg;
        for (int j0 = blockIdx.x * AM_T; j0 < n; j0 += gridDim.x * AM_T) {
            const int j = j0 + tid;
            float hi = 0.f, lo = 0.f;
            float vh[A_NBMAX], vl[A_NBMAX];
#pragma unroll
            for (int b = 0; b < A_NBMAX; ++b) vh[b] = vl[b] = 0.f;
            for (int i0 = 0; i0 < Rg; i0 += AM_T) {
                const int cnt = min(AM_T, Rg - i0);
                __syncthreads();
                if (tid < cnt) {
                    const int64_t r = g * Rg + i0 + tid;
                    sM[tid] = a.M[r];
                    sZ[tid] = 1.f / a.Z[r];
                }
                __syncthreads();
                if (j < n) {
                    const float *col = lg + (int64_t)i0 * n + j;
                    for (int i = 0; i < cnt; ++i) {
                        const float p = __expf(__ldg(col + (int64_t)i * n) - sM[i]) * sZ[i];
                        float t = hi + p, bb = t - hi;
                        lo += (hi - (t - bb)) + (p - bb);
                        hi = t;
#pragma unroll
                        for (int b = 0; b < A_NBMAX; ++b)
                            if (i0 + i >= wfirst[b]) {
                                t = vh[b] + p;
                                bb = t - vh[b];
                                vl[b] += (vh[b] - (t - bb)) + (p - bb);
                                vh[b] = t;
                            }
                    }
                }
            }
            if (j < n) {
                a.G[g * a.R.max_n + j] = hi + lo;
                for (int b = 0; b < a.nb; ++b) a.vote[(g * a.nb + b) * a.R.max_n + j] = vh[b] + vl[b];
            }
        }
    }
}

// ------------------------------------------------------- group-level sets
__global__ void __launch_bounds__(AS_T) k_aud_select(AudArgs a)
{
    __shared__ TopmSmem S;
    const int tid = threadIdx.x;
    for (int64_t g = blockIdx.x; g < a.R.num_groups; g += gridDim.x) {
        const int n = a.R.n[g];
        const float *G = a.G + g * a.R.max_n;
        for (int b = 0; b < a.nb; ++b) {
            const int s = a.s[b];
            uint32_t *hb = a.gbits + ((g * a.nb + b) * 2 + 0) * a.words;
            uint32_t *sb = a.gbits + ((g * a.nb + b) * 2 + 1) * a.words;
            if (s < 1 || s > n) {
                for (int w = tid; w < a.words; w += AS_T) hb[w] = sb[w] = 0u;
                continue;
            }
            // H2O: the last r positions, then the s - r of largest accumulated mass
            const int r = s / 2, mh = s - r;
            uint32_t Th = 0u;
            int Lh = -1;
            block_topm(n - r, mh, [&](int j) { return order_key(G[j]); }, S, Th, Lh);
            // SnapKV: the last w positions, then the s - w of largest pooled vote
            const int w = snap_w(s), ms = s - w, lim = n - w;
            const float *vt = a.vote + (g * a.nb + b) * a.R.max_n;
            auto pooled = [&](int j) {
                float v = vt[j];
                for (int q = max(0, j - 3); q <= min(lim - 1, j + 3); ++q) v = fmaxf(v, vt[q]);
                return order_key(v);
            };
            uint32_t Ts = 0u;
            int Ls = -1;
            if (ms > 0) block_topm(lim, ms, pooled, S, Ts, Ls);
            for (int wd = tid; wd < a.words; wd += AS_T) {
                uint32_t mh_bits = 0u, ms_bits = 0u;
                for (int e = 0; e < 32; ++e) {
                    const int j = wd * 32 + e;
                    if (j >= n) break;
                    bool kh = j >= n - r;
                    if (!kh) {
                        const uint32_t k = order_key(G[j]);
                        kh = k > Th || (k == Th && j <= Lh);
                    }
                    bool ks = j >= lim;
                    if (!ks && ms > 0) {
                        const uint32_t k = pooled(j);
                        ks = k > Ts || (k == Ts && j <= Ls);
                    }
                    mh_bits |= (uint32_t)kh << e;
                    ms_bits |= (uint32_t)ks << e;
                }
                hb[wd] = mh_bits;
                sb[wd] = ms_bits;
            }
            __syncthreads();
        }
    }
}

// ---------------------------------------------------------- rows: score sets
template <int DPL, typename VT>
__global__ void __launch_bounds__(AR_T) k_aud_row(AudArgs a)
{
    extern __shared__ uint32_t smw[];  // [nb][2][words] Quest sets, then the page maxima
    __shared__ TopmSmem S;
    constexpr int d = DPL * 32;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    uint32_t *qbits = smw;
    float *pm = reinterpret_cast<float *>(smw + a.nb * 2 * a.words);
    for (int64_t row = blockIdx.x; row < a.R.rows; row += gridDim.x) {
        const int64_t g = row / a.R.R;
        const int n = a.R.n[g];
        const float *l = a.R.logits + a.R.logit_off[g] + (row - g * a.R.R) * n;
        const VT *V = static_cast<const VT *>(a.R.v) + a.R.v_off[g];
        const float M = a.M[row], Zi = 1.f / a.Z[row];
        // Quest sets: page maxima, the top pages, the pages' keys as bits
        for (int b = 0; b < a.nb; ++b)
            for (int q = 0; q < 2; ++q) {
                const int s = a.s[b];
                const int P = quest_p(q, s);
                const int np = (n + P - 1) / P, mp = s / P;
                uint32_t *qb = qbits + (b * 2 + q) * a.words;
                const bool valid = s >= 1 && s <= n && mp >= 1 && (q == 0 || s >= 16);
                if (!valid) {
                    __syncthreads();
                    for (int w = tid; w < a.words; w += AR_T) qb[w] = 0u;
                    continue;
                }
                __syncthreads();  // pm is free
                for (int p = tid; p < np; p += AR_T) {
                    float m = -INFINITY;
                    for (int j = p * P; j < min(n, p * P + P); ++j) m = fmaxf(m, __ldg(l + j));
                    pm[p] = m;
                }
                __syncthreads();
                uint32_t T = 0u;
                int L = -1;
                block_topm(np, min(mp, np), [&](int p) { return order_key(pm[p]); }, S, T, L);
                for (int w = tid; w < a.words; w += AR_T) {
                    uint32_t bits = 0u;
                    for (int e = 0; e < 32; ++e) {
                        const int j = w * 32 + e;
                        if (j >= n) break;
                        const int p = j / P;
                        const uint32_t k = order_key(pm[p]);
                        bits |= (uint32_t)(k > T || (k == T && p <= L)) << e;
                    }
                    qb[w] = bits;
                }
            }
        __syncthreads();
        // one warp per (rule, budget): gather the members, form es
        float ol[DPL];
#pragma unroll
        for (int c = 0; c < DPL; ++c) ol[c] = a.o[row * d + lane * DPL + c];
        for (int set = wid; set < NSEL * a.nb; set += AR_T / 32) {
            const int sel = set / a.nb, b = set - sel * a.nb;
            const int s = a.s[b];
            const uint32_t *src = nullptr;
            if (sel == FW_SEL_H2O) src = a.gbits + ((g * a.nb + b) * 2 + 0) * a.words;
            if (sel == FW_SEL_SNAPKV) src = a.gbits + ((g * a.nb + b) * 2 + 1) * a.words;
            if (sel == FW_SEL_QUEST) src = qbits + (b * 2 + 0) * a.words;
            if (sel == FW_SEL_QUEST16) src = qbits + (b * 2 + 1) * a.words;
            const int sinks = min(4, s / 2);
            float N[DPL];
#pragma unroll
            for (int c = 0; c < DPL; ++c) N[c] = 0.f;
            float pA = 0.f;
            int cnt = 0;
            const int nw = (n + 31) / 32;
            for (int w0 = 0; w0 < nw; w0 += 32) {
                const int w = w0 + lane;
                uint32_t word = 0u;
                if (w < nw) {
                    if (sel == FW_SEL_STREAMING) {
                        for (int e = 0; e < 32; ++e) {
                            const int j = w * 32 + e;
                            if (j < n && s >= 1 && s <= n && (j < sinks || j >= n - (s - sinks))) word |= 1u << e;
                        }
                    } else {
                        word = src[w];
                    }
                }
                if (a.bits) {
                    if (w < nw) a.bits[((row * NSEL + sel) * a.nb + b) * (int64_t)a.words + w] = word;
                }
                // members of the 32 words, one at a time across the warp
                for (int src_lane = 0; src_lane < 32; ++src_lane) {
                    uint32_t mw = __shfl_sync(FW_FULL, word, src_lane);
                    while (mw) {
                        const int j = (w0 + src_lane) * 32 + __ffs(mw) - 1;
                        mw &= mw - 1;
                        const float p = __expf(__ldg(l + j) - M) * Zi;
                        pA += p;
                        ++cnt;
#pragma unroll
                        for (int c = 0; c < DPL; ++c) N[c] = fmaf(p, load_v(V, (int64_t)j * d + lane * DPL + c), N[c]);
                    }
                }
            }
            float e2 = 0.f;
#pragma unroll
            for (int c = 0; c < DPL; ++c) {
                const float diff = N[c] / pA - ol[c];
                e2 = fmaf(diff, diff, e2);
            }
            e2 = warp_sum(e2);
            if (lane == 0) a.es[(row * NSEL + sel) * a.nb + b] = cnt > 0 ? sqrtf(e2) : __int_as_float(0x7fc00000);
        }
        __syncthreads();
    }
}

}  // namespace

static size_t aud_words(const RowsDev &R) { return (size_t)(R.max_n + 31) / 32; }

size_t selector_audit_workspace(const RowsDev &R, int nb)
{
    return align256((size_t)R.num_groups * R.max_n * 4) + align256((size_t)R.num_groups * nb * R.max_n * 4) +
           align256((size_t)R.num_groups * nb * 2 * aud_words(R) * 4);
}

fw_status selector_audit(const RowsDev &R, const int32_t *s, int nb, const fw_gap_out &topk, float *es,
                         uint32_t *bits, int words, void *ws, cudaStream_t st)
{
    AudArgs a;
    a.R = R;
    a.nb = nb;
    for (int b = 0; b < A_NBMAX; ++b) a.s[b] = b < nb ? s[b] : 0;
    a.M = topk.row_max;
    a.Z = topk.row_sum;
    a.o = topk.o;
    char *w = (char *)ws;
    a.G = (float *)w;
    w += align256((size_t)R.num_groups * R.max_n * 4);
    a.vote = (float *)w;
    w += align256((size_t)R.num_groups * nb * R.max_n * 4);
    a.gbits = (uint32_t *)w;
    a.words = (int)aud_words(R);
    a.es = es;
    a.bits = bits;
    if (bits && words != a.words) return FW_ERR_INVALID_ARG;
    int sms = 0;
    if (device_sms(&sms) != FW_OK) return FW_ERR_CUDA;
    const int64_t chunks = (R.max_n + AM_T - 1) / AM_T;
    const int64_t per_group = std::max<int64_t>(1, ((int64_t)sms * 8 + R.num_groups - 1) / R.num_groups);
    const dim3 gm((unsigned)std::min(chunks, per_group), (unsigned)std::min<int64_t>(R.num_groups, 65535));
    FW_LAUNCH(k_aud_mass, gm, AM_T, 0, st, a);
    FW_LAUNCH(k_aud_select, (unsigned)std::min<int64_t>(R.num_groups, 1 << 20), AS_T, 0, st, a);
    const size_t smem = ((size_t)nb * 2 * a.words + (size_t)(R.max_n + 1) / 2 + 1) * 4;
    FW_DISPATCH(R.d, R.v_dtype, {
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_aud_row<DPL, VT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        FW_LAUNCH((k_aud_row<DPL, VT>), (unsigned)std::min<int64_t>(R.rows, (int64_t)sms * 16), AR_T, smem, st, a);
    });
    return FW_OK;
}

}  // namespace fw
