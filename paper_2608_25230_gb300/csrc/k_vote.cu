// k_vote.cu -- the group vote (Sec. 2.1, shared kept sets).
//
// Deployment keeps one set per KV head for every query row that shares it.
// The vote keeps the s keys of largest mass summed over the group's rows,
//     G_j = sum_{rows i of the group} p_ij,   p_ij = exp(l_ij - M_i) / Z_i,
// equal G -> lower index first, and scores every row of the group against that
// set with Definition 2.1's quantities (es(A) = ||m_A - mu|| and the dropped
// mass of the row's own masses).  Three launches, each one pass over HBM:
//   k_vote_mass    G of every group: one thread per key walks the group's rows
//                  in order (loads coalesced over keys) with a compensated sum;
//                  flags non-finite logits.
//                  Each mass is the fast exponential times 1/Z of its row (a few
//                  ulp): an accurate exp and a divide per (row, key) would make
//                  this pass and the scoring pass instruction-bound.
//   k_vote_select  per group and budget (a block each), the order key T of the s-th largest G
//                  (three-pass radix select over G staged in shared memory) and
//                  the index L of the last tied key taken; the set is
//                  {j : key(G_j) > T} + {j : key(G_j) == T, j <= L}.
//   k_vote_eval    one warp per row streams the row's logits once; each key
//                  falls in the band of the nested sets (budgets in ascending
//                  order) that first contains it; members add p_j v_j to their
//                  band.  Prefix sums over the bands give every budget's m_A,
//                  suffix sums its dropped mass.
// For bf16 values with d = 64 or 128 the scoring runs instead on the long-row
// path's tensor-core P.V kernels in their vote mode (k_long_tc.cu): the rows
// of a group share V and the nested sets, so the band-masked products of all
// the group's rows are one contraction, and V is streamed once per tile of
// rows rather than gathered once per row.
#include <algorithm>
#include <climits>

#include "fw_internal.h"

namespace fw {
namespace {

constexpr int VM_T = 256;      // k_vote_mass: threads per block, one key each
constexpr int VS_T = 512;      // k_vote_select: threads per group
constexpr int VE_W = 8;        // k_vote_eval: warps (rows) per block
constexpr int V_NBMAX = 4;     // budgets per call
constexpr int VS_STAGE_MAX = 49152;  // groups up to this many keys select from shared memory

struct VoteArgs {
    RowsDev R;
    const int32_t *s;     // [groups][nb] budgets
    int nb;
    const float *M, *Z;   // [rows] softmax statistics of the gap call
    const float *o;       // [rows][d] dense outputs of the gap call
    float *mass;          // [groups][max_n] G
    uint32_t *thr;        // [groups][nb] order key of the s-th largest G
    int32_t *tidx;        // [groups][nb] largest index taken at thr; -1: budget out of range
    int32_t *gflag;       // [groups] nonzero: a logit of the group is not finite
    uint32_t *bits;       // [groups][nb][words] or null
    int words;
    float *gap;           // [rows][nb]
    float *dropped;       // [rows][nb] or null
    int32_t *row_status;  // [rows] or null
    int staged;           // k_vote_select keeps G in shared memory
};

// ------------------------------------------------------------------ G

__global__ void __launch_bounds__(VM_T) k_vote_mass(VoteArgs a)
{
    __shared__ float sM[VM_T], sZ[VM_T];  // M and 1 / Z of the rows in the chunk
    const int tid = threadIdx.x;
    const int Rg = a.R.R;
    for (int64_t g = blockIdx.y; g < a.R.num_groups; g += gridDim.y) {
        const int n = a.R.n[g];
        const float *lg = a.R.logits + a.R.logit_off[g];
        float *G = a.mass + g * (int64_t)a.R.max_n;
        bool bad = false;
        for (int j0 = blockIdx.x * VM_T; j0 < n; j0 += gridDim.x * VM_T) {
            const int j = j0 + tid;
            // compensated sum (TwoSum, errors carried in lo): the rounding of the
            // sum stays at about one ulp of G whatever the group size
            float hi = 0.f, lo = 0.f;
            for (int i0 = 0; i0 < Rg; i0 += VM_T) {
                const int cnt = min(VM_T, Rg - i0);
                __syncthreads();
                if (tid < cnt) {
                    const int64_t r = g * Rg + i0 + tid;
                    sM[tid] = a.M[r];
                    sZ[tid] = 1.f / a.Z[r];
                }
                __syncthreads();
                if (j < n) {
                    const float *col = lg + (int64_t)i0 * n + j;
#pragma unroll 8
                    for (int i = 0; i < cnt; ++i) {
                        const float l = __ldg(col + (int64_t)i * n);
                        bad |= !isfinite(l);
                        const float p = __expf(l - sM[i]) * sZ[i];
                        const float t = hi + p, bb = t - hi;
                        lo += (hi - (t - bb)) + (p - bb);
                        hi = t;
                    }
                }
            }
            if (j < n) G[j] = hi + lo;
        }
        if (__syncthreads_or(bad) && tid == 0) a.gflag[g] = FW_ERR_NONFINITE;
    }
}

// --------------------------------------------------------- the vote set

__global__ void __launch_bounds__(VS_T) k_vote_select(VoteArgs a)
{
    extern __shared__ float sG[];
    __shared__ uint32_t hist[2048];
    __shared__ int wcnt[VS_T / 32];
    __shared__ uint32_t s_digit;
    __shared__ int s_rem, s_L;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    // a block per (group, budget): the budgets of a group select side by side
    for (int64_t item = blockIdx.x; item < a.R.num_groups * a.nb; item += gridDim.x) {
        const int64_t g = item / a.nb;
        const int b = (int)(item - g * a.nb);
        const int n = a.R.n[g];
        const float *Gg = a.mass + g * (int64_t)a.R.max_n;
        const float *G = Gg;
        if (a.staged) {
            __syncthreads();
            for (int j = tid; j < n; j += VS_T) sG[j] = Gg[j];
            __syncthreads();
            G = sG;
        }
        {
            const int64_t gb = g * a.nb + b;
            const int s = a.s[gb];
            uint32_t T = 0;
            int L = -1;
            if (s >= 1 && s <= n) {
                uint32_t prefix = 0, pmask = 0;
                int rem = s;
                // digits of 11, 11 and 10 bits from the top of the order key
                for (int pass = 0; pass < 3; ++pass) {
                    const int shift = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
                    const int nbin = pass < 2 ? 2048 : 1024;
                    for (int i = tid; i < 2048; i += VS_T) hist[i] = 0u;
                    __syncthreads();
                    for (int j = tid; j < n; j += VS_T) {
                        const uint32_t u = order_key(G[j]);
                        if ((u & pmask) == prefix) atomicAdd(&hist[(u >> shift) & (uint32_t)(nbin - 1)], 1u);
                    }
                    __syncthreads();
                    if (wid == 0) {
                        // lane 0 sums the top nbin/32 bins, lane 31 the bottom ones
                        const int per = nbin / 32;
                        const int top = nbin - 1 - lane * per;
                        int c = 0;
                        for (int q = 0; q < per; ++q) c += (int)hist[top - q];
                        int incl = c;
#pragma unroll
                        for (int off = 1; off < 32; off <<= 1) {
                            const int y = __shfl_up_sync(FW_FULL, incl, off);
                            if (lane >= off) incl += y;
                        }
                        const int excl = incl - c;
                        if (excl < rem && rem <= incl) {
                            int acc = excl;
                            for (int q = 0; q < per; ++q) {
                                const int h = (int)hist[top - q];
                                if (acc + h >= rem) {
                                    s_digit = (uint32_t)(top - q);
                                    s_rem = rem - acc;
                                    break;
                                }
                                acc += h;
                            }
                        }
                    }
                    __syncthreads();
                    prefix |= s_digit << shift;
                    pmask |= (uint32_t)(nbin - 1) << shift;
                    rem = s_rem;
                    __syncthreads();
                }
                T = prefix;
                // L: the rem-th key (in index order) whose order key is T
                if (tid == 0) s_L = -1;
                __syncthreads();
                int run = 0;
                for (int j0 = 0; j0 < n; j0 += VS_T) {
                    const int j = j0 + tid;
                    const bool eq = j < n && order_key(G[j]) == T;
                    const unsigned m = __ballot_sync(FW_FULL, eq);
                    if (lane == 0) wcnt[wid] = __popc(m);
                    __syncthreads();
                    int before = run, tot = 0;
#pragma unroll
                    for (int w = 0; w < VS_T / 32; ++w) {
                        if (w < wid) before += wcnt[w];
                        tot += wcnt[w];
                    }
                    before += __popc(m & ((1u << lane) - 1u));
                    if (eq && before + 1 == rem) s_L = j;
                    run += tot;
                    __syncthreads();
                    if (s_L >= 0) break;  // every thread reads it after the barrier
                }
                L = s_L;
                __syncthreads();
            }
            if (tid == 0) {
                a.thr[gb] = T;
                a.tidx[gb] = L;
            }
            if (a.bits) {
                uint32_t *w = a.bits + gb * (int64_t)a.words;
                for (int j0 = 0; j0 < a.words * 32; j0 += VS_T) {
                    const int j = j0 + tid;
                    bool in = false;
                    if (L >= 0 && j < n) {
                        const uint32_t u = order_key(G[j]);
                        in = u > T || (u == T && j <= L);
                    }
                    const unsigned m = __ballot_sync(FW_FULL, in);
                    if (lane == 0 && (j0 >> 5) + wid < a.words) w[(j0 >> 5) + wid] = m;
                }
            }
        }
    }
}

// ------------------------------------------------------ every row's score

// DPL consecutive value columns starting at p (aligned to their own size)
template <int DPL> __device__ __forceinline__ void load_cols(const float *p, float (&x)[DPL])
{
    if constexpr (DPL % 4 == 0) {
#pragma unroll
        for (int q = 0; q < DPL / 4; ++q) {
            const float4 t = __ldg(reinterpret_cast<const float4 *>(p) + q);
            x[4 * q] = t.x;
            x[4 * q + 1] = t.y;
            x[4 * q + 2] = t.z;
            x[4 * q + 3] = t.w;
        }
    } else if constexpr (DPL == 2) {
        const float2 t = __ldg(reinterpret_cast<const float2 *>(p));
        x[0] = t.x;
        x[1] = t.y;
    } else {
        x[0] = __ldg(p);
    }
}

__device__ __forceinline__ void bf16_pair(uint32_t w, float &lo, float &hi)
{
    lo = __uint_as_float(w << 16);
    hi = __uint_as_float(w & 0xffff0000u);
}

template <int DPL> __device__ __forceinline__ void load_cols(const uint16_t *p, float (&x)[DPL])
{
    if constexpr (DPL == 8) {
        const uint4 t = __ldg(reinterpret_cast<const uint4 *>(p));
        bf16_pair(t.x, x[0], x[1]);
        bf16_pair(t.y, x[2], x[3]);
        bf16_pair(t.z, x[4], x[5]);
        bf16_pair(t.w, x[6], x[7]);
    } else if constexpr (DPL == 4) {
        const uint2 t = __ldg(reinterpret_cast<const uint2 *>(p));
        bf16_pair(t.x, x[0], x[1]);
        bf16_pair(t.y, x[2], x[3]);
    } else if constexpr (DPL == 2) {
        bf16_pair(__ldg(reinterpret_cast<const unsigned int *>(p)), x[0], x[1]);
    } else {
        x[0] = bf16_to_f32(__ldg(p));
    }
}

template <int DPL, typename VT>
__global__ void __launch_bounds__(VE_W * 32) k_vote_eval(VoteArgs a)
{
    constexpr int QB = DPL >= 8 ? 4 : 8;  // member value rows in flight per batch
    constexpr int d = DPL * 32;
    const int lane = threadIdx.x & 31;
    const int nb = a.nb;
    for (int64_t r = (int64_t)blockIdx.x * VE_W + (threadIdx.x >> 5); r < a.R.rows;
         r += (int64_t)gridDim.x * VE_W) {
        const int64_t g = r / a.R.R;
        const int64_t i = r - g * a.R.R;
        const int n = a.R.n[g];
        const float *l = a.R.logits + a.R.logit_off[g] + i * n;
        const VT *V = static_cast<const VT *>(a.R.v) + a.R.v_off[g];
        const float *G = a.mass + g * (int64_t)a.R.max_n;
        const float M = a.M[r], Zi = 1.f / a.Z[r];

        // the group's budgets in ascending order of s: the sets are nested along it
        int sv[V_NBMAX], ord[V_NBMAX];
#pragma unroll
        for (int t = 0; t < V_NBMAX; ++t) {
            sv[t] = t < nb ? a.s[g * nb + t] : INT_MAX;
            ord[t] = t;
        }
#define FW_VOTE_CX(x, y)                                                                  \
    if (sv[y] < sv[x]) {                                                                  \
        const int ts = sv[x], to = ord[x];                                                \
        sv[x] = sv[y], ord[x] = ord[y], sv[y] = ts, ord[y] = to;                          \
    }
        FW_VOTE_CX(0, 1) FW_VOTE_CX(2, 3) FW_VOTE_CX(0, 2) FW_VOTE_CX(1, 3) FW_VOTE_CX(1, 2)
#undef FW_VOTE_CX
        uint32_t T[V_NBMAX];
        int L[V_NBMAX];
        bool invalid = false;
#pragma unroll
        for (int t = 0; t < V_NBMAX; ++t) {
            T[t] = 0u;
            L[t] = -1;
            if (t < nb) {
                T[t] = a.thr[g * nb + ord[t]];
                L[t] = a.tidx[g * nb + ord[t]];
                invalid |= L[t] < 0;
            }
        }

        float tacc[V_NBMAX][DPL];
        df acc[V_NBMAX][DPL];
        df pm[V_NBMAX + 1];
#pragma unroll
        for (int t = 0; t < V_NBMAX; ++t)
#pragma unroll
            for (int c = 0; c < DPL; ++c) acc[t][c] = df_zero();
#pragma unroll
        for (int t = 0; t <= V_NBMAX; ++t) pm[t] = df_zero();

        // the next tile's logit and mass are loaded one tile ahead
        float ln = lane < n ? __ldg(l + lane) : 0.f;
        float gn = lane < n ? G[lane] : 0.f;
        for (int j0 = 0; j0 < n; j0 += 32) {
            const int j = j0 + lane;
            const float lc = ln, gc = gn;
            if (j + 32 < n) {
                ln = __ldg(l + j + 32);
                gn = G[j + 32];
            }
            float p = 0.f;
            int band = nb;  // number of (ascending) budgets whose set leaves key j out
            if (j < n) {
                p = __expf(lc - M) * Zi;
                const uint32_t u = order_key(gc);
                band = 0;
#pragma unroll
                for (int t = 0; t < V_NBMAX; ++t)
                    if (t < nb && !(u > T[t] || (u == T[t] && j <= L[t]))) ++band;
            }
#pragma unroll
            for (int t = 0; t <= V_NBMAX; ++t)
                if (band == t) pm[t] = df_add(pm[t], df{p, 0.f});

            unsigned mem = __ballot_sync(FW_FULL, band < nb);
            if (!mem) continue;
#pragma unroll
            for (int t = 0; t < V_NBMAX; ++t)
#pragma unroll
                for (int c = 0; c < DPL; ++c) tacc[t][c] = 0.f;
            while (mem) {
                int src[QB];
#pragma unroll
                for (int q = 0; q < QB; ++q) {
                    src[q] = mem ? __ffs(mem) - 1 : -1;
                    mem = mem ? (mem & (mem - 1u)) : 0u;
                }
                float x[QB][DPL];
#pragma unroll
                for (int q = 0; q < QB; ++q) {
                    if (src[q] >= 0) {
                        load_cols<DPL>(V + (int64_t)(j0 + src[q]) * d + lane * DPL, x[q]);
                    } else {
#pragma unroll
                        for (int c = 0; c < DPL; ++c) x[q][c] = 0.f;
                    }
                }
#pragma unroll
                for (int q = 0; q < QB; ++q) {
                    const int sq = src[q] < 0 ? 0 : src[q];
                    const float pq = __shfl_sync(FW_FULL, p, sq);
                    const int bq = __shfl_sync(FW_FULL, band, sq);
                    if (src[q] >= 0) {
#pragma unroll
                        for (int t = 0; t < V_NBMAX; ++t)
                            if (bq == t)
#pragma unroll
                                for (int c = 0; c < DPL; ++c) tacc[t][c] = fmaf(pq, x[q][c], tacc[t][c]);
                    }
                }
            }
#pragma unroll
            for (int t = 0; t < V_NBMAX; ++t)
#pragma unroll
                for (int c = 0; c < DPL; ++c) acc[t][c] = df_add(acc[t][c], df{tacc[t][c], 0.f});
        }
#pragma unroll
        for (int t = 0; t <= V_NBMAX; ++t) pm[t] = warp_sum_df(pm[t]);

        float oc[DPL];
        load_cols<DPL>(a.o + r * d + lane * DPL, oc);
        df Prun = df_zero();
        df Nrun[DPL];
#pragma unroll
        for (int c = 0; c < DPL; ++c) Nrun[c] = df_zero();
#pragma unroll
        for (int t = 0; t < V_NBMAX; ++t) {
            if (t >= nb) break;
            // the set of the t-th smallest budget holds bands 0..t
            Prun = df_add(Prun, pm[t]);
            df drop = df_zero();
#pragma unroll
            for (int u = 0; u <= V_NBMAX; ++u)
                if (u > t && u <= nb) drop = df_add(drop, pm[u]);
            float e2 = 0.f;
#pragma unroll
            for (int c = 0; c < DPL; ++c) {
                Nrun[c] = df_add(Nrun[c], acc[t][c]);
                // m_A - mu = (N_A - p(A) mu) / p(A), the numerator formed with fused products
                const float num = fmaf(-Prun.hi, oc[c], Nrun[c].hi) + fmaf(-Prun.lo, oc[c], Nrun[c].lo);
                const float diff = num / Prun.hi;
                e2 = fmaf(diff, diff, e2);
            }
            e2 = warp_sum(e2);
            if (lane == 0) {
                const int64_t rb = r * nb + ord[t];
                a.gap[rb] = sqrtf(e2);
                if (a.dropped) a.dropped[rb] = drop.hi + drop.lo;
            }
        }
        if (a.row_status && lane == 0)
            a.row_status[r] = a.gflag[g] ? FW_ERR_NONFINITE : (invalid ? FW_ERR_INVALID_ARG : FW_OK);
    }
}

}  // namespace

static size_t vote_mass_bytes(const RowsDev &R) { return align256((size_t)R.num_groups * R.max_n * 4); }
static size_t vote_thr_bytes(const RowsDev &R, int nb) { return align256((size_t)R.num_groups * nb * 4); }

size_t group_vote_workspace(const RowsDev &R, int nb)
{
    return vote_mass_bytes(R) + 2 * vote_thr_bytes(R, nb) + align256((size_t)R.num_groups * 4);
}

fw_status group_vote(const RowsDev &R, const int32_t *s, int nb, const fw_gap_out &topk, float *gap,
                     float *dropped, uint32_t *bits, int words, int32_t *row_status, void *ws, size_t ws_bytes,
                     cudaStream_t st)
{
    (void)ws_bytes;
    VoteArgs a;
    a.R = R;
    a.s = s;
    a.nb = nb;
    a.M = topk.row_max;
    a.Z = topk.row_sum;
    a.o = topk.o;
    char *w = (char *)ws;
    a.mass = (float *)w;
    w += vote_mass_bytes(R);
    a.thr = (uint32_t *)w;
    w += vote_thr_bytes(R, nb);
    a.tidx = (int32_t *)w;
    w += vote_thr_bytes(R, nb);
    a.gflag = (int32_t *)w;
    a.bits = bits;
    a.words = words;
    a.gap = gap;
    a.dropped = dropped;
    a.row_status = row_status;
    a.staged = R.max_n <= VS_STAGE_MAX;
    FW_CUDA_CHECK(cudaMemsetAsync(a.gflag, 0, (size_t)R.num_groups * 4, st));

    int sms = 0;
    if (device_sms(&sms) != FW_OK) return FW_ERR_CUDA;
    const int64_t chunks = (R.max_n + VM_T - 1) / VM_T;
    const int64_t per_group = std::max<int64_t>(1, ((int64_t)sms * 8 + R.num_groups - 1) / R.num_groups);
    const dim3 gm((unsigned)std::min(chunks, per_group), (unsigned)std::min<int64_t>(R.num_groups, 65535));
    FW_LAUNCH(k_vote_mass, gm, VM_T, 0, st, a);

    const size_t sel_smem = a.staged ? (size_t)R.max_n * 4 : 0;
    FW_CUDA_CHECK(cudaFuncSetAttribute(k_vote_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sel_smem));
    FW_LAUNCH(k_vote_select, (unsigned)std::min<int64_t>(R.num_groups * nb, 1 << 20), VS_T, sel_smem, st, a);

    // bf16 values: the scoring as band-masked P.V products on the tensor cores
    // (the rows of a group share V and the set); otherwise one warp per row
    {
        const fw_status vs = long_pv_vote(R, nb, a.M, a.Z, a.mass, R.max_n, a.thr, a.tidx, a.s, a.gflag, gap,
                                          dropped, row_status, st);
        if (vs != FW_ERR_UNSUPPORTED) return vs;
    }
    const unsigned ge = (unsigned)std::min<int64_t>((R.rows + VE_W - 1) / VE_W, 1 << 24);
    FW_DISPATCH(R.d, R.v_dtype, { FW_LAUNCH((k_vote_eval<DPL, VT>), ge, VE_W * 32, 0, st, a); });
    return FW_OK;
}

}  // namespace fw
