// k_pool.cu -- ES_pool (Definition 2.2): the exact best size-s subset of the
// candidate set -- the top-mass set plus the E dropped keys of largest
// single-key error p_j ||v_j - mu|| (ties -> lower index) -- for rows of any
// length up to 49,152 keys and budgets s <= 32 (pools of at most 64 keys).
//
//   k_pool_build  one CTA per row: p_j and e_j^2 = p_j^2 ||v_j - o||^2 of every
//                 key (o = the dense output of the gap call; a warp per key,
//                 lanes across the value row), then per budget a 3-pass radix
//                 select (11/11/10 bits) of the top E among the dropped keys
//                 (equal errors: lower index first) and the pool in ascending
//                 key order.
//   k_pool_enum   one warp per (row, budget): the pool's Gram matrix
//                 G_ab = u_a . u_b, u = p (v - o), in shared memory; the
//                 smaller side (the s kept keys, or the P - s keys left out)
//                 is enumerated in colex order, lanes taking rank ranges, with
//                 the sums over all members but the lowest held while the
//                 lowest member runs (O(m) shared-memory reads per subset).
//                 Every subset gets an fp32 score es^2 and a rigorous interval
//                 around it (the rounding of the Gram sums, bounded by
//                 (sum_pool |u|)^2); the subsets whose lower end does not
//                 exceed the least upper end are buffered (4,096 per warp, in
//                 the workspace) and re-scored in fp64 as
//                 es^2 = (sum_{a,b in A} G_ab) / p(A)^2 from an fp64 copy of
//                 the Gram matrix (the products u_a . u_b formed in fp64 from
//                 the fp32 masses, the bf16 / fp32 values and o), and the least
//                 es wins, exact ties to the smallest colex rank of the
//                 members' pool positions.  (Re-scoring from the value rows
//                 cost |A| dependent row loads per candidate; flat rows send
//                 ~1,000 candidates per item.)
//
// Nothing waits on another block; a buffer of re-scoring candidates that
// overflows falls back to a per-lane re-scoring pass over the same
// candidates, so the answer stays exact.
#include <algorithm>
#include <climits>

#include "fw_internal.h"

namespace fw {
namespace {

constexpr int PB_T = 256;            // k_pool_build: threads per row
constexpr int PE_W = 4;              // k_pool_enum: warps per block, one (row, budget) each
constexpr int PMAX = 64;             // pool keys
constexpr int PSMAX = 32;            // largest budget
constexpr int PB_STAGE_MAX = 49152;  // keys per row staged in shared memory
constexpr int GCAP = 4096;           // re-scoring candidates buffered per warp (workspace)
constexpr int PE_BPS = 4;            // k_pool_enum blocks per SM in the launch (each warp owns workspace)
constexpr uint64_t PE_MAX_SUBSETS = 1ull << 32;
constexpr int GLD = PMAX + 1;        // Gram row stride (odd: conflict-free columns)

// C(a, b) for a <= 64, b <= 32 (all below 2^63), by Pascal's rule at compile time.
struct Binom64Table {
    uint64_t v[65][33];
};
constexpr Binom64Table make_binom64()
{
    Binom64Table t{};
    for (int a = 0; a <= 64; ++a) {
        t.v[a][0] = 1;
        for (int b = 1; b <= 32; ++b) t.v[a][b] = a == 0 ? 0 : t.v[a - 1][b - 1] + t.v[a - 1][b];
    }
    return t;
}
static __constant__ Binom64Table c_b64 = make_binom64();

__device__ __forceinline__ uint64_t cb(int a, int b) { return (b < 0 || b > 32 || a < b) ? 0 : c_b64.v[a][b]; }

struct PoolArgs {
    RowsDev R;
    const int32_t *k;          // [rows][nb]
    int nb;
    int E[4];                  // extras of each budget slot
    const uint32_t *thr_key;   // [rows][nb] from the gap call
    const int32_t *thr_idx;
    const float *o, *M, *Z;    // [rows][d], [rows], [rows]
    int32_t *pool;             // ws [rows][nb][PMAX] ascending key indices
    int32_t *pool_n;           // ws [rows][nb] pool size; -1 invalid budget, -2 pool too large
    float *best_gap;           // [rows][nb]
    int32_t *best_idx;         // [rows][nb][k_max]
    int k_max;
    float *topk_gap;           // [rows][nb] or null
    int32_t *row_status;       // [rows] or null
    int64_t *n_cand;           // [rows][nb] re-scored subsets, or null
    uint64_t *gcand;           // ws [gridDim.x * PE_W][GCAP] candidate masks of each warp
    double *g64;               // ws [gridDim.x * PE_W][PMAX * PMAX] fp64 Gram matrix of each warp
};

// ------------------------------------------------------------ the pool

template <int DPL, typename VT>
__device__ __forceinline__ void load_row_part(const VT *V, int64_t j, int lane, float (&x)[DPL])
{
    constexpr int d = DPL * 32;
#pragma unroll
    for (int c = 0; c < DPL; ++c) x[c] = load_v(V, j * d + lane * DPL + c);
}

template <int DPL, typename VT>
__global__ void __launch_bounds__(PB_T) k_pool_build(PoolArgs a)
{
    extern __shared__ float sm[];
    float *e2 = sm;  // [max_n] single-key errors squared
    __shared__ uint32_t hist[2048];
    __shared__ int wcnt[PB_T / 32];
    __shared__ uint32_t s_digit;
    __shared__ int s_rem, s_L;
    constexpr int d = DPL * 32;
    constexpr int NW = PB_T / 32;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    for (int64_t r = blockIdx.x; r < a.R.rows; r += gridDim.x) {
        const int64_t g = r / a.R.R;
        const int n = a.R.n[g];
        const float *l = a.R.logits + a.R.logit_off[g] + (r - g * a.R.R) * n;
        const VT *V = static_cast<const VT *>(a.R.v) + a.R.v_off[g];
        const float M = a.M[r], Zi = 1.f / a.Z[r];
        float so[DPL];
#pragma unroll
        for (int c = 0; c < DPL; ++c) so[c] = a.o[r * d + lane * DPL + c];
        __syncthreads();  // the previous row's e2 is no longer read
        // a warp per key, two keys in flight: lanes hold DPL consecutive dims
        for (int j = wid * 2; j < n; j += NW * 2) {
            float x0[DPL], x1[DPL];
            const bool two = j + 1 < n;
            load_row_part<DPL, VT>(V, j, lane, x0);
            if (two) load_row_part<DPL, VT>(V, j + 1, lane, x1);
            float s0 = 0.f, s1 = 0.f;
#pragma unroll
            for (int c = 0; c < DPL; ++c) {
                const float w0 = x0[c] - so[c];
                s0 = fmaf(w0, w0, s0);
                if (two) {
                    const float w1 = x1[c] - so[c];
                    s1 = fmaf(w1, w1, s1);
                }
            }
            s0 = warp_sum(s0);
            s1 = warp_sum(s1);
            if (lane == 0) {
                const float p0 = __expf(__ldg(l + j) - M) * Zi;
                e2[j] = p0 * p0 * s0;
            } else if (lane == 1 && two) {
                const float p1 = __expf(__ldg(l + j + 1) - M) * Zi;
                e2[j + 1] = p1 * p1 * s1;
            }
        }
        __syncthreads();
        for (int b = 0; b < a.nb; ++b) {
            const int64_t rb = r * a.nb + b;
            const int s = a.k[rb];
            const uint32_t tk = a.thr_key[rb];
            const int ti = a.thr_idx[rb];
            if (s < 1 || s > n || s > PSMAX || s > a.k_max || a.E[b] < 0) {
                if (tid == 0) a.pool_n[rb] = -1;
                continue;
            }
            const int Ee = min(a.E[b], n - s);
            if (s + Ee > PMAX) {
                if (tid == 0) a.pool_n[rb] = -2;
                continue;
            }
            // top Ee of the dropped keys by e2 (order key of a non-negative float)
            uint32_t T = 0xffffffffu;
            int L = -1;
            if (Ee > 0) {
                if (tid == 0) {
                    s_digit = 0u;
                    s_rem = 1;
                }
                uint32_t prefix = 0, pmask = 0;
                int rem = Ee;
                for (int pass = 0; pass < 3; ++pass) {
                    const int shift = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
                    const int nbin = pass < 2 ? 2048 : 1024;
                    for (int i = tid; i < 2048; i += PB_T) hist[i] = 0u;
                    __syncthreads();
                    for (int j = tid; j < n; j += PB_T) {
                        const uint32_t kl = order_key(__ldg(l + j));
                        const bool kept = kl > tk || (kl == tk && j <= ti);
                        const uint32_t u = order_key(e2[j]);
                        if (!kept && (u & pmask) == prefix) atomicAdd(&hist[(u >> shift) & (uint32_t)(nbin - 1)], 1u);
                    }
                    __syncthreads();
                    if (wid == 0) {
                        // bins in descending order, nbin / 32 consecutive bins per lane
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
                // the rem-th dropped key (index order) whose key equals T
                if (tid == 0) s_L = -1;
                __syncthreads();
                int run = 0;
                for (int j0 = 0; j0 < n; j0 += PB_T) {
                    const int j = j0 + tid;
                    bool eq = false;
                    if (j < n) {
                        const uint32_t kl = order_key(__ldg(l + j));
                        const bool kept = kl > tk || (kl == tk && j <= ti);
                        eq = !kept && order_key(e2[j]) == T;
                    }
                    const unsigned m = __ballot_sync(FW_FULL, eq);
                    if (lane == 0) wcnt[wid] = __popc(m);
                    __syncthreads();
                    int before = run, tot = 0;
#pragma unroll
                    for (int w = 0; w < NW; ++w) {
                        if (w < wid) before += wcnt[w];
                        tot += wcnt[w];
                    }
                    before += __popc(m & ((1u << lane) - 1u));
                    if (eq && before + 1 == rem) s_L = j;
                    run += tot;
                    __syncthreads();
                    if (s_L >= 0) break;
                }
                L = s_L;
                __syncthreads();
            }
            // the pool in ascending key order: kept keys and the extras
            int run = 0;
            int32_t *pl = a.pool + rb * PMAX;
            for (int j0 = 0; j0 < n; j0 += PB_T) {
                const int j = j0 + tid;
                bool in = false;
                if (j < n) {
                    const uint32_t kl = order_key(__ldg(l + j));
                    const bool kept = kl > tk || (kl == tk && j <= ti);
                    const uint32_t u = order_key(e2[j]);
                    in = kept || (Ee > 0 && (u > T || (u == T && j <= L)));
                }
                const unsigned m = __ballot_sync(FW_FULL, in);
                if (lane == 0) wcnt[wid] = __popc(m);
                __syncthreads();
                int before = run, tot = 0;
#pragma unroll
                for (int w = 0; w < NW; ++w) {
                    if (w < wid) before += wcnt[w];
                    tot += wcnt[w];
                }
                before += __popc(m & ((1u << lane) - 1u));
                if (in && before < PMAX) pl[before] = j;
                run += tot;
                __syncthreads();
            }
            if (tid == 0) a.pool_n[rb] = run <= PMAX ? run : -2;
        }
    }
}

// ------------------------------------------------------------ enumeration

// next m-combination of 0..P-1 in colex order (the lowest member moves fastest)
__device__ __forceinline__ bool colex_next(int *c, int m, int P)
{
    int i = 0;
    while (i < m && c[i] + 1 == (i + 1 < m ? c[i + 1] : P)) ++i;
    if (i == m) return false;
    ++c[i];
    for (int t = 0; t < i; ++t) c[t] = t;
    return true;
}

// the m-combination of 0..P-1 of colex rank `rank`
__device__ __forceinline__ void colex_unrank(uint64_t rank, int m, int P, int *c)
{
    for (int i = m - 1; i >= 0; --i) {
        int x = i;
        while (x + 1 < P && cb(x + 1, i + 1) <= rank) ++x;
        c[i] = x;
        rank -= cb(x, i + 1);
    }
}

// colex rank of the set bits of a 64-bit mask (positions ascending)
__device__ __forceinline__ uint64_t colex_rank64(uint64_t A)
{
    uint64_t rank = 0;
    int i = 1;
    for (uint64_t w = A; w; w &= w - 1, ++i) rank += cb(__ffsll((long long)w) - 1, i);
    return rank;
}

// per-warp enumeration state in shared memory
struct EnumSm {
    float G[PMAX * GLD];
    float pp[PMAX];
    float t[PMAX];        // t_x = sum_y G_xy = u_x . U
    int32_t pidx[PMAX];
    int ncand;
};

// es of the pool positions in A, from the definition in fp64: the warp forms
// N_A = sum_A p_j v_j across the value dims (lane c covers DPL of them).
template <int DPL, typename VT>
__device__ __forceinline__ double es_warp(const VT *V, const float *o_lane, const EnumSm &S, uint64_t A, int lane)
{
    constexpr int d = DPL * 32;
    double PA = 0.0;
    double N[DPL];
#pragma unroll
    for (int c = 0; c < DPL; ++c) N[c] = 0.0;
    for (uint64_t w = A; w; w &= w - 1) {
        const int x = __ffsll((long long)w) - 1;
        const double px = (double)S.pp[x];
        PA += px;
        float v[DPL];
#pragma unroll
        for (int c = 0; c < DPL; ++c) v[c] = load_v(V, (int64_t)S.pidx[x] * d + lane * DPL + c);
#pragma unroll
        for (int c = 0; c < DPL; ++c) N[c] = fma(px, (double)v[c], N[c]);
    }
    double e2 = 0.0;
#pragma unroll
    for (int c = 0; c < DPL; ++c) {
        const double diff = N[c] / PA - (double)o_lane[c];
        e2 = fma(diff, diff, e2);
    }
    e2 = warp_sum_d(e2);
    return sqrt(e2);
}

// es of the pool positions in A from the fp64 Gram matrix: lane i sums the row
// of A's i-th member over A (|A| <= 32), the warp adds the rows.
__device__ __forceinline__ double es_gram_warp(const double *g, const EnumSm &S, uint64_t A, int lane)
{
    double rs = 0.0, pa = 0.0;
    int i = 0;
    for (uint64_t w = A; w; w &= w - 1, ++i) {
        if (i != lane) continue;
        const int x = __ffsll((long long)w) - 1;
        pa = (double)S.pp[x];
        for (uint64_t w2 = A; w2; w2 &= w2 - 1) rs += g[x * PMAX + __ffsll((long long)w2) - 1];
    }
    const double Q = warp_sum_d(rs), PA = warp_sum_d(pa);
    return sqrt(fmax(Q, 0.0)) / PA;
}

// the same by one lane alone (fallback when the candidate buffer overflows)
__device__ double es_gram_lane(const double *g, const EnumSm &S, uint64_t A)
{
    double Q = 0.0, PA = 0.0;
    for (uint64_t w = A; w; w &= w - 1) {
        const int x = __ffsll((long long)w) - 1;
        PA += (double)S.pp[x];
        for (uint64_t w2 = A; w2; w2 &= w2 - 1) Q += g[x * PMAX + __ffsll((long long)w2) - 1];
    }
    return sqrt(fmax(Q, 0.0)) / PA;
}

// Walks the colex ranks [lo, hi) of m-subsets C of the pool and calls
// f(Cmask, lower, upper) with the interval that holds the exact es^2 of the
// subset A (A = C in the direct form, pool \ C otherwise).
template <typename F>
__device__ __forceinline__ void walk(const EnumSm &S, int P, int m, bool direct, uint64_t lo, uint64_t hi, float UU,
                                     float PU, float Eabs, float pe, F &&f)
{
    if (lo >= hi) return;
    int c[PSMAX];
    colex_unrank(lo, m, P, c);
    uint64_t q = lo;
    for (;;) {
        // sums over the members above the lowest
        float g2o = 0.f, pao = 0.f, lino = 0.f;
        uint64_t om = 0;
        for (int i = 1; i < m; ++i) {
            const int x = c[i];
            om |= 1ull << x;
            pao += S.pp[x];
            lino += S.t[x];
            g2o += S.G[x * GLD + x];
            for (int j = 1; j < i; ++j) g2o = fmaf(2.f, S.G[x * GLD + c[j]], g2o);
        }
        const int lim = m > 1 ? c[1] : P;
        for (int x = c[0]; x < lim && q < hi; ++x, ++q) {
            float rs = S.G[x * GLD + x];
            for (int i = 1; i < m; ++i) rs = fmaf(2.f, S.G[x * GLD + c[i]], rs);
            float g2 = g2o + rs, pa = pao + S.pp[x];
            if (!direct) {
                g2 = fmaf(-2.f, lino + S.t[x], UU) + g2;
                pa = PU - pa;
            }
            const float num_lo = fmaxf(g2 - Eabs, 0.f), num_hi = g2 + Eabs;
            const float pl = pa + pe, ph = pa - pe;
            const float lower = num_lo / (pl * pl) * (1.f - 1e-6f);
            const float upper = ph > 0.f ? num_hi / (ph * ph) * (1.f + 1e-6f) : INFINITY;
            f(om | (1ull << x), lower, upper);
        }
        if (q >= hi) return;
        c[0] = lim - 1;
        if (!colex_next(c, m, P)) return;
    }
}

template <int DPL, typename VT>
__global__ void __launch_bounds__(PE_W * 32) k_pool_enum(PoolArgs a)
{
    extern __shared__ __align__(16) unsigned char smraw[];
    constexpr int d = DPL * 32;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    EnumSm &S = reinterpret_cast<EnumSm *>(smraw)[wid];
    const int64_t wslot = (int64_t)blockIdx.x * PE_W + wid;
    uint64_t *gc = a.gcand + wslot * GCAP;
    double *g64 = a.g64 + wslot * (PMAX * PMAX);
    const int64_t items = a.R.rows * a.nb;
    for (int64_t it = (int64_t)blockIdx.x * PE_W + wid; it < items; it += (int64_t)gridDim.x * PE_W) {
        const int64_t r = it / a.nb;
        const int64_t g = r / a.R.R;
        const int n = a.R.n[g];
        const float *l = a.R.logits + a.R.logit_off[g] + (r - g * a.R.R) * n;
        const VT *V = static_cast<const VT *>(a.R.v) + a.R.v_off[g];
        const float M = a.M[r], Zi = 1.f / a.Z[r];
        const int s = a.k[it];
        const int P = a.pool_n[it];
        int32_t *bi = a.best_idx + it * a.k_max;
        const bool direct = s <= P - s;
        const int m = direct ? s : P - s;
        // refused items: an out-of-range budget (P = -1), a pool over PMAX keys
        // (P = -2), or more subsets than the enumeration takes
        int refuse = P == -1 ? FW_ERR_INVALID_ARG : (P < 0 ? FW_ERR_UNSUPPORTED : 0);
        if (!refuse && P < s) refuse = FW_ERR_INVALID_ARG;  // thresholds that keep fewer than s keys
        const uint64_t T = refuse ? 0 : cb(P, m);
        if (!refuse && T > PE_MAX_SUBSETS) refuse = FW_ERR_UNSUPPORTED;
        if (refuse) {
            if (lane == 0) {
                if (a.row_status) atomicMax(a.row_status + r, refuse);
                a.best_gap[it] = __int_as_float(0x7fc00000);
                if (a.topk_gap) a.topk_gap[it] = __int_as_float(0x7fc00000);
                if (a.n_cand) a.n_cand[it] = 0;
            }
            for (int q = lane; q < a.k_max; q += 32) bi[q] = -1;
            continue;
        }
        float ol[DPL];
#pragma unroll
        for (int c = 0; c < DPL; ++c) ol[c] = a.o[r * d + lane * DPL + c];
        for (int q = lane; q < P; q += 32) {
            const int j = a.pool[it * PMAX + q];
            S.pidx[q] = j;
            S.pp[q] = __expf(__ldg(l + j) - M) * Zi;
        }
        if (lane == 0) S.ncand = 0;
        __syncwarp();
        // Gram matrix of u = p (v - o) in fp64 (the warp forms each product
        // across d): the fp64 copy for the re-scoring, its fp32 rounding for
        // the walk
        for (int x = 0; x < P; ++x) {
            float vx[DPL];
            load_row_part<DPL, VT>(V, S.pidx[x], lane, vx);
            double dx[DPL];
#pragma unroll
            for (int c = 0; c < DPL; ++c) dx[c] = (double)vx[c] - (double)ol[c];
            for (int y = x; y < P; ++y) {
                float vy[DPL];
                load_row_part<DPL, VT>(V, S.pidx[y], lane, vy);
                double acc = 0.0;
#pragma unroll
                for (int c = 0; c < DPL; ++c) acc = fma(dx[c], (double)vy[c] - (double)ol[c], acc);
                acc = warp_sum_d(acc) * (double)S.pp[x] * (double)S.pp[y];
                if (lane == 0) {
                    S.G[x * GLD + y] = S.G[y * GLD + x] = (float)acc;
                    g64[x * PMAX + y] = g64[y * PMAX + x] = acc;
                }
            }
        }
        __syncwarp();
        float S1 = 0.f;
        for (int x = lane; x < P; x += 32) {
            float sx = 0.f;
            for (int y = 0; y < P; ++y) sx += S.G[x * GLD + y];
            S.t[x] = sx;
            S1 += sqrtf(fmaxf(S.G[x * GLD + x], 0.f));
        }
        __syncwarp();
        float UU = 0.f, PU = 0.f;
        for (int x = lane; x < P; x += 32) {
            UU += S.t[x];
            PU += S.pp[x];
        }
        UU = warp_sum(UU);
        PU = warp_sum(PU);
        S1 = warp_sum(S1) * 1.0001f;
        // Rounding bound: every Gram entry, partial sum and t_x is bounded by
        // S1^2 (|G_xy| <= |u_x||u_y|); the products carry <= DPL + 8 roundings,
        // the score's chains <= 2P + m^2 + 2m more; twice that for safety.
        const float Eabs = (float)(2 * DPL + 32 + 4 * P + 2 * m * m + 4 * m) * 5.9604645e-8f * S1 * S1;
        const float pe = (float)(2 * P + 2 * m + 8) * 5.9604645e-8f * PU;
        // lane ranges of colex ranks
        const uint64_t qn = T / 32, rm = T % 32;
        uint64_t lo = qn * lane + min((uint64_t)lane, rm);
        const uint64_t hi = lo + qn + ((uint64_t)lane < rm ? 1 : 0);
        const uint64_t all = P == 64 ? ~0ull : ((1ull << P) - 1ull);
        // pass 1: the least upper end (m = 0: the pool itself is the only subset)
        float U = INFINITY;
        if (m == 0) lo = hi;
        walk(S, P, m, direct, lo, hi, UU, PU, Eabs, pe, [&](uint64_t, float, float up) { U = fminf(U, up); });
        U = warp_min(U);
        // pass 2: buffer every subset whose interval reaches down to U
        int over = 0;
        int64_t ncand = 0;
        walk(S, P, m, direct, lo, hi, UU, PU, Eabs, pe, [&](uint64_t Cm, float low, float) {
            if (low <= U) {
                ++ncand;
                const int slot = atomicAdd(&S.ncand, 1);
                if (slot < GCAP) gc[slot] = direct ? Cm : (all & ~Cm);
                else over = 1;
            }
        });
        __syncwarp();
        over = __any_sync(FW_FULL, over);
        double bes = INFINITY;
        uint64_t brank = ~0ull, bmask = 0;
        if (m == 0) {
            // the pool is the kept set itself: one subset
            bmask = all;
            bes = es_warp<DPL, VT>(V, ol, S, all, lane);
        } else if (!over) {
            const int nc = S.ncand;
            for (int q = 0; q < nc; ++q) {
                const uint64_t A = gc[q];
                const double es = es_gram_warp(g64, S, A, lane);
                const uint64_t rank = colex_rank64(A);
                if (es < bes || (es == bes && rank < brank)) {
                    bes = es;
                    brank = rank;
                    bmask = A;
                }
            }
        } else {
            // every lane re-scores its own candidates alone
            walk(S, P, m, direct, lo, hi, UU, PU, Eabs, pe, [&](uint64_t Cm, float low, float) {
                if (low <= U) {
                    const uint64_t A = direct ? Cm : (all & ~Cm);
                    const double es = es_gram_lane(g64, S, A);
                    const uint64_t rank = colex_rank64(A);
                    if (es < bes || (es == bes && rank < brank)) {
                        bes = es;
                        brank = rank;
                        bmask = A;
                    }
                }
            });
            for (int off = 16; off; off >>= 1) {
                const double oe = __shfl_xor_sync(FW_FULL, bes, off);
                const uint64_t orank = __shfl_xor_sync(FW_FULL, brank, off);
                const uint64_t omask = __shfl_xor_sync(FW_FULL, bmask, off);
                if (oe < bes || (oe == bes && orank < brank)) {
                    bes = oe;
                    brank = orank;
                    bmask = omask;
                }
            }
        }
        // the top-mass set: the pool's kept keys
        uint64_t K = 0;
        {
            const uint32_t tk = a.thr_key[it];
            const int ti = a.thr_idx[it];
            for (int x = lane; x < P; x += 32) {
                const uint32_t kl = order_key(__ldg(l + S.pidx[x]));
                if (kl > tk || (kl == tk && S.pidx[x] <= ti)) K |= 1ull << x;
            }
            for (int off = 16; off; off >>= 1) K |= __shfl_xor_sync(FW_FULL, K, off);
        }
        const double tes = a.topk_gap ? es_warp<DPL, VT>(V, ol, S, K, lane) : 0.0;
        ncand = (int64_t)warp_sum_d((double)ncand);
        if (lane == 0) {
            a.best_gap[it] = (float)bes;
            if (a.topk_gap) a.topk_gap[it] = (float)tes;
            if (a.n_cand) a.n_cand[it] = ncand;
        }
        bmask = __shfl_sync(FW_FULL, bmask, 0);
        for (int x = lane; x < P; x += 32)
            if ((bmask >> x) & 1ull) bi[__popcll(bmask & ((1ull << x) - 1ull))] = S.pidx[x];
        for (int q = s + lane; q < a.k_max; q += 32) bi[q] = -1;
        __syncwarp();
    }
}

}  // namespace

static size_t pool_bytes(const RowsDev &R, int nb) { return align256((size_t)R.rows * nb * PMAX * 4); }

// blocks of the enumeration launch: PE_BPS per SM, fewer when there are fewer items
static int64_t pool_enum_blocks(const RowsDev &R, int nb)
{
    int sms = 0;
    if (device_sms(&sms) != FW_OK) sms = 152;  // no device: the size query still answers
    const int64_t items = R.rows * nb;
    return std::max<int64_t>(1, std::min<int64_t>((items + PE_W - 1) / PE_W, (int64_t)sms * PE_BPS));
}

// per warp of the enumeration launch: the candidate buffer and the fp64 Gram matrix
static size_t warp_ws_bytes(const RowsDev &R, int nb)
{
    return align256((size_t)pool_enum_blocks(R, nb) * PE_W * (GCAP + PMAX * PMAX) * 8);
}

size_t pool_best_subset_workspace(const RowsDev &R, int nb)
{
    return pool_bytes(R, nb) + align256((size_t)R.rows * nb * 4) + warp_ws_bytes(R, nb);
}

fw_status pool_best_subset(const RowsDev &R, const int32_t *k, int nb, const int32_t *E, const fw_gap_out &topk,
                           float *best_gap, int32_t *best_idx, int k_max, float *topk_gap, int64_t *n_cand,
                           int32_t *row_status, void *ws, cudaStream_t st)
{
    if (R.max_n > PB_STAGE_MAX) return FW_ERR_UNSUPPORTED;
    PoolArgs a;
    a.R = R;
    a.k = k;
    a.nb = nb;
    for (int b = 0; b < 4; ++b) a.E[b] = b < nb ? E[b] : 0;
    a.thr_key = topk.thr_key;
    a.thr_idx = topk.thr_idx;
    a.o = topk.o;
    a.M = topk.row_max;
    a.Z = topk.row_sum;
    a.pool = (int32_t *)ws;
    a.pool_n = (int32_t *)((char *)ws + pool_bytes(R, nb));
    {
        char *w = (char *)ws + pool_bytes(R, nb) + align256((size_t)R.rows * nb * 4);
        a.gcand = (uint64_t *)w;
        a.g64 = (double *)(w + (size_t)pool_enum_blocks(R, nb) * PE_W * GCAP * 8);
    }
    a.best_gap = best_gap;
    a.best_idx = best_idx;
    a.k_max = k_max;
    a.topk_gap = topk_gap;
    a.row_status = row_status;
    a.n_cand = n_cand;
    int sms = 0;
    if (device_sms(&sms) != FW_OK) return FW_ERR_CUDA;
    if (row_status) FW_CUDA_CHECK(cudaMemsetAsync(row_status, 0, (size_t)R.rows * 4, st));
    FW_DISPATCH(R.d, R.v_dtype, {
        const size_t sb = (size_t)R.max_n * 4;
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_pool_build<DPL, VT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sb));
        FW_LAUNCH((k_pool_build<DPL, VT>), (unsigned)std::min<int64_t>(R.rows, (int64_t)sms * 4), PB_T, sb, st, a);
        const size_t se = (size_t)PE_W * sizeof(EnumSm);
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_pool_enum<DPL, VT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)se));
        FW_LAUNCH((k_pool_enum<DPL, VT>), (unsigned)pool_enum_blocks(R, nb), PE_W * 32, se, st, a);
    });
    return FW_OK;
}

}  // namespace fw
