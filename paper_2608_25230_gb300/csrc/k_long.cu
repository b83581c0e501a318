// k_long.cu -- rows of any length: softmax statistics, exact top-k thresholds
// and the P.V products behind the dense output, forced-weight output, gap and
// dropped mass (Definition 2.1, Sec. 2.1, Lemma 2.1).
//
// Kernel 1 (one CTA per row): online max/sum-exp, then a 4 x 8-bit radix
// select of the k-th largest order key for every budget, then the index of
// the last kept key among equal ones (ties keep lower indices first).
// Kernel 2 (one CTA per (group, tile of rows sharing V)): streams V once per
// tile and accumulates, per row, the sums S_b = sum p_j v_j over the "bands"
// of nested kept sets (band of key j = number of budgets that drop it).  Then
// N_A = sum of the bands inside A, N_{A^c} = the rest, and
//   o_A - mu = (pbar(A) N_A - p(A) N_{A^c}) / p(A),
// which never subtracts two rounded outputs and keeps the gap accurate when it
// is small; pbar(A) is summed over the dropped keys.
#include "fw_internal.h"

namespace fw {
namespace {

constexpr int LT = 256;  // threads of the select kernel
constexpr int kSelStageMax = 32768;  // longest row whose keys the select kernel stages (128 KB)
constexpr int RT = 8;    // rows per P.V tile
constexpr int JT = 64;   // keys per staged chunk

struct SelArgs {
    RowsDev R;
    const int32_t *k;
    int nb;
    fw_gap_out out;
    LongWs ws;
};

__device__ __forceinline__ void block_max_sum(float &m, float &s, float *red_m, float *red_s)
{
    // combine (m, s) pairs: s = sum exp(x - m)
    for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(FW_FULL, m, o);
        const float s2 = __shfl_xor_sync(FW_FULL, s, o);
        const float mm = fmaxf(m, m2);
        s = (m == -INFINITY ? 0.f : s * expf(m - mm)) + (m2 == -INFINITY ? 0.f : s2 * expf(m2 - mm));
        m = mm;
    }
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        red_m[w] = m;
        red_s[w] = s;
    }
    __syncthreads();
    if (w == 0) {
        m = lane < (int)(blockDim.x >> 5) ? red_m[lane] : -INFINITY;
        s = lane < (int)(blockDim.x >> 5) ? red_s[lane] : 0.f;
        for (int o = 16; o > 0; o >>= 1) {
            const float m2 = __shfl_xor_sync(FW_FULL, m, o);
            const float s2 = __shfl_xor_sync(FW_FULL, s, o);
            const float mm = fmaxf(m, m2);
            s = (m == -INFINITY ? 0.f : s * expf(m - mm)) + (m2 == -INFINITY ? 0.f : s2 * expf(m2 - mm));
            m = mm;
        }
        if (lane == 0) {
            red_m[0] = m;
            red_s[0] = s;
        }
    }
    __syncthreads();
    m = red_m[0];
    s = red_s[0];
    __syncthreads();
}

// STAGED: the row's order keys are kept in shared memory (rows of at most
// kSelStageMax keys), so the logits are read from HBM once; otherwise every
// pass re-reads them.
// The float of an order key (inverse of order_key; -0 comes back as +0).
__device__ __forceinline__ float key_float(uint32_t k)
{
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

template <bool STAGED>
__global__ void __launch_bounds__(LT) k_long_select(const SelArgs a)
{
    extern __shared__ uint32_t skeys[];  // [n] order keys when STAGED
    __shared__ uint32_t hist[4][256];
    __shared__ uint32_t whist[LT / 32][4][256];  // per-warp histograms (32 KB)
    __shared__ float red_m[32], red_s[32];
    __shared__ uint32_t s_prefix[4], s_rem[4];
    __shared__ int s_bad;
    __shared__ uint32_t wcnt[LT / 32];
    __shared__ int s_found;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int64_t row = blockIdx.x;
    const int64_t g = row / a.R.R;
    const int64_t ri = row - g * a.R.R;
    const int n = a.R.n[g];
    const int nb = a.nb;
    const float *lg = a.R.logits + a.R.logit_off[g] + ri * n;
    auto key_at = [&](int j) -> uint32_t { return STAGED ? skeys[j] : order_key(lg[j]); };
    if (tid == 0) s_bad = 0;
    __syncthreads();
    float m = -INFINITY, s = 0.f;
    bool bad = n < 1;
    if (STAGED) {
        // max and staged keys (independent loads, no branch), then sum of exp from shared memory
#pragma unroll 8
        for (int j = tid; j < n; j += LT) {
            const float x = lg[j];
            skeys[j] = order_key(x);
            bad |= !isfinite(x);
            m = fmaxf(m, x);
        }
        if (bad) atomicOr(&s_bad, 1);
        m = warp_max(m);
        if (lane == 0) red_m[wid] = m;
        __syncthreads();
        m = red_m[0];
        for (int w = 1; w < LT / 32; ++w) m = fmaxf(m, red_m[w]);
        for (int j = tid; j < n; j += LT) s += expf(key_float(skeys[j]) - m);
        s = warp_sum(s);
        if (lane == 0) red_s[wid] = s;
        __syncthreads();
        s = 0.f;
        for (int w = 0; w < LT / 32; ++w) s += red_s[w];
    } else {
        // online max / sum of exp
        for (int j = tid; j < n; j += LT) {
            const float x = lg[j];
            if (!isfinite(x)) {
                bad = true;
                continue;
            }
            if (x > m) {
                s = s * expf(m - x) + 1.f;
                m = x;
            } else {
                s += expf(x - m);
            }
        }
        if (bad) atomicOr(&s_bad, 1);
        block_max_sum(m, s, red_m, red_s);
    }
    int status = s_bad ? FW_ERR_NONFINITE : FW_OK;
    if (status == FW_OK) {
        for (int b = 0; b < nb; ++b) {
            const int kb = a.k[row * nb + b];
            if (kb < 1 || kb > n) status = FW_ERR_INVALID_ARG;
        }
    }
    if (tid == 0) {
        a.ws.M[row] = m;
        a.ws.Z[row] = s;
        a.ws.status[row] = status;
        if (a.out.row_max) a.out.row_max[row] = m;
        if (a.out.row_sum) a.out.row_sum[row] = s;
        if (a.out.row_status) a.out.row_status[row] = status;
    }
    if (status != FW_OK) return;
    // radix select of the kb-th largest key, 8 bits at a time from the top.
    // Per-warp histograms.  Pass 0 (the top byte, where a row's keys share a
    // handful of values) has one histogram for every budget and counts each
    // warp's equal bins once; later passes use shared atomics.
    if (tid < nb) {
        s_prefix[tid] = 0u;
        s_rem[tid] = (uint32_t)a.k[row * nb + tid];
    }
    uint32_t pmask = 0u;
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        const int nh = pass == 0 ? 1 : nb;  // histograms this pass
        for (int i = tid; i < (LT / 32) * 4 * 256; i += LT) (&whist[0][0][0])[i] = 0u;
        __syncthreads();
        uint32_t pre[4];
#pragma unroll
        for (int b = 0; b < 4; ++b) pre[b] = b < nb ? s_prefix[b] : 0u;
        for (int j0 = 0; j0 < n; j0 += LT) {
            const int j = j0 + tid;
            const uint32_t key = j < n ? key_at(j) : 0u;
            if (pass == 0) {  // top bytes: few distinct values, aggregate them in the warp first
                const uint32_t bin = j < n ? key >> 24 : 256u + lane;  // lone lanes skip
                const uint32_t grp = __match_any_sync(FW_FULL, bin);
                if (j < n && lane == __ffs(grp) - 1) whist[wid][0][bin] += __popc(grp);
            } else {
#pragma unroll
                for (int b = 0; b < 4; ++b)
                    if (b < nb && j < n && (key & pmask) == pre[b]) atomicAdd(&whist[wid][b][(key >> shift) & 255u], 1u);
            }
        }
        __syncthreads();
        // merge the warps' histograms (bins split over the threads)
        for (int e = tid; e < nh * 256; e += LT) {
            uint32_t c = 0;
            for (int w = 0; w < LT / 32; ++w) c += whist[w][e >> 8][e & 255];
            hist[e >> 8][e & 255] = c;
        }
        __syncthreads();
        if (tid < nb) {
            const int hb = pass == 0 ? 0 : tid;
            uint32_t cum = 0, rem = s_rem[tid];
            for (int v = 255; v >= 0; --v) {
                const uint32_t c = hist[hb][v];
                if (cum + c >= rem) {
                    s_prefix[tid] |= (uint32_t)v << shift;
                    s_rem[tid] = rem - cum;
                    break;
                }
                cum += c;
            }
        }
        pmask |= 255u << shift;
        __syncthreads();
    }
    // the s_rem[b]-th key equal to the threshold, in index order
    for (int b = 0; b < nb; ++b) {
        const uint32_t T = s_prefix[b];
        const uint32_t want = s_rem[b];
        uint32_t base = 0;
        if (tid == 0) s_found = -1;
        __syncthreads();
        for (int j0 = 0; j0 < n; j0 += LT) {
            const int j = j0 + tid;
            const bool match = j < n && key_at(j) == T;
            const uint32_t bal = __ballot_sync(FW_FULL, match);
            if (lane == 0) wcnt[wid] = __popc(bal);
            __syncthreads();
            uint32_t before = 0, total = 0;
            for (int w = 0; w < LT / 32; ++w) {
                if (w < wid) before += wcnt[w];
                total += wcnt[w];
            }
            if (match) {
                const uint32_t r = base + before + __popc(bal & ((1u << lane) - 1u)) + 1u;
                if (r == want) s_found = j;
            }
            __syncthreads();
            base += total;
            if (base >= want) break;
        }
        __syncthreads();
        if (tid == 0) {
            a.ws.tk[row * nb + b] = T;
            a.ws.ti[row * nb + b] = s_found;
            if (a.out.thr_key) a.out.thr_key[row * nb + b] = T;
            if (a.out.thr_idx) a.out.thr_idx[row * nb + b] = s_found;
        }
        __syncthreads();
        if (a.out.kept_bits) {
            const int ti = s_found;
            uint32_t *wbits = a.out.kept_bits + (row * nb + b) * (int64_t)a.out.kept_words;
            const int nw = a.out.kept_words;
            for (int w0 = 0; w0 < nw * 32; w0 += LT) {
                const int j = w0 + tid;
                bool kept = false;
                if (j < n) {
                    const uint32_t key = key_at(j);
                    kept = key > T || (key == T && j <= ti);
                }
                const uint32_t bal = __ballot_sync(FW_FULL, kept);
                if (lane == 0 && (j >> 5) < nw) wbits[j >> 5] = bal;
            }
        }
    }
}

// ------------------------------------------------------------------- P . V
struct PvArgs {
    RowsDev R;
    const int32_t *k;
    int nb;
    fw_gap_out out;
    LongWs ws;
    int tiles_per_group;
};

template <int DPL, typename VT>
__global__ void __launch_bounds__(DPL * 32) k_long_pv(const PvArgs a)
{
    constexpr int d = DPL * 32;
    constexpr int NT = d;  // one thread per value dimension
    __shared__ float pst[RT][JT];
    __shared__ uint8_t bst[RT][JT];
    __shared__ float rowM[RT], rowZi[RT];
    __shared__ uint32_t rtk[RT][4];
    __shared__ int32_t rti[RT][4];
    __shared__ int rok[RT];
    __shared__ float bmass[RT][5];
    __shared__ float red[RT][5][d / 32 > 0 ? d / 32 : 1];
    const int tid = threadIdx.x;
    const int nb = a.nb;
    const int64_t g = blockIdx.x / a.tiles_per_group;
    const int tile = blockIdx.x - (int)(g * a.tiles_per_group);
    const int r0 = tile * RT;
    const int nr = min(RT, a.R.R - r0);
    const int n = a.R.n[g];
    const VT *V = reinterpret_cast<const VT *>(a.R.v) + a.R.v_off[g];
    if (tid < RT) {
        const int r = tid;
        rok[r] = 0;
        if (r < nr) {
            const int64_t row = g * a.R.R + r0 + r;
            rok[r] = a.ws.status[row] == FW_OK;
            rowM[r] = a.ws.M[row];
            rowZi[r] = 1.f / a.ws.Z[row];
            for (int b = 0; b < 4; ++b) {
                rtk[r][b] = b < nb ? a.ws.tk[row * nb + b] : 0u;
                rti[r][b] = b < nb ? a.ws.ti[row * nb + b] : -1;
            }
        }
        for (int b = 0; b < 5; ++b) bmass[r][b] = 0.f;
    }
    __syncthreads();
    float acc[RT][5];
#pragma unroll
    for (int r = 0; r < RT; ++r)
#pragma unroll
        for (int b = 0; b < 5; ++b) acc[r][b] = 0.f;
    float mloc[RT * JT / NT > 0 ? RT * JT / NT : 1][5];
    constexpr int PER = (RT * JT + NT - 1) / NT;
#pragma unroll
    for (int i = 0; i < PER; ++i)
#pragma unroll
        for (int b = 0; b < 5; ++b) mloc[i][b] = 0.f;
    for (int j0 = 0; j0 < n; j0 += JT) {
        // stage p and the band of RT x JT (row, key) pairs
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const int e = tid + i * NT;
            if (e < RT * JT) {
                const int r = e / JT, jj = e % JT, j = j0 + jj;
                float p = 0.f;
                int band = 0;
                if (r < nr && j < n && rok[r]) {
                    const int64_t row = g * a.R.R + r0 + r;
                    const float x = a.R.logits[a.R.logit_off[g] + (int64_t)(r0 + r) * n + j];
                    (void)row;
                    p = expf(x - rowM[r]) * rowZi[r];
                    const uint32_t key = order_key(x);
                    for (int b = 0; b < nb; ++b)
                        band += !(key > rtk[r][b] || (key == rtk[r][b] && j <= rti[r][b]));
                    mloc[i][0] += band == 0 ? p : 0.f;
#pragma unroll
                    for (int b = 1; b < 5; ++b) mloc[i][b] += band == b ? p : 0.f;
                }
                pst[r][jj] = p;
                bst[r][jj] = (uint8_t)band;
            }
        }
        __syncthreads();
        const int jl = min(JT, n - j0);
        for (int jj = 0; jj < jl; ++jj) {
            const float v = load_v(V, (int64_t)(j0 + jj) * d + tid);
#pragma unroll
            for (int r = 0; r < RT; ++r) {
                const float p = pst[r][jj];
                const int band = bst[r][jj];
#pragma unroll
                for (int b = 0; b < 5; ++b) acc[r][b] = fmaf(band == b ? p : 0.f, v, acc[r][b]);
            }
        }
        __syncthreads();
    }
    // band masses: each thread's staged rows are fixed: row of element (tid + i*NT)
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        const int e = tid + i * NT;
        if (e < RT * JT) {
            const int r = e / JT;
#pragma unroll
            for (int b = 0; b < 5; ++b) atomicAdd(&bmass[r][b], mloc[i][b]);
        }
    }
    __syncthreads();
    // epilogue per row and budget
    const int lane = tid & 31, wid = tid >> 5;
    for (int r = 0; r < nr; ++r) {
        if (!rok[r]) continue;
        const int64_t row = g * a.R.R + r0 + r;
        float o = 0.f;
#pragma unroll
        for (int b = 0; b < 5; ++b) o += acc[r][b];
        if (a.out.o) a.out.o[row * d + tid] = o;
        for (int b = 0; b < nb; ++b) {
            // sorted position of budget b among the row's budgets
            const int kb = a.k[row * nb + b];
            int sb = 0;
            for (int b2 = 0; b2 < nb; ++b2) {
                const int k2 = a.k[row * nb + b2];
                sb += (k2 < kb) || (k2 == kb && b2 < b);
            }
            float NA = 0.f, NC = 0.f, PA = 0.f, PC = 0.f;
#pragma unroll
            for (int q = 0; q < 5; ++q) {
                if (q <= sb) {
                    NA += acc[r][q];
                    PA += bmass[r][q];
                } else {
                    NC += acc[r][q];
                    PC += bmass[r][q];
                }
            }
            const float diff = PC * NA - PA * NC;  // p(A) (m_A - mu)
            float s2 = warp_sum(diff * diff);
            if (lane == 0) red[r][b][wid] = s2;
            __syncthreads();
            if (tid == 0) {
                float t = 0.f;
                for (int w = 0; w < NT / 32; ++w) t += red[r][b][w];
                const float phi = sqrtf(t);
                a.out.gap[row * nb + b] = phi / PA;
                a.out.dropped[row * nb + b] = PC;
                if (a.out.phi) a.out.phi[row * nb + b] = phi;
            }
            if (a.out.o_kept) a.out.o_kept[(row * nb + b) * d + tid] = NA / PA;
            __syncthreads();
        }
    }
}

}  // namespace

static LongWs carve(const RowsDev &R, int nb, void *ws)
{
    char *w = (char *)ws;
    LongWs L;
    L.M = (float *)w;
    w += align256(R.rows * 4);
    L.Z = (float *)w;
    w += align256(R.rows * 4);
    L.tk = (uint32_t *)w;
    w += align256(R.rows * nb * 4);
    L.ti = (int32_t *)w;
    w += align256(R.rows * nb * 4);
    L.status = (int32_t *)w;
    return L;
}

size_t long_gap_workspace(const RowsDev &R, int nb)
{
    return align256(R.rows * 4) * 2 + align256(R.rows * nb * 4) * 2 + align256(R.rows * 4);
}

fw_status long_gap(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &out, void *ws, size_t ws_bytes,
                   cudaStream_t s)
{
    (void)ws_bytes;
    const LongWs L = carve(R, nb, ws);
    const SelArgs sa{R, k, nb, out, L};
    if (R.max_n <= kSelStageMax) {
        const size_t smem = (size_t)R.max_n * 4;
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_long_select<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        FW_LAUNCH(k_long_select<true>, (unsigned)R.rows, LT, smem, s, sa);
    } else {
        FW_LAUNCH(k_long_select<false>, (unsigned)R.rows, LT, 0, s, sa);
    }
    if (long_pv_tc_supported(R, nb)) return long_pv_tc(R, k, nb, out, L, s);
    PvArgs pa{R, k, nb, out, L, (R.R + RT - 1) / RT};
    const unsigned grid = (unsigned)(R.num_groups * pa.tiles_per_group);
    FW_DISPATCH(R.d, R.v_dtype, FW_LAUNCH((k_long_pv<DPL, VT>), grid, DPL * 32, 0, s, pa));
    return FW_OK;
}

}  // namespace fw
