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
#include <algorithm>

#include "fw_internal.h"
#include "tc_sm100.cuh"

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
    int32_t *redo_list;   // rows the register select leaves to the radix select
    int32_t *redo_count;  // (device) entries of redo_list; NULL: one CTA per row
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
__device__ __forceinline__ void select_row(const SelArgs &a, const int64_t row)
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

template <bool STAGED>
__global__ void __launch_bounds__(LT) k_long_select(const SelArgs a)
{
    if (!a.redo_count) {
        select_row<STAGED>(a, blockIdx.x);
        return;
    }
    const int cnt = *a.redo_count;
    for (int i = blockIdx.x; i < cnt; i += gridDim.x) {
        select_row<STAGED>(a, a.redo_list[i]);
        __syncthreads();
    }
}

// ------------------------------------------------------ linear-bin select
// Rows of at most SEL_MAX_N keys.  Persistent CTAs walk rows, and a row's
// logits stay in registers: thread t holds keys 4 (t + NT q) + c (q < VPT / 4,
// c < 4).  While a row is processed, the CTA's next row arrives in shared
// memory by bulk copy (rows that are whole 16-byte vectors; others are read
// from global memory directly), so its HBM time overlaps this row's work.  The k-th largest key of every budget comes
// from one histogram of SNB linear bins over [min, max] of the row (a monotone
// map of the float, so the bins split the key order), the bin holding the
// k-th key, and an exact rank among that bin's keys.  Rows whose threshold
// bin holds more than SCAP keys (heavy ties) are listed for the radix select,
// which runs on them after this kernel.  (A first version kept the row in
// shared memory, loaded after the previous row was done, with every pass a
// shared-memory sweep and a divergent candidate test; it ran at 13 % of HBM
// bandwidth.)
constexpr int SEL_MAX_N = 32768;  // longest row of the linear-bin select
constexpr int SNB = 2048;         // linear bins
constexpr int SCAP = 512;         // keys of a threshold bin ranked directly
constexpr int WCAP = 64;          // threshold-bin keys one warp gathers
constexpr uint32_t SEL_CHUNK = 32768;  // bytes per bulk-copy instruction
constexpr uint32_t SEL_WAIT = 1u << 22;  // polls of a row-copy wait before it gives up

template <int NT> __host__ __device__ constexpr int sel_minb() { return NT >= 1024 ? 1 : (NT >= 512 ? 2 : 4); }

template <int NT, int VPT>
__global__ void __launch_bounds__(NT, sel_minb<NT>()) k_long_select_reg(const SelArgs a)
{
    constexpr int NW = NT / 32;
    constexpr int V4 = VPT / 4;
    constexpr int BPT = SNB / NT;  // bins per thread in the scan
    static_assert(SNB % NT == 0 && VPT % 4 == 0, "layout");
    __shared__ uint32_t hist[SNB];
    __shared__ uint32_t ckey[4][SCAP];
    __shared__ int32_t cidx[4][SCAP];
    __shared__ uint32_t wkey[NW][WCAP];  // each warp's hits: order key, index, bin
    __shared__ int32_t widx[NW][WCAP];
    __shared__ int16_t wbin[NW][WCAP];
    __shared__ int wnum[NW], wbud[NW][4];
    __shared__ float red_a[NW], red_b[NW];
    __shared__ uint32_t wsum[NW];
    __shared__ int s_tb[4], s_ti[4], s_kv[4], s_rem[4], s_bcnt[4];
    __shared__ uint32_t s_T[4];
    __shared__ int s_staged, s_err;
    __shared__ __align__(8) uint64_t full;
    extern __shared__ __align__(16) float sbuf[];  // [max_n] the CTA's next row, by bulk copy
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int nb = a.nb;
    // the bulk copy of row r into sbuf (thread 0; rows that are not 16-byte
    // aligned whole vectors are read from global memory instead)
    auto stage = [&](int64_t r) -> int {
        if (r >= a.R.rows) return 0;
        const int64_t g2 = r / a.R.R;
        const int n2 = a.R.n[g2];
        const float *lg2 = a.R.logits + a.R.logit_off[g2] + (r - g2 * a.R.R) * n2;
        if ((n2 & 3) != 0 || (reinterpret_cast<uintptr_t>(lg2) & 15) != 0 || n2 < 1) return 0;
        const uint32_t bytes = (uint32_t)n2 * 4u;
        tc::fence_async_smem();
        tc::mbar_arrive_expect_tx(&full, bytes);
        for (uint32_t o = 0; o < bytes; o += SEL_CHUNK)
            tc::bulk_g2s(reinterpret_cast<char *>(sbuf) + o, reinterpret_cast<const char *>(lg2) + o,
                         bytes - o < SEL_CHUNK ? bytes - o : SEL_CHUNK, &full);
        return 1;
    };
    if (tid == 0) {
        tc::mbar_init(&full, 1);
        tc::mbar_init_fence();
        s_err = 0;
        s_staged = stage(blockIdx.x);
    }
    __syncthreads();
    uint32_t phase = 0;
    int64_t fail_row = -1;
    for (int64_t row = blockIdx.x; row < a.R.rows; row += gridDim.x) {
        const int64_t g = row / a.R.R;
        const int n = a.R.n[g];
        const float *lg = a.R.logits + a.R.logit_off[g] + (row - g * a.R.R) * n;
        const bool staged = s_staged != 0;
        if (staged) {
            if (wid == 0 && !tc::mbar_wait(&full, phase, SEL_WAIT)) s_err = 1;  // (every writer stores 1)
            phase ^= 1u;
            __syncthreads();
            if (s_err) {
                fail_row = row;
                break;
            }
        }
        // ---- the row into registers (zero past its end)
        float x[VPT];
#pragma unroll
        for (int q = 0; q < V4; ++q) {
            const int j0 = 4 * (tid + NT * q);
            if (staged) {
                float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
                if (j0 < n) v = reinterpret_cast<const float4 *>(sbuf)[tid + NT * q];
                x[4 * q] = v.x, x[4 * q + 1] = v.y, x[4 * q + 2] = v.z, x[4 * q + 3] = v.w;
            } else {
#pragma unroll
                for (int c = 0; c < 4; ++c) x[4 * q + c] = j0 + c < n ? __ldg(lg + j0 + c) : 0.f;
            }
        }
        __syncthreads();  // sbuf is read and s_staged consumed: the next row may land
        if (tid == 0) s_staged = stage(row + gridDim.x);
        // f(j, x) for every key of the row; a vector slot q is whole when all
        // threads' keys in it are inside the row (uniform test)
        auto for_keys = [&](auto &&f) {
#pragma unroll
            for (int q = 0; q < V4; ++q) {
                const int j0 = 4 * (tid + NT * q);
                if (4 * NT * (q + 1) <= n) {
#pragma unroll
                    for (int c = 0; c < 4; ++c) f(j0 + c, x[4 * q + c]);
                } else if (4 * NT * q < n) {
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        if (j0 + c < n) f(j0 + c, x[4 * q + c]);
                }
            }
        };
        float m = -INFINITY, mn = INFINITY;
        bool nan = false;
        for_keys([&](int, float v) {
            nan |= v != v;
            m = fmaxf(m, v);
            mn = fminf(mn, v);
        });
        m = warp_max(m);
        mn = warp_min(mn);
        if (lane == 0) {
            red_a[wid] = m;
            red_b[wid] = mn;
        }
        for (int i = tid; i < SNB; i += NT) hist[i] = 0u;
        if (tid < nb) s_kv[tid] = a.k[row * nb + tid];
        bool bad = __syncthreads_or(nan) || n < 1;
        m = warp_max(lane < NW ? red_a[lane] : -INFINITY);  // (every warp, every lane: the same)
        mn = warp_min(lane < NW ? red_b[lane] : INFINITY);
        bad |= !isfinite(m) || !isfinite(mn);  // (an infinite key is the max or the min)
        int status = bad ? FW_ERR_NONFINITE : FW_OK;
        for (int b = 0; b < nb; ++b) {
            const int kb = s_kv[b];
            if (kb < 1 || kb > n) status = status == FW_OK ? FW_ERR_INVALID_ARG : status;
        }
        // ---- sum of exponentials and the histogram of linear bins over [mn, m]
        // (halves keep m - mn finite)
        const float hmn = mn * 0.5f, den = m * 0.5f - hmn;
        float scl = den > 0.f ? (float)SNB / den : 0.f;
        if (!(scl < 1e30f)) scl = 0.f;
        auto bin_of = [&](float v) { return (int)fminf((v * 0.5f - hmn) * scl, (float)(SNB - 1)); };
        float se = 0.f;
        if (status == FW_OK) {
            for_keys([&](int, float v) {
                se += __expf(v - m);
                atomicAdd(&hist[bin_of(v)], 1u);
            });
        }
        se = warp_sum(se);
        __syncthreads();  // red_a reads above are done
        if (lane == 0) red_a[wid] = se;
        __syncthreads();
        const float Z = warp_sum(lane < NW ? red_a[lane] : 0.f);
        if (tid == 0) {
            a.ws.M[row] = m;
            a.ws.Z[row] = Z;
            a.ws.status[row] = status;
            if (a.out.row_max) a.out.row_max[row] = m;
            if (a.out.row_sum) a.out.row_sum[row] = Z;
            if (a.out.row_status) a.out.row_status[row] = status;
        }
        if (status != FW_OK) {  // (uniform)
            __syncthreads();
            continue;
        }
        // ---- keys above each bin (bins from the top), the bin of each budget's k-th key
        uint32_t hv[BPT], loc = 0;
#pragma unroll
        for (int i = 0; i < BPT; ++i) {
            hv[i] = hist[SNB - 1 - (tid * BPT + i)];
            loc += hv[i];
        }
        uint32_t inc = loc;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(FW_FULL, inc, o);
            if (lane >= o) inc += y;
        }
        if (lane == 31) wsum[wid] = inc;
        __syncthreads();
        uint32_t above = inc - loc + __reduce_add_sync(FW_FULL, lane < wid ? wsum[lane] : 0u);
#pragma unroll
        for (int i = 0; i < BPT; ++i) {
            const int bn = SNB - 1 - (tid * BPT + i);
            for (int b = 0; b < nb; ++b) {
                const uint32_t kb = (uint32_t)s_kv[b];
                if (above < kb && kb <= above + hv[i]) {
                    s_tb[b] = bn;
                    s_rem[b] = (int)(kb - above);
                    s_bcnt[b] = (int)hv[i];
                }
            }
            above += hv[i];
        }
        __syncthreads();
        // a budget whose threshold bin is crowded (heavy ties) leaves the row to
        // the radix select, which runs after this kernel on the listed rows
        bool crowded = false;
        for (int b = 0; b < nb; ++b) crowded |= s_bcnt[b] > SCAP;
        if (crowded) {
            if (tid == 0) a.redo_list[atomicAdd(a.redo_count, 1)] = (int32_t)row;
            __syncthreads();
            continue;
        }
        // ---- the threshold bins' keys.  Each warp gathers its hits in its own
        // buffer (ballot offsets, no atomics: the hits are sparse, and
        // same-address shared atomics from many warps serialise), then the
        // buffers are concatenated per budget.
        int gb[4];
#pragma unroll
        for (int b = 0; b < 4; ++b) gb[b] = b < nb ? s_tb[b] : -1;
        {
            int wc = 0;                 // this warp's hits (uniform)
            int bc[4] = {0, 0, 0, 0};   // ... per budget
            const uint32_t lt = (1u << lane) - 1u;
#pragma unroll
            for (int q = 0; q < V4; ++q) {
                if (4 * NT * q >= n) break;  // (uniform)
                const int j0 = 4 * (tid + NT * q);
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const float v = x[4 * q + c];
                    const int bn = bin_of(v);
                    const bool in = j0 + c < n;
                    bool h[4];
#pragma unroll
                    for (int b = 0; b < 4; ++b) h[b] = in && bn == gb[b];
                    const bool hit = h[0] | h[1] | h[2] | h[3];
                    const uint32_t mk = __ballot_sync(FW_FULL, hit);
                    if (mk) {
                        const int pos = wc + __popc(mk & lt);
                        if (hit && pos < WCAP) {
                            wkey[wid][pos] = order_key(v);
                            widx[wid][pos] = j0 + c;
                            wbin[wid][pos] = (int16_t)bn;
                        }
                        wc += __popc(mk);
#pragma unroll
                        for (int b = 0; b < 4; ++b) bc[b] += __popc(__ballot_sync(FW_FULL, h[b]));
                    }
                }
            }
            if (lane == 0) {
                wnum[wid] = wc;
#pragma unroll
                for (int b = 0; b < 4; ++b) wbud[wid][b] = bc[b];
            }
        }
        __syncthreads();
        // a warp with more hits than its buffer holds (keys of a threshold bin
        // bunched in one warp's stretch) leaves the row to the radix select
        if (__syncthreads_or(tid < NW && wnum[tid] > WCAP)) {
            if (tid == 0) a.redo_list[atomicAdd(a.redo_count, 1)] = (int32_t)row;
            __syncthreads();
            continue;
        }
        {
            const uint32_t lt = (1u << lane) - 1u;
            int off[4], run[4];
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                off[b] = (int)__reduce_add_sync(FW_FULL, lane < wid ? (uint32_t)wbud[lane][b] : 0u);  // (NW <= 32)
                run[b] = 0;
            }
            const int nw_ = wnum[wid];
            for (int e0 = 0; e0 < nw_; e0 += 32) {
                const int e = e0 + lane;
                const int bn = e < nw_ ? wbin[wid][e] : -2;
#pragma unroll
                for (int b = 0; b < 4; ++b) {
                    const bool mt = bn == gb[b];
                    const uint32_t bm = __ballot_sync(FW_FULL, mt);
                    const int p = off[b] + run[b] + __popc(bm & lt);
                    if (mt && p < SCAP) {  // (p < s_bcnt[b] <= SCAP: the bins match the histogram's)
                        ckey[b][p] = wkey[wid][e];
                        cidx[b][p] = widx[wid][e];
                    }
                    run[b] += __popc(bm);
                }
            }
        }
        __syncthreads();
        // the exact rank of every candidate among its budget's, a warp per
        // candidate (lanes split the comparisons)
        {
            const int p1 = s_bcnt[0], p2 = p1 + (nb > 1 ? s_bcnt[1] : 0), p3 = p2 + (nb > 2 ? s_bcnt[2] : 0),
                      p4 = p3 + (nb > 3 ? s_bcnt[3] : 0);
            for (int t = wid; t < p4; t += NW) {
                const int b = (t >= p1) + (t >= p2) + (t >= p3);
                const int base = b == 0 ? 0 : (b == 1 ? p1 : (b == 2 ? p2 : p3));
                const int cb = s_bcnt[b];
                const int c = t - base;
                const uint32_t kc = ckey[b][c];
                const int ic = cidx[b][c];
                uint32_t r = 0;
                for (int c2 = lane; c2 < cb; c2 += 32) {
                    const uint32_t k2 = ckey[b][c2];
                    r += k2 > kc || (k2 == kc && cidx[b][c2] < ic);
                }
                r = __reduce_add_sync(FW_FULL, r);
                if (lane == 0 && (int)r == s_rem[b] - 1) {
                    s_T[b] = kc;
                    s_ti[b] = ic;
                }
            }
        }
        __syncthreads();
        // ---- thresholds and kept bits
        if (tid < nb) {
            a.ws.tk[row * nb + tid] = s_T[tid];
            a.ws.ti[row * nb + tid] = s_ti[tid];
            if (a.out.thr_key) a.out.thr_key[row * nb + tid] = s_T[tid];
            if (a.out.thr_idx) a.out.thr_idx[row * nb + tid] = s_ti[tid];
        }
        if (a.out.kept_bits) {
            // keys strictly above each threshold by one compare; a warp's 4 keys
            // per lane in slot q are 128 consecutive keys, so the 8 lanes of an
            // octet make one 32-bit word.  The keys equal to the threshold (all
            // in its bin, so among the candidates) up to the tie index are
            // added after.
            const int nw = a.out.kept_words;
            float xt[4];
#pragma unroll
            for (int b = 0; b < 4; ++b) xt[b] = b < nb ? key_float(s_T[b]) : INFINITY;
#pragma unroll
            for (int q = 0; q < V4; ++q) {
                const int j0 = 4 * (tid + NT * q);
                const int w = j0 >> 5;
#pragma unroll
                for (int b = 0; b < 4; ++b) {
                    if (b >= nb) break;
                    uint32_t bits = 0u;
#pragma unroll
                    for (int c = 0; c < 4; ++c) bits |= (uint32_t)(j0 + c < n && x[4 * q + c] > xt[b]) << c;
                    bits <<= (j0 & 31);
                    bits |= __shfl_xor_sync(FW_FULL, bits, 1);
                    bits |= __shfl_xor_sync(FW_FULL, bits, 2);
                    bits |= __shfl_xor_sync(FW_FULL, bits, 4);
                    if ((lane & 7) == 0 && w < nw) a.out.kept_bits[(row * nb + b) * (int64_t)nw + w] = bits;
                }
            }
            __syncthreads();  // the words above are visible to the block
            constexpr int CPB = NT / 4;
            const int b = tid / CPB;
            if (b < nb) {
                const uint32_t T = s_T[b];
                const int ti = s_ti[b];
                for (int c = tid % CPB; c < s_bcnt[b]; c += CPB) {
                    const int ic = cidx[b][c];
                    if (ckey[b][c] == T && ic <= ti)
                        atomicOr(&a.out.kept_bits[(row * nb + b) * (int64_t)nw + (ic >> 5)], 1u << (ic & 31));
                }
            }
        }
        __syncthreads();  // s_T, s_ti, hist and candidates are reused by the next row
    }
    if (fail_row >= 0 && tid == 0) {
        // a row copy did not arrive in time: after a last bounded wait for it,
        // that row and the rest of this CTA's rows are marked
        (void)tc::mbar_wait(&full, phase ^ 1u, SEL_WAIT);
        for (int64_t row = fail_row; row < a.R.rows; row += gridDim.x) {
            a.ws.status[row] = FW_ERR_TIMEOUT;
            if (a.out.row_status) a.out.row_status[row] = FW_ERR_TIMEOUT;
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

// after the LongWs arrays: the redo list [rows] and its count
static size_t carve_bytes(const RowsDev &R, int nb)
{
    return align256(R.rows * 4) * 2 + align256(R.rows * nb * 4) * 2 + align256(R.rows * 4);
}

size_t long_gap_workspace(const RowsDev &R, int nb) { return carve_bytes(R, nb) + align256(R.rows * 4) + 256; }

fw_status long_gap(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &out, void *ws, size_t ws_bytes,
                   cudaStream_t s)
{
    (void)ws_bytes;
    const LongWs L = carve(R, nb, ws);
    int32_t *redo_list = (int32_t *)((char *)ws + carve_bytes(R, nb));
    int32_t *redo_count = (int32_t *)((char *)redo_list + align256(R.rows * 4));
    SelArgs sa{R, k, nb, out, L, redo_list, nullptr};
    if (R.max_n <= SEL_MAX_N) {
        FW_CUDA_CHECK(cudaMemsetAsync(redo_count, 0, sizeof(int32_t), s));
        sa.redo_count = redo_count;
        int dev = 0, sms = 0;
        FW_CUDA_CHECK(cudaGetDevice(&dev));
        FW_CUDA_CHECK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
        auto launch = [&](auto kernel, int nt) -> fw_status {
            const size_t smem = (size_t)R.max_n * 4;
            FW_CUDA_CHECK(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
            int per_sm = 0;
            FW_CUDA_CHECK(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, nt, smem));
            const int64_t grid = std::min<int64_t>(R.rows, (int64_t)sms * std::max(per_sm, 1));
            FW_LAUNCH(kernel, (unsigned)grid, nt, smem, s, sa);
            return FW_OK;
        };
        const fw_status st = R.max_n <= 1024    ? launch(k_long_select_reg<256, 4>, 256)
                             : R.max_n <= 2048  ? launch(k_long_select_reg<256, 8>, 256)
                             : R.max_n <= 4096  ? launch(k_long_select_reg<256, 16>, 256)
                             : R.max_n <= 8192  ? launch(k_long_select_reg<512, 16>, 512)
                             : R.max_n <= 16384 ? launch(k_long_select_reg<512, 32>, 512)
                                                : launch(k_long_select_reg<1024, 32>, 1024);
        if (st != FW_OK) return st;
        // the listed rows (crowded threshold bins) by the radix select
        const size_t smem = (size_t)R.max_n * 4;
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_long_select<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        FW_LAUNCH(k_long_select<true>, (unsigned)std::min<int64_t>(R.rows, sms), LT, smem, s, sa);
    } else if (R.max_n <= kSelStageMax) {
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
