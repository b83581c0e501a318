// k_wscore.cu -- the observation-window importance score that Sec. 4 runs
// ContourKV with (SnapKV's score): the last w query rows of a cell (KV head)
// vote for the keys they attend to, and the votes are max-pooled along the
// positions.  For cell c with keys k_j (j < T) and window queries q_i
// (i < w, query i at position T - w + i, so it sees keys j <= T - w + i):
//   a_ij   = softmax over the visible j of scale * q_i . k_j,
//   vote_j = sum_i a_ij,
//   r_j    = max of vote over [j - h, j + h] clipped to the prefix [0, T - w)
//            for prefix positions (h = pool / 2), r_j = vote_j in the window.
//
// One CTA per cell, two passes over its keys (per-query softmax statistics,
// then the votes); each pass is a GEMM of 128-key tiles against the window:
// D[128 keys][32 queries] = K_tile (128 x d, K-major) x Q^T (d x 32, K-major)
// on tcgen05 (bf16 x bf16 -> fp32 in TMEM), the K tiles brought in by TMA
// (128-byte swizzle, three stages), the window queries by TMA once per cell.
// Warp 0 issues the TMA loads, warp 1 the MMAs (and owns the TMEM: two
// accumulators of 32 columns), warps 2-5 read the accumulators (one TMEM lane
// quarter each: 32 keys x 32 queries per thread row) and keep per-query
// running max / sum (pass 1) or add up the votes (pass 2).  Every wait is
// bounded; a wait that gives up marks the cell FW_ERR_TIMEOUT, the warps keep
// their loop shape (so named barriers still meet), in-flight copies are waited
// for, and the TMEM is freed.
#include <cuda.h>  // CUtensorMap and its enums (the encoder comes from the driver at run time)

#include "fw_internal.h"
#include "tc_sm100.cuh"

namespace fw {
namespace {

constexpr int WS_KT = 128;                 // keys per tile: the MMA's M
constexpr int WS_N = 32;                   // window queries per tile: the MMA's N (w <= 32, padded)
constexpr int WS_STAGES = 3;               // K tiles in flight
constexpr int WS_THREADS = 192;            // TMA warp, MMA warp, four epilogue warps
constexpr uint32_t WS_WAIT = 1u << 22;     // polls before a wait gives up

struct WsArgs {
    int cells, T, w, ph;  // ph: half-width of the max pool
    float scale2;         // scale * log2(e): logits in base-2 units
    float *votes;         // workspace [cells][T]
    float *scores;        // [cells][T]
    int32_t *status;      // [cells] or null
};

__device__ __forceinline__ void ws_named_barrier() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// 2^x by the hardware approximation (ex2.approx.ftz: ~2 ulp, well inside the
// score's 1e-4 tolerance); the per-(key, query) exponentials are most of the
// epilogue's work
__device__ __forceinline__ float ex2a(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// combine two (max, sum of 2^(x - max)) pairs
__device__ __forceinline__ void ms_merge(float &m, float &z, float m2, float z2)
{
    const float mn = fmaxf(m, m2);
    const float a = m == -INFINITY ? 0.f : z * exp2f(m - mn);
    const float b = m2 == -INFINITY ? 0.f : z2 * exp2f(m2 - mn);
    m = mn;
    z = a + b;
}

template <int D>
__global__ void __launch_bounds__(WS_THREADS, 2) k_wscore(const __grid_constant__ CUtensorMap tmK,
                                                       const __grid_constant__ CUtensorMap tmQ, const WsArgs a)
{
    constexpr int NBOX = D / 64;          // 128-byte boxes across d
    constexpr int KBOX = WS_KT * 128;     // bytes of one K box
    constexpr int KSTAGE = NBOX * KBOX;   // bytes of one K tile
    constexpr int QBOX = WS_N * 128;      // bytes of one Q box
    extern __shared__ uint8_t smraw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~(uintptr_t)1023);
    uint8_t *sK = sm;                            // [STAGES][NBOX][128 rows x 128 B]
    uint8_t *sQ = sm + WS_STAGES * KSTAGE;       // [NBOX][32 rows x 128 B]
    __shared__ __align__(8) uint64_t full[WS_STAGES], empty[WS_STAGES], accfull[2], accempty[2], qfull;
    __shared__ uint32_t s_taddr;
    __shared__ int s_err;
    __shared__ float s_m[4][WS_N], s_z[4][WS_N];

    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int c = blockIdx.x;
    const int T = a.T, w = a.w;
    const int ntiles = (T + WS_KT - 1) / WS_KT;
    const int total = 2 * ntiles;
    if (tid == 0) {
        for (int s = 0; s < WS_STAGES; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            tc::mbar_init(&accfull[b], 1);
            tc::mbar_init(&accempty[b], 4);
        }
        tc::mbar_init(&qfull, 1);
        tc::mbar_init_fence();
        s_err = 0;
    }
    if (wid == 1) tc::tmem_alloc(&s_taddr, 64);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t taddr = s_taddr;

    if (wid == 0) {
        // -------------------------------------------------------------- TMA
        if (lane == 0) {
            tc::tma_prefetch_desc(&tmK);
            tc::tma_prefetch_desc(&tmQ);
            tc::mbar_arrive_expect_tx(&qfull, NBOX * QBOX);
            for (int h = 0; h < NBOX; ++h) tc::tma_load_2d(sQ + h * QBOX, &tmQ, 64 * h, c * w, &qfull);
            int issued = 0;
            bool ok = true;
            for (int it = 0; it < total; ++it) {
                const int s = it % WS_STAGES;
                if (it >= WS_STAGES && !tc::mbar_wait(&empty[s], (uint32_t)((it / WS_STAGES) - 1) & 1u, WS_WAIT)) {
                    ok = false;
                    break;
                }
                const int t = it % ntiles;
                tc::mbar_arrive_expect_tx(&full[s], KSTAGE);
                for (int h = 0; h < NBOX; ++h)
                    tc::tma_load_2d(sK + s * KSTAGE + h * KBOX, &tmK, 64 * h, c * T + t * WS_KT, &full[s]);
                ++issued;
            }
            if (!ok) atomicOr(&s_err, 1);
            // every copy this thread started has landed before the CTA moves on
            // (already so when the MMAs consumed them)
            for (int it = issued - WS_STAGES < 0 ? 0 : issued - WS_STAGES; it < issued; ++it)
                if (!tc::mbar_wait(&full[it % WS_STAGES], (uint32_t)(it / WS_STAGES) & 1u, WS_WAIT)) atomicOr(&s_err, 1);
            if (!tc::mbar_wait(&qfull, 0, WS_WAIT)) atomicOr(&s_err, 1);
        }
        __syncwarp();
    } else if (wid == 1) {
        // -------------------------------------------------------------- MMA
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_bf16_f32(WS_KT, WS_N, false, false);
            const uint32_t k0 = tc::smem_u32(sK), q0 = tc::smem_u32(sQ);
            bool ok = tc::mbar_wait(&qfull, 0, WS_WAIT);
            int last = -1;
            for (int it = 0; ok && it < total; ++it) {
                const int s = it % WS_STAGES, b = it & 1;
                ok = tc::mbar_wait(&full[s], (uint32_t)(it / WS_STAGES) & 1u, WS_WAIT);
                if (ok && it >= 2) ok = tc::mbar_wait(&accempty[b], (uint32_t)((it >> 1) - 1) & 1u, WS_WAIT);
                if (!ok) break;
                tc::fence_after_sync();
#pragma unroll
                for (int ks = 0; ks < D / 16; ++ks) {
                    const int h = ks >> 2, off = (ks & 3) * 32;
                    const uint64_t ad = tc::sdesc_sw128(k0 + s * KSTAGE + h * KBOX + off, 16, 1024);
                    const uint64_t bd = tc::sdesc_sw128(q0 + h * QBOX + off, 16, 1024);
                    tc::mma_bf16(taddr + (uint32_t)(b * 32), ad, bd, idesc, ks > 0);
                }
                tc::commit(&empty[s]);
                tc::commit(&accfull[b]);
                last = it;
            }
            if (!ok) atomicOr(&s_err, 1);
            // the last MMAs have completed before the TMEM can be freed
            if (last >= 0 && !tc::mbar_wait(&accfull[last & 1], (uint32_t)(last >> 1) & 1u, WS_WAIT))
                atomicOr(&s_err, 1);
        }
        __syncwarp();
    } else {
        // --------------------------------------------------------- epilogue
        const int q4 = wid & 3;  // the TMEM lane quarter this warp may read
        const int ew = wid - 2;  // epilogue warp 0..3
        const float scale2 = a.scale2;
        float m[WS_N], z[WS_N];  // pass 1: running max / sum; pass 2: max and 1 / sum
#pragma unroll
        for (int i = 0; i < WS_N; ++i) {
            m[i] = -INFINITY;
            z[i] = 0.f;
        }
        bool ok = true;
        for (int it = 0; it < total; ++it) {
            const int b = it & 1, pass = it / ntiles, t = it - pass * ntiles;
            if (pass == 1 && t == 0) {
                // the softmax statistics of every query over all keys of the cell
#pragma unroll
                for (int i = 0; i < WS_N; ++i) {
                    float mi = m[i], zi = z[i];
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1)
                        ms_merge(mi, zi, __shfl_xor_sync(FW_FULL, mi, o), __shfl_xor_sync(FW_FULL, zi, o));
                    if (lane == 0) {
                        s_m[ew][i] = mi;
                        s_z[ew][i] = zi;
                    }
                }
                ws_named_barrier();
#pragma unroll
                for (int i = 0; i < WS_N; ++i) {
                    float mi = s_m[0][i], zi = s_z[0][i];
                    for (int e = 1; e < 4; ++e) ms_merge(mi, zi, s_m[e][i], s_z[e][i]);
                    m[i] = mi;
                    z[i] = zi > 0.f ? 1.f / zi : 0.f;
                }
            }
            if (ok) ok = tc::mbar_wait(&accfull[b], (uint32_t)(it >> 1) & 1u, WS_WAIT);
            float v[WS_N];
            if (ok) {
                tc::fence_after_sync();
                tc::ld32(taddr + ((uint32_t)(q4 * 32) << 16) + (uint32_t)(b * 32), v);
                tc::fence_before_sync();
            }
            __syncwarp();
            if (ok && lane == 0) tc::mbar_arrive(&accempty[b]);
            if (!ok) continue;
            const int j = t * WS_KT + q4 * 32 + lane;
            const int lim = T - w;  // query i sees keys j <= lim + i
            // a tile whose keys every query sees (all but the cell's last) skips the masks
            const bool open = t * WS_KT + WS_KT - 1 <= lim && w == WS_N;
            if (pass == 0) {
                // running (max, sum) with one exponential per element: when x
                // raises the max the old sum is scaled by 2^(m - x), else
                // 2^(x - m) is added
#pragma unroll
                for (int i = 0; i < WS_N; ++i) {
                    if (open || (j < T && i < w && j <= lim + i)) {
                        const float x = v[i] * scale2;
                        const float dx = x - m[i];
                        const float e = ex2a(-fabsf(dx));
                        z[i] = dx > 0.f ? fmaf(z[i], e, 1.f) : z[i] + e;
                        m[i] = fmaxf(m[i], x);
                    }
                }
            } else if (j < T) {
                float vote = 0.f;
#pragma unroll
                for (int i = 0; i < WS_N; ++i)
                    if (open || (i < w && j <= lim + i)) vote = fmaf(ex2a(fmaf(v[i], scale2, -m[i])), z[i], vote);
                a.votes[(int64_t)c * T + j] = vote;
            }
        }
        if (!ok) atomicOr(&s_err, 1);
        // max pooling along the prefix positions (the cell's votes are in global
        // memory, written by these four warps)
        __threadfence_block();
        ws_named_barrier();
        const float *vc = a.votes + (int64_t)c * T;
        const int lim = T - w;
        for (int j = ew * 32 + lane; j < T; j += 128) {
            float r = vc[j];
            if (j < lim) {
                const int lo = j - a.ph < 0 ? 0 : j - a.ph, hi = j + a.ph < lim ? j + a.ph : lim - 1;
                for (int q = lo; q <= hi; ++q) r = fmaxf(r, vc[q]);
            }
            a.scores[(int64_t)c * T + j] = r;
        }
    }
    tc::fence_before_sync();
    __syncthreads();
    if (tid == 0 && a.status) a.status[c] = s_err ? FW_ERR_TIMEOUT : FW_OK;
    if (wid == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(taddr, 64);
    }
}

}  // namespace

size_t window_score_workspace(int cells, int T) { return align256((size_t)cells * T * 4); }

fw_status window_score(const void *Qw, const void *K, int cells, int T, int d, int w, float scale, int pool,
                       float *scores, void *ws, int32_t *status, cudaStream_t s)
{
    CUtensorMap mk, mq;
    if (!make_tma_2d_bf16(&mk, K, (uint64_t)cells * T, (uint64_t)d, WS_KT)) return FW_ERR_CUDA;
    if (!make_tma_2d_bf16(&mq, Qw, (uint64_t)cells * w, (uint64_t)d, WS_N)) return FW_ERR_CUDA;
    WsArgs a;
    a.cells = cells;
    a.T = T;
    a.w = w;
    a.ph = pool / 2;
    a.scale2 = scale * 1.4426950408889634f;
    a.votes = (float *)ws;
    a.scores = scores;
    a.status = status;
    auto launch = [&](auto kernel, int nbox) -> fw_status {
        const size_t smem = 1024 + (size_t)WS_STAGES * nbox * WS_KT * 128 + (size_t)nbox * WS_N * 128;
        FW_CUDA_CHECK(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        FW_LAUNCH(kernel, (unsigned)cells, WS_THREADS, smem, s, mk, mq, a);
        return FW_OK;
    };
    return d == 128 ? launch(k_wscore<128>, 2) : launch(k_wscore<64>, 1);
}

}  // namespace fw
