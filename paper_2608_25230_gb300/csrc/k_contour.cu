// k_contour.cu -- ContourKV allocation and ragged per-head storage (Sec. 4).
//
// One importance score per (cell, position); one global threshold tau shared
// by every cell; each cell keeps its recency floor (last min(floor, T)
// positions) plus its non-floor positions ranked among the best
// K = budget - cells*floor non-floor entries of the whole cache.  The order is
// (score desc, cell asc, position asc), so ties at tau are split exactly.
//
// tau is found by a global radix select (4 passes x 8 bits).  Every pass is a
// histogram launch over all cells followed by a one-block scan launch: no
// kernel ever waits on another block.  Then per-cell counts, an exclusive
// prefix sum into ragged offsets, and per-cell ordered compaction of the kept
// positions.  The compaction copy moves 16-byte vectors, a row per 16 lanes.
#include <algorithm>
#include <mutex>

#include "fw_internal.h"

namespace fw {
namespace {

constexpr int CT = 256;  // threads per block

struct CState {
    uint32_t prefix;   // bits of tau's key fixed so far
    uint32_t rem;      // rank still to find inside the current prefix
    uint32_t K_lo;     // K (low 32 bits; K < 2^32 checked on the host)
    uint32_t pad;
};

struct CArgs {
    const float *scores;
    int cells, T, F;
    int64_t K;
    uint32_t *hist;      // [256]
    CState *st;          // [1]
    int32_t *gt;         // [cells] non-floor keys above tau
    int32_t *eq;         // [cells] non-floor keys equal to tau
    int32_t *take;       // [cells] ties taken
    int32_t *counts;
    int64_t *offsets;
    int32_t *kept_pos;
    float *tau;
    float *dropped_uniform, *dropped_alloc;
    int uniform_s;
};

__global__ void k_c_init(CArgs a)
{
    if (threadIdx.x == 0) {
        a.st->prefix = 0u;
        a.st->rem = (uint32_t)a.K;
        a.st->K_lo = (uint32_t)a.K;
    }
    for (int i = threadIdx.x; i < 256; i += blockDim.x) a.hist[i] = 0u;
}

// histogram of digit `pass` among non-floor keys matching the prefix
__global__ void __launch_bounds__(CT) k_c_hist(CArgs a, int pass)
{
    __shared__ uint32_t h[256];
    for (int i = threadIdx.x; i < 256; i += CT) h[i] = 0u;
    __syncthreads();
    const int shift = 24 - 8 * pass;
    const uint32_t pmask = pass == 0 ? 0u : (0xffffffffu << (32 - 8 * pass));
    const uint32_t prefix = a.st->prefix;
    const int64_t per_cell = a.T - a.F;
    const int64_t total = (int64_t)a.cells * per_cell;
    for (int64_t e = (int64_t)blockIdx.x * CT + threadIdx.x; e < total; e += (int64_t)gridDim.x * CT) {
        const int64_t c = e / per_cell, j = e - c * per_cell;
        const uint32_t key = order_key(__ldg(a.scores + c * a.T + j));
        if ((key & pmask) == prefix) atomicAdd(&h[(key >> shift) & 255u], 1u);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < 256; i += CT)
        if (h[i]) atomicAdd(&a.hist[i], h[i]);
}

__global__ void k_c_scan(CArgs a, int pass)
{
    // one thread: walk bins from the top
    if (threadIdx.x == 0) {
        const int shift = 24 - 8 * pass;
        uint32_t cum = 0, rem = a.st->rem;
        for (int v = 255; v >= 0; --v) {
            const uint32_t c = a.hist[v];
            if (cum + c >= rem) {
                a.st->prefix |= (uint32_t)v << shift;
                a.st->rem = rem - cum;
                break;
            }
            cum += c;
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < 256; i += blockDim.x) a.hist[i] = 0u;
}

// per cell: keys above / equal to tau among the non-floor positions
__global__ void __launch_bounds__(CT) k_c_count(CArgs a)
{
    __shared__ int s_gt, s_eq;
    const int c = blockIdx.x;
    if (threadIdx.x == 0) s_gt = s_eq = 0;
    __syncthreads();
    const uint32_t tk = a.st->prefix;
    int gt = 0, eq = 0;
    if (a.K > 0) {
        for (int j = threadIdx.x; j < a.T - a.F; j += CT) {
            const uint32_t key = order_key(__ldg(a.scores + (int64_t)c * a.T + j));
            gt += key > tk;
            eq += key == tk;
        }
    }
    for (int o = 16; o > 0; o >>= 1) {
        gt += __shfl_xor_sync(FW_FULL, gt, o);
        eq += __shfl_xor_sync(FW_FULL, eq, o);
    }
    if ((threadIdx.x & 31) == 0) {
        atomicAdd(&s_gt, gt);
        atomicAdd(&s_eq, eq);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        a.gt[c] = s_gt;
        a.eq[c] = s_eq;
    }
}

// one block: ties taken per cell (in cell order), counts, offsets, tau
__global__ void __launch_bounds__(1024) k_c_offsets(CArgs a)
{
    __shared__ int64_t part[1024];
    __shared__ int64_t part2[1024];
    const int tid = threadIdx.x;
    const int nt = blockDim.x;
    const int per = (a.cells + nt - 1) / nt;
    const int c0 = tid * per, c1 = min(a.cells, c0 + per);
    // ties: exclusive prefix of eq over cells
    int64_t se = 0, sc = 0;
    for (int c = c0; c < c1; ++c) se += a.eq[c];
    part[tid] = se;
    __syncthreads();
    for (int o = 1; o < nt; o <<= 1) {
        const int64_t v = tid >= o ? part[tid - o] : 0;
        __syncthreads();
        part[tid] += v;
        __syncthreads();
    }
    int64_t ebefore = part[tid] - se;
    int64_t gt_total = 0;
    // total above tau
    {
        int64_t sg = 0;
        for (int c = c0; c < c1; ++c) sg += a.gt[c];
        part2[tid] = sg;
        __syncthreads();
        for (int o = nt / 2; o > 0; o >>= 1) {
            if (tid < o) part2[tid] += part2[tid + o];
            __syncthreads();
        }
        gt_total = part2[0];
        __syncthreads();
    }
    const int64_t ties_taken = a.K > 0 ? a.K - gt_total : 0;
    for (int c = c0; c < c1; ++c) {
        int64_t t = ties_taken - ebefore;
        t = t < 0 ? 0 : (t > a.eq[c] ? a.eq[c] : t);
        a.take[c] = (int32_t)t;
        ebefore += a.eq[c];
        const int cnt = a.F + (a.K > 0 ? a.gt[c] : 0) + (int)t;
        a.counts[c] = cnt;
        sc += cnt;
    }
    part[tid] = sc;
    __syncthreads();
    for (int o = 1; o < nt; o <<= 1) {
        const int64_t v = tid >= o ? part[tid - o] : 0;
        __syncthreads();
        part[tid] += v;
        __syncthreads();
    }
    int64_t off = part[tid] - sc;
    for (int c = c0; c < c1; ++c) {
        a.offsets[c] = off;
        off += a.counts[c];
    }
    if (tid == nt - 1) a.offsets[a.cells] = part[tid];
    if (tid == 0) {
        const uint32_t tk = a.st->prefix;
        const uint32_t u = (tk & 0x80000000u) ? (tk & 0x7fffffffu) : ~tk;
        *a.tau = a.K > 0 ? __uint_as_float(u) : INFINITY;
    }
}

// per cell: ordered compaction of kept positions + dropped mass of the allocation
__global__ void __launch_bounds__(CT) k_c_emit(CArgs a)
{
    __shared__ int wc[CT / 32], wt[CT / 32];
    __shared__ double red[CT / 32], red2[CT / 32];
    const int c = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const uint32_t tk = a.st->prefix;
    const int take = a.take[c];
    const int64_t base = a.offsets[c];
    const float *s = a.scores + (int64_t)c * a.T;
    int written = 0, ties_seen = 0;
    double tot = 0.0, drop = 0.0;
    for (int j0 = 0; j0 < a.T; j0 += CT) {
        const int j = j0 + tid;
        bool kept = false, tie = false;
        float x = 0.f;
        if (j < a.T) {
            x = __ldg(s + j);
            if (j >= a.T - a.F) {
                kept = true;
            } else if (a.K > 0) {
                const uint32_t key = order_key(x);
                kept = key > tk;
                tie = key == tk;
            }
        }
        // rank of this tie among the cell's ties, in position order
        const uint32_t tb = __ballot_sync(FW_FULL, tie);
        if (lane == 0) wt[wid] = __popc(tb);
        __syncthreads();
        int tbefore = 0, ttotal = 0;
        for (int w = 0; w < CT / 32; ++w) {
            if (w < wid) tbefore += wt[w];
            ttotal += wt[w];
        }
        if (tie) kept = (ties_seen + tbefore + __popc(tb & ((1u << lane) - 1u))) < take;
        ties_seen += ttotal;
        const uint32_t kb = __ballot_sync(FW_FULL, kept);
        if (lane == 0) wc[wid] = __popc(kb);
        __syncthreads();
        int before = 0, total = 0;
        for (int w = 0; w < CT / 32; ++w) {
            if (w < wid) before += wc[w];
            total += wc[w];
        }
        if (kept) a.kept_pos[base + written + before + __popc(kb & ((1u << lane) - 1u))] = j;
        written += total;
        if (j < a.T) {
            tot += (double)x;
            if (!kept) drop += (double)x;
        }
        __syncthreads();
    }
    tot = warp_sum_d(tot);
    drop = warp_sum_d(drop);
    if (lane == 0) {
        red[wid] = tot;
        red2[wid] = drop;
    }
    __syncthreads();
    if (tid == 0 && a.dropped_alloc) {
        double t = 0.0, dd = 0.0;
        for (int w = 0; w < CT / 32; ++w) {
            t += red[w];
            dd += red2[w];
        }
        a.dropped_alloc[c] = t > 0.0 ? (float)(dd / t) : 0.f;
    }
}

// per cell: dropped mass outside the cell's own top-s set (ties -> lower position)
__global__ void __launch_bounds__(CT) k_c_uniform(CArgs a)
{
    __shared__ uint32_t hist[256];
    __shared__ uint32_t s_prefix, s_rem;
    __shared__ uint32_t wcnt[CT / 32];
    __shared__ int s_found;
    __shared__ double red[CT / 32], red2[CT / 32];
    const int c = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int T = a.T;
    const float *s = a.scores + (int64_t)c * T;
    const int su = a.uniform_s < T ? a.uniform_s : T;
    uint32_t tk = 0u;
    int ti = -1;
    if (su > 0) {
        if (tid == 0) {
            s_prefix = 0u;
            s_rem = (uint32_t)su;
        }
        uint32_t pmask = 0u;
        for (int pass = 0; pass < 4; ++pass) {
            const int shift = 24 - 8 * pass;
            for (int i = tid; i < 256; i += CT) hist[i] = 0u;
            __syncthreads();
            const uint32_t pre = s_prefix;
            for (int j = tid; j < T; j += CT) {
                const uint32_t key = order_key(__ldg(s + j));
                if ((key & pmask) == pre) atomicAdd(&hist[(key >> shift) & 255u], 1u);
            }
            __syncthreads();
            if (tid == 0) {
                uint32_t cum = 0, rem = s_rem;
                for (int v = 255; v >= 0; --v) {
                    const uint32_t cc = hist[v];
                    if (cum + cc >= rem) {
                        s_prefix |= (uint32_t)v << shift;
                        s_rem = rem - cum;
                        break;
                    }
                    cum += cc;
                }
            }
            pmask |= 255u << shift;
            __syncthreads();
        }
        tk = s_prefix;
        const uint32_t want = s_rem;
        if (tid == 0) s_found = -1;
        __syncthreads();
        uint32_t base = 0;
        for (int j0 = 0; j0 < T; j0 += CT) {
            const int j = j0 + tid;
            const bool match = j < T && order_key(__ldg(s + j)) == tk;
            const uint32_t bal = __ballot_sync(FW_FULL, match);
            if (lane == 0) wcnt[wid] = __popc(bal);
            __syncthreads();
            uint32_t before = 0, total = 0;
            for (int w = 0; w < CT / 32; ++w) {
                if (w < wid) before += wcnt[w];
                total += wcnt[w];
            }
            if (match && base + before + __popc(bal & ((1u << lane) - 1u)) + 1u == want) s_found = j;
            __syncthreads();
            base += total;
            if (base >= want) break;
        }
        __syncthreads();
        ti = s_found;
    }
    double tot = 0.0, drop = 0.0;
    for (int j = tid; j < T; j += CT) {
        const float x = __ldg(s + j);
        const uint32_t key = order_key(x);
        const bool kept = su > 0 && (key > tk || (key == tk && j <= ti));
        tot += (double)x;
        if (!kept) drop += (double)x;
    }
    tot = warp_sum_d(tot);
    drop = warp_sum_d(drop);
    if (lane == 0) {
        red[wid] = tot;
        red2[wid] = drop;
    }
    __syncthreads();
    if (tid == 0) {
        double t = 0.0, dd = 0.0;
        for (int w = 0; w < CT / 32; ++w) {
            t += red[w];
            dd += red2[w];
        }
        a.dropped_uniform[c] = t > 0.0 ? (float)(dd / t) : 0.f;
    }
}

// ragged compaction: block (cell, chunk) copies rows [offsets[c] + chunk*RPB, ...)
constexpr int RPB = 256;  // rows per block
__global__ void __launch_bounds__(256) k_compact(const uint4 *K, const uint4 *V, int T, int vec_per_row,
                                                 const int64_t *offsets, const int32_t *kept_pos, uint4 *Ko,
                                                 uint4 *Vo, int chunks)
{
    const int c = blockIdx.x / chunks;
    const int chunk = blockIdx.x - c * chunks;
    const int64_t beg = offsets[c] + (int64_t)chunk * RPB;
    const int64_t end = min(offsets[c + 1], beg + RPB);
    if (beg >= end) return;
    const int64_t nvec = (end - beg) * vec_per_row;
    for (int64_t e = threadIdx.x; e < nvec; e += blockDim.x) {
        const int64_t q = beg + e / vec_per_row;
        const int part = (int)(e % vec_per_row);
        const int64_t src = ((int64_t)c * T + kept_pos[q]) * vec_per_row + part;
        const int64_t dst = q * vec_per_row + part;
        Ko[dst] = __ldg(K + src);
        Vo[dst] = __ldg(V + src);
    }
}

}  // namespace

size_t contour_workspace(int cells, int T)
{
    (void)T;
    return align256(256 * 4) + align256(sizeof(CState)) + 3 * align256((size_t)cells * 4);
}

fw_status contour_alloc(const float *scores, int cells, int T, int floor_, int64_t total_budget, int uniform_s,
                        int32_t *counts, int64_t *offsets, int32_t *kept_pos, float *tau, float *dropped_uniform,
                        float *dropped_alloc, void *ws, size_t ws_bytes, cudaStream_t s)
{
    (void)ws_bytes;
    CArgs a;
    a.scores = scores;
    a.cells = cells;
    a.T = T;
    a.F = floor_ < T ? floor_ : T;
    a.K = total_budget - (int64_t)cells * a.F;
    if (a.K >= ((int64_t)1 << 32)) return FW_ERR_UNSUPPORTED;
    char *w = (char *)ws;
    a.hist = (uint32_t *)w;
    w += align256(256 * 4);
    a.st = (CState *)w;
    w += align256(sizeof(CState));
    a.gt = (int32_t *)w;
    w += align256((size_t)cells * 4);
    a.eq = (int32_t *)w;
    w += align256((size_t)cells * 4);
    a.take = (int32_t *)w;
    a.counts = counts;
    a.offsets = offsets;
    a.kept_pos = kept_pos;
    a.tau = tau;
    a.dropped_uniform = dropped_uniform;
    a.dropped_alloc = dropped_alloc;
    a.uniform_s = uniform_s;
    FW_LAUNCH(k_c_init, 1, 256, 0, s, a);
    if (a.K > 0) {
        const int64_t keys = (int64_t)cells * (T - a.F);
        const unsigned hb = (unsigned)std::max<int64_t>(1, std::min<int64_t>(152 * 8, (keys + CT - 1) / CT));
        for (int pass = 0; pass < 4; ++pass) {
            FW_LAUNCH(k_c_hist, hb, CT, 0, s, a, pass);
            FW_LAUNCH(k_c_scan, 1, 256, 0, s, a, pass);
        }
    }
    FW_LAUNCH(k_c_count, (unsigned)cells, CT, 0, s, a);
    FW_LAUNCH(k_c_offsets, 1, 1024, 0, s, a);
    FW_LAUNCH(k_c_emit, (unsigned)cells, CT, 0, s, a);
    if (dropped_uniform) FW_LAUNCH(k_c_uniform, (unsigned)cells, CT, 0, s, a);
    return FW_OK;
}

fw_status ragged_compact(const void *K, const void *V, int cells, int T, int row_bytes, const int64_t *offsets,
                         const int32_t *kept_pos, int64_t total, void *K_out, void *V_out, cudaStream_t s)
{
    if (total == 0) return FW_OK;
    const int vec = row_bytes / 16;
    const int chunks = (T + RPB - 1) / RPB;
    const int64_t grid = (int64_t)cells * chunks;
    if (grid >= ((int64_t)1 << 31)) return FW_ERR_UNSUPPORTED;
    FW_LAUNCH(k_compact, (unsigned)grid, 256, 0, s, (const uint4 *)K, (const uint4 *)V, T, vec, offsets, kept_pos,
              (uint4 *)K_out, (uint4 *)V_out, chunks);
    return FW_OK;
}

}  // namespace fw

// ------------------------------------------------------------------------
// Allocation-free variant: the scratch lives in a fixed device array.
namespace fw {
namespace {

constexpr size_t kNoallocBytes = 256 * 4 + 256 + 3 * (size_t)FW_CONTOUR_NOALLOC_MAX_CELLS * 4;  // >= contour_workspace
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocBytes + 3 * 256];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
void *g_noalloc_ptr[kMaxDevices] = {};

// Device address of the scratch array for the current device (looked up once per device).
fw_status noalloc_scratch(void **ptr)
{
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return FW_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return FW_ERR_CUDA;
        g_noalloc_ptr[dev] = p;
    }
    *ptr = g_noalloc_ptr[dev];
    return FW_OK;
}

}  // namespace
}  // namespace fw

extern "C" fw_status fw_contour_alloc_noalloc(const float *scores, int32_t cells, int32_t T, int32_t floor_,
                                              int64_t total_budget, int32_t uniform_s, int32_t *counts,
                                              int64_t *offsets, int32_t *kept_pos, float *tau,
                                              float *dropped_uniform, float *dropped_alloc, void *stream)
{
    if (cells > FW_CONTOUR_NOALLOC_MAX_CELLS) return FW_ERR_WORKSPACE;
    if (cells >= 1 && T >= 1 && fw::contour_workspace(cells, T) > sizeof(fw::g_noalloc_scratch))
        return FW_ERR_WORKSPACE;
    void *ws = nullptr;
    if (cells >= 1 && T >= 1) {
        const fw_status st = fw::noalloc_scratch(&ws);
        if (st != FW_OK) return st;
    }
    return fw_contour_alloc(scores, cells, T, floor_, total_budget, uniform_s, counts, offsets, kept_pos, tau,
                            dropped_uniform, dropped_alloc, ws, sizeof(fw::g_noalloc_scratch), stream);
}
