// k_contour.cu -- ContourKV allocation and ragged per-head storage (Sec. 4).
//
// One importance score per (cell, position); one global threshold tau shared
// by every cell; each cell keeps its recency floor (last min(floor, T)
// positions) plus its non-floor positions ranked among the best
// K = budget - cells*floor non-floor entries of the whole cache.  The order is
// (score desc, cell asc, position asc), so ties at tau are split exactly.
//
// Every kernel of the allocation splits a cell into S slices of consecutive
// positions, a block each (up to 8, so that a few hundred cells still spread
// over every SM), and the kernels are specialised on what the call asks for
// (tau, the uniform-budget set, the cap), which keeps the per-score work to a
// few instructions.
//   - tau is found by a global radix select (4 passes x 8 bits).  A pass
//     launches the slices of a cell as one thread-block cluster: each block
//     builds its slice's histograms in shared memory, the cluster's first
//     block sums them through distributed shared memory and adds the sum to
//     the pass's global histogram, then takes a ticket; the cluster with the
//     last ticket scans the completed histogram and records the radix state
//     (digits fixed so far, rank left) that every block of the next launch
//     reads.  Nothing ever waits on another block.  The same passes carry each
//     cell's own top-uniform_s select (the uniform-budget dropped mass): its
//     histogram is the cell's alone, so the cluster's first block fixes its
//     digit at the end of the pass.
//   - A count kernel, clustered the same way, records per slice the non-floor
//     keys above and equal to the deciding thresholds, and per cell those
//     counts and the sums of the scores below each threshold; the cluster with
//     the last ticket then turns them into the ties each cell takes, the
//     counts, the ragged offsets and both dropped masses (the dropped set is
//     "below the threshold" plus the ties not taken, every tie worth the
//     threshold's own score).
//   - An emit kernel writes each slice's kept positions in order, starting
//     from the kept entries and ties of the cell's earlier slices.
// The compaction copy moves 16-byte vectors, a row per 16 lanes.
//
// The capped variant (the enforcement of Sec. 4: no cell keeps more than a
// cap, e.g. a uniform method's per-head count) truncates each cell to its
// floor plus its best cap - floor non-floor entries of the allocation; the
// passes carry a third, per-cell select of the (cap - floor)-th non-floor key.
// The global threshold and the cap's threshold both keep a prefix of the
// cell's order (score desc, position asc), so the kept set is the shorter of
// the two prefixes: each cell is decided by one key, tau's or the cap's.
#include <algorithm>

#include "fw_internal.h"

namespace fw {
namespace {

constexpr int CT = 128;             // threads of a pass, count or emit block
constexpr int PER = 32;             // scores per thread of a 4,096-position slice
constexpr int SMAX = 8;             // slices per cell at most (a portable cluster)
constexpr int SLICE_MIN = 4096;     // positions per slice at least, where the cell has that many
constexpr int SLOT_TARGET = 2048;   // slices over all cells that the split aims for

struct CState {
    uint32_t prefix;   // bits of tau's key fixed so far
    uint32_t rem;      // rank still to find inside the current prefix
    uint32_t ticket[5];  // clusters done with each pass and with the count
    uint32_t pad;
};

// One slice of a cell: its non-floor keys against the deciding thresholds.
struct Slot {
    int32_t gt, eq;    // above / equal to tau's key (both 0 when K = 0)
    int32_t cgt, ceq;  // above / equal to the cell's cap key (both 0 without a cap select)
};

// One cell: its slices' counts and sums.
struct CellRec {
    int32_t gt, eq, ceq, ueq;  // as Slot; ueq: keys equal to the uniform-budget key (0 without a uniform set)
    double tot;                // the cell's scores summed
    double lt;                 // non-floor scores below tau's key (every non-floor score when K = 0)
    double clt;                // non-floor scores below the cap key (every one when the cap keeps none)
    double ult;                // scores below the uniform-budget key (every one without a uniform set)
};

struct CArgs {
    const float *scores;
    int cells, T, F;
    int S, L;            // slices per cell, positions per slice (the last one may be shorter)
    int64_t K;
    uint32_t *hist;      // [4][256] global histograms of the four passes
    CState *st;          // [1]
    Slot *slot;          // [cells][S]
    CellRec *rec;        // [cells]
    int32_t *take;       // [cells] ties of the cell's deciding key that it keeps
    int32_t *emode;      // [cells] 0: tau decides, 1: the cap decides, 2: no non-floor entry is kept
    int32_t *counts;
    int64_t *offsets;
    int32_t *kept_pos;
    float *tau;
    float *dropped_uniform, *dropped_alloc;
    int uniform_s;
    uint32_t *uprefix;   // [cells] bits of the cell's uniform-budget threshold fixed so far
    uint32_t *urem;      // [cells] rank still to find inside that prefix (0: no uniform set)
    int capnf;           // cap - floor on non-floor entries per cell; < 0: no cap
    uint32_t *cprefix;   // [cells] bits of the cell's cap threshold (non-floor keys) fixed so far
    uint32_t *crem;      // [cells] rank still to find inside that prefix (0: the cap truncates nothing)
};

// Slices per cell: up to SMAX, none shorter than SLICE_MIN positions, and at
// most SLOT_TARGET slices over all cells (one per cell beyond that many cells).
int n_slices(int cells, int T)
{
    int s = (int)std::min<int64_t>(SMAX, ((int64_t)T + SLICE_MIN - 1) / SLICE_MIN);
    s = std::min(s, std::max(1, SLOT_TARGET / std::max(cells, 1)));
    return std::max(s, 1);
}
// Positions per slice: T / S rounded up to a multiple of 4 (16-byte vectors).
int slice_len(int T, int S) { return (int)((((int64_t)T + S - 1) / S + 3) & ~(int64_t)3); }

__device__ __forceinline__ void slice_bounds(const CArgs &a, int r, int &lo, int &hi)
{
    lo = (int)min((int64_t)a.T, (int64_t)r * a.L);
    hi = (int)min((int64_t)a.T, (int64_t)lo + a.L);
}

// The cap keeps every non-floor entry (no select needed), none, or a prefix.
__host__ __device__ __forceinline__ bool cap_selects(const CArgs &a)
{
    return a.cprefix && a.capnf > 0 && a.capnf < a.T - a.F;
}
// 0: no cap, 1: the cap keeps no non-floor entry, 2: the cap's threshold decides
__host__ __device__ __forceinline__ int cap_mode(const CArgs &a)
{
    return a.capnf < 0 || a.capnf >= a.T - a.F ? 0 : (a.capnf == 0 ? 1 : 2);
}

// The order key of a score x >= 0 (or -0, which gets +0's key): its bits with
// the sign bit set, increasing with x.  Scores are finite and >= 0 by the
// contract of the entry points, so this is order_key on every valid input.
__device__ __forceinline__ uint32_t score_key(float x) { return __float_as_uint(x) | 0x80000000u; }

// The score whose order key is k (the inverse of order_key on scores >= 0).
__device__ __forceinline__ float key_score(uint32_t k)
{
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// Every thread of every block of the cluster arrives, then waits for all;
// shared-memory writes before it are visible to the cluster after it.
__device__ __forceinline__ void cluster_barrier()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// The address of p's counterpart in the shared memory of the cluster's block `rank`.
__device__ __forceinline__ uint32_t cluster_addr(const void *p, uint32_t rank)
{
    const uint32_t local = (uint32_t)__cvta_generic_to_shared(p);
    uint32_t remote;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(rank));
    return remote;
}
// Loads of another block's shared memory; the cluster barriers around them
// order them against its writes, so they carry no memory clobber and several
// can be in flight at once.
__device__ __forceinline__ uint32_t ld_cluster_u32(const void *p, uint32_t rank)
{
    uint32_t v;
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(cluster_addr(p, rank)));
    return v;
}
__device__ __forceinline__ double ld_cluster_f64(const void *p, uint32_t rank)
{
    double v;
    asm volatile("ld.shared::cluster.f64 %0, [%1];" : "=d"(v) : "r"(cluster_addr(p, rank)));
    return v;
}

// Programmatic dependent launch: a kernel of the chain lets the next one be
// scheduled at once (its blocks then wait in grid_wait until this grid has
// finished and its writes are visible), so launches overlap the tails.
__device__ __forceinline__ void grid_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_release() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

__global__ void k_c_init(CArgs a)
{
    grid_release();
    grid_wait();
    if (threadIdx.x == 0) {
        a.st->prefix = 0u;
        a.st->rem = (uint32_t)a.K;
        for (int i = 0; i < 5; ++i) a.st->ticket[i] = 0u;
    }
    for (int i = threadIdx.x; i < 4 * 256; i += blockDim.x) a.hist[i] = 0u;
    const uint32_t su = a.dropped_uniform ? (uint32_t)max(min(a.uniform_s, a.T), 0) : 0u;
    for (int c = threadIdx.x; c < a.cells; c += blockDim.x) {
        a.uprefix[c] = 0u;
        a.urem[c] = su;
        if (a.cprefix) {
            a.cprefix[c] = 0u;
            a.crem[c] = cap_selects(a) ? (uint32_t)a.capnf : 0u;
        }
    }
}

// Given lane l's counts c[i] of bins 255 - 8l - i (i < 8) of a 256-bin
// histogram: the bin where the count from the top bin down first reaches rem,
// and the rank left inside that bin (bin 0 and rank 0 when rem is 0 or above
// the total).  One warp.
__device__ __forceinline__ void warp_pick(const uint32_t (&c)[8], uint32_t rem, uint32_t &bin, uint32_t &nrem)
{
    const int lane = threadIdx.x & 31;
    uint32_t loc = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) loc += c[i];
    uint32_t inc = loc;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(FW_FULL, inc, o);
        if (lane >= o) inc += y;
    }
    const uint32_t exc = inc - loc;
    const bool mine = exc < rem && rem <= inc;
    uint32_t v = 0u, nr = 0u;
    if (mine) {
        uint32_t cum = exc;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            if (v == 0u && cum + c[i] >= rem) {
                v = 256u + 255u - 8u * lane - i;  // (+256: found)
                nr = rem - cum;
            }
            cum += c[i];
        }
    }
    const int src = __ffs(__ballot_sync(FW_FULL, mine)) - 1;
    bin = __shfl_sync(FW_FULL, v, src < 0 ? 0 : src) & 255u;
    nrem = __shfl_sync(FW_FULL, nr, src < 0 ? 0 : src);
}

// Calls f(j, score) for the positions j of [lo, hi) of a cell's scores sc,
// a block's NT threads striding over them with LD 16-byte loads each in
// flight before any is used (vectors when T % 4 == 0, the row is 16-byte
// aligned and lo, hi are multiples of 4).
template <int NT, int LD, typename F>
__device__ __forceinline__ void for_range(const float *sc, int T, int lo, int hi, F &&f)
{
    if ((T & 3) == 0 && (reinterpret_cast<uintptr_t>(sc) & 15) == 0 && ((lo | hi) & 3) == 0) {
        const float4 *v4 = reinterpret_cast<const float4 *>(sc + lo);
        const int nq = (hi - lo) / 4;
        for (int q0 = threadIdx.x; q0 < nq; q0 += LD * NT) {
            float4 v[LD];
#pragma unroll
            for (int u = 0; u < LD; ++u) {
                const int q = q0 + u * NT;
                v[u] = q < nq ? __ldg(v4 + q) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int u = 0; u < LD; ++u) {
                const int q = q0 + u * NT;
                if (q < nq) {
                    const int j = lo + 4 * q;
                    f(j, v[u].x);
                    f(j + 1, v[u].y);
                    f(j + 2, v[u].z);
                    f(j + 3, v[u].w);
                }
            }
        }
    } else {
        for (int j = lo + (int)threadIdx.x; j < hi; j += NT) f(j, __ldg(sc + j));
    }
}

// The slice [lo, hi) as its non-floor part (positions before nf, cut at a
// multiple of 4) with no per-position floor test, then the rest with one.
template <typename FN, typename FC>
__device__ __forceinline__ void for_slice(const float *sc, int T, int lo, int hi, int nf, FN &&f_nonfloor,
                                          FC &&f_checked)
{
    const int m = max(lo, min(hi, nf) & ~3);
    for_range<CT, PER / 4>(sc, T, lo, m, f_nonfloor);
    if (m < hi) for_range<CT, 1>(sc, T, m, hi, f_checked);
}

// One radix pass, a cluster of S blocks per cell, a block per slice.  The
// slice's non-floor keys matching tau's prefix go to the global histogram of
// digit `pass`; its keys matching the cell's uniform prefix (all positions)
// and its non-floor keys matching the cap prefix go to the cell's own
// histograms, which the cluster's first block sums and scans at once.
template <bool GLOB, bool UNI, bool CAP>
__global__ void __launch_bounds__(CT) k_c_pass(CArgs a, int pass)
{
    __shared__ uint32_t hg[GLOB ? 256 : 1], hu[UNI ? 256 : 1], hc[CAP ? 256 : 1];
    __shared__ uint32_t s_last;
    grid_release();
    for (int i = threadIdx.x; i < 256; i += CT) {
        if (GLOB) hg[i] = 0u;
        if (UNI) hu[i] = 0u;
        if (CAP) hc[i] = 0u;
    }
    grid_wait();
    __syncthreads();
    const int c = blockIdx.x / a.S, r = blockIdx.x - c * a.S;  // r: the block's rank in its cluster
    int lo, hi;
    slice_bounds(a, r, lo, hi);
    const int shift = 24 - 8 * pass;
    const uint32_t pmask = pass == 0 ? 0u : (0xffffffffu << (32 - 8 * pass));
    const uint32_t prefix = GLOB ? a.st->prefix : 0u;  // tau's digits from the earlier passes
    const uint32_t upre = UNI ? a.uprefix[c] : 0u;
    const uint32_t cpre = CAP ? a.cprefix[c] : 0u;
    const int nf = a.T - a.F;
    auto nonfloor = [&](int, float x) {
        const uint32_t key = score_key(x);
        const uint32_t dg = (key >> shift) & 255u;
        const uint32_t km = key & pmask;
        if (GLOB && km == prefix) atomicAdd(&hg[dg], 1u);
        if (UNI && km == upre) atomicAdd(&hu[dg], 1u);
        if (CAP && km == cpre) atomicAdd(&hc[dg], 1u);
    };
    auto checked = [&](int j, float x) {
        const uint32_t key = score_key(x);
        const uint32_t dg = (key >> shift) & 255u;
        const uint32_t km = key & pmask;
        if (GLOB && j < nf && km == prefix) atomicAdd(&hg[dg], 1u);
        if (UNI && km == upre) atomicAdd(&hu[dg], 1u);
        if (CAP && j < nf && km == cpre) atomicAdd(&hc[dg], 1u);
    };
    for_slice(a.scores + (int64_t)c * a.T, a.T, lo, hi, nf, nonfloor, checked);
    cluster_barrier();  // every slice's histograms are complete
    if (r == 0) {
        for (int i = threadIdx.x; i < 256; i += CT) {
            uint32_t vg[SMAX], vu[SMAX], vk[SMAX];  // every rank's bin i, loaded before any is summed
#pragma unroll
            for (int q = 0; q < SMAX; ++q) {
                vg[q] = vu[q] = vk[q] = 0u;
                if (q < a.S) {
                    if (GLOB) vg[q] = ld_cluster_u32(&hg[i], (uint32_t)q);
                    if (UNI) vu[q] = ld_cluster_u32(&hu[i], (uint32_t)q);
                    if (CAP) vk[q] = ld_cluster_u32(&hc[i], (uint32_t)q);
                }
            }
            uint32_t g = 0u, u = 0u, k = 0u;
#pragma unroll
            for (int q = 0; q < SMAX; ++q) g += vg[q], u += vu[q], k += vk[q];
            if (GLOB && g) atomicAdd(&a.hist[pass * 256 + i], g);
            if (UNI) hu[i] = u;  // the cell's sums, in the first block's own arrays
            if (CAP) hc[i] = k;
        }
        if (GLOB) {
            __threadfence();  // this block's histogram adds before its ticket
            __syncthreads();
            if (threadIdx.x == 0) s_last = atomicAdd(&a.st->ticket[pass], 1u) == (uint32_t)a.cells - 1u;
        }
    }
    cluster_barrier();  // the first block is done reading the others (and has its sums)
    if (r != 0) return;
    const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint32_t cnt[8], v, nr;
    if (UNI && wid == 0) {
#pragma unroll
        for (int i = 0; i < 8; ++i) cnt[i] = hu[255 - 8 * lane - i];
        warp_pick(cnt, a.urem[c], v, nr);
        if (lane == 0) {
            a.uprefix[c] = upre | (v << shift);
            a.urem[c] = nr;
        }
    }
    if (CAP && wid == 1) {
#pragma unroll
        for (int i = 0; i < 8; ++i) cnt[i] = hc[255 - 8 * lane - i];
        warp_pick(cnt, a.crem[c], v, nr);
        if (lane == 0) {
            a.cprefix[c] = cpre | (v << shift);
            a.crem[c] = nr;
        }
    }
    if (GLOB && wid == 2 && s_last) {  // every cluster's adds are in: tau's digit of this pass
        __threadfence();
#pragma unroll
        for (int i = 0; i < 8; ++i) cnt[i] = __ldcg(&a.hist[pass * 256 + 255 - 8 * lane - i]);
        warp_pick(cnt, a.st->rem, v, nr);
        if (lane == 0) {
            a.st->prefix = prefix | (v << shift);
            a.st->rem = nr;
        }
    }
}

// Exclusive prefix (over the block's threads, in thread order) and total of v.
template <int NW, typename U>
__device__ __forceinline__ void block_scan(U v, U *wsum, int wid, int lane, U &before, U &total)
{
    U inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const U y = __shfl_up_sync(FW_FULL, inc, o);
        if (lane >= o) inc += y;
    }
    if (lane == 31) wsum[wid] = inc;
    __syncthreads();
    U winc = 0, w = 0;
#pragma unroll
    for (int i = 0; i < NW; ++i) {
        const U x = wsum[i];
        if (i < wid) winc += x;
        w += x;
    }
    before = winc + inc - v;
    total = w;
    __syncthreads();  // wsum is rewritten by the next scan
}

// The cells' ties at tau, deciding keys, counts, offsets and dropped masses
// from their records; tau.  Run by one block after every cell's record is in.
__device__ void finish_offsets(const CArgs &a)
{
    constexpr int NW = CT / 32;
    __shared__ long long wsum[NW];
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int per = (a.cells + CT - 1) / CT;
    const int c0 = min(a.cells, tid * per), c1 = min(a.cells, c0 + per);
    long long se = 0, sg = 0;
    for (int c = c0; c < c1; ++c) {
        se += __ldcg(&a.rec[c].eq);
        sg += __ldcg(&a.rec[c].gt);
    }
    long long ebefore, etot, gbef, gt_total;
    block_scan<NW>(se, wsum, wid, lane, ebefore, etot);
    block_scan<NW>(sg, wsum, wid, lane, gbef, gt_total);
    const long long ties_taken = a.K > 0 ? a.K - gt_total : 0;
    const uint32_t tk = a.st->prefix;
    const int cmode = cap_mode(a);
    long long sc = 0;
    for (int c = c0; c < c1; ++c) {
        const CellRec *R = &a.rec[c];
        const int gt = __ldcg(&R->gt), eq = __ldcg(&R->eq), ceq = __ldcg(&R->ceq), ueq = __ldcg(&R->ueq);
        const double tot = __ldcg(&R->tot), lt = __ldcg(&R->lt), clt = __ldcg(&R->clt), ult = __ldcg(&R->ult);
        long long t = ties_taken - ebefore;
        t = t < 0 ? 0 : (t > eq ? eq : t);
        ebefore += eq;
        const int gk = gt + (int)t;  // non-floor entries tau keeps (gt = 0 when K = 0)
        const bool capped = cmode != 0 && gk > a.capnf;
        const int cwant = cmode == 2 ? (int)a.crem[c] : 0;
        const int nonf = capped ? a.capnf : gk;
        a.take[c] = capped ? cwant : (int)t;
        a.emode[c] = nonf == 0 ? 2 : (capped ? 1 : 0);
        const int cnt = a.F + nonf;
        a.counts[c] = cnt;
        sc += cnt;
        if (a.dropped_alloc) {  // below the deciding key, plus its ties not taken
            double d;
            if (capped) {
                const int n = ceq - cwant;
                d = clt + (n > 0 ? (double)n * (double)key_score(a.cprefix[c]) : 0.0);
            } else {
                const int n = eq - (int)t;
                d = lt + (n > 0 ? (double)n * (double)key_score(tk) : 0.0);
            }
            a.dropped_alloc[c] = tot > 0.0 ? (float)(d / tot) : 0.f;
        }
        if (a.dropped_uniform) {
            const int n = ueq - (int)a.urem[c];
            const double d = ult + (n > 0 ? (double)n * (double)key_score(a.uprefix[c]) : 0.0);
            a.dropped_uniform[c] = tot > 0.0 ? (float)(d / tot) : 0.f;
        }
    }
    long long off, total;
    block_scan<NW>(sc, wsum, wid, lane, off, total);
    for (int c = c0; c < c1; ++c) {
        a.offsets[c] = off;
        off += a.counts[c];
    }
    if (tid == 0) {
        a.offsets[a.cells] = total;
        *a.tau = a.K > 0 ? key_score(tk) : INFINITY;
    }
}

// A cluster per cell, a block per slice: the slice's keys against tau's key,
// the cap's and the uniform set's, counted, and the scores below each summed;
// the cluster's first block gathers the cell's record, and the cluster with
// the last ticket finishes the offsets of every cell.
template <bool GLOB, bool UNI, int CMODE>
__global__ void __launch_bounds__(CT) k_c_count(CArgs a)
{
    constexpr int NW = CT / 32;
    __shared__ int32_t si[5][NW];
    __shared__ double sd[4][NW];
    __shared__ int32_t s_i[5];  // the slice's gt, eq, cgt, ceq, ueq
    __shared__ double s_d[4];   // and its tot, lt, clt, ult
    __shared__ uint32_t s_last;
    const int c = blockIdx.x / a.S, r = blockIdx.x - c * a.S;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    grid_release();
    grid_wait();
    const uint32_t tk = a.st->prefix;  // tau's key (K > 0)
    const uint32_t cT = CMODE == 2 ? a.cprefix[c] : 0u;
    const uint32_t uT = a.uprefix[c];
    const int nf = a.T - a.F;
    int lo, hi;
    slice_bounds(a, r, lo, hi);
    // per-thread sums of (hi - lo) / CT scores in fp32, the sums over threads in fp64
    int gt = 0, eq = 0, cgt = 0, ceq = 0, ueq = 0;
    float tot = 0.f, lt = 0.f, clt = 0.f, ult = 0.f;
    auto all = [&](uint32_t key, float x) {
        tot += x;
        if constexpr (UNI) {
            ueq += key == uT;
            ult += key < uT ? x : 0.f;
        } else {
            ult += x;
        }
    };
    auto nonfloor = [&](uint32_t key, float x) {
        if constexpr (GLOB) {
            gt += key > tk;
            eq += key == tk;
            lt += key < tk ? x : 0.f;
        } else {
            lt += x;
        }
        if constexpr (CMODE == 2) {
            cgt += key > cT;
            ceq += key == cT;
            clt += key < cT ? x : 0.f;
        } else if constexpr (CMODE == 1) {
            clt += x;
        }
    };
    for_slice(
        a.scores + (int64_t)c * a.T, a.T, lo, hi, nf,
        [&](int, float x) {
            const uint32_t key = score_key(x);
            all(key, x);
            nonfloor(key, x);
        },
        [&](int j, float x) {
            const uint32_t key = score_key(x);
            all(key, x);
            if (j < nf) nonfloor(key, x);
        });
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        if (GLOB) {
            gt += __shfl_xor_sync(FW_FULL, gt, o);
            eq += __shfl_xor_sync(FW_FULL, eq, o);
        }
        if (CMODE == 2) {
            cgt += __shfl_xor_sync(FW_FULL, cgt, o);
            ceq += __shfl_xor_sync(FW_FULL, ceq, o);
        }
        if (UNI) ueq += __shfl_xor_sync(FW_FULL, ueq, o);
    }
    const double dt = warp_sum_d((double)tot), dl = warp_sum_d((double)lt);
    const double dc = CMODE != 0 ? warp_sum_d((double)clt) : 0.0, du = warp_sum_d((double)ult);
    if (lane == 0) {
        si[0][wid] = gt, si[1][wid] = eq, si[2][wid] = cgt, si[3][wid] = ceq, si[4][wid] = ueq;
        sd[0][wid] = dt, sd[1][wid] = dl, sd[2][wid] = dc, sd[3][wid] = du;
    }
    __syncthreads();
    if (threadIdx.x < 5) {
        int v = 0;
        for (int w = 0; w < NW; ++w) v += si[threadIdx.x][w];
        s_i[threadIdx.x] = v;
    } else if (threadIdx.x >= 32 && threadIdx.x < 36) {
        double v = 0.0;
        for (int w = 0; w < NW; ++w) v += sd[threadIdx.x - 32][w];
        s_d[threadIdx.x - 32] = v;
    }
    __syncthreads();
    if (threadIdx.x == 0) a.slot[blockIdx.x] = Slot{s_i[0], s_i[1], s_i[2], s_i[3]};
    cluster_barrier();  // every slice's sums are in its block's shared memory
    if (r == 0) {
        // thread 8q + f loads field f of rank q (all at once), then 8 threads sum over the ranks
        __shared__ double g_d[SMAX][4];
        __shared__ int32_t g_i[SMAX][4];
        const int q = threadIdx.x >> 3, f = threadIdx.x & 7;
        if (q < SMAX) {
            if (f < 4) {
                g_i[q][f] = q < a.S ? (int32_t)ld_cluster_u32(&s_i[f == 0 ? 0 : f == 1 ? 1 : f == 2 ? 3 : 4], (uint32_t)q)
                                    : 0;
            } else {
                g_d[q][f - 4] = q < a.S ? ld_cluster_f64(&s_d[f - 4], (uint32_t)q) : 0.0;
            }
        }
        __syncthreads();
        __shared__ int32_t t_i[4];
        __shared__ double t_d[4];
        if (threadIdx.x < 8) {
            const int ff = threadIdx.x;
            if (ff < 4) {
                int v = 0;
                for (int qq = 0; qq < SMAX; ++qq) v += g_i[qq][ff];
                t_i[ff] = v;
            } else {
                double v = 0.0;
                for (int qq = 0; qq < SMAX; ++qq) v += g_d[qq][ff - 4];
                t_d[ff - 4] = v;
            }
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            a.rec[c] = CellRec{t_i[0], t_i[1], t_i[2], t_i[3], t_d[0], t_d[1], t_d[2], t_d[3]};
            __threadfence();  // the record before the ticket
            s_last = atomicAdd(&a.st->ticket[4], 1u) == (uint32_t)a.cells - 1u;
        }
    }
    cluster_barrier();  // the first block is done reading the others
    if (r == 0 && s_last) {
        __threadfence();
        finish_offsets(a);
    }
}

// A block per slice: the slice's kept positions, in order, behind those of
// the cell's earlier slices.  A thread takes EPT consecutive positions of a
// chunk of CT * EPT; a chunk costs one block scan of the kept counts, and a
// second one of the ties at the deciding key in the slices that hold any.
constexpr int EPT = PER;  // positions per thread and chunk (a bit mask of 32)

__global__ void __launch_bounds__(CT) k_c_emit(CArgs a)
{
    constexpr int NW = CT / 32;
    constexpr int CH = CT * EPT;  // positions per chunk
    __shared__ uint32_t wsum32[NW];
    __shared__ int s_tb, s_kb, s_te;
    const int c = blockIdx.x / a.S, r = blockIdx.x - c * a.S;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int nfe = a.T - a.F;  // positions before the floor
    int lo, hi;
    slice_bounds(a, r, lo, hi);
    const float *s = a.scores + (int64_t)c * a.T;
    const bool vec = (a.T & 3) == 0 && (reinterpret_cast<uintptr_t>(s) & 15) == 0;
    auto load = [&](int j, float (&x)[EPT]) {
        if (vec && j + EPT <= hi) {
#pragma unroll
            for (int h = 0; h < EPT; h += 4) {
                const float4 v = __ldg(reinterpret_cast<const float4 *>(s + j + h));
                x[h] = v.x, x[h + 1] = v.y, x[h + 2] = v.z, x[h + 3] = v.w;
            }
        } else {
#pragma unroll
            for (int u = 0; u < EPT; ++u) x[u] = j + u < hi ? __ldg(s + j + u) : 0.f;
        }
    };
    grid_release();
    grid_wait();  // every earlier kernel of the stream is complete from here on (scores included)
    float x[EPT];
    load(lo + EPT * tid, x);
    const int mode = a.emode[c];
    const int want = a.take[c];
    if (wid == 0) {  // ties of the deciding key and kept entries in the cell's earlier slices: lane q, slice q
        int e = 0, g = 0, fl = 0;
        if (lane <= r) {
            const Slot sq = a.slot[(int64_t)c * a.S + lane];
            e = mode == 2 ? 0 : (mode == 1 ? sq.ceq : sq.eq);
            g = mode == 2 ? 0 : (mode == 1 ? sq.cgt : sq.gt);
            int qlo, qhi;
            slice_bounds(a, lane, qlo, qhi);
            fl = max(0, qhi - max(qlo, nfe));  // floor positions
        }
        int inc = e;  // ties in slices 0..lane
#pragma unroll
        for (int o = 1; o < SMAX; o <<= 1) {
            const int y = __shfl_up_sync(FW_FULL, inc, o);
            if (lane >= o) inc += y;
        }
        const int tb = inc - e;
        int kept = lane < r ? fl + g + (mode == 2 ? 0 : min(max(want - tb, 0), e)) : 0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) kept += __shfl_xor_sync(FW_FULL, kept, o);
        if (lane == r) {
            s_te = e;
            s_tb = tb;
            s_kb = kept;
        }
    }
    const uint32_t eT = mode == 1 ? a.cprefix[c] : a.st->prefix;
    const int64_t wend = a.offsets[c + 1];  // the cell's end: no write beyond it
    __syncthreads();
    const bool ties = s_te > 0;  // the slice holds keys equal to the deciding key
    const int64_t base = a.offsets[c] + s_kb;
    int ties_seen = s_tb;
    int64_t written = 0;
    for (int j0 = lo; j0 < hi; j0 += CH) {
        const int jt = j0 + EPT * tid;  // this thread's first position
        if (j0 > lo) load(jt, x);
        // flags as bit masks (bit u: position jt + u)
        uint32_t kept = 0u, tie = 0u;
        if (mode != 2 && jt + EPT <= min(hi, nfe)) {  // every position in range and before the floor
#pragma unroll
            for (int u = 0; u < EPT; ++u) {
                const uint32_t key = score_key(x[u]);
                kept |= (key > eT ? 1u : 0u) << u;
                if (ties) tie |= (key == eT ? 1u : 0u) << u;
            }
        } else {
#pragma unroll
            for (int u = 0; u < EPT; ++u) {
                const int j = jt + u;
                if (j < hi) {
                    if (j >= nfe) {
                        kept |= 1u << u;
                    } else if (mode != 2) {
                        const uint32_t key = score_key(x[u]);
                        kept |= (key > eT ? 1u : 0u) << u;
                        tie |= (key == eT ? 1u : 0u) << u;
                    }
                }
            }
        }
        if (ties) {  // ranks of the ties among the cell's, in position order
            uint32_t tb, ttot;
            block_scan<NW>((uint32_t)__popc(tie), wsum32, wid, lane, tb, ttot);
            int rt = ties_seen + (int)tb;
            for (uint32_t m = tie; m; m &= m - 1) {
                const int u = __ffs(m) - 1;
                if (rt++ < want) kept |= 1u << u;
            }
            ties_seen += (int)ttot;
        }
        uint32_t kbef, ktot;
        block_scan<NW>((uint32_t)__popc(kept), wsum32, wid, lane, kbef, ktot);
        int64_t w = base + written + kbef;
        for (uint32_t m = kept; m; m &= m - 1) {
            if (w < wend) a.kept_pos[w] = jt + __ffs(m) - 1;
            ++w;
        }
        written += ktot;
    }
}

// ragged compaction: block (cell, chunk) copies rows [offsets[c] + chunk*RPB, ...).
// With dst_base, cell c's rows go to rows dst_base[c] + (q - offsets[c]) of the
// output instead (a store with room per cell), provided they fit its capacity.
constexpr int RPB = 256;  // rows per block
__global__ void __launch_bounds__(256) k_compact(const uint4 *K, const uint4 *V, int T, int vec_per_row,
                                                 const int64_t *offsets, const int32_t *kept_pos, uint4 *Ko,
                                                 uint4 *Vo, int chunks, const int64_t *dst_base,
                                                 const int32_t *capacity, int32_t *status)
{
    grid_wait();  // launched chained: the offsets and positions of the kernel before are complete from here on
    const int c = blockIdx.x / chunks;
    const int chunk = blockIdx.x - c * chunks;
    const int64_t cnt = offsets[c + 1] - offsets[c];
    int64_t shift = 0;
    if (dst_base) {
        const bool fits = cnt <= capacity[c];
        if (chunk == 0 && threadIdx.x == 0 && status) status[c] = fits ? FW_OK : FW_ERR_WORKSPACE;
        if (!fits) return;
        shift = dst_base[c] - offsets[c];
    }
    const int64_t beg = offsets[c] + (int64_t)chunk * RPB;
    const int64_t end = min(offsets[c + 1], beg + RPB);
    if (beg >= end) return;
    const int64_t nvec = (end - beg) * vec_per_row;
    for (int64_t e = threadIdx.x; e < nvec; e += blockDim.x) {
        const int64_t q = beg + e / vec_per_row;
        const int part = (int)(e % vec_per_row);
        const int64_t src = ((int64_t)c * T + kept_pos[q]) * vec_per_row + part;
        const int64_t dst = (q + shift) * vec_per_row + part;
        Ko[dst] = __ldg(K + src);
        Vo[dst] = __ldg(V + src);
    }
}

// decode-time append: block c copies cell c's m new rows behind its filled
// rows when they fit, then advances its count
__global__ void __launch_bounds__(256) k_append(uint4 *Ks, uint4 *Vs, const int64_t *base, const int32_t *capacity,
                                                int32_t *counts, const uint4 *nK, const uint4 *nV, int m,
                                                int vec_per_row, int32_t *status)
{
    __shared__ int s_cnt;
    const int c = blockIdx.x;
    if (threadIdx.x == 0) s_cnt = counts[c];
    __syncthreads();
    const int cnt = s_cnt;
    const bool fits = cnt >= 0 && (int64_t)cnt + m <= (int64_t)capacity[c];
    if (fits) {
        const int64_t dst0 = (base[c] + cnt) * vec_per_row;
        const int64_t src0 = (int64_t)c * m * vec_per_row;
        const int nvec = m * vec_per_row;
        for (int e = threadIdx.x; e < nvec; e += blockDim.x) {
            Ks[dst0 + e] = __ldg(nK + src0 + e);
            Vs[dst0 + e] = __ldg(nV + src0 + e);
        }
    }
    __syncthreads();  // every thread has read the old count
    if (threadIdx.x == 0) {
        if (fits) counts[c] = cnt + m;
        if (status) status[c] = fits ? FW_OK : FW_ERR_WORKSPACE;
    }
}

}  // namespace

// Workspace: the four histograms, the radix state, four per-cell arrays
// (take, emode, uprefix, urem), the cell records and the slice records; the
// capped variant adds two per-cell arrays (cprefix, crem).
size_t contour_workspace(int cells, int T)
{
    const size_t slots = (size_t)cells * n_slices(cells, T);
    return align256(4 * 256 * 4) + align256(sizeof(CState)) + 4 * align256((size_t)cells * 4) +
           align256((size_t)cells * sizeof(CellRec)) + align256(slots * sizeof(Slot));
}

size_t contour_capped_workspace(int cells, int T) { return contour_workspace(cells, T) + 2 * align256((size_t)cells * 4); }

// A launch of `grid` blocks (in clusters of `cl` consecutive blocks when
// cl > 1) that the stream may start while the kernel before it is finishing:
// every kernel launched this way waits for its predecessor (grid_wait) before
// it reads what that one wrote.
template <typename... Args>
static fw_status launch_chained(void (*kernel)(Args...), unsigned grid, unsigned block, unsigned cl, cudaStream_t s,
                                Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(block);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = cl;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = cl > 1 ? 2 : 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, args...);
    ::fw::g_launches.fetch_add(1, std::memory_order_relaxed);
    if (e != cudaSuccess || cudaGetLastError() != cudaSuccess) return FW_ERR_CUDA;
    return FW_OK;
}

template <bool G, bool U, bool C>
static fw_status run_passes(const CArgs &a, cudaStream_t s)
{
    for (int pass = 0; pass < 4; ++pass) {
        const fw_status st = launch_chained(k_c_pass<G, U, C>, (unsigned)(a.cells * a.S), CT, (unsigned)a.S, s, a, pass);
        if (st != FW_OK) return st;
    }
    return FW_OK;
}

template <bool G, bool U, int CM>
static fw_status run_count(const CArgs &a, cudaStream_t s)
{
    return launch_chained(k_c_count<G, U, CM>, (unsigned)(a.cells * a.S), CT, (unsigned)a.S, s, a);
}

fw_status contour_alloc(const float *scores, int cells, int T, int floor_, int64_t total_budget, int uniform_s,
                        int32_t *counts, int64_t *offsets, int32_t *kept_pos, float *tau, float *dropped_uniform,
                        float *dropped_alloc, void *ws, size_t ws_bytes, cudaStream_t s, int cap)
{
    (void)ws_bytes;
    CArgs a;
    a.scores = scores;
    a.cells = cells;
    a.T = T;
    a.F = floor_ < T ? floor_ : T;
    a.S = n_slices(cells, T);
    a.L = slice_len(T, a.S);
    a.K = total_budget - (int64_t)cells * a.F;
    if (a.K >= ((int64_t)1 << 32)) return FW_ERR_UNSUPPORTED;
    if ((int64_t)cells * a.S >= ((int64_t)1 << 31)) return FW_ERR_UNSUPPORTED;
    char *w = (char *)ws;
    a.hist = (uint32_t *)w;
    w += align256(4 * 256 * 4);
    a.st = (CState *)w;
    w += align256(sizeof(CState));
    a.take = (int32_t *)w;
    w += align256((size_t)cells * 4);
    a.emode = (int32_t *)w;
    w += align256((size_t)cells * 4);
    a.uprefix = (uint32_t *)w;
    w += align256((size_t)cells * 4);
    a.urem = (uint32_t *)w;
    w += align256((size_t)cells * 4);
    a.rec = (CellRec *)w;
    w += align256((size_t)cells * sizeof(CellRec));
    a.slot = (Slot *)w;
    w += align256((size_t)cells * a.S * sizeof(Slot));
    a.capnf = -1;
    a.cprefix = a.crem = nullptr;
    if (cap >= 0) {  // the capped variant: two more per-cell arrays after the uncapped layout
        a.cprefix = (uint32_t *)w;
        w += align256((size_t)cells * 4);
        a.crem = (uint32_t *)w;
        a.capnf = cap - a.F;
    }
    a.counts = counts;
    a.offsets = offsets;
    a.kept_pos = kept_pos;
    a.tau = tau;
    a.dropped_uniform = dropped_uniform;
    a.dropped_alloc = dropped_alloc;
    a.uniform_s = uniform_s;
    const bool G = a.K > 0;
    const bool U = dropped_uniform && std::min(uniform_s, T) > 0;  // every cell has a uniform set
    const bool C = cap_selects(a);
    const int CM = cap_mode(a);
    {
        const fw_status st = launch_chained(k_c_init, 1u, 1024u, 1u, s, a);
        if (st != FW_OK) return st;
    }
    if (G || U || C) {
        using PassFn = fw_status (*)(const CArgs &, cudaStream_t);
        static const PassFn passes[8] = {run_passes<false, false, false>, run_passes<false, false, true>,
                                         run_passes<false, true, false>,  run_passes<false, true, true>,
                                         run_passes<true, false, false>,  run_passes<true, false, true>,
                                         run_passes<true, true, false>,   run_passes<true, true, true>};
        const fw_status st = passes[(G ? 4 : 0) + (U ? 2 : 0) + (C ? 1 : 0)](a, s);
        if (st != FW_OK) return st;
    }
    using CountFn = fw_status (*)(const CArgs &, cudaStream_t);
    static const CountFn count[12] = {run_count<false, false, 0>, run_count<false, false, 1>, run_count<false, false, 2>,
                                      run_count<false, true, 0>,  run_count<false, true, 1>,  run_count<false, true, 2>,
                                      run_count<true, false, 0>,  run_count<true, false, 1>,  run_count<true, false, 2>,
                                      run_count<true, true, 0>,   run_count<true, true, 1>,   run_count<true, true, 2>};
    const fw_status st = count[(G ? 6 : 0) + (U ? 3 : 0) + CM](a, s);
    if (st != FW_OK) return st;
    return launch_chained(k_c_emit, (unsigned)(cells * a.S), CT, 1u, s, a);
}

fw_status ragged_compact(const void *K, const void *V, int cells, int T, int row_bytes, const int64_t *offsets,
                         const int32_t *kept_pos, int64_t total, void *K_out, void *V_out, cudaStream_t s)
{
    if (total == 0) return FW_OK;
    const int vec = row_bytes / 16;
    const int chunks = (T + RPB - 1) / RPB;
    const int64_t grid = (int64_t)cells * chunks;
    if (grid >= ((int64_t)1 << 31)) return FW_ERR_UNSUPPORTED;
    return launch_chained(k_compact, (unsigned)grid, 256u, 1u, s, (const uint4 *)K, (const uint4 *)V, T, vec, offsets,
                          kept_pos, (uint4 *)K_out, (uint4 *)V_out, chunks, (const int64_t *)nullptr,
                          (const int32_t *)nullptr, (int32_t *)nullptr);
}

fw_status ragged_compact_to(const void *K, const void *V, int cells, int T, int row_bytes, const int64_t *offsets,
                            const int32_t *kept_pos, const int64_t *base, const int32_t *capacity, void *K_store,
                            void *V_store, int32_t *status, cudaStream_t s)
{
    const int vec = row_bytes / 16;
    const int chunks = (T + RPB - 1) / RPB;
    const int64_t grid = (int64_t)cells * chunks;
    if (grid >= ((int64_t)1 << 31)) return FW_ERR_UNSUPPORTED;
    return launch_chained(k_compact, (unsigned)grid, 256u, 1u, s, (const uint4 *)K, (const uint4 *)V, T, vec, offsets,
                          kept_pos, (uint4 *)K_store, (uint4 *)V_store, chunks, base, capacity, status);
}

fw_status ragged_append(void *K_store, void *V_store, const int64_t *base, const int32_t *capacity, int32_t *counts,
                        const void *new_K, const void *new_V, int cells, int m, int row_bytes, int32_t *status,
                        cudaStream_t s)
{
    FW_LAUNCH(k_append, (unsigned)cells, 256, 0, s, (uint4 *)K_store, (uint4 *)V_store, base, capacity, counts,
              (const uint4 *)new_K, (const uint4 *)new_V, m, row_bytes / 16, status);
    return FW_OK;
}

}  // namespace fw

// ------------------------------------------------------------------------
// Allocation-free variant: the scratch lives in a fixed device array.
namespace fw {
namespace {

// >= contour_workspace for every T at the largest cell count: the slices
// over all cells never outnumber max(cells, SLOT_TARGET) <= the maximum
static_assert(SLOT_TARGET <= FW_CONTOUR_NOALLOC_MAX_CELLS, "slice records sized by the cell maximum");
constexpr size_t kNoallocBytes = 4 * 256 * 4 + 256 + 4 * (size_t)FW_CONTOUR_NOALLOC_MAX_CELLS * 4 +
                                 (size_t)FW_CONTOUR_NOALLOC_MAX_CELLS * (sizeof(CellRec) + sizeof(Slot));
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocBytes + 6 * 256];

// Device address of the scratch array in the current device's context.  It is
// looked up on every call (a host-side query, no launch): after a device reset
// or a re-created primary context the module is loaded anew and the array may
// sit elsewhere, so no address is kept between calls.
fw_status noalloc_scratch(void **ptr)
{
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return FW_ERR_CUDA;
    *ptr = p;
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
