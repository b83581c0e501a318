// k_contour.cu -- ContourKV allocation and ragged per-head storage (Sec. 4).
//
// One importance score per (cell, position); one global threshold tau shared
// by every cell; each cell keeps its recency floor (last min(floor, T)
// positions) plus its non-floor positions ranked among the best
// K = budget - cells*floor non-floor entries of the whole cache.  The order is
// (score desc, cell asc, position asc), so ties at tau are split exactly.
//
// tau is found by a global radix select (4 passes x 8 bits).  Every pass is a
// histogram launch (a block per cell) into its own global histogram; each
// block of the next launch derives the digits fixed so far from those
// histograms (a warp scan), so no kernel ever waits on another block.  The same passes carry each cell's own
// top-uniform_s select (the uniform-budget dropped mass): its histogram is
// the cell's alone, so the cell's block fixes its digit at the end of the pass.  Then per-cell counts, an exclusive
// prefix sum into ragged offsets, and per-cell ordered compaction of the kept
// positions.  The compaction copy moves 16-byte vectors, a row per 16 lanes.
//
// The capped variant (the enforcement of Sec. 4: no cell keeps more than a
// cap, e.g. a uniform method's per-head count) truncates each cell to its
// floor plus its best cap - floor non-floor entries of the allocation; the
// passes carry a third, per-cell select of the (cap - floor)-th non-floor key,
// and a non-floor position is kept when both the global threshold and the
// cell's cap threshold keep it (both are prefixes of the cell's order).
#include <algorithm>

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
    uint32_t *hist;      // [4][256] global histograms of the four passes
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
    uint32_t *uprefix;   // [cells] bits of the cell's uniform-budget threshold fixed so far
    uint32_t *urem;      // [cells] rank still to find inside that prefix (0: no uniform set)
    int capnf;           // cap - floor on non-floor entries per cell; < 0: no cap
    uint32_t *cprefix;   // [cells] bits of the cell's cap threshold (non-floor keys) fixed so far
    uint32_t *crem;      // [cells] rank still to find inside that prefix (0: the cap truncates nothing)
};

// The cap keeps every non-floor entry (no select needed), none, or a prefix.
__device__ __forceinline__ bool cap_selects(const CArgs &a) { return a.capnf > 0 && a.capnf < a.T - a.F; }

__global__ void k_c_init(CArgs a)
{
    if (threadIdx.x == 0) {
        a.st->prefix = 0u;
        a.st->rem = (uint32_t)a.K;
        a.st->K_lo = (uint32_t)a.K;
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

// The radix state after `npass` passes: the bits of tau's key fixed so far
// and the rank still to find inside them, from the passes' global
// histograms.  One warp; lane l takes bins 255 - 8l .. 248 - 8l of a pass.
__device__ __forceinline__ void select_state(const uint32_t *hist4, int npass, uint32_t K, uint32_t &prefix,
                                             uint32_t &rem)
{
    const int lane = threadIdx.x & 31;
    prefix = 0u;
    rem = K;
    for (int p = 0; p < npass; ++p) {
        uint32_t c[8], loc = 0;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            c[i] = hist4[p * 256 + 255 - 8 * lane - i];
            loc += c[i];
        }
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
        v = __shfl_sync(FW_FULL, v, src < 0 ? 0 : src);
        nr = __shfl_sync(FW_FULL, nr, src < 0 ? 0 : src);
        prefix |= (v & 255u) << (24 - 8 * p);
        rem = nr;
    }
}

// One radix pass, a block per cell.  The cell's non-floor keys matching the
// global prefix go to the global histogram of digit `pass` (the threshold
// tau); all of the cell's keys matching its own uniform prefix go to a cell
// histogram, which the block scans at once to fix the digit of the cell's own
// top-uniform_s threshold (the uniform-budget dropped mass).
constexpr int CPT = 512;  // threads of a pass block
__global__ void __launch_bounds__(CPT) k_c_pass(CArgs a, int pass)
{
    __shared__ uint32_t hg[256], hu[256], hc[256];
    __shared__ uint32_t s_prefix;
    for (int i = threadIdx.x; i < 256; i += CPT) hg[i] = hu[i] = hc[i] = 0u;
    const bool glob = a.K > 0;
    if (threadIdx.x < 32) {  // the global state after the earlier passes
        uint32_t pf = 0u, rm = 0u;
        if (glob) select_state(a.hist, pass, (uint32_t)a.K, pf, rm);
        if (threadIdx.x == 0) s_prefix = pf;
    }
    __syncthreads();
    const int c = blockIdx.x;
    const int shift = 24 - 8 * pass;
    const uint32_t pmask = pass == 0 ? 0u : (0xffffffffu << (32 - 8 * pass));
    const uint32_t prefix = s_prefix;
    const uint32_t upre = a.uprefix[c];
    const bool uni = a.urem[c] > 0u;
    const bool cap = a.cprefix && cap_selects(a);
    const uint32_t cpre = cap ? a.cprefix[c] : 0u;
    const int nf = a.T - a.F;
    const float *sc = a.scores + (int64_t)c * a.T;
    auto visit = [&](int j, float x) {
        const uint32_t key = order_key(x);
        const uint32_t dg = (key >> shift) & 255u;
        if (glob && j < nf && (key & pmask) == prefix) atomicAdd(&hg[dg], 1u);
        if (uni && (key & pmask) == upre) atomicAdd(&hu[dg], 1u);
        if (cap && j < nf && (key & pmask) == cpre) atomicAdd(&hc[dg], 1u);
    };
    if ((a.T & 3) == 0 && (reinterpret_cast<uintptr_t>(sc) & 15) == 0) {
        // LD vectors per thread in flight before any is used (one at a time
        // left each block waiting on a memory round trip per vector: a block
        // per cell, 256 cells, too few bytes in flight per SM)
        constexpr int LD = 8;
        const int nq = a.T / 4;
        for (int q0 = threadIdx.x; q0 < nq; q0 += LD * CPT) {
            float4 v[LD];
#pragma unroll
            for (int u = 0; u < LD; ++u) {
                const int q = q0 + u * CPT;
                v[u] = q < nq ? __ldg(reinterpret_cast<const float4 *>(sc) + q) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int u = 0; u < LD; ++u) {
                const int q = q0 + u * CPT;
                if (q < nq) {
                    visit(4 * q, v[u].x);
                    visit(4 * q + 1, v[u].y);
                    visit(4 * q + 2, v[u].z);
                    visit(4 * q + 3, v[u].w);
                }
            }
        }
    } else {
        for (int j = threadIdx.x; j < a.T; j += CPT) visit(j, __ldg(sc + j));
    }
    __syncthreads();
    if (glob)
        for (int i = threadIdx.x; i < 256; i += CPT)
            if (hg[i]) atomicAdd(&a.hist[pass * 256 + i], hg[i]);
    if (uni && threadIdx.x == 0) {
        uint32_t cum = 0, rem = a.urem[c];
        for (int v = 255; v >= 0; --v) {
            const uint32_t cc = hu[v];
            if (cum + cc >= rem) {
                a.uprefix[c] = upre | ((uint32_t)v << shift);
                a.urem[c] = rem - cum;
                break;
            }
            cum += cc;
        }
    }
    if (cap && threadIdx.x == 32) {
        uint32_t cum = 0, rem = a.crem[c];
        for (int v = 255; v >= 0; --v) {
            const uint32_t cc = hc[v];
            if (cum + cc >= rem) {
                a.cprefix[c] = cpre | ((uint32_t)v << shift);
                a.crem[c] = rem - cum;
                break;
            }
            cum += cc;
        }
    }
}

// per cell: keys above / equal to tau among the non-floor positions
__global__ void __launch_bounds__(CT) k_c_count(CArgs a)
{
    __shared__ int s_gt, s_eq;
    __shared__ uint32_t s_tk;
    const int c = blockIdx.x;
    if (threadIdx.x < 32) {  // tau's key from the four passes; block 0 records it
        uint32_t pf = 0u, rm = 0u;
        if (a.K > 0) select_state(a.hist, 4, (uint32_t)a.K, pf, rm);
        if (threadIdx.x == 0) {
            s_tk = pf;
            s_gt = s_eq = 0;
            if (c == 0) {
                a.st->prefix = pf;
                a.st->rem = rm;
            }
        }
    }
    __syncthreads();
    const uint32_t tk = s_tk;
    int gt = 0, eq = 0;
    if (a.K > 0) {
        // eight 16-byte loads per thread in flight before any is used
        const float *sc = a.scores + (int64_t)c * a.T;
        const int nf = a.T - a.F;
        auto tally = [&](int j, float x) {
            if (j < nf) {
                const uint32_t key = order_key(x);
                gt += key > tk;
                eq += key == tk;
            }
        };
        if ((a.T & 3) == 0 && (reinterpret_cast<uintptr_t>(sc) & 15) == 0) {
            const int nq = (nf + 3) / 4;
            for (int q0 = threadIdx.x; q0 < nq; q0 += 8 * CT) {
                float4 v[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int q = q0 + u * CT;
                    v[u] = q < nq ? __ldg(reinterpret_cast<const float4 *>(sc) + q) : make_float4(0.f, 0.f, 0.f, 0.f);
                }
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int j = 4 * (q0 + u * CT);
                    tally(j, v[u].x);
                    tally(j + 1, v[u].y);
                    tally(j + 2, v[u].z);
                    tally(j + 3, v[u].w);
                }
            }
        } else {
            for (int j = threadIdx.x; j < nf; j += CT) tally(j, __ldg(sc + j));
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
        int nonf = (a.K > 0 ? a.gt[c] : 0) + (int)t;
        if (a.capnf >= 0) nonf = min(nonf, a.capnf);
        const int cnt = a.F + nonf;
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

// per cell, positions in order: the ordered compaction of the kept positions,
// the dropped mass of the allocation, and the cell's own top-uniform_s set
// (keys above its threshold, then the first equal ones in position order) with
// the dropped mass outside it.  A thread takes EPT consecutive positions of a
// chunk of CTE * EPT, so a chunk costs two block scans: the tie counts (the
// global threshold's, the uniform set's and the cap's, packed in one 64-bit
// word) and the kept counts.
constexpr int CTE = 512;  // threads of an emit block (two per SM: the cells fit one wave)
constexpr int EPT = 8;    // positions per thread and chunk

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
    const U w = lane < NW ? wsum[lane] : (U)0;
    U winc = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const U y = __shfl_up_sync(FW_FULL, winc, o);
        if (lane >= o) winc += y;
    }
    before = __shfl_sync(FW_FULL, winc - w, wid) + inc - v;
    total = __shfl_sync(FW_FULL, winc, 31);
    __syncthreads();  // wsum is rewritten by the next scan
}

__global__ void __launch_bounds__(CTE, 2) k_c_emit(CArgs a)
{
    constexpr int NW = CTE / 32;
    constexpr int CH = CTE * EPT;  // positions per chunk
    __shared__ unsigned long long wsum64[NW];
    __shared__ uint32_t wsum32[NW];
    __shared__ double red[NW], red2[NW], red3[NW];
    const int c = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const uint32_t tk = a.st->prefix;
    const int take = a.take[c];
    const int64_t base = a.offsets[c];
    const uint32_t uT = a.uprefix[c];
    const int uwant = (int)a.urem[c];  // 0: no uniform set (every key dropped)
    // the cap: none (every non-floor entry passes it), zero entries, or its threshold
    const int cmode = a.capnf < 0 || a.capnf >= a.T - a.F ? 0 : (a.capnf == 0 ? 1 : 2);
    const uint32_t cT = cmode == 2 ? a.cprefix[c] : 0u;
    const int cwant = cmode == 2 ? (int)a.crem[c] : 0;
    const float *s = a.scores + (int64_t)c * a.T;
    const bool vec = (a.T & 3) == 0 && (reinterpret_cast<uintptr_t>(s) & 15) == 0;
    const int nfe = a.T - a.F;  // positions before the floor
    int64_t written = 0;
    int ties_seen = 0, uties_seen = 0, cties_seen = 0;
    // per-thread sums of T / CTE positive terms in fp32 (relative error below
    // 1e-5); the sums over threads in fp64
    float tot = 0.f, drop = 0.f, udrop = 0.f;
    auto load4 = [&](int j, float (&x)[EPT]) {
        if (vec && j + EPT <= a.T) {
#pragma unroll
            for (int h = 0; h < EPT; h += 4) {
                const float4 v = __ldg(reinterpret_cast<const float4 *>(s + j + h));
                x[h] = v.x, x[h + 1] = v.y, x[h + 2] = v.z, x[h + 3] = v.w;
            }
        } else {
#pragma unroll
            for (int u = 0; u < EPT; ++u) x[u] = j + u < a.T ? __ldg(s + j + u) : 0.f;
        }
    };
    float xn[EPT];
    load4(EPT * tid, xn);  // the next chunk's scores, loaded a chunk ahead
    for (int j0 = 0; j0 < a.T; j0 += CH) {
        const int jt = j0 + EPT * tid;  // this thread's first position
        float x[EPT];
#pragma unroll
        for (int u = 0; u < EPT; ++u) x[u] = xn[u];
        if (j0 + CH < a.T) load4(jt + CH, xn);
        // flags as bit masks (bit u: position jt + u)
        uint32_t kept = 0u, tie = 0u, ukept = 0u, utie = 0u, ckept = 0u, ctie = 0u;
#pragma unroll
        for (int u = 0; u < EPT; ++u) {
            const int j = jt + u;
            const uint32_t bit = 1u << u;
            bool k_ = false, t_ = false, uk_ = false, ut_ = false, ck_ = true, ct_ = false;
            if (j < a.T) {
                const uint32_t key = order_key(x[u]);
                if (j >= nfe) {
                    k_ = true;
                } else {
                    if (a.K > 0) {
                        k_ = key > tk;
                        t_ = key == tk;
                    }
                    if (cmode == 1) {
                        ck_ = false;
                    } else if (cmode == 2) {
                        ck_ = key > cT;
                        ct_ = key == cT;
                    }
                }
                if (uwant > 0) {
                    uk_ = key > uT;
                    ut_ = key == uT;
                }
            }
            kept |= k_ ? bit : 0u;
            tie |= t_ ? bit : 0u;
            ukept |= uk_ ? bit : 0u;
            utie |= ut_ ? bit : 0u;
            ckept |= ck_ ? bit : 0u;
            ctie |= ct_ ? bit : 0u;
        }
        // ranks of the ties among the cell's ties, in position order
        unsigned long long tb, ttot;
        block_scan<NW>((unsigned long long)__popc(tie) | ((unsigned long long)__popc(utie) << 21) |
                           ((unsigned long long)__popc(ctie) << 42),
                       wsum64, wid, lane, tb, ttot);
        int rt = ties_seen + (int)(tb & 0x1fffffu), ru = uties_seen + (int)((tb >> 21) & 0x1fffffu),
            rc = cties_seen + (int)(tb >> 42);
#pragma unroll
        for (int u = 0; u < EPT; ++u) {
            const uint32_t bit = 1u << u;
            if (tie & bit) kept = rt++ < take ? (kept | bit) : (kept & ~bit);
            if (utie & bit) ukept = ru++ < uwant ? (ukept | bit) : (ukept & ~bit);
            if (ctie & bit) ckept = rc++ < cwant ? (ckept | bit) : (ckept & ~bit);
        }
        kept &= ckept;
        ties_seen += (int)(ttot & 0x1fffffu);
        uties_seen += (int)((ttot >> 21) & 0x1fffffu);
        cties_seen += (int)(ttot >> 42);
        uint32_t kbef, ktot;
        block_scan<NW>((uint32_t)__popc(kept), wsum32, wid, lane, kbef, ktot);
        int64_t w = base + written + kbef;
#pragma unroll
        for (int u = 0; u < EPT; ++u) {
            const int j = jt + u;
            const uint32_t bit = 1u << u;
            if (kept & bit) a.kept_pos[w++] = j;
            if (j < a.T) {
                tot += x[u];
                if (!(kept & bit)) drop += x[u];
                if (!(ukept & bit)) udrop += x[u];
            }
        }
        written += ktot;
    }
    const double tsum = warp_sum_d((double)tot), dsum = warp_sum_d((double)drop), usum = warp_sum_d((double)udrop);
    if (lane == 0) {
        red[wid] = tsum;
        red2[wid] = dsum;
        red3[wid] = usum;
    }
    __syncthreads();
    if (tid == 0) {
        double t = 0.0, dd = 0.0, du = 0.0;
        for (int w = 0; w < NW; ++w) {
            t += red[w];
            dd += red2[w];
            du += red3[w];
        }
        if (a.dropped_alloc) a.dropped_alloc[c] = t > 0.0 ? (float)(dd / t) : 0.f;
        if (a.dropped_uniform) a.dropped_uniform[c] = t > 0.0 ? (float)(du / t) : 0.f;
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

size_t contour_workspace(int cells, int T)
{
    (void)T;
    return align256(4 * 256 * 4) + align256(sizeof(CState)) + 5 * align256((size_t)cells * 4);
}

size_t contour_capped_workspace(int cells, int T) { return contour_workspace(cells, T) + 2 * align256((size_t)cells * 4); }

static bool cap_selects_host(const CArgs &a) { return a.cprefix && a.capnf > 0 && a.capnf < a.T - a.F; }

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
    a.K = total_budget - (int64_t)cells * a.F;
    if (a.K >= ((int64_t)1 << 32)) return FW_ERR_UNSUPPORTED;
    char *w = (char *)ws;
    a.hist = (uint32_t *)w;
    w += align256(4 * 256 * 4);
    a.st = (CState *)w;
    w += align256(sizeof(CState));
    a.gt = (int32_t *)w;
    w += align256((size_t)cells * 4);
    a.eq = (int32_t *)w;
    w += align256((size_t)cells * 4);
    a.take = (int32_t *)w;
    w += align256((size_t)cells * 4);
    a.uprefix = (uint32_t *)w;
    w += align256((size_t)cells * 4);
    a.urem = (uint32_t *)w;
    a.capnf = -1;
    a.cprefix = a.crem = nullptr;
    if (cap >= 0) {  // the capped variant: two more per-cell arrays after the uncapped layout
        w += align256((size_t)cells * 4);
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
    FW_LAUNCH(k_c_init, 1, 1024, 0, s, a);
    if (a.K > 0 || (dropped_uniform && uniform_s > 0) || cap_selects_host(a)) {
        for (int pass = 0; pass < 4; ++pass) FW_LAUNCH(k_c_pass, (unsigned)cells, CPT, 0, s, a, pass);
    }
    FW_LAUNCH(k_c_count, (unsigned)cells, CT, 0, s, a);
    FW_LAUNCH(k_c_offsets, 1, 1024, 0, s, a);
    FW_LAUNCH(k_c_emit, (unsigned)cells, CTE, 0, s, a);
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
              (uint4 *)K_out, (uint4 *)V_out, chunks, (const int64_t *)nullptr, (const int32_t *)nullptr,
              (int32_t *)nullptr);
    return FW_OK;
}

fw_status ragged_compact_to(const void *K, const void *V, int cells, int T, int row_bytes, const int64_t *offsets,
                            const int32_t *kept_pos, const int64_t *base, const int32_t *capacity, void *K_store,
                            void *V_store, int32_t *status, cudaStream_t s)
{
    const int vec = row_bytes / 16;
    const int chunks = (T + RPB - 1) / RPB;
    const int64_t grid = (int64_t)cells * chunks;
    if (grid >= ((int64_t)1 << 31)) return FW_ERR_UNSUPPORTED;
    FW_LAUNCH(k_compact, (unsigned)grid, 256, 0, s, (const uint4 *)K, (const uint4 *)V, T, vec, offsets, kept_pos,
              (uint4 *)K_store, (uint4 *)V_store, chunks, base, capacity, status);
    return FW_OK;
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

constexpr size_t kNoallocBytes = 4 * 256 * 4 + 256 + 5 * (size_t)FW_CONTOUR_NOALLOC_MAX_CELLS * 4;  // >= contour_workspace
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocBytes + 5 * 256];

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
