// k_long_tc.cu -- the P.V products of the long-row path (dense output mu,
// forced-weight outputs m_A, gaps and dropped mass; Definition 2.1, Sec. 2.1,
// Lemma 2.1) on the 5th-generation tensor cores, for bf16 values.
//
// For a tile of RT rows of one group (rows sharing V) the kernel forms
//   S[b][r][:] = sum_j [band(r, j) = b] p_rj v_j,   b = 0..nb,
// where band(r, j) = number of budgets of row r that drop key j, as one GEMM:
// A = (band, row) x keys, 128 x 64 per stage, B = keys x d (V itself), the
// fp32 accumulator D = 128 x d in tensor memory.  Each probability is split
// into three bf16 terms (hi + mid + lo reproduce the fp32 value to ~2^-24), so
// with bf16 V every product is exact and only the fp32 accumulation rounds,
// as on the CUDA cores.  The A tiles are written by the producer warps
// (exp, band, split) in the 128-byte-swizzled K-major layout; V tiles arrive
// by cp.async in the 128-byte-swizzled MN-major layout; one thread issues
// tcgen05.mma and tcgen05.commit frees each stage.  The tensor core rounds its
// fp32 accumulation toward zero, which over thousands of additions into one
// accumulator biases the sums by ~1e-3; so every chunk of CH = 8 stages (512
// keys, about 100 accumulation steps: a bias below ~1e-5 of the partial sums)
// accumulates into a fresh TMEM buffer (two in rotation) and the producers add
// it into fp32 registers with round-to-nearest two stages after the chunk ends,
// when its MMAs have long completed, so that no producer ever waits on the MMAs
// it has just enabled.  The epilogue combines
// the bands exactly as the CUDA-core kernel does (the TMA-fed kernels below
// also serve the group vote, whose bands come from the group's summed masses
// and shared thresholds instead of each row's own):
//   N_A = sum of the bands inside A, N_{A^c} = the rest,
//   p(A) (m_A - mu) = pbar(A) N_A - p(A) N_{A^c}.
#include <cuda_bf16.h>

#include "fw_internal.h"
#include "tc_sm100.cuh"

namespace fw {
namespace {

constexpr int TM = 128;       // rows of the MMA tile: (band, row) pairs, band-major
constexpr int KS = 64;        // keys per stage: one 128-byte swizzle atom of bf16
// producer warps: 16 for d = 128, 8 for d = 64 (each warp flushes 32 TMEM columns)
template <int D> __host__ __device__ constexpr int prod_warps() { return D == 128 ? 16 : 8; }
template <int D> __host__ __device__ constexpr int pv_threads() { return (prod_warps<D>() + 1) * 32; }
constexpr int NSPLIT = 3;     // bf16 terms per probability
constexpr int ASLOTS = 2;     // A tiles in flight
constexpr int BSLOTS = 4;     // V / logit tiles in flight (prefetch distance 2)
constexpr int NACC = 2;       // chunk accumulators in TMEM (added two stages after a chunk ends)
constexpr int CH = 8;         // stages (of KS keys) accumulated in TMEM between flushes
constexpr int MAXRT = 32;     // rows per tile
constexpr uint32_t WAIT_POLLS = 1u << 20;  // polls before a wait gives up (well over a second)
constexpr int A_SPLIT_BYTES = TM * 128;            // 16 KB
constexpr int A_SLOT_BYTES = NSPLIT * A_SPLIT_BYTES;  // 48 KB

struct TcArgs {
    RowsDev R;
    const int32_t *k;
    int nb;
    fw_gap_out out;
    LongWs ws;
    int tiles_per_group;
    int RT;
    // the group vote (vmass != NULL): one kept set per group, key j kept by
    // budget b when key(G_j) > vthr[b] or (key(G_j) == vthr[b] and j <= vtidx[b]);
    // the budgets are vs (per group), ws.M / ws.Z the rows' softmax statistics
    const float *vmass;     // [groups][vmstride] summed masses G
    int64_t vmstride;
    const uint32_t *vthr;   // [groups][nb]
    const int32_t *vtidx;   // [groups][nb] (-1: budget out of range)
    const int32_t *vs;      // [groups][nb]
    const int32_t *vgflag;  // [groups] nonzero: a logit of the group is not finite
};

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, uint32_t src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async4(uint32_t dst, const void *src, uint32_t src_bytes)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait2() { asm volatile("cp.async.wait_group 2;" ::: "memory"); }

__device__ __forceinline__ uint32_t bf16_bits_rn(float x)
{
    return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(x));
}

template <int D>
__global__ void __launch_bounds__(pv_threads<D>(), 1) k_long_pv_tc(const TcArgs a)
{
    constexpr int PW = prod_warps<D>();
    constexpr int NT = pv_threads<D>();
    constexpr int NPROD = PW * 32;
    constexpr int TPR = NPROD / MAXRT;  // producer threads per row
    constexpr int KPTH = KS / TPR;      // keys per producer thread and stage (4 or 8)
    constexpr int B_SLOT_BYTES = D * 128;  // KS keys x D bf16
    constexpr int MCOL = NACC * D;  // first TMEM column of the band-mass accumulators (16 per buffer)
    constexpr uint32_t TCOLS = NACC * (D + 16) <= 256 ? 256u : 512u;  // TMEM columns (a power of two)
    constexpr int NC = D / 8;              // 16-byte chunks per V row
    extern __shared__ uint8_t smraw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~(uintptr_t)1023);
    uint8_t *sOnes = sm;                               // [16 x 128 B] bf16 ones: B of the band-mass MMA
    uint8_t *sA = sm + 2048;                           // [ASLOTS][NSPLIT][TM x 128 B]
    uint8_t *sB = sA + ASLOTS * A_SLOT_BYTES;          // [BSLOTS][D/64][KS x 128 B]
    float *sL = reinterpret_cast<float *>(sB + BSLOTS * B_SLOT_BYTES);  // [BSLOTS][RT][KS] raw logits
    float *acc = reinterpret_cast<float *>(sA);       // epilogue: [TM][D + 1]
    __shared__ __align__(8) uint64_t full[BSLOTS], empty[BSLOTS], accfree[NACC];
    __shared__ uint32_t s_taddr;
    __shared__ int s_err;
    __shared__ float rowM[MAXRT], rowZi[MAXRT];
    __shared__ uint32_t rtk[MAXRT][4];
    __shared__ int32_t rti[MAXRT][4];
    __shared__ int rok[MAXRT];
    __shared__ float bmass[MAXRT][5];

    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int nb = a.nb, nbb = nb + 1, RT = a.RT;
    const int64_t g = blockIdx.x / a.tiles_per_group;
    const int tile = (int)(blockIdx.x - g * a.tiles_per_group);
    const int r0 = tile * RT;
    const int nr = min(RT, a.R.R - r0);
    const int n = a.R.n[g];
    const uint16_t *V = reinterpret_cast<const uint16_t *>(a.R.v) + a.R.v_off[g];
    const float *LG = a.R.logits + a.R.logit_off[g];
    // rows start on 16-byte boundaries: logit copies of 16 bytes
    const bool lg16 = (n & 3) == 0 && (reinterpret_cast<uintptr_t>(LG) & 15) == 0;
    const int nst = (n + KS - 1) / KS;

    if (tid < MAXRT) {
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
    }
    if (tid == 0) {
        s_err = 0;
        for (int s = 0; s < BSLOTS; ++s) {
            tc::mbar_init(&full[s], NPROD);
            tc::mbar_init(&empty[s], 1);
        }
        for (int x = 0; x < NACC; ++x) tc::mbar_init(&accfree[x], NPROD);
        tc::mbar_init_fence();
    }
    // rows of A past nbb * RT stay zero in every slot; the ones tile is
    // constant (any swizzle of it reads 1.0)
    for (int e = tid; e < 2048 / 16; e += NT)
        reinterpret_cast<uint4 *>(sOnes)[e] = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
    if (tid < MAXRT)
        for (int b = 0; b < 5; ++b) bmass[tid][b] = 0.f;
    for (int e = tid; e < ASLOTS * NSPLIT * TM * 8; e += NT) {
        const int m = (e / 8) % TM;
        if (m >= nbb * RT) reinterpret_cast<uint4 *>(sA)[e] = make_uint4(0u, 0u, 0u, 0u);
    }
    tc::fence_async_smem();
    if (wid == PW) tc::tmem_alloc(&s_taddr, TCOLS);  // NACC stage accumulators
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t taddr = s_taddr;

    if (wid == PW) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_bf16_f32(TM, D, false, true);
            constexpr uint32_t idesc_m = tc::idesc_bf16_f32(TM, 16, false, false);
            const uint32_t a0 = tc::smem_u32(sA), b0 = tc::smem_u32(sB), o0 = tc::smem_u32(sOnes);
            bool ok = true;
            for (int it = 0; it < nst && ok; ++it) {
                const int bs = it % BSLOTS, as = it % ASLOTS;
                ok = tc::mbar_wait(&full[bs], (uint32_t)(it / BSLOTS) & 1u, WAIT_POLLS);
                // chunk c = it / CH accumulates in buffer c % NACC, last read by the
                // producers when they flushed chunk c - NACC
                const int ch = it / CH;
                if (ok && it % CH == 0 && ch >= NACC)
                    ok = tc::mbar_wait(&accfree[ch % NACC], (uint32_t)((ch - NACC) / NACC) & 1u, WAIT_POLLS);
                if (!ok) break;
                tc::fence_after_sync();
                const uint32_t dacc = taddr + (uint32_t)(((it / CH) % NACC) * D);
                const uint32_t dmass = taddr + (uint32_t)(MCOL + ((it / CH) % NACC) * 16);
                const bool fresh = it % CH == 0;  // first stage of a chunk overwrites the buffer
#pragma unroll
                for (int ks = 0; ks < KS / 16; ++ks) {
                    const uint64_t bd = tc::sdesc_sw128(b0 + bs * B_SLOT_BYTES + ks * 2048, KS * 128, 1024);
#pragma unroll
                    for (int sp = 0; sp < NSPLIT; ++sp) {
                        const uint64_t ad =
                            tc::sdesc_sw128(a0 + as * A_SLOT_BYTES + sp * A_SPLIT_BYTES + ks * 32, 16, 1024);
                        tc::mma_bf16(dacc, ad, bd, idesc, !fresh || ks > 0 || sp > 0);
                        // band masses: the same A tile times a K x 16 tile of ones
                        tc::mma_bf16(dmass, ad, tc::sdesc_sw128(o0 + ks * 32, 16, 1024), idesc_m,
                                     !fresh || ks > 0 || sp > 0);
                    }
                }
                tc::commit(&empty[bs]);
            }
            if (!ok) atomicOr(&s_err, 1);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ producers
        const int ptid = tid;                       // 0..NPROD-1
        const int rr0 = ptid / TPR;                 // the row handled (tiles have at most 32 rows)
        const int kc = (ptid % TPR) * KPTH / 8;     // 8-key chunk of the stage
        const int hk = (ptid % TPR) * KPTH % 8;     // first key of this thread in the chunk
        bool ok = true;
        const uint32_t bbase = tc::smem_u32(sB), lbase = tc::smem_u32(sL);
        // this thread's accumulator entries: TMEM lane 32 (wid % 4) + lane, the
        // 32 columns of part wid / 4
        const int quarter = wid & 3, part = wid >> 2;
        float racc[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) racc[i] = 0.f;
        float rmass = 0.f;  // band mass of TMEM lane 32 quarter + lane (warps of part 0)
        // stage st closes its chunk: the chunk's buffer is added once its MMAs completed
        auto chunk_end = [&](int st) { return st % CH == CH - 1 || st == nst - 1; };
        auto flush = [&](int st) {
            if (ok) ok = tc::mbar_wait(&empty[st % BSLOTS], (uint32_t)(st / BSLOTS) & 1u, WAIT_POLLS);
            tc::fence_after_sync();
            const uint32_t base =
                taddr + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(((st / CH) % NACC) * D + part * 32);
            float v[32];
            tc::ld32(base, v);
#pragma unroll
            for (int i = 0; i < 32; ++i) racc[i] += v[i];
            if (part == 0)
                rmass += tc::ld1(taddr + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(MCOL + ((st / CH) % NACC) * 16));
            tc::fence_before_sync();
            tc::mbar_arrive(&accfree[(st / CH) % NACC]);
        };
        auto issue = [&](int st) {  // cp.async of stage st's V tile and this thread's logits
            if (st < nst) {
                const int bs = st % BSLOTS, j0 = st * KS;
                for (int e = ptid; e < KS * NC; e += NPROD) {
                    const int kk = e / NC, nc = e % NC;
                    const int j = j0 + kk;
                    const int n2 = nc >> 3, c = nc & 7;
                    const uint32_t dst = bbase + bs * B_SLOT_BYTES + n2 * (KS * 128) + (kk >> 3) * 1024 +
                                         (kk & 7) * 128 + ((c ^ (kk & 7)) << 4);
                    const bool in = j < n;
                    cp_async16(dst, V + (int64_t)(in ? j : 0) * D + nc * 8, in ? 16u : 0u);
                }
                for (int r = rr0; r < RT; r += 32) {
                    const bool live = r < nr && rok[r];
                    const float *lrow = LG + (int64_t)(r0 + (live ? r : 0)) * n;
                    const uint32_t ldst = lbase + ((bs * RT + r) * KS + kc * 8 + hk) * 4;
                    if (lg16) {  // 16-byte copies, zero-filled past the row's end
#pragma unroll
                        for (int h = 0; h < KPTH / 4; ++h) {
                            const int j = j0 + kc * 8 + hk + 4 * h;
                            const int nv = live ? min(max(n - j, 0), 4) : 0;
                            cp_async16(ldst + 16 * h, lrow + (nv > 0 ? j : 0), 4u * (uint32_t)nv);
                        }
                    } else {
#pragma unroll
                        for (int u = 0; u < KPTH; ++u) {
                            const int j = j0 + kc * 8 + hk + u;
                            const bool in = live && j < n;
                            cp_async4(ldst + 4 * u, lrow + (in ? j : 0), in ? 4u : 0u);
                        }
                    }
                }
            }
            cp_async_commit();
        };
        // this thread's row: thresholds, softmax statistics and the band rows of its chunk
        const bool live = rr0 < nr && rok[rr0];
        const float Mr = live ? rowM[rr0] : 0.f, Zr = live ? rowZi[rr0] : 0.f;
        // thresholds as floats: key > T <=> x > xT and key == T <=> x == xT
        // for finite logits (order keys fold -0 onto +0, as float compares do)
        float mxt[4];
        int mti[4];
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const uint32_t tk = live ? rtk[rr0][b] : 0u;
            mxt[b] = __uint_as_float((tk & 0x80000000u) ? (tk & 0x7fffffffu) : ~tk);
            mti[b] = live ? rti[rr0][b] : -1;
        }
        uint32_t boff[5];
#pragma unroll
        for (int b = 0; b < 5; ++b) {
            const int m = b * RT + rr0;
            boff[b] = (uint32_t)((m >> 3) * 1024 + (m & 7) * 128 + ((kc ^ (m & 7)) << 4));
        }
        issue(0);
        issue(1);
        for (int it = 0; it < nst; ++it) {
            const int bs = it % BSLOTS, as = it % ASLOTS;
            // the V / logit slot of stage it + 2 and the A slot of stage it were
            // last read by the MMAs of stage it - 2
            if (ok && it >= 2) {
                const int pst = it - 2;
                ok = tc::mbar_wait(&empty[pst % BSLOTS], (uint32_t)(pst / BSLOTS) & 1u, WAIT_POLLS);
            }
            issue(it + 2);
            cp_async_wait2();  // this thread's copies of stage it are in shared memory
            uint8_t *aslot = sA + as * A_SLOT_BYTES;
            const int j0 = it * KS;
            if (rr0 < RT) {  // (threads past the tile's rows have no band rows)
                const float *lr = sL + (bs * RT + rr0) * KS + kc * 8 + hk;
                // this thread's KPTH keys of its row: mass, band and three bf16
                // terms (keys past the row's end or in a dead row get mass 0)
                float xs[KPTH];
#pragma unroll
                for (int q = 0; q < KPTH / 4; ++q) {
                    const float4 x4 = *reinterpret_cast<const float4 *>(lr + 4 * q);
                    xs[4 * q] = x4.x, xs[4 * q + 1] = x4.y, xs[4 * q + 2] = x4.z, xs[4 * q + 3] = x4.w;
                }
                uint32_t h16[KPTH], m16[KPTH], l16[KPTH];
                int bdv[KPTH];
#pragma unroll
                for (int u = 0; u < KPTH; ++u) {
                    const int j = j0 + kc * 8 + hk + u;
                    const float x = xs[u];
                    const float p = (live && j < n) ? __expf(x - Mr) * Zr : 0.f;
                    int bd = 0;
#pragma unroll
                    for (int b = 0; b < 4; ++b)
                        if (b < nb) bd += !(x > mxt[b] || (x == mxt[b] && j <= mti[b]));
                    bdv[u] = bd;
                    h16[u] = bf16_bits_rn(p);
                    const float r1 = p - __uint_as_float(h16[u] << 16);
                    m16[u] = bf16_bits_rn(r1);
                    l16[u] = bf16_bits_rn(r1 - __uint_as_float(m16[u] << 16));
                }
                // one vector per (band row, term): each key's terms in its own
                // band's row, zeros in the others.  Keys 2q and 2q + 1 share a
                // 32-bit word; a 2 x 16-bit compare of their bands gives the mask.
                uint32_t ph[KPTH / 2], pm[KPTH / 2], pl[KPTH / 2], pb[KPTH / 2];
#pragma unroll
                for (int q = 0; q < KPTH / 2; ++q) {
                    ph[q] = h16[2 * q] | (h16[2 * q + 1] << 16);
                    pm[q] = m16[2 * q] | (m16[2 * q + 1] << 16);
                    pl[q] = l16[2 * q] | (l16[2 * q + 1] << 16);
                    pb[q] = (uint32_t)bdv[2 * q] | ((uint32_t)bdv[2 * q + 1] << 16);
                }
#pragma unroll
                for (int b = 0; b < 5; ++b) {
                    if (b >= nbb) continue;
                    uint32_t wh[KPTH / 2], wm[KPTH / 2], wl[KPTH / 2];
#pragma unroll
                    for (int q = 0; q < KPTH / 2; ++q) {
                        const uint32_t msk = __vcmpeq2(pb[q], (uint32_t)b * 0x00010001u);
                        wh[q] = ph[q] & msk;
                        wm[q] = pm[q] & msk;
                        wl[q] = pl[q] & msk;
                    }
                    uint8_t *dst = aslot + boff[b] + 2 * hk;
                    if constexpr (KPTH == 8) {
                        *reinterpret_cast<uint4 *>(dst) = make_uint4(wh[0], wh[1], wh[2], wh[3]);
                        *reinterpret_cast<uint4 *>(dst + A_SPLIT_BYTES) = make_uint4(wm[0], wm[1], wm[2], wm[3]);
                        *reinterpret_cast<uint4 *>(dst + 2 * A_SPLIT_BYTES) = make_uint4(wl[0], wl[1], wl[2], wl[3]);
                    } else {
                        *reinterpret_cast<uint2 *>(dst) = make_uint2(wh[0], wh[1]);
                        *reinterpret_cast<uint2 *>(dst + A_SPLIT_BYTES) = make_uint2(wm[0], wm[1]);
                        *reinterpret_cast<uint2 *>(dst + 2 * A_SPLIT_BYTES) = make_uint2(wl[0], wl[1]);
                    }
                }
            }
            tc::fence_async_smem();
            tc::mbar_arrive(&full[bs]);
            if (it >= 2 && chunk_end(it - 2)) flush(it - 2);
        }
        for (int st = nst - 2 < 0 ? 0 : nst - 2; st < nst; ++st)
            if (chunk_end(st)) flush(st);
        // band masses from the ones MMA: TMEM lane m = (band, row) = (m / RT, m % RT)
        if (part == 0) {
            const int m = quarter * 32 + lane;
            if (m < nbb * RT) bmass[m % RT][m / RT] = rmass;
        }
        // accumulators -> shared for the per-row epilogue (the stage buffers are idle now)
        if (!ok) atomicOr(&s_err, 1);
        {
            const int m = quarter * 32 + lane;
#pragma unroll
            for (int i = 0; i < 32; ++i) acc[m * (D + 1) + part * 32 + i] = racc[i];
        }
    }
    tc::fence_before_sync();
    __syncthreads();
    if (wid == PW) {
        tc::fence_after_sync();
        tc::tmem_dealloc(taddr, TCOLS);
        return;
    }
    // --------------------------------------------------------------- epilogue
    const bool failed = s_err != 0;
    constexpr int CPT = D / 32;
    for (int r = wid; r < nr; r += PW) {
        const int64_t row = g * a.R.R + r0 + r;
        if (failed) {
            if (lane == 0 && a.out.row_status) a.out.row_status[row] = FW_ERR_TIMEOUT;
            continue;
        }
        if (!rok[r]) continue;
        float S[5][CPT];
#pragma unroll
        for (int b = 0; b < 5; ++b)
#pragma unroll
            for (int t = 0; t < CPT; ++t)
                S[b][t] = b < nbb ? acc[(b * RT + r) * (D + 1) + lane + 32 * t] : 0.f;
        if (a.out.o) {
#pragma unroll
            for (int t = 0; t < CPT; ++t) {
                float o = 0.f;
#pragma unroll
                for (int b = 0; b < 5; ++b) o += S[b][t];
                a.out.o[row * D + lane + 32 * t] = o;
            }
        }
        for (int b = 0; b < nb; ++b) {
            const int kb = a.k[row * nb + b];
            int sb = 0;
            for (int b2 = 0; b2 < nb; ++b2) {
                const int k2 = a.k[row * nb + b2];
                sb += (k2 < kb) || (k2 == kb && b2 < b);
            }
            float PA = 0.f, PC = 0.f;
            for (int q = 0; q < 5; ++q) {
                if (q <= sb) PA += bmass[r][q];
                else PC += bmass[r][q];
            }
            float s2 = 0.f;
            float NAv[CPT];
#pragma unroll
            for (int t = 0; t < CPT; ++t) {
                float NA = 0.f, NC = 0.f;
#pragma unroll
                for (int q = 0; q < 5; ++q) {
                    if (q <= sb) NA += S[q][t];
                    else NC += S[q][t];
                }
                NAv[t] = NA;
                const float diff = PC * NA - PA * NC;  // p(A) (m_A - mu)
                s2 = fmaf(diff, diff, s2);
            }
            s2 = warp_sum(s2);
            if (lane == 0) {
                const float phi = sqrtf(s2);
                a.out.gap[row * nb + b] = phi / PA;
                a.out.dropped[row * nb + b] = PC;
                if (a.out.phi) a.out.phi[row * nb + b] = phi;
            }
            if (a.out.o_kept)
#pragma unroll
                for (int t = 0; t < CPT; ++t) a.out.o_kept[(row * nb + b) * D + lane + 32 * t] = NAv[t] / PA;
        }
    }
}

// ---------------------------------------------------------------------------
// The same P.V with one copy warp: V tiles arrive by TMA (64 keys x 64 dims
// boxes, 128-byte swizzle: the MN-major operand layout) and the stage's
// logits (64 per row) by 16-byte cp.async, half a warp per row, so the
// producer warps only build A.  (One bulk copy per 256-byte logit row was
// tried first: 32 small TMA requests per stage kept the stage time near
// 1.3 us, about three times the MMA time.)  Warp 0 copies, warp 1 issues the
// MMAs, the other warps produce: a thread takes KPTH consecutive keys of one
// row (NB budgets known at compile time) and writes one vector per (band row,
// term).  Stages whose V rows would cross the end of the group's block (the
// partial last stage, or a block not aligned to whole rows) go through
// per-thread cp.async with zero fill instead, and logit rows that are not
// 16-byte aligned (n not a multiple of 4, misaligned base) through 4-byte
// cp.async; the barrier tracks every kind.
template <int D> __host__ __device__ constexpr int pvm_pw() { return D == 128 ? 16 : 8; }  // producer warps
template <int D> __host__ __device__ constexpr int pvm_nt() { return (pvm_pw<D>() + 2) * 32; }
constexpr int PVM_BS = 3;                      // copy slots (V + ones + logits)

__device__ __forceinline__ uint32_t cvt_bf16x2(float hi_elem, float lo_elem)
{
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi_elem), "f"(lo_elem));
    return r;
}
__device__ __forceinline__ void cp_async_mbar_arrive(uint64_t *bar)
{
    asm volatile("cp.async.mbarrier.arrive.shared.b64 [%0];" ::"r"(tc::smem_u32(bar)) : "memory");
}

template <int D, int NB>
__global__ void __launch_bounds__(pvm_nt<D>(), 1) k_long_pv_tma(const __grid_constant__ CUtensorMap tmV, const TcArgs a)
{
    constexpr int NBB = NB + 1;                 // bands
    constexpr int RT = TM / NBB < MAXRT ? TM / NBB : MAXRT;
    constexpr int PW = pvm_pw<D>();
    constexpr int NT = pvm_nt<D>();
    constexpr int NPROD = PW * 32;
    constexpr int TPR = NPROD / MAXRT;          // producer threads per row
    constexpr int KPTH = KS / TPR;              // keys per producer thread and stage (4 or 8)
    constexpr int NVBOX = D / 64;               // 64-dim groups of V
    constexpr int NG = NVBOX + 1;               // ... and one group of ones (the band masses)
    constexpr int B_SLOT_BYTES = NG * KS * 128;
    constexpr int DN = D + 16;                  // MMA N: the value dims, then 16 columns of masses
    constexpr uint32_t TCOLS = NACC * DN <= 256 ? 256u : 512u;
    constexpr int NC = D / 8;
    constexpr int FCOLS = D / (PW / 4);         // accumulator columns flushed per warp (32)
    extern __shared__ uint8_t smraw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~(uintptr_t)1023);
    uint8_t *sA = sm;                                     // [ASLOTS][NSPLIT][TM x 128 B]
    uint8_t *sB = sA + ASLOTS * A_SLOT_BYTES;             // [PVM_BS][NG][64 keys x 128 B]
    float *sL = reinterpret_cast<float *>(sB + PVM_BS * B_SLOT_BYTES);  // [PVM_BS][32][64]
    float *sG = sL + PVM_BS * MAXRT * KS;                 // [PVM_BS][64] the vote's G
    float *acc = reinterpret_cast<float *>(sA);           // epilogue: [TM][D + 1]
    __shared__ __align__(8) uint64_t fullB[PVM_BS], freeB[PVM_BS], fullA[ASLOTS], freeA[ASLOTS], accfree[NACC];
    __shared__ uint32_t s_taddr;
    __shared__ int s_err;
    __shared__ float rowM[MAXRT], rowZi[MAXRT];
    __shared__ uint32_t rtk[MAXRT][4];
    __shared__ int32_t rti[MAXRT][4];
    __shared__ int rok[MAXRT];
    __shared__ float bmass[MAXRT][5];
    __shared__ uint32_t vT[4];   // the vote's thresholds, budgets ascending
    __shared__ int32_t vL[4];
    __shared__ int rstat[MAXRT];

    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int64_t g = blockIdx.x / a.tiles_per_group;
    const int tile = (int)(blockIdx.x - g * a.tiles_per_group);
    const int r0 = tile * RT;
    const int nr = min(RT, a.R.R - r0);
    const int n = a.R.n[g];
    const int64_t voff = a.R.v_off[g];
    const uint16_t *V = reinterpret_cast<const uint16_t *>(a.R.v) + voff;
    const float *LG = a.R.logits + a.R.logit_off[g];
    const bool vote = a.vmass != nullptr;
    const float *GB = vote ? a.vmass + g * a.vmstride : nullptr;
    const bool vrows = voff % D == 0;  // the block starts on a whole row of the V tensor map
    const bool lbulk = (n & 3) == 0 && (reinterpret_cast<uintptr_t>(LG) & 15) == 0;
    const int nst = (n + KS - 1) / KS;

    if (tid < MAXRT) {
        const int r = tid;
        rok[r] = 0;
        if (r < nr) {
            const int64_t row = g * a.R.R + r0 + r;
            if (vote) {
                bool inv = false;
                for (int b = 0; b < NB; ++b) inv |= a.vtidx[g * NB + b] < 0;
                rstat[r] = a.vgflag[g] ? FW_ERR_NONFINITE : (inv ? FW_ERR_INVALID_ARG : FW_OK);
                rok[r] = rstat[r] == FW_OK;
            } else {
                rok[r] = a.ws.status[row] == FW_OK;
            }
            rowM[r] = a.ws.M[row];
            rowZi[r] = 1.f / a.ws.Z[row];
            for (int b = 0; b < 4; ++b) {
                rtk[r][b] = b < NB && !vote ? a.ws.tk[row * NB + b] : 0u;
                rti[r][b] = b < NB && !vote ? a.ws.ti[row * NB + b] : -1;
            }
        }
        for (int b = 0; b < 5; ++b) bmass[r][b] = 0.f;
    }
    if (vote && tid == MAXRT) {  // the group's budgets in ascending order (the sets are nested along it)
        int sv[4], ov[4];
        for (int b = 0; b < 4; ++b) {
            sv[b] = b < NB ? a.vs[g * NB + b] : 0x7fffffff;
            ov[b] = b;
        }
        for (int x = 1; x < NB; ++x)
            for (int y = x; y > 0 && sv[y] < sv[y - 1]; --y) {
                const int t1 = sv[y], t2 = ov[y];
                sv[y] = sv[y - 1], ov[y] = ov[y - 1];
                sv[y - 1] = t1, ov[y - 1] = t2;
            }
        for (int b = 0; b < 4; ++b) {
            vT[b] = b < NB ? a.vthr[g * NB + ov[b]] : 0u;
            vL[b] = b < NB ? a.vtidx[g * NB + ov[b]] : -1;
        }
    }
    if (tid == 0) {
        s_err = 0;
        for (int x = 0; x < PVM_BS; ++x) {
            tc::mbar_init(&fullB[x], 1);
            tc::mbar_init(&freeB[x], PW + 1);
        }
        for (int x = 0; x < ASLOTS; ++x) {
            tc::mbar_init(&fullA[x], PW);
            tc::mbar_init(&freeA[x], 1);
        }
        for (int x = 0; x < NACC; ++x) tc::mbar_init(&accfree[x], PW);
        tc::mbar_init_fence();
    }
    // the ones group of every copy slot (constant; any swizzle of it reads 1.0)
    for (int e = tid; e < PVM_BS * KS * 8; e += NT) {
        const int slot = e / (KS * 8), q = e % (KS * 8);
        reinterpret_cast<uint4 *>(sB + slot * B_SLOT_BYTES + NVBOX * (KS * 128))[q] =
            make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
    }
    // rows of A past NBB * RT stay zero in every slot
    for (int e = tid; e < ASLOTS * NSPLIT * TM * 8; e += NT) {
        const int m = (e / 8) % TM;
        if (m >= NBB * RT) reinterpret_cast<uint4 *>(sA)[e] = make_uint4(0u, 0u, 0u, 0u);
    }
    tc::fence_async_smem();
    if (wid == 1) tc::tmem_alloc(&s_taddr, TCOLS);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t taddr = s_taddr;

    if (wid == 0) {
        // ---------------------------------------------------------- copies
        const uint32_t bbase = tc::smem_u32(sB), lbase = tc::smem_u32(sL);
        const uint32_t livemask = __ballot_sync(FW_FULL, lane < nr && rok[lane]);
        const int lc = lane & 15, lh = lane >> 4;  // 16-byte chunk of a logit row, row parity
        int issued = 0;
        bool ok = true;
        for (int it = 0; it < nst; ++it) {
            const int bs = it % PVM_BS, j0 = it * KS;
            if (it >= PVM_BS) {
                if (lane == 0) ok = tc::mbar_wait(&freeB[bs], (uint32_t)((it / PVM_BS) - 1) & 1u, WAIT_POLLS);
                ok = __shfl_sync(FW_FULL, ok, 0);
                if (!ok) break;
            }
            const int kn = min(KS, n - j0);  // keys of this stage
            const bool vtma = vrows && kn == KS;
            const bool live_row = (livemask >> lane) & 1u;
            // (1) the per-thread copies, each lane's tracked by the barrier: its
            // pending count rises now and falls when they land, so the phase
            // cannot complete before them whatever the order of what follows
            if (!vtma) {  // V rows past the block's end are zero-filled
                for (int e = lane; e < KS * NC; e += 32) {
                    const int kk = e / NC, nc = e % NC;
                    const int n2 = nc >> 3, c = nc & 7;
                    const uint32_t dst = bbase + bs * B_SLOT_BYTES + n2 * (KS * 128) + (kk >> 3) * 1024 +
                                         (kk & 7) * 128 + ((c ^ (kk & 7)) << 4);
                    const bool in = kk < kn;
                    cp_async16(dst, V + (int64_t)(in ? j0 + kk : 0) * D + nc * 8, in ? 16u : 0u);
                }
            }
            if (lbulk) {  // 16-byte copies, half a warp per row (kn is a multiple of 4)
                const bool cin = lc * 4 < kn;
                for (int rp = 0; rp < nr; rp += 2) {
                    const int r = rp + lh;
                    if ((livemask >> r) & 1u)
                        cp_async16(lbase + (uint32_t)(((bs * MAXRT + r) * KS + lc * 4) * 4),
                                   LG + (int64_t)(r0 + r) * n + j0 + (cin ? lc * 4 : 0), cin ? 16u : 0u);
                }
            } else if (live_row) {
                const uint32_t d0 = lbase + (uint32_t)((bs * MAXRT + lane) * KS * 4);
                const float *lsrc = LG + (int64_t)(r0 + lane) * n + j0;
                for (int u = 0; u < kn; ++u) cp_async4(d0 + 4 * u, lsrc + u, 4u);
            }
            if (vote)  // the stage's summed masses (zero past the row)
                for (int e = lane; e < KS; e += 32)
                    cp_async4(tc::smem_u32(sG + bs * KS + e), GB + j0 + (e < kn ? e : 0), e < kn ? 4u : 0u);
            cp_async_mbar_arrive(&fullB[bs]);
            // (2) the barrier's one expected arrival, with the bytes of the V boxes
            const uint32_t tx = vtma ? (uint32_t)(NVBOX * 64 * 128) : 0u;
            __syncwarp();
            if (lane == 0) tc::mbar_arrive_expect_tx(&fullB[bs], tx);
            __syncwarp();
            // (3) the V boxes by TMA
            if (vtma && lane == 0)
                for (int h = 0; h < NVBOX; ++h)
                    tc::tma_load_2d(sB + bs * B_SLOT_BYTES + h * (KS * 128), &tmV, 64 * h, (int32_t)(voff / D + j0),
                                    &fullB[bs]);
            ++issued;
        }
        if (!ok && lane == 0) atomicOr(&s_err, 1);
        // the copies still in flight land before the CTA moves on
        if (lane == 0)
            for (int it = issued - PVM_BS < 0 ? 0 : issued - PVM_BS; it < issued; ++it)
                if (!tc::mbar_wait(&fullB[it % PVM_BS], (uint32_t)(it / PVM_BS) & 1u, WAIT_POLLS)) atomicOr(&s_err, 1);
        __syncwarp();
    } else if (wid == 1) {
        // -------------------------------------------------------------- MMA
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_bf16_f32(TM, DN, false, true);
            // descriptors of slot 0, k-step 0, term 0; the others differ by an
            // address offset (>> 4) in the start field, which never carries out
            // of it (shared memory stays below 256 KB)
            const uint64_t ad0 = tc::sdesc_sw128(tc::smem_u32(sA), 16, 1024);
            const uint64_t bd0 = tc::sdesc_sw128(tc::smem_u32(sB), KS * 128, 1024);
            bool ok = true;
            int last = -1;
            for (int it = 0; it < nst && ok; ++it) {
                const int bs = it % PVM_BS, as = it % ASLOTS;
                ok = tc::mbar_wait(&fullB[bs], (uint32_t)(it / PVM_BS) & 1u, WAIT_POLLS);
                if (ok) ok = tc::mbar_wait(&fullA[as], (uint32_t)(it / ASLOTS) & 1u, WAIT_POLLS);
                const int ch = it / CH;
                if (ok && it % CH == 0 && ch >= NACC)
                    ok = tc::mbar_wait(&accfree[ch % NACC], (uint32_t)((ch - NACC) / NACC) & 1u, WAIT_POLLS);
                if (!ok) break;
                tc::fence_after_sync();
                const uint32_t dacc = taddr + (uint32_t)((ch % NACC) * DN);
                const bool fresh = it % CH == 0;
                const uint64_t abase = ad0 + (uint64_t)((as * A_SLOT_BYTES) >> 4);
                const uint64_t bbs = bd0 + (uint64_t)((bs * B_SLOT_BYTES) >> 4);
#pragma unroll
                for (int ks = 0; ks < KS / 16; ++ks) {
                    const uint64_t bd = bbs + (uint64_t)((ks * 2048) >> 4);
#pragma unroll
                    for (int sp = 0; sp < NSPLIT; ++sp)
                        tc::mma_bf16(dacc, abase + (uint64_t)((sp * A_SPLIT_BYTES + ks * 32) >> 4), bd, idesc,
                                     !fresh || ks > 0 || sp > 0);
                }
                tc::commit(&freeA[as]);
                tc::commit(&freeB[bs]);
                last = it;
            }
            if (!ok) atomicOr(&s_err, 1);
            if (last >= 0 && !tc::mbar_wait(&freeA[last % ASLOTS], (uint32_t)(last / ASLOTS) & 1u, WAIT_POLLS))
                atomicOr(&s_err, 1);
        }
        __syncwarp();
    } else {
        // --------------------------------------------------------- producers
        const int pw = wid - 2;                  // 0..PW-1
        const int ptid = tid - 64;               // 0..NPROD-1
        const int rr = ptid / TPR;               // row of the tile (0..31)
        const int kq = ptid % TPR;               // this thread's KPTH keys of the stage
        const int kc = kq * KPTH / 8, hk = (kq * KPTH) % 8;  // 8-key chunk and first key in it
        const int quarter = wid & 3, part = pw >> 2;  // TMEM lanes / columns this warp flushes
        float racc[FCOLS];
#pragma unroll
        for (int i = 0; i < FCOLS; ++i) racc[i] = 0.f;
        float rmass = 0.f;
        const bool live = rr < nr && rok[rr];
        const float Mr = live ? rowM[rr] : 0.f, Zr = live ? rowZi[rr] : 0.f;
        float xt[NB];
        int tix[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const uint32_t tk = live ? rtk[rr][b] : 0u;
            xt[b] = __uint_as_float((tk & 0x80000000u) ? (tk & 0x7fffffffu) : ~tk);
            tix[b] = live ? rti[rr][b] : -1;
        }
        uint32_t boff[NBB];
#pragma unroll
        for (int b = 0; b < NBB; ++b) {
            const int m = b * RT + rr;
            boff[b] = (uint32_t)((m >> 3) * 1024 + (m & 7) * 128 + ((kc ^ (m & 7)) << 4) + 2 * hk);
        }
        bool ok = true;
        auto chunk_end = [&](int st) { return st % CH == CH - 1 || st == nst - 1; };
        auto flush = [&](int st) {
            tc::fence_after_sync();
            const int buf = (st / CH) % NACC;
            const uint32_t lanes = (uint32_t)(quarter * 32) << 16;
            float v[32];
            tc::ld32(taddr + lanes + (uint32_t)(buf * DN + part * FCOLS), v);
#pragma unroll
            for (int i = 0; i < FCOLS; ++i) racc[i] += v[i];
            if (part == 0) rmass += tc::ld1(taddr + lanes + (uint32_t)(buf * DN + D));
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&accfree[buf]);
        };
        for (int it = 0; it < nst; ++it) {
            const int bs = it % PVM_BS, as = it % ASLOTS, j0 = it * KS;
            if (ok) ok = tc::mbar_wait(&fullB[bs], (uint32_t)(it / PVM_BS) & 1u, WAIT_POLLS);
            // the A slot was last read by the MMAs of stage it - ASLOTS (which also
            // closes chunk it - ASLOTS for the flush below)
            if (ok && it >= ASLOTS) ok = tc::mbar_wait(&freeA[as], (uint32_t)((it / ASLOTS) - 1) & 1u, WAIT_POLLS);
            if (!ok) break;
            uint8_t *aslot = sA + as * A_SLOT_BYTES;
            if (rr < RT) {
                const float *lr = sL + (bs * MAXRT + rr) * KS + kq * KPTH;
                float xs[KPTH];
#pragma unroll
                for (int q = 0; q < KPTH / 4; ++q) {
                    const float4 x4 = *reinterpret_cast<const float4 *>(lr + 4 * q);
                    xs[4 * q] = x4.x, xs[4 * q + 1] = x4.y, xs[4 * q + 2] = x4.z, xs[4 * q + 3] = x4.w;
                }
                float pv[KPTH];
                uint32_t bdp[KPTH / 2];  // bands of keys 2q, 2q + 1 as 2 x 16 bits
                bool tie = false;
#pragma unroll
                for (int u = 0; u < KPTH; ++u) {
                    const int j = j0 + kq * KPTH + u;
                    const float x = xs[u];
                    pv[u] = (live && j < n) ? __expf(x - Mr) * Zr : 0.f;
                    int bd = 0;
                    if (vote) {
                        const uint32_t gk = order_key(sG[bs * KS + kq * KPTH + u]);
#pragma unroll
                        for (int b = 0; b < NB; ++b) bd += !(gk > vT[b] || (gk == vT[b] && j <= vL[b]));
                    } else {
#pragma unroll
                        for (int b = 0; b < NB; ++b) {
                            bd += x < xt[b];
                            tie |= x == xt[b];
                        }
                    }
                    if (u & 1) bdp[u >> 1] |= (uint32_t)bd << 16;
                    else bdp[u >> 1] = (uint32_t)bd;
                }
                if (tie) {  // a key equal to a threshold: its index decides (rare)
#pragma unroll
                    for (int u = 0; u < KPTH; ++u) {
                        const int j = j0 + kq * KPTH + u;
                        const float x = xs[u];
                        int bd = 0;
#pragma unroll
                        for (int b = 0; b < NB; ++b) bd += (x < xt[b]) | ((x == xt[b]) & (j > tix[b]));
                        const uint32_t sh = (u & 1) ? 16u : 0u;
                        bdp[u >> 1] = (bdp[u >> 1] & ~(0xffffu << sh)) | ((uint32_t)bd << sh);
                    }
                }
                // three bf16 terms per mass, two keys per 32-bit word (key 2q low)
                uint32_t ph[KPTH / 2], pm[KPTH / 2], pl[KPTH / 2];
#pragma unroll
                for (int q = 0; q < KPTH / 2; ++q) {
                    const float a0 = pv[2 * q], a1 = pv[2 * q + 1];
                    ph[q] = cvt_bf16x2(a1, a0);
                    const float e0 = a0 - __uint_as_float(ph[q] << 16), e1 = a1 - __uint_as_float(ph[q] & 0xffff0000u);
                    pm[q] = cvt_bf16x2(e1, e0);
                    const float f0 = e0 - __uint_as_float(pm[q] << 16), f1 = e1 - __uint_as_float(pm[q] & 0xffff0000u);
                    pl[q] = cvt_bf16x2(f1, f0);
                }
#pragma unroll
                for (int b = 0; b < NBB; ++b) {
                    uint32_t wh[KPTH / 2], wm[KPTH / 2], wl[KPTH / 2];
#pragma unroll
                    for (int q = 0; q < KPTH / 2; ++q) {
                        const uint32_t msk = __vcmpeq2(bdp[q], (uint32_t)b * 0x00010001u);
                        wh[q] = ph[q] & msk;
                        wm[q] = pm[q] & msk;
                        wl[q] = pl[q] & msk;
                    }
                    uint8_t *dst = aslot + boff[b];
                    if constexpr (KPTH == 8) {
                        *reinterpret_cast<uint4 *>(dst) = make_uint4(wh[0], wh[1], wh[2], wh[3]);
                        *reinterpret_cast<uint4 *>(dst + A_SPLIT_BYTES) = make_uint4(wm[0], wm[1], wm[2], wm[3]);
                        *reinterpret_cast<uint4 *>(dst + 2 * A_SPLIT_BYTES) = make_uint4(wl[0], wl[1], wl[2], wl[3]);
                    } else {
                        *reinterpret_cast<uint2 *>(dst) = make_uint2(wh[0], wh[1]);
                        *reinterpret_cast<uint2 *>(dst + A_SPLIT_BYTES) = make_uint2(wm[0], wm[1]);
                        *reinterpret_cast<uint2 *>(dst + 2 * A_SPLIT_BYTES) = make_uint2(wl[0], wl[1]);
                    }
                }
            }
            tc::fence_async_smem();
            __syncwarp();
            if (lane == 0) {
                tc::mbar_arrive(&fullA[as]);
                tc::mbar_arrive(&freeB[bs]);  // this warp has read the stage's logits
            }
            if (it >= ASLOTS && chunk_end(it - ASLOTS)) flush(it - ASLOTS);
        }
        // the last chunks: their MMAs complete before they are read
        for (int st = nst - ASLOTS < 0 ? 0 : nst - ASLOTS; st < nst && ok; ++st) {
            ok = tc::mbar_wait(&freeA[st % ASLOTS], (uint32_t)(st / ASLOTS) & 1u, WAIT_POLLS);
            if (ok && chunk_end(st)) flush(st);
        }
        if (!ok && lane == 0) atomicOr(&s_err, 1);
        const int m = quarter * 32 + lane;
        if (part == 0 && m < NBB * RT) bmass[m % RT][m / RT] = rmass;
        // accumulators -> shared for the per-row epilogue: every MMA has completed,
        // so the A slots (which acc overlays) are idle
#pragma unroll
        for (int i = 0; i < FCOLS; ++i) acc[m * (D + 1) + part * FCOLS + i] = racc[i];
    }
    tc::fence_before_sync();
    __syncthreads();
    if (wid == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(taddr, TCOLS);
    }
    if (wid < 2) return;
    // --------------------------------------------------------------- epilogue
    const bool failed = s_err != 0;
    constexpr int CPT = D / 32;
    for (int r = wid - 2; r < nr; r += PW) {
        const int64_t row = g * a.R.R + r0 + r;
        if (failed) {
            if (lane == 0 && a.out.row_status) a.out.row_status[row] = FW_ERR_TIMEOUT;
            continue;
        }
        if (vote && lane == 0 && a.out.row_status) a.out.row_status[row] = rstat[r];
        if (!rok[r]) {
            if (vote && lane < NB) {  // no set to score
                a.out.gap[row * NB + lane] = __int_as_float(0x7fc00000);
                if (a.out.dropped) a.out.dropped[row * NB + lane] = __int_as_float(0x7fc00000);
            }
            continue;
        }
        float S[NBB][CPT];
#pragma unroll
        for (int b = 0; b < NBB; ++b)
#pragma unroll
            for (int t = 0; t < CPT; ++t) S[b][t] = acc[(b * RT + r) * (D + 1) + lane + 32 * t];
        if (a.out.o) {
#pragma unroll
            for (int t = 0; t < CPT; ++t) {
                float o = 0.f;
#pragma unroll
                for (int b = 0; b < NBB; ++b) o += S[b][t];
                a.out.o[row * D + lane + 32 * t] = o;
            }
        }
        for (int b = 0; b < NB; ++b) {
            const int kb = vote ? a.vs[g * NB + b] : a.k[row * NB + b];
            int sb = 0;
            for (int b2 = 0; b2 < NB; ++b2) {
                const int k2 = vote ? a.vs[g * NB + b2] : a.k[row * NB + b2];
                sb += (k2 < kb) || (k2 == kb && b2 < b);
            }
            float PA = 0.f, PC = 0.f;
#pragma unroll
            for (int q = 0; q < NBB; ++q) {
                if (q <= sb) PA += bmass[r][q];
                else PC += bmass[r][q];
            }
            float s2 = 0.f;
            float NAv[CPT];
#pragma unroll
            for (int t = 0; t < CPT; ++t) {
                float NA = 0.f, NCs = 0.f;
#pragma unroll
                for (int q = 0; q < NBB; ++q) {
                    if (q <= sb) NA += S[q][t];
                    else NCs += S[q][t];
                }
                NAv[t] = NA;
                const float diff = PC * NA - PA * NCs;  // p(A) (m_A - mu)
                s2 = fmaf(diff, diff, s2);
            }
            s2 = warp_sum(s2);
            if (lane == 0) {
                const float phi = sqrtf(s2);
                a.out.gap[row * NB + b] = phi / PA;
                if (a.out.dropped) a.out.dropped[row * NB + b] = PC;
                if (a.out.phi) a.out.phi[row * NB + b] = phi;
            }
            if (a.out.o_kept)
#pragma unroll
                for (int t = 0; t < CPT; ++t) a.out.o_kept[(row * NB + b) * D + lane + 32 * t] = NAv[t] / PA;
        }
    }
}

// ---------------------------------------------------------------------------
// P.V for small groups (at most 8 rows share V, as under grouped-query
// attention): the same band-expanded products, transposed,
//   S^T[dim][(band, row)] = sum_j V[j][dim] P[(band, row)][j],
// so that the value dimension is the MMA's M (128: the d = 128 dims, or the
// d = 64 dims and 64 rows of zeros) and the NBB x RT (band, row) pairs its N
// (16, 32 or 48 columns).  With the (band, row) pairs on M, a group of 4 rows
// with one budget would fill 8 of the 128 tile rows and the tensor work would
// be 16 times the useful work; here it is at most 3 split terms x the
// padding of N, and the kernel streams V at the memory's pace.  The band
// masses are summed by the producers (compensated, in registers) instead of
// by a column of ones.  Warp 0 copies (V boxes by TMA, logits by cp.async),
// warp 1 issues the MMAs, warps 2..5 build P^T (K-major, 128-byte swizzle)
// and flush the TMEM chunk accumulators, each warp its 32 TMEM lanes (dims).
constexpr int TN_BS = 3;                 // copy slots (V + logits): small CTAs, three or four per SM
constexpr int TN_PW = 4;                 // producer / flush warps
constexpr int TN_NT = (TN_PW + 2) * 32;  // threads
template <int NB, int RT> __host__ __device__ constexpr int tn_cols() { return ((NB + 1) * RT + 15) / 16 * 16; }
template <int NB, int RT> __host__ __device__ constexpr uint32_t tn_tcols()
{
    return NACC * tn_cols<NB, RT>() <= 32 ? 32u : (NACC * tn_cols<NB, RT>() <= 64 ? 64u : 128u);
}

template <int D, int NB, int RT>
__global__ void __launch_bounds__(TN_NT, 3) k_long_pv_tn(const __grid_constant__ CUtensorMap tmV, const TcArgs a)
{
    constexpr int NBB = NB + 1;                 // bands
    constexpr int NP = NBB * RT;                // (band, row) pairs
    constexpr int N = tn_cols<NB, RT>();        // MMA N
    constexpr int NPROD = TN_PW * 32;
    constexpr int TPR = NPROD / RT;             // producer threads per row (32 or 16)
    constexpr int KPTH = KS / TPR;              // keys per producer thread and stage (2 or 4)
    constexpr int NVBOX = D / 64;               // 64-dim blocks of V
    // a V slot holds the d = 128 dims as two 64-row blocks of the M = 128
    // operand; for d = 64 it holds one, and every slot's second block is one
    // shared zero block behind the slots (each slot's descriptor points its
    // leading byte offset there)
    constexpr int V_SLOT = NVBOX * KS * 128;
    constexpr int P_TERM = N * 128;             // one split term of P^T: N rows x 64 keys
    constexpr int P_SLOT = NSPLIT * P_TERM;
    constexpr uint32_t TCOLS = tn_tcols<NB, RT>();
    constexpr int NC = D / 8;
    static_assert(KPTH == 2 || KPTH == 4, "producer layout");
    static_assert(NP * (D + 1) * 4 <= TN_BS * V_SLOT, "epilogue staging fits the V slots");
    extern __shared__ uint8_t smraw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~(uintptr_t)1023);
    uint8_t *sV = sm;                                     // [TN_BS][NVBOX][64 keys x 128 B] (+ zero block)
    uint8_t *sP = sV + TN_BS * V_SLOT + (NVBOX == 1 ? KS * 128 : 0);  // [ASLOTS][NSPLIT][N x 128 B]
    float *sL = reinterpret_cast<float *>(sP + ASLOTS * P_SLOT);  // [TN_BS][RT][64]
    float *sG = sL + TN_BS * RT * KS;                     // [TN_BS][64] the vote's G
    float *acc = reinterpret_cast<float *>(sV);           // epilogue: [NP][D + 1]
    __shared__ __align__(8) uint64_t fullB[TN_BS], freeB[TN_BS], fullA[ASLOTS], freeA[ASLOTS], accfree[NACC];
    __shared__ uint32_t s_taddr;
    __shared__ int s_err;
    __shared__ float rowM[RT], rowZi[RT];
    __shared__ uint32_t rtk[RT][4];
    __shared__ int32_t rti[RT][4];
    __shared__ int rok[RT];
    __shared__ float bmass[RT][5];
    __shared__ uint32_t vT[4];   // the vote's thresholds, budgets ascending
    __shared__ int32_t vL[4];
    __shared__ int rstat[RT];

    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int64_t g = blockIdx.x / a.tiles_per_group;
    const int tile = (int)(blockIdx.x - g * a.tiles_per_group);
    const int r0 = tile * RT;
    const int nr = min(RT, a.R.R - r0);
    const int n = a.R.n[g];
    const int64_t voff = a.R.v_off[g];
    const uint16_t *V = reinterpret_cast<const uint16_t *>(a.R.v) + voff;
    const float *LG = a.R.logits + a.R.logit_off[g];
    const bool vote = a.vmass != nullptr;
    const float *GB = vote ? a.vmass + g * a.vmstride : nullptr;
    const bool vrows = voff % D == 0;  // the block starts on a whole row of the V tensor map
    const bool l16 = (n & 3) == 0 && (reinterpret_cast<uintptr_t>(LG) & 15) == 0;
    const int nst = (n + KS - 1) / KS;

    if (tid < RT) {
        const int r = tid;
        rok[r] = 0;
        if (r < nr) {
            const int64_t row = g * a.R.R + r0 + r;
            if (vote) {
                bool inv = false;
                for (int b = 0; b < NB; ++b) inv |= a.vtidx[g * NB + b] < 0;
                rstat[r] = a.vgflag[g] ? FW_ERR_NONFINITE : (inv ? FW_ERR_INVALID_ARG : FW_OK);
                rok[r] = rstat[r] == FW_OK;
            } else {
                rok[r] = a.ws.status[row] == FW_OK;
            }
            rowM[r] = a.ws.M[row];
            rowZi[r] = 1.f / a.ws.Z[row];
            for (int b = 0; b < 4; ++b) {
                rtk[r][b] = b < NB && !vote ? a.ws.tk[row * NB + b] : 0u;
                rti[r][b] = b < NB && !vote ? a.ws.ti[row * NB + b] : -1;
            }
        }
        for (int b = 0; b < 5; ++b) bmass[r][b] = 0.f;
    }
    if (vote && tid == RT) {  // the group's budgets in ascending order (the sets are nested along it)
        int sv[4], ov[4];
        for (int b = 0; b < 4; ++b) {
            sv[b] = b < NB ? a.vs[g * NB + b] : 0x7fffffff;
            ov[b] = b;
        }
        for (int x = 1; x < NB; ++x)
            for (int y = x; y > 0 && sv[y] < sv[y - 1]; --y) {
                const int t1 = sv[y], t2 = ov[y];
                sv[y] = sv[y - 1], ov[y] = ov[y - 1];
                sv[y - 1] = t1, ov[y - 1] = t2;
            }
        for (int b = 0; b < 4; ++b) {
            vT[b] = b < NB ? a.vthr[g * NB + ov[b]] : 0u;
            vL[b] = b < NB ? a.vtidx[g * NB + ov[b]] : -1;
        }
    }
    if (tid == 0) {
        s_err = 0;
        for (int x = 0; x < TN_BS; ++x) {
            tc::mbar_init(&fullB[x], 1);
            tc::mbar_init(&freeB[x], TN_PW + 1);
        }
        for (int x = 0; x < ASLOTS; ++x) {
            tc::mbar_init(&fullA[x], TN_PW);
            tc::mbar_init(&freeA[x], 1);
        }
        for (int x = 0; x < NACC; ++x) tc::mbar_init(&accfree[x], TN_PW);
        tc::mbar_init_fence();
    }
    // d = 64: the second 64-row block of every slot is the shared zero block (M = 128 rows)
    if (NVBOX == 1)
        for (int e = tid; e < KS * 8; e += TN_NT)
            reinterpret_cast<uint4 *>(sV + TN_BS * V_SLOT)[e] = make_uint4(0u, 0u, 0u, 0u);
    // rows of P^T past the NP pairs stay zero in every slot and term
    for (int e = tid; e < ASLOTS * NSPLIT * N * 8; e += TN_NT) {
        const int m = (e / 8) % N;
        if (m >= NP) reinterpret_cast<uint4 *>(sP)[e] = make_uint4(0u, 0u, 0u, 0u);
    }
    tc::fence_async_smem();
    if (wid == 1) tc::tmem_alloc(&s_taddr, TCOLS);
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t taddr = s_taddr;

    if (wid == 0) {
        // ---------------------------------------------------------- copies
        const uint32_t vbase = tc::smem_u32(sV), lbase = tc::smem_u32(sL);
        const uint32_t livemask = __ballot_sync(FW_FULL, lane < nr && rok[lane]);
        int issued = 0;
        bool ok = true;
        for (int it = 0; it < nst; ++it) {
            const int bs = it % TN_BS, j0 = it * KS;
            if (it >= TN_BS) {
                if (lane == 0) ok = tc::mbar_wait(&freeB[bs], (uint32_t)((it / TN_BS) - 1) & 1u, WAIT_POLLS);
                ok = __shfl_sync(FW_FULL, ok, 0);
                if (!ok) break;
            }
            const int kn = min(KS, n - j0);  // keys of this stage
            const bool vtma = vrows && kn == KS;
            // (1) the per-thread copies, each lane's tracked by the barrier
            if (!vtma) {  // V rows past the block's end are zero-filled
                for (int e = lane; e < KS * NC; e += 32) {
                    const int kk = e / NC, nc = e % NC;
                    const int n2 = nc >> 3, c = nc & 7;
                    const uint32_t dst = vbase + bs * V_SLOT + n2 * (KS * 128) + (kk >> 3) * 1024 +
                                         (kk & 7) * 128 + ((c ^ (kk & 7)) << 4);
                    const bool in = kk < kn;
                    cp_async16(dst, V + (int64_t)(in ? j0 + kk : 0) * D + nc * 8, in ? 16u : 0u);
                }
            }
            if (l16) {  // 16-byte chunks, 16 per row (kn is a multiple of 4)
                for (int e = lane; e < RT * 16; e += 32) {
                    const int r = e >> 4, c = e & 15;
                    const bool cin = c * 4 < kn;
                    if ((livemask >> r) & 1u)
                        cp_async16(lbase + (uint32_t)(((bs * RT + r) * KS + c * 4) * 4),
                                   LG + (int64_t)(r0 + r) * n + j0 + (cin ? c * 4 : 0), cin ? 16u : 0u);
                }
            } else {
                for (int e = lane; e < RT * KS; e += 32) {
                    const int r = e / KS, u = e % KS;
                    if (((livemask >> r) & 1u) && u < kn)
                        cp_async4(lbase + (uint32_t)(((bs * RT + r) * KS + u) * 4), LG + (int64_t)(r0 + r) * n + j0 + u,
                                  4u);
                }
            }
            if (vote)  // the stage's summed masses (zero past the row)
                for (int e = lane; e < KS; e += 32)
                    cp_async4(tc::smem_u32(sG + bs * KS + e), GB + j0 + (e < kn ? e : 0), e < kn ? 4u : 0u);
            cp_async_mbar_arrive(&fullB[bs]);
            // (2) the barrier's one expected arrival, with the bytes of the V boxes
            const uint32_t tx = vtma ? (uint32_t)(NVBOX * 64 * 128) : 0u;
            __syncwarp();
            if (lane == 0) tc::mbar_arrive_expect_tx(&fullB[bs], tx);
            __syncwarp();
            // (3) the V boxes by TMA
            if (vtma && lane == 0)
                for (int h = 0; h < NVBOX; ++h)
                    tc::tma_load_2d(sV + bs * V_SLOT + h * (KS * 128), &tmV, 64 * h, (int32_t)(voff / D + j0),
                                    &fullB[bs]);
            ++issued;
        }
        if (!ok && lane == 0) atomicOr(&s_err, 1);
        // the copies still in flight land before the CTA moves on
        if (lane == 0)
            for (int it = issued - TN_BS < 0 ? 0 : issued - TN_BS; it < issued; ++it)
                if (!tc::mbar_wait(&fullB[it % TN_BS], (uint32_t)(it / TN_BS) & 1u, WAIT_POLLS)) atomicOr(&s_err, 1);
        __syncwarp();
    } else if (wid == 1) {
        // -------------------------------------------------------------- MMA
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_bf16_f32(128, N, true, false);
            // V^T: MN-major, the two 64-row blocks KS * 128 bytes apart; P^T:
            // K-major.  Other slots, k-steps and terms differ by an address
            // offset (>> 4) in the start field, which never carries out of it.
            const uint64_t ad0 = tc::sdesc_sw128(tc::smem_u32(sV), KS * 128, 1024);
            const uint64_t bd0 = tc::sdesc_sw128(tc::smem_u32(sP), 16, 1024);
            bool ok = true;
            int last = -1;
            for (int it = 0; it < nst && ok; ++it) {
                const int bs = it % TN_BS, as = it % ASLOTS;
                ok = tc::mbar_wait(&fullB[bs], (uint32_t)(it / TN_BS) & 1u, WAIT_POLLS);
                if (ok) ok = tc::mbar_wait(&fullA[as], (uint32_t)(it / ASLOTS) & 1u, WAIT_POLLS);
                const int ch = it / CH;
                if (ok && it % CH == 0 && ch >= NACC)
                    ok = tc::mbar_wait(&accfree[ch % NACC], (uint32_t)((ch - NACC) / NACC) & 1u, WAIT_POLLS);
                if (!ok) break;
                tc::fence_after_sync();
                const uint32_t dacc = taddr + (uint32_t)((ch % NACC) * N);
                const bool fresh = it % CH == 0;
                // V^T of the slot; d = 64: the second block is the zero block
                const uint64_t abs_ = NVBOX == 2
                                          ? ad0 + (uint64_t)((bs * V_SLOT) >> 4)
                                          : tc::sdesc_sw128(tc::smem_u32(sV) + bs * V_SLOT, (TN_BS - bs) * V_SLOT, 1024);
                const uint64_t bas = bd0 + (uint64_t)((as * P_SLOT) >> 4);
#pragma unroll
                for (int ks = 0; ks < KS / 16; ++ks) {
                    const uint64_t ad = abs_ + (uint64_t)((ks * 2048) >> 4);
#pragma unroll
                    for (int sp = 0; sp < NSPLIT; ++sp)
                        tc::mma_bf16(dacc, ad, bas + (uint64_t)((sp * P_TERM + ks * 32) >> 4), idesc,
                                     !fresh || ks > 0 || sp > 0);
                }
                tc::commit(&freeA[as]);
                tc::commit(&freeB[bs]);
                last = it;
            }
            if (!ok) atomicOr(&s_err, 1);
            if (last >= 0 && !tc::mbar_wait(&freeA[last % ASLOTS], (uint32_t)(last / ASLOTS) & 1u, WAIT_POLLS))
                atomicOr(&s_err, 1);
        }
        __syncwarp();
    } else {
        // --------------------------------------------------------- producers
        const int ptid = tid - 64;               // 0..NPROD-1
        const int rr = ptid / TPR;               // row of the tile
        const int kq = ptid % TPR;               // this thread's KPTH keys of the stage
        const int kc = kq * KPTH / 8, hk = (kq * KPTH) % 8;  // 8-key chunk and first key in it
        const int quarter = wid & 3;             // TMEM lanes (dims) this warp flushes
        const bool fl = quarter < 2 * NVBOX;     // d = 64: lanes 64..127 hold zero rows
        float racc[N];
#pragma unroll
        for (int i = 0; i < N; ++i) racc[i] = 0.f;
        float ms[NBB], mc[NBB];                  // band masses, compensated
#pragma unroll
        for (int b = 0; b < NBB; ++b) ms[b] = mc[b] = 0.f;
        const bool live = rr < nr && rok[rr];
        const float Mr = live ? rowM[rr] : 0.f, Zr = live ? rowZi[rr] : 0.f;
        float xt[NB];
        int tix[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const uint32_t tk = live ? rtk[rr][b] : 0u;
            xt[b] = __uint_as_float((tk & 0x80000000u) ? (tk & 0x7fffffffu) : ~tk);
            tix[b] = live ? rti[rr][b] : -1;
        }
        uint32_t boff[NBB];
#pragma unroll
        for (int b = 0; b < NBB; ++b) {
            const int m = b * RT + rr;
            boff[b] = (uint32_t)((m >> 3) * 1024 + (m & 7) * 128 + ((kc ^ (m & 7)) << 4) + 2 * hk);
        }
        bool ok = true;
        auto chunk_end = [&](int st) { return st % CH == CH - 1 || st == nst - 1; };
        auto flush = [&](int st) {
            tc::fence_after_sync();
            const int buf = (st / CH) % NACC;
            if (fl) {
                const uint32_t lanes = (uint32_t)(quarter * 32) << 16;
#pragma unroll
                for (int c0 = 0; c0 < N; c0 += 16) {
                    float v[16];
                    tc::ld16(taddr + lanes + (uint32_t)(buf * N + c0), v);
#pragma unroll
                    for (int i = 0; i < 16; ++i) racc[c0 + i] += v[i];
                }
            }
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&accfree[buf]);
        };
        for (int it = 0; it < nst; ++it) {
            const int bs = it % TN_BS, as = it % ASLOTS, j0 = it * KS;
            if (ok) ok = tc::mbar_wait(&fullB[bs], (uint32_t)(it / TN_BS) & 1u, WAIT_POLLS);
            // the P^T slot was last read by the MMAs of stage it - ASLOTS
            if (ok && it >= ASLOTS) ok = tc::mbar_wait(&freeA[as], (uint32_t)((it / ASLOTS) - 1) & 1u, WAIT_POLLS);
            if (!ok) break;
            uint8_t *pslot = sP + as * P_SLOT;
            const float *lr = sL + (bs * RT + rr) * KS + kq * KPTH;
            float xs[KPTH];
            if constexpr (KPTH == 4) {
                const float4 x4 = *reinterpret_cast<const float4 *>(lr);
                xs[0] = x4.x, xs[1] = x4.y, xs[2] = x4.z, xs[3] = x4.w;
            } else {
                const float2 x2 = *reinterpret_cast<const float2 *>(lr);
                xs[0] = x2.x, xs[1] = x2.y;
            }
            float pv[KPTH];
            uint32_t bdp[KPTH / 2];  // bands of keys 2q, 2q + 1 as 2 x 16 bits
            bool tie = false;
#pragma unroll
            for (int u = 0; u < KPTH; ++u) {
                const int j = j0 + kq * KPTH + u;
                const float x = xs[u];
                pv[u] = (live && j < n) ? __expf(x - Mr) * Zr : 0.f;
                int bd = 0;
                if (vote) {
                    const uint32_t gk = order_key(sG[bs * KS + kq * KPTH + u]);
#pragma unroll
                    for (int b = 0; b < NB; ++b) bd += !(gk > vT[b] || (gk == vT[b] && j <= vL[b]));
                } else {
#pragma unroll
                    for (int b = 0; b < NB; ++b) {
                        bd += x < xt[b];
                        tie |= x == xt[b];
                    }
                }
                if (u & 1) bdp[u >> 1] |= (uint32_t)bd << 16;
                else bdp[u >> 1] = (uint32_t)bd;
            }
            if (tie) {  // a key equal to a threshold: its index decides (rare)
#pragma unroll
                for (int u = 0; u < KPTH; ++u) {
                    const int j = j0 + kq * KPTH + u;
                    const float x = xs[u];
                    int bd = 0;
#pragma unroll
                    for (int b = 0; b < NB; ++b) bd += (x < xt[b]) | ((x == xt[b]) & (j > tix[b]));
                    const uint32_t sh = (u & 1) ? 16u : 0u;
                    bdp[u >> 1] = (bdp[u >> 1] & ~(0xffffu << sh)) | ((uint32_t)bd << sh);
                }
            }
            // band masses (Kahan-compensated: up to n / KPTH additions per thread)
#pragma unroll
            for (int u = 0; u < KPTH; ++u) {
                const int bd = (int)((bdp[u >> 1] >> ((u & 1) * 16)) & 0xffffu);
#pragma unroll
                for (int b = 0; b < NBB; ++b) {
                    const float y = (bd == b ? pv[u] : 0.f) - mc[b];
                    const float t = ms[b] + y;
                    mc[b] = (t - ms[b]) - y;
                    ms[b] = t;
                }
            }
            // three bf16 terms per mass, two keys per 32-bit word (key 2q low)
            uint32_t ph[KPTH / 2], pm[KPTH / 2], pl[KPTH / 2];
#pragma unroll
            for (int q = 0; q < KPTH / 2; ++q) {
                const float a0 = pv[2 * q], a1 = pv[2 * q + 1];
                ph[q] = cvt_bf16x2(a1, a0);
                const float e0 = a0 - __uint_as_float(ph[q] << 16), e1 = a1 - __uint_as_float(ph[q] & 0xffff0000u);
                pm[q] = cvt_bf16x2(e1, e0);
                const float f0 = e0 - __uint_as_float(pm[q] << 16), f1 = e1 - __uint_as_float(pm[q] & 0xffff0000u);
                pl[q] = cvt_bf16x2(f1, f0);
            }
#pragma unroll
            for (int b = 0; b < NBB; ++b) {
                uint32_t wh[KPTH / 2], wm[KPTH / 2], wl[KPTH / 2];
#pragma unroll
                for (int q = 0; q < KPTH / 2; ++q) {
                    const uint32_t msk = __vcmpeq2(bdp[q], (uint32_t)b * 0x00010001u);
                    wh[q] = ph[q] & msk;
                    wm[q] = pm[q] & msk;
                    wl[q] = pl[q] & msk;
                }
                uint8_t *dst = pslot + boff[b];
                if constexpr (KPTH == 4) {
                    *reinterpret_cast<uint2 *>(dst) = make_uint2(wh[0], wh[1]);
                    *reinterpret_cast<uint2 *>(dst + P_TERM) = make_uint2(wm[0], wm[1]);
                    *reinterpret_cast<uint2 *>(dst + 2 * P_TERM) = make_uint2(wl[0], wl[1]);
                } else {
                    *reinterpret_cast<uint32_t *>(dst) = wh[0];
                    *reinterpret_cast<uint32_t *>(dst + P_TERM) = wm[0];
                    *reinterpret_cast<uint32_t *>(dst + 2 * P_TERM) = wl[0];
                }
            }
            tc::fence_async_smem();
            __syncwarp();
            if (lane == 0) {
                tc::mbar_arrive(&fullA[as]);
                tc::mbar_arrive(&freeB[bs]);  // this warp has read the stage's logits
            }
            if (it >= ASLOTS && chunk_end(it - ASLOTS)) flush(it - ASLOTS);
        }
        // the last chunks: their MMAs complete before they are read
        for (int st = nst - ASLOTS < 0 ? 0 : nst - ASLOTS; st < nst && ok; ++st) {
            ok = tc::mbar_wait(&freeA[st % ASLOTS], (uint32_t)(st / ASLOTS) & 1u, WAIT_POLLS);
            if (ok && chunk_end(st)) flush(st);
        }
        if (!ok && lane == 0) atomicOr(&s_err, 1);
        // band masses: the TPR threads of a row (a warp, or half of one) combine
#pragma unroll
        for (int b = 0; b < NBB; ++b) {
            float v = ms[b] - mc[b];
#pragma unroll
            for (int o = TPR / 2; o >= 1; o >>= 1) v += __shfl_xor_sync(FW_FULL, v, o);
            if (kq == 0 && rr < RT) bmass[rr][b] = v;
        }
        // accumulators -> shared for the per-row epilogue: every MMA has
        // completed and every copy has landed, so the V slots (which acc
        // overlays) are idle
        if (fl) {
            const int dim = quarter * 32 + lane;
#pragma unroll
            for (int m = 0; m < NP; ++m) acc[m * (D + 1) + dim] = racc[m];
        }
    }
    tc::fence_before_sync();
    __syncthreads();
    if (wid == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(taddr, TCOLS);
    }
    if (wid < 2) return;
    // --------------------------------------------------------------- epilogue
    const bool failed = s_err != 0;
    constexpr int CPT = D / 32;
    for (int r = wid - 2; r < nr; r += TN_PW) {
        const int64_t row = g * a.R.R + r0 + r;
        if (failed) {
            if (lane == 0 && a.out.row_status) a.out.row_status[row] = FW_ERR_TIMEOUT;
            continue;
        }
        if (vote && lane == 0 && a.out.row_status) a.out.row_status[row] = rstat[r];
        if (!rok[r]) {
            if (vote && lane < NB) {  // no set to score
                a.out.gap[row * NB + lane] = __int_as_float(0x7fc00000);
                if (a.out.dropped) a.out.dropped[row * NB + lane] = __int_as_float(0x7fc00000);
            }
            continue;
        }
        float S[NBB][CPT];
#pragma unroll
        for (int b = 0; b < NBB; ++b)
#pragma unroll
            for (int t = 0; t < CPT; ++t) S[b][t] = acc[(b * RT + r) * (D + 1) + lane + 32 * t];
        if (a.out.o) {
#pragma unroll
            for (int t = 0; t < CPT; ++t) {
                float o = 0.f;
#pragma unroll
                for (int b = 0; b < NBB; ++b) o += S[b][t];
                a.out.o[row * D + lane + 32 * t] = o;
            }
        }
        for (int b = 0; b < NB; ++b) {
            const int kb = vote ? a.vs[g * NB + b] : a.k[row * NB + b];
            int sb = 0;
            for (int b2 = 0; b2 < NB; ++b2) {
                const int k2 = vote ? a.vs[g * NB + b2] : a.k[row * NB + b2];
                sb += (k2 < kb) || (k2 == kb && b2 < b);
            }
            float PA = 0.f, PC = 0.f;
#pragma unroll
            for (int q = 0; q < NBB; ++q) {
                if (q <= sb) PA += bmass[r][q];
                else PC += bmass[r][q];
            }
            float s2 = 0.f;
            float NAv[CPT];
#pragma unroll
            for (int t = 0; t < CPT; ++t) {
                float NA = 0.f, NCs = 0.f;
#pragma unroll
                for (int q = 0; q < NBB; ++q) {
                    if (q <= sb) NA += S[q][t];
                    else NCs += S[q][t];
                }
                NAv[t] = NA;
                const float diff = PC * NA - PA * NCs;  // p(A) (m_A - mu)
                s2 = fmaf(diff, diff, s2);
            }
            s2 = warp_sum(s2);
            if (lane == 0) {
                const float phi = sqrtf(s2);
                a.out.gap[row * NB + b] = phi / PA;
                if (a.out.dropped) a.out.dropped[row * NB + b] = PC;
                if (a.out.phi) a.out.phi[row * NB + b] = phi;
            }
            if (a.out.o_kept)
#pragma unroll
                for (int t = 0; t < CPT; ++t) a.out.o_kept[(row * NB + b) * D + lane + 32 * t] = NAv[t] / PA;
        }
    }
}

template <int D, int NB, int RT> size_t pv_tn_smem()
{
    return 1024 + (size_t)TN_BS * (D / 64) * KS * 128 + (D == 64 ? KS * 128 : 0) +
           (size_t)ASLOTS * NSPLIT * tn_cols<NB, RT>() * 128 + (size_t)TN_BS * RT * KS * 4 + (size_t)TN_BS * KS * 4;
}

template <int D> size_t pv_tma_smem()
{
    return 1024 + (size_t)ASLOTS * A_SLOT_BYTES + (size_t)PVM_BS * (D / 64 + 1) * KS * 128 +
           (size_t)PVM_BS * MAXRT * KS * 4 + (size_t)PVM_BS * KS * 4;
}

template <int D> size_t tc_smem(int RT)
{
    return 1024 + 2048 + (size_t)ASLOTS * A_SLOT_BYTES + (size_t)BSLOTS * D * 128 + (size_t)BSLOTS * RT * KS * 4;
}

}  // namespace

bool long_pv_tc_supported(const RowsDev &R, int nb)
{
    return R.v_dtype == FW_BF16 && (R.d == 64 || R.d == 128) && nb >= 1 && nb <= 4;
}

namespace {

// The TMA-fed kernels (transposed products for groups of at most 8 rows);
// FW_ERR_UNSUPPORTED when no instantiation fits.
fw_status launch_pv_tma(TcArgs a, const CUtensorMap &mv, cudaStream_t s)
{
    const RowsDev &R = a.R;
    const int nb = a.nb;
    if (R.R <= 8) {  // small groups: the transposed products
        const int rt = R.R <= 4 ? 4 : 8;
        a.RT = rt;
        a.tiles_per_group = 1;
        const unsigned grid = (unsigned)R.num_groups;
        auto launch_tn = [&](auto kernel, size_t smem) -> fw_status {
            FW_CUDA_CHECK(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
            FW_LAUNCH(kernel, grid, TN_NT, smem, s, mv, a);
            return FW_OK;
        };
#define FW_PV_TN(DD, NN, RR) \
    if (R.d == DD && nb == NN && rt == RR) return launch_tn(k_long_pv_tn<DD, NN, RR>, pv_tn_smem<DD, NN, RR>());
#define FW_PV_TN_D(DD) \
    FW_PV_TN(DD, 1, 4) FW_PV_TN(DD, 2, 4) FW_PV_TN(DD, 3, 4) FW_PV_TN(DD, 4, 4) \
    FW_PV_TN(DD, 1, 8) FW_PV_TN(DD, 2, 8) FW_PV_TN(DD, 3, 8) FW_PV_TN(DD, 4, 8)
        FW_PV_TN_D(128) FW_PV_TN_D(64)
#undef FW_PV_TN_D
#undef FW_PV_TN
        return FW_ERR_UNSUPPORTED;
    }
    a.RT = TM / (nb + 1) < MAXRT ? TM / (nb + 1) : MAXRT;
    a.tiles_per_group = (R.R + a.RT - 1) / a.RT;
    const unsigned grid = (unsigned)(R.num_groups * a.tiles_per_group);
    auto launch = [&](auto kernel, size_t smem) -> fw_status {
        FW_CUDA_CHECK(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        FW_LAUNCH(kernel, grid, (R.d == 128 ? pvm_nt<128>() : pvm_nt<64>()), smem, s, mv, a);
        return FW_OK;
    };
#define FW_PV_NB(DD, NN) \
    if (R.d == DD && nb == NN) return launch(k_long_pv_tma<DD, NN>, pv_tma_smem<DD>());
    FW_PV_NB(128, 1) FW_PV_NB(128, 2) FW_PV_NB(128, 3) FW_PV_NB(128, 4)
    FW_PV_NB(64, 1) FW_PV_NB(64, 2) FW_PV_NB(64, 3) FW_PV_NB(64, 4)
#undef FW_PV_NB
    return FW_ERR_UNSUPPORTED;
}

TcArgs base_args(const RowsDev &R, int nb, const fw_gap_out &out, const LongWs &L)
{
    TcArgs a;
    a.R = R;
    a.k = nullptr;
    a.nb = nb;
    a.out = out;
    a.ws = L;
    a.RT = TM / (nb + 1) < MAXRT ? TM / (nb + 1) : MAXRT;
    a.tiles_per_group = (R.R + a.RT - 1) / a.RT;
    a.vmass = nullptr;
    a.vmstride = 0;
    a.vthr = nullptr;
    a.vtidx = nullptr;
    a.vs = nullptr;
    a.vgflag = nullptr;
    return a;
}

}  // namespace

fw_status long_pv_tc(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &out, const LongWs &L,
                     cudaStream_t s)
{
    TcArgs a = base_args(R, nb, out, L);
    a.k = k;
    // the copy-warp kernels (TMA for V) when the driver can encode the V
    // tensor map; the rows of the map are every whole row the block may
    // address (boxes are only issued inside a group's own block)
    CUtensorMap mv;
    if (make_tma_2d_bf16(&mv, R.v, (uint64_t)1 << 31, (uint64_t)R.d, 64)) {
        const fw_status st = launch_pv_tma(a, mv, s);
        if (st != FW_ERR_UNSUPPORTED) return st;
    }
    const unsigned grid = (unsigned)(R.num_groups * a.tiles_per_group);
    if (R.d == 128) {
        const size_t smem = tc_smem<128>(a.RT);
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_long_pv_tc<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        FW_LAUNCH(k_long_pv_tc<128>, grid, pv_threads<128>(), smem, s, a);
    } else {
        const size_t smem = tc_smem<64>(a.RT);
        FW_CUDA_CHECK(cudaFuncSetAttribute(k_long_pv_tc<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        FW_LAUNCH(k_long_pv_tc<64>, grid, pv_threads<64>(), smem, s, a);
    }
    return FW_OK;
}

fw_status long_pv_vote(const RowsDev &R, int nb, const float *M, const float *Z, const float *mass,
                       int64_t mass_stride, const uint32_t *thr, const int32_t *tidx, const int32_t *s_budget,
                       const int32_t *gflag, float *gap, float *dropped, int32_t *row_status, cudaStream_t s)
{
    if (!long_pv_tc_supported(R, nb)) return FW_ERR_UNSUPPORTED;
    fw_gap_out out{};
    out.gap = gap;
    out.dropped = dropped;
    out.row_status = row_status;
    LongWs L{};
    L.M = const_cast<float *>(M);
    L.Z = const_cast<float *>(Z);
    TcArgs a = base_args(R, nb, out, L);
    a.vmass = mass;
    a.vmstride = mass_stride;
    a.vthr = thr;
    a.vtidx = tidx;
    a.vs = s_budget;
    a.vgflag = gflag;
    CUtensorMap mv;
    if (!make_tma_2d_bf16(&mv, R.v, (uint64_t)1 << 31, (uint64_t)R.d, 64)) return FW_ERR_UNSUPPORTED;
    return launch_pv_tma(a, mv, s);
}

}  // namespace fw
