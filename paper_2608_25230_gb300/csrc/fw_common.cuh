// fw_common.cuh -- device helpers shared by the library's kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <cmath>

#include "fw.h"

#define FW_FULL 0xffffffffu

namespace fw {

// ------------------------------------------------------------ launch accounting
extern std::atomic<uint64_t> g_launches;

// Launch a kernel, count it, and turn a launch error into FW_ERR_CUDA.
#define FW_LAUNCH(kernel, grid, block, smem, stream, ...)                                      \
    do {                                                                                       \
        kernel<<<(grid), (block), (smem), (cudaStream_t)(stream)>>>(__VA_ARGS__);              \
        ::fw::g_launches.fetch_add(1, std::memory_order_relaxed);                              \
        cudaError_t _e = cudaGetLastError();                                                   \
        if (_e != cudaSuccess) return FW_ERR_CUDA;                                             \
    } while (0)

#define FW_CUDA_CHECK(expr)                                                                    \
    do {                                                                                       \
        if ((expr) != cudaSuccess) return FW_ERR_CUDA;                                         \
    } while (0)

// ------------------------------------------------------------------- order keys
// Unsigned key with the order of the float, after folding -0 onto +0, so that
// equal logits tie (and are then ordered by index).
__device__ __forceinline__ uint32_t order_key(float x)
{
    uint32_t u = __float_as_uint(x == 0.0f ? 0.0f : x);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float bf16_to_f32(uint16_t b) { return __uint_as_float(((uint32_t)b) << 16); }

template <typename VT> __device__ __forceinline__ float load_v(const VT *p, int64_t i);
template <> __device__ __forceinline__ float load_v<float>(const float *p, int64_t i) { return __ldg(p + i); }
template <> __device__ __forceinline__ float load_v<uint16_t>(const uint16_t *p, int64_t i)
{
    return bf16_to_f32(__ldg(p + i));
}

// --------------------------------------------------------- double-float (df)
// A value hi + lo held in two floats (|lo| <= ulp(hi)/2), about 44 bits of
// precision on the fp32 pipe.  Built from the classical error-free transforms:
// Knuth's TwoSum, the Dekker/Fast2Sum renormalisation, and the FMA-based exact
// product a*b = p + fma(a, b, -p).  GB300 runs fp64 at a small fraction of its
// fp32 rate, so vector sums that need more than fp32 use this instead.
struct df {
    float hi, lo;
};

__device__ __forceinline__ df df_two_sum(float a, float b)
{
    float s = a + b;
    float bb = s - a;
    float e = (a - (s - bb)) + (b - bb);
    return {s, e};
}
__device__ __forceinline__ df df_fast_two_sum(float a, float b)
{
    float s = a + b;
    float e = b - (s - a);
    return {s, e};
}
__device__ __forceinline__ df df_add(df x, df y)
{
    df s = df_two_sum(x.hi, y.hi);
    df t = df_two_sum(x.lo, y.lo);
    float e = s.lo + t.hi;
    s = df_fast_two_sum(s.hi, e);
    e = t.lo + s.lo;
    return df_fast_two_sum(s.hi, e);
}
__device__ __forceinline__ df df_neg(df x) { return {-x.hi, -x.lo}; }
__device__ __forceinline__ df df_sub(df x, df y) { return df_add(x, df_neg(y)); }
__device__ __forceinline__ df df_mul(df x, df y)
{
    float p = x.hi * y.hi;
    float e = fmaf(x.hi, y.hi, -p);
    e = fmaf(x.hi, y.lo, e);
    e = fmaf(x.lo, y.hi, e);
    return df_fast_two_sum(p, e);
}
__device__ __forceinline__ df df_mul_f(df x, float y)
{
    float p = x.hi * y;
    float e = fmaf(x.hi, y, -p);
    e = fmaf(x.lo, y, e);
    return df_fast_two_sum(p, e);
}
// f - x for a float f and df x
__device__ __forceinline__ df df_rsub_f(float f, df x)
{
    df s = df_two_sum(f, -x.hi);
    float e = s.lo - x.lo;
    return df_fast_two_sum(s.hi, e);
}
__device__ __forceinline__ df df_from_double(double x)
{
    float hi = (float)x;
    float lo = (float)(x - (double)hi);
    return {hi, lo};
}
__device__ __forceinline__ double df_to_double(df x) { return (double)x.hi + (double)x.lo; }
__device__ __forceinline__ df df_zero() { return {0.0f, 0.0f}; }

// ----------------------------------------------------------- warp reductions
__device__ __forceinline__ float warp_max(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(FW_FULL, v, o));
    return v;
}
__device__ __forceinline__ float warp_min(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(FW_FULL, v, o));
    return v;
}
__device__ __forceinline__ float warp_sum(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FW_FULL, v, o);
    return v;
}
__device__ __forceinline__ double warp_sum_d(double v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FW_FULL, v, o);
    return v;
}
__device__ __forceinline__ df warp_sum_df(df v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        df w = {__shfl_xor_sync(FW_FULL, v.hi, o), __shfl_xor_sync(FW_FULL, v.lo, o)};
        v = df_add(v, w);
    }
    return v;
}
__device__ __forceinline__ df shfl_df(df v, int src)
{
    return {__shfl_sync(FW_FULL, v.hi, src), __shfl_sync(FW_FULL, v.lo, src)};
}

// Binomial coefficients C(a, b) for a <= 32 (all below 2^32), built by
// Pascal's rule at compile time; per translation unit in constant memory.
struct BinomTable {
    uint32_t v[33][33];
};
constexpr BinomTable make_binom_table()
{
    BinomTable t{};
    for (int a = 0; a <= 32; ++a) {
        t.v[a][0] = 1u;
        for (int b = 1; b <= a; ++b) t.v[a][b] = t.v[a - 1][b - 1] + (b <= a - 1 ? t.v[a - 1][b] : 0u);
    }
    return t;
}
static __constant__ BinomTable c_binom = make_binom_table();

__device__ __forceinline__ uint64_t binom64(int a, int b)
{
    if (b < 0 || b > a) return 0;
    if (a <= 32) return c_binom.v[a][b];
    uint64_t r = 1;
    for (int t = 1; t <= b; ++t) r = r * (uint64_t)(a - b + t) / (uint64_t)t;
    return r;
}
// colex rank of the set bits of a 32-bit mask: sum_i C(c_i, i), i = 1.. in ascending order
__device__ __forceinline__ uint64_t colex_rank_mask(uint32_t m)
{
    uint64_t r = 0;
    int i = 1;
    while (m) {
        const int c = __ffs(m) - 1;
        r += c_binom.v[c][i];  // c <= 31, i <= 32; C(c, i) = 0 for i > c
        ++i;
        m &= m - 1;
    }
    return r;
}

// Columns [c0, c0 + DC) of the n value rows into st[j][DC + 1], fp32; the warp
// issues all its loads before it stores any (8 elements per lane per step).
template <int DC, typename VT>
__device__ __forceinline__ void stage_value_cols(const VT *V, int n, int d, int c0, float *st, int lane)
{
    const int tot = n * DC;
    for (int e0 = 0; e0 < tot; e0 += 32 * 8) {
        float v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int e = e0 + lane + 32 * u;
            v[u] = e < tot ? load_v(V, (int64_t)(e / DC) * d + c0 + e % DC) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int e = e0 + lane + 32 * u;
            if (e < tot) st[(e / DC) * (DC + 1) + e % DC] = v[u];
        }
    }
}

// CTA-wide selection of the m largest of n unsigned order keys, equal keys
// taken in ascending index order: on return (every thread) T is the m-th
// largest key and L the largest index taken among the keys equal to T; key j
// is selected iff key(j) > T or (key(j) == T and j <= L).  1 <= m <= n.
// Three radix passes (11, 11, 10 bits) over a 2048-bin shared histogram, then
// an index-order scan of the keys equal to T.  key(j) is called for j < n by
// every thread of the block (all threads must call this function).
struct TopmSmem {
    uint32_t hist[2048];
    int wcnt[32];
    uint32_t digit;
    int rem, L;
};
template <typename KeyFn>
__device__ __forceinline__ void block_topm(int n, int m, KeyFn key, TopmSmem &S, uint32_t &T, int &L)
{
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5, nt = blockDim.x, nw = nt >> 5;
    uint32_t prefix = 0, pmask = 0;
    int rem = m;
    if (tid == 0) {
        S.digit = 0u;
        S.rem = 1;
    }
    for (int pass = 0; pass < 3; ++pass) {
        const int shift = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
        const int nbin = pass < 2 ? 2048 : 1024;
        for (int i = tid; i < 2048; i += nt) S.hist[i] = 0u;
        __syncthreads();
        for (int j = tid; j < n; j += nt) {
            const uint32_t u = key(j);
            if ((u & pmask) == prefix) atomicAdd(&S.hist[(u >> shift) & (uint32_t)(nbin - 1)], 1u);
        }
        __syncthreads();
        if (wid == 0) {
            const int per = nbin / 32;  // bins in descending order, per lanes
            const int top = nbin - 1 - lane * per;
            int c = 0;
            for (int q = 0; q < per; ++q) c += (int)S.hist[top - q];
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
                    const int h = (int)S.hist[top - q];
                    if (acc + h >= rem) {
                        S.digit = (uint32_t)(top - q);
                        S.rem = rem - acc;
                        break;
                    }
                    acc += h;
                }
            }
        }
        __syncthreads();
        prefix |= S.digit << shift;
        pmask |= (uint32_t)(nbin - 1) << shift;
        rem = S.rem;
        __syncthreads();
    }
    T = prefix;
    // the rem-th key equal to T in index order
    if (tid == 0) S.L = -1;
    __syncthreads();
    int run = 0;
    for (int j0 = 0; j0 < n; j0 += nt) {
        const int j = j0 + tid;
        const bool eq = j < n && key(j) == T;
        const unsigned bm = __ballot_sync(FW_FULL, eq);
        if (lane == 0) S.wcnt[wid] = __popc(bm);
        __syncthreads();
        int before = run, tot = 0;
        for (int w = 0; w < nw; ++w) {
            if (w < wid) before += S.wcnt[w];
            tot += S.wcnt[w];
        }
        before += __popc(bm & ((1u << lane) - 1u));
        if (eq && before + 1 == rem) S.L = j;
        run += tot;
        __syncthreads();
        if (S.L >= 0) break;
    }
    L = S.L;
    __syncthreads();
}

// Dispatch on the value width d (multiples of 32 supported: 32, 64, 128, 256)
// and the value dtype; binds DPL (dims per lane) and VT (element type).
#define FW_DISPATCH(d, vdt, ...)                                                              \
    do {                                                                                       \
        if ((vdt) == FW_F32) {                                                                 \
            using VT = float;                                                                  \
            FW_DISPATCH_D(d, __VA_ARGS__);                                                            \
        } else if ((vdt) == FW_BF16) {                                                         \
            using VT = uint16_t;                                                               \
            FW_DISPATCH_D(d, __VA_ARGS__);                                                            \
        } else {                                                                               \
            return FW_ERR_INVALID_ARG;                                                         \
        }                                                                                      \
    } while (0)
#define FW_DISPATCH_D(d, ...)                                                                 \
    switch (d) {                                                                               \
    case 32: { constexpr int DPL = 1; __VA_ARGS__; } break;                                           \
    case 64: { constexpr int DPL = 2; __VA_ARGS__; } break;                                           \
    case 128: { constexpr int DPL = 4; __VA_ARGS__; } break;                                          \
    case 256: { constexpr int DPL = 8; __VA_ARGS__; } break;                                          \
    default: return FW_ERR_UNSUPPORTED;                                                        \
    }

}  // namespace fw
