// fw_internal.h -- launcher interfaces between the C ABI (fw_api.cu) and the
// kernel translation units.
#pragma once

#include <cuda.h>  // CUtensorMap (types only; the encoder is fetched from the driver at run time)

#include "fw_common.cuh"

namespace fw {

// Device-side copy of fw_rows plus the derived row count.
struct RowsDev {
    int64_t num_groups;
    int64_t rows;
    int32_t R;      // rows per group
    int32_t d;
    int32_t max_n;
    int32_t v_dtype;
    const float *logits;
    const int64_t *logit_off;
    const int32_t *n;
    const void *v;
    const int64_t *v_off;
};

// Rows with n <= 32 ("small rows": exact-enumeration workloads).
fw_status small_gap(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &out,
                    cudaStream_t s);
fw_status small_swap(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &topk,
                     int E, int max_swaps, int32_t *n_swaps, int32_t *swap_out, int32_t *swap_in,
                     float *refined_gap, float *topk_gap, int32_t *capped, cudaStream_t s);
size_t enum_workspace(const RowsDev &R);
fw_status best_subset(const RowsDev &R, const int32_t *k, uint64_t *best_rank, float *best_gap,
                      int32_t *best_idx, int k_max, float *topk_gap, int32_t *row_status,
                      void *ws, size_t ws_bytes, cudaStream_t s);
fw_status best_subset_stats(const RowsDev &R, const void *ws, fw_best_subset_stats *out, cudaStream_t s);

// Long rows (any n): row statistics + radix top-k, then the P.V products.
// Per-row results of the select kernel that the P.V kernels read.
struct LongWs {
    float *M, *Z;          // [rows]
    uint32_t *tk;          // [rows][nb]
    int32_t *ti;           // [rows][nb]
    int32_t *status;       // [rows]
};
bool long_pv_tc_supported(const RowsDev &R, int nb);
fw_status long_pv_tc(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &out, const LongWs &L,
                     cudaStream_t s);
// The group vote's scoring on the same tensor-core kernels: every row of a
// group against the group's nested sets (key j kept by budget b when
// key(mass_j) > thr[b], or equal and j <= tidx[b]); writes gap, dropped and
// row_status.  FW_ERR_UNSUPPORTED when the rows do not fit them.
fw_status long_pv_vote(const RowsDev &R, int nb, const float *M, const float *Z, const float *mass,
                       int64_t mass_stride, const uint32_t *thr, const int32_t *tidx, const int32_t *s_budget,
                       const int32_t *gflag, float *gap, float *dropped, int32_t *row_status, cudaStream_t s);
size_t long_gap_workspace(const RowsDev &R, int nb);
fw_status long_gap(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &out, void *ws,
                   size_t ws_bytes, cudaStream_t s);
constexpr int kLongSwapMaxE = 96;  // largest pool the long-row selector stages in shared memory
size_t long_swap_workspace(const RowsDev &R, int nb, int E, int max_swaps);
fw_status long_swap(const RowsDev &R, const int32_t *k, int nb, const fw_gap_out &topk, int E,
                    int max_swaps, int32_t *n_swaps, int32_t *swap_out, int32_t *swap_in,
                    float *refined_gap, float *topk_gap, int32_t *capped, void *ws,
                    size_t ws_bytes, cudaStream_t s);

// The group vote: one kept set per group of rows by summed mass, every row scored.
size_t group_vote_workspace(const RowsDev &R, int nb);
fw_status group_vote(const RowsDev &R, const int32_t *s, int nb, const fw_gap_out &topk, float *gap,
                     float *dropped, uint32_t *bits, int words, int32_t *row_status, void *ws, size_t ws_bytes,
                     cudaStream_t st);

// ContourKV allocation and ragged compaction.
size_t contour_workspace(int cells, int T);
size_t contour_capped_workspace(int cells, int T);
// cap < 0: no cap (the plain allocation); otherwise each cell keeps at most cap entries
fw_status contour_alloc(const float *scores, int cells, int T, int floor_, int64_t total_budget,
                        int uniform_s, int32_t *counts, int64_t *offsets, int32_t *kept_pos,
                        float *tau, float *dropped_uniform, float *dropped_alloc, void *ws,
                        size_t ws_bytes, cudaStream_t s, int cap = -1);
fw_status ragged_compact(const void *K, const void *V, int cells, int T, int row_bytes,
                         const int64_t *offsets, const int32_t *kept_pos, int64_t total,
                         void *K_out, void *V_out, cudaStream_t s);
fw_status ragged_compact_to(const void *K, const void *V, int cells, int T, int row_bytes, const int64_t *offsets,
                            const int32_t *kept_pos, const int64_t *base, const int32_t *capacity, void *K_store,
                            void *V_store, int32_t *status, cudaStream_t s);
fw_status ragged_append(void *K_store, void *V_store, const int64_t *base, const int32_t *capacity, int32_t *counts,
                        const void *new_K, const void *new_V, int cells, int m, int row_bytes, int32_t *status,
                        cudaStream_t s);

// ES_pool (Definition 2.2): exact best subset of the candidate set, any row length.
size_t pool_best_subset_workspace(const RowsDev &R, int nb);
fw_status pool_best_subset(const RowsDev &R, const int32_t *k, int nb, const int32_t *E, const fw_gap_out &topk,
                           float *best_gap, int32_t *best_idx, int k_max, float *topk_gap, int64_t *n_cand,
                           int32_t *row_status, void *ws, cudaStream_t st);

// The observation-window importance score (TMA + tcgen05).
size_t window_score_workspace(int cells, int T);
fw_status window_score(const void *Qw, const void *K, int cells, int T, int d, int w, float scale, int pool,
                       float *scores, void *ws, int32_t *status, cudaStream_t s);

// The deployed selectors' kept sets, scored (Sec. 2.3, App. C).
size_t selector_audit_workspace(const RowsDev &R, int nb);
fw_status selector_audit(const RowsDev &R, const int32_t *s, int nb, const fw_gap_out &topk, float *es,
                         uint32_t *bits, int words, void *ws, cudaStream_t st);

// A TMA map of a 2-D bf16 tensor [rows][cols] (cols innermost, row stride
// cols * 2 bytes) read in boxes of box_rows x 64 elements with the 128-byte
// swizzle.  False if the driver's encoder is unavailable or refuses the map.
bool make_tma_2d_bf16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows);

// The fp32 FMA throughput probe (a measurement aid).
fw_status fp32_fma_probe(int blocks, int iters, float *out, cudaStream_t s);

// Number of SMs of the current device (queried once per device).
fw_status device_sms(int *sms);

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

}  // namespace fw
