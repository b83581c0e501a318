// fw_api.cu -- the C ABI: host-side validation, workspace carving, dispatch.
#include <cstring>

#include "fw_internal.h"

namespace fw {
std::atomic<uint64_t> g_launches{0};

static bool aligned(const void *p, size_t a) { return ((uintptr_t)p % a) == 0; }

using EncodeTiled = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                 const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiled tma_encoder()
{
    static std::atomic<EncodeTiled> fn{nullptr};
    EncodeTiled f = fn.load(std::memory_order_acquire);
    if (!f) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess) {
            f = reinterpret_cast<EncodeTiled>(p);
            fn.store(f, std::memory_order_release);
        }
    }
    return f;
}

bool make_tma_2d_bf16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows)
{
    EncodeTiled enc = tma_encoder();
    if (!enc) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols * 2};
    const cuuint32_t box[2] = {64, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

fw_status device_sms(int *sms)
{
    static std::atomic<int> cache[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return FW_ERR_CUDA;
    if (dev >= 0 && dev < 64) {
        const int c = cache[dev].load(std::memory_order_relaxed);
        if (c > 0) {
            *sms = c;
            return FW_OK;
        }
    }
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) return FW_ERR_CUDA;
    if (dev >= 0 && dev < 64) cache[dev].store(n, std::memory_order_relaxed);
    *sms = n;
    return FW_OK;
}

static fw_status check_rows(const fw_rows *r, RowsDev &R)
{
    if (!r) return FW_ERR_INVALID_ARG;
    if (r->num_groups < 0 || r->rows_per_group < 1 || r->max_n < 1) return FW_ERR_INVALID_ARG;
    if (r->d != 32 && r->d != 64 && r->d != 128 && r->d != 256) return FW_ERR_UNSUPPORTED;
    if (r->v_dtype != FW_F32 && r->v_dtype != FW_BF16) return FW_ERR_INVALID_ARG;
    if (r->num_groups > 0 && (!r->logits || !r->logit_off || !r->n || !r->v || !r->v_off))
        return FW_ERR_INVALID_ARG;
    if (((uintptr_t)r->v & 15u) != 0) return FW_ERR_INVALID_ARG;  // rows are read in 16-byte vectors
    R.num_groups = r->num_groups;
    R.R = r->rows_per_group;
    R.rows = r->num_groups * (int64_t)r->rows_per_group;
    R.d = r->d;
    R.max_n = r->max_n;
    R.v_dtype = r->v_dtype;
    R.logits = r->logits;
    R.logit_off = r->logit_off;
    R.n = r->n;
    R.v = r->v;
    R.v_off = r->v_off;
    return FW_OK;
}

}  // namespace fw

using namespace fw;

extern "C" {

const char *fw_status_string(fw_status s)
{
    switch (s) {
    case FW_OK: return "ok";
    case FW_ERR_INVALID_ARG: return "invalid argument";
    case FW_ERR_UNSUPPORTED: return "unsupported configuration";
    case FW_ERR_CUDA: return "CUDA error";
    case FW_ERR_TIMEOUT: return "timeout";
    case FW_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    case FW_ERR_NONFINITE: return "non-finite logit";
    default: return "unknown status";
    }
}

uint64_t fw_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

size_t fw_dense_and_topk_gap_workspace(const fw_rows *rows, int32_t nb)
{
    RowsDev R;
    if (check_rows(rows, R) != FW_OK || nb < 1 || nb > 4) return 0;
    if (R.max_n <= 32) return 0;
    return long_gap_workspace(R, nb);
}

fw_status fw_dense_and_topk_gap(const fw_rows *rows, const int32_t *k, int32_t nb, const fw_gap_out *out,
                                void *workspace, size_t workspace_bytes, void *stream)
{
    RowsDev R;
    fw_status st = check_rows(rows, R);
    if (st != FW_OK) return st;
    if (nb < 1 || nb > 4 || !k || !out || !out->gap || !out->dropped) return FW_ERR_INVALID_ARG;
    if (out->kept_bits && out->kept_words < (R.max_n + 31) / 32) return FW_ERR_INVALID_ARG;
    if (R.rows == 0) return FW_OK;
    cudaStream_t s = (cudaStream_t)stream;
    if (R.max_n <= 32) return small_gap(R, k, nb, *out, s);
    if (workspace_bytes < long_gap_workspace(R, nb) || !workspace || !aligned(workspace, 256))
        return FW_ERR_WORKSPACE;
    return long_gap(R, k, nb, *out, workspace, workspace_bytes, s);
}

size_t fw_swap_refine_workspace(const fw_rows *rows, int32_t nb, const fw_swap_params *prm)
{
    RowsDev R;
    if (check_rows(rows, R) != FW_OK || nb < 1 || nb > 4 || !prm) return 0;
    if (R.max_n <= 32) return 0;
    return long_swap_workspace(R, nb, prm->E, prm->max_swaps);
}

fw_status fw_swap_refine(const fw_rows *rows, const int32_t *k, int32_t nb, const fw_gap_out *topk,
                         const fw_swap_params *prm, int32_t *n_swaps, int32_t *swap_out, int32_t *swap_in,
                         float *refined_gap, float *topk_gap, int32_t *capped, void *workspace,
                         size_t workspace_bytes, void *stream)
{
    RowsDev R;
    fw_status st = check_rows(rows, R);
    if (st != FW_OK) return st;
    if (nb < 1 || nb > 4 || !k || !topk || !prm || !n_swaps || !swap_out || !swap_in || !refined_gap)
        return FW_ERR_INVALID_ARG;
    if (!topk->thr_key || !topk->thr_idx || !topk->o || !topk->row_max || !topk->row_sum)
        return FW_ERR_INVALID_ARG;
    if (prm->E < 0 || prm->max_swaps < 1) return FW_ERR_INVALID_ARG;
    if (R.rows == 0) return FW_OK;
    cudaStream_t s = (cudaStream_t)stream;
    if (R.max_n <= 32)
        return small_swap(R, k, nb, *topk, prm->E, prm->max_swaps, n_swaps, swap_out, swap_in,
                          refined_gap, topk_gap, capped, s);
    if (prm->E > kLongSwapMaxE) return FW_ERR_UNSUPPORTED;
    if (workspace_bytes < long_swap_workspace(R, nb, prm->E, prm->max_swaps) || !workspace ||
        !aligned(workspace, 256))
        return FW_ERR_WORKSPACE;
    return long_swap(R, k, nb, *topk, prm->E, prm->max_swaps, n_swaps, swap_out, swap_in, refined_gap,
                     topk_gap, capped, workspace, workspace_bytes, s);
}

size_t fw_group_vote_workspace(const fw_rows *rows, int32_t nb)
{
    RowsDev R;
    if (check_rows(rows, R) != FW_OK || nb < 1 || nb > 4) return 0;
    return group_vote_workspace(R, nb);
}

fw_status fw_group_vote(const fw_rows *rows, const int32_t *s, int32_t nb, const fw_gap_out *topk, float *vote_gap,
                        float *vote_dropped, uint32_t *vote_bits, int32_t kept_words, int32_t *row_status,
                        void *workspace, size_t workspace_bytes, void *stream)
{
    RowsDev R;
    fw_status st = check_rows(rows, R);
    if (st != FW_OK) return st;
    if (nb < 1 || nb > 4 || !s || !topk || !vote_gap) return FW_ERR_INVALID_ARG;
    if (!topk->o || !topk->row_max || !topk->row_sum) return FW_ERR_INVALID_ARG;
    if (vote_bits && kept_words < (R.max_n + 31) / 32) return FW_ERR_INVALID_ARG;
    if (R.rows == 0) return FW_OK;
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < group_vote_workspace(R, nb))
        return FW_ERR_WORKSPACE;
    return group_vote(R, s, nb, *topk, vote_gap, vote_dropped, vote_bits, kept_words, row_status, workspace,
                      workspace_bytes, (cudaStream_t)stream);
}

size_t fw_best_subset_workspace(const fw_rows *rows)
{
    RowsDev R;
    if (check_rows(rows, R) != FW_OK) return 0;
    return enum_workspace(R);
}

fw_status fw_best_subset(const fw_rows *rows, const int32_t *k, uint64_t *best_rank, float *best_gap,
                         int32_t *best_idx, int32_t k_max, float *topk_gap, int32_t *row_status,
                         void *workspace, size_t workspace_bytes, void *stream)
{
    RowsDev R;
    fw_status st = check_rows(rows, R);
    if (st != FW_OK) return st;
    if (R.max_n > 32) return FW_ERR_UNSUPPORTED;
    if (!k || !best_rank || !best_gap || !best_idx || k_max < 1 || k_max > 32) return FW_ERR_INVALID_ARG;
    if (R.rows == 0) return FW_OK;
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < enum_workspace(R)) return FW_ERR_WORKSPACE;
    return best_subset(R, k, best_rank, best_gap, best_idx, k_max, topk_gap, row_status, workspace,
                       workspace_bytes, (cudaStream_t)stream);
}

size_t fw_pool_best_subset_workspace(const fw_rows *rows, int32_t nb)
{
    RowsDev R;
    if (check_rows(rows, R) != FW_OK || nb < 1 || nb > 4) return 0;
    return pool_best_subset_workspace(R, nb);
}

fw_status fw_pool_best_subset(const fw_rows *rows, const int32_t *k, int32_t nb, const int32_t *E,
                              const fw_gap_out *topk, float *best_gap, int32_t *best_idx, int32_t k_max,
                              float *topk_gap, int64_t *n_cand, int32_t *row_status, void *workspace,
                              size_t workspace_bytes, void *stream)
{
    RowsDev R;
    fw_status st = check_rows(rows, R);
    if (st != FW_OK) return st;
    if (nb < 1 || nb > 4 || !k || !E || !topk || !best_gap || !best_idx || k_max < 1 || k_max > 32)
        return FW_ERR_INVALID_ARG;
    for (int b = 0; b < nb; ++b)
        if (E[b] < 0) return FW_ERR_INVALID_ARG;
    if (!topk->thr_key || !topk->thr_idx || !topk->o || !topk->row_max || !topk->row_sum) return FW_ERR_INVALID_ARG;
    if (R.rows == 0) return FW_OK;
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < pool_best_subset_workspace(R, nb))
        return FW_ERR_WORKSPACE;
    return pool_best_subset(R, k, nb, E, *topk, best_gap, best_idx, k_max, topk_gap, n_cand, row_status, workspace,
                            (cudaStream_t)stream);
}

fw_status fw_sync_status(const int32_t *row_status, int64_t rows, int64_t *first_row, void *stream)
{
    if (first_row) *first_row = -1;
    if (rows < 0 || (rows > 0 && !row_status)) return FW_ERR_INVALID_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaStreamSynchronize(s) != cudaSuccess) return FW_ERR_CUDA;
    int32_t buf[4096];
    for (int64_t r0 = 0; r0 < rows; r0 += 4096) {
        const int64_t cnt = rows - r0 < 4096 ? rows - r0 : 4096;
        if (cudaMemcpyAsync(buf, row_status + r0, (size_t)cnt * 4, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
            cudaStreamSynchronize(s) != cudaSuccess)
            return FW_ERR_CUDA;
        for (int64_t i = 0; i < cnt; ++i)
            if (buf[i] != FW_OK) {
                if (first_row) *first_row = r0 + i;
                return (fw_status)buf[i];
            }
    }
    return FW_OK;
}

fw_status fw_fp32_fma_probe(int32_t blocks, int32_t iters, float *out, void *stream)
{
    if (blocks < 1 || iters < 1 || !out) return FW_ERR_INVALID_ARG;
    return fp32_fma_probe(blocks, iters, out, (cudaStream_t)stream);
}

fw_status fw_best_subset_read_stats(const fw_rows *rows, const void *workspace, fw_best_subset_stats *stats,
                                    void *stream)
{
    RowsDev R;
    fw_status st = check_rows(rows, R);
    if (st != FW_OK) return st;
    if (!stats || !workspace || !aligned(workspace, 256)) return FW_ERR_INVALID_ARG;
    if (R.max_n > 32) return FW_ERR_UNSUPPORTED;
    return best_subset_stats(R, workspace, stats, (cudaStream_t)stream);
}

size_t fw_contour_alloc_workspace(int32_t cells, int32_t T)
{
    if (cells < 1 || T < 1) return 0;
    return contour_workspace(cells, T);
}

fw_status fw_contour_alloc(const float *scores, int32_t cells, int32_t T, int32_t floor_, int64_t total_budget,
                           int32_t uniform_s, int32_t *counts, int64_t *offsets, int32_t *kept_pos, float *tau,
                           float *dropped_uniform, float *dropped_alloc, void *workspace, size_t workspace_bytes,
                           void *stream)
{
    if (!scores || cells < 1 || T < 1 || floor_ < 0 || uniform_s < 0) return FW_ERR_INVALID_ARG;
    const int F = floor_ < T ? floor_ : T;
    if (total_budget < (int64_t)cells * F || total_budget > (int64_t)cells * T) return FW_ERR_INVALID_ARG;
    if (!counts || !offsets || !kept_pos || !tau) return FW_ERR_INVALID_ARG;
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < contour_workspace(cells, T))
        return FW_ERR_WORKSPACE;
    return contour_alloc(scores, cells, T, floor_, total_budget, uniform_s, counts, offsets, kept_pos, tau,
                         dropped_uniform, dropped_alloc, workspace, workspace_bytes, (cudaStream_t)stream);
}

size_t fw_contour_alloc_capped_workspace(int32_t cells, int32_t T)
{
    if (cells < 1 || T < 1) return 0;
    return contour_capped_workspace(cells, T);
}

fw_status fw_contour_alloc_capped(const float *scores, int32_t cells, int32_t T, int32_t floor_, int64_t total_budget,
                                  int32_t uniform_s, int32_t cap, int32_t *counts, int64_t *offsets, int32_t *kept_pos,
                                  float *tau, float *dropped_uniform, float *dropped_alloc, void *workspace,
                                  size_t workspace_bytes, void *stream)
{
    if (!scores || cells < 1 || T < 1 || floor_ < 0 || uniform_s < 0) return FW_ERR_INVALID_ARG;
    const int F = floor_ < T ? floor_ : T;
    if (total_budget < (int64_t)cells * F || total_budget > (int64_t)cells * T) return FW_ERR_INVALID_ARG;
    if (cap < F) return FW_ERR_INVALID_ARG;
    if (!counts || !offsets || !kept_pos || !tau) return FW_ERR_INVALID_ARG;
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < contour_capped_workspace(cells, T))
        return FW_ERR_WORKSPACE;
    return contour_alloc(scores, cells, T, floor_, total_budget, uniform_s, counts, offsets, kept_pos, tau,
                         dropped_uniform, dropped_alloc, workspace, workspace_bytes, (cudaStream_t)stream, cap);
}

fw_status fw_ragged_compact(const void *K, const void *V, int32_t cells, int32_t T, int32_t row_bytes,
                            const int64_t *offsets, const int32_t *kept_pos, int64_t total, void *K_out,
                            void *V_out, void *stream)
{
    if (!K || !V || !offsets || !kept_pos || cells < 1 || T < 1 || total < 0) return FW_ERR_INVALID_ARG;
    if (row_bytes <= 0 || row_bytes % 16 != 0) return FW_ERR_INVALID_ARG;
    if (total > 0 && (!K_out || !V_out)) return FW_ERR_INVALID_ARG;
    if (!aligned(K, 16) || !aligned(V, 16) || (total > 0 && (!aligned(K_out, 16) || !aligned(V_out, 16))))
        return FW_ERR_INVALID_ARG;
    return ragged_compact(K, V, cells, T, row_bytes, offsets, kept_pos, total, K_out, V_out,
                          (cudaStream_t)stream);
}

fw_status fw_ragged_compact_to(const void *K, const void *V, int32_t cells, int32_t T, int32_t row_bytes,
                               const int64_t *offsets, const int32_t *kept_pos, const int64_t *base,
                               const int32_t *capacity, void *K_store, void *V_store, int32_t *status, void *stream)
{
    if (!K || !V || !offsets || !kept_pos || !base || !capacity || !K_store || !V_store || cells < 1 || T < 1)
        return FW_ERR_INVALID_ARG;
    if (row_bytes <= 0 || row_bytes % 16 != 0) return FW_ERR_INVALID_ARG;
    if (!aligned(K, 16) || !aligned(V, 16) || !aligned(K_store, 16) || !aligned(V_store, 16)) return FW_ERR_INVALID_ARG;
    return ragged_compact_to(K, V, cells, T, row_bytes, offsets, kept_pos, base, capacity, K_store, V_store, status,
                             (cudaStream_t)stream);
}

fw_status fw_ragged_append(void *K_store, void *V_store, const int64_t *base, const int32_t *capacity, int32_t *counts,
                           const void *new_K, const void *new_V, int32_t cells, int32_t m, int32_t row_bytes,
                           int32_t *status, void *stream)
{
    if (!K_store || !V_store || !base || !capacity || !counts || !new_K || !new_V || cells < 1 || m < 1)
        return FW_ERR_INVALID_ARG;
    if (row_bytes <= 0 || row_bytes % 16 != 0) return FW_ERR_INVALID_ARG;
    if ((int64_t)m * (row_bytes / 16) >= ((int64_t)1 << 31)) return FW_ERR_INVALID_ARG;
    if (!aligned(K_store, 16) || !aligned(V_store, 16) || !aligned(new_K, 16) || !aligned(new_V, 16))
        return FW_ERR_INVALID_ARG;
    return ragged_append(K_store, V_store, base, capacity, counts, new_K, new_V, cells, m, row_bytes, status,
                         (cudaStream_t)stream);
}

size_t fw_window_score_workspace(int32_t cells, int32_t T)
{
    if (cells < 1 || T < 1) return 0;
    return window_score_workspace(cells, T);
}

fw_status fw_window_score(const void *Qw, const void *K, int32_t cells, int32_t T, int32_t d, int32_t w, float scale,
                          int32_t pool, float *scores, int32_t *status, void *workspace, size_t workspace_bytes,
                          void *stream)
{
    if (!Qw || !K || !scores || cells < 1 || T < 1 || w < 1 || w > 32 || w > T) return FW_ERR_INVALID_ARG;
    if (pool < 1 || pool % 2 == 0 || !(scale > 0.f) || !(scale < 1e30f)) return FW_ERR_INVALID_ARG;
    if (d != 64 && d != 128) return FW_ERR_UNSUPPORTED;
    if ((int64_t)cells * T >= ((int64_t)1 << 31) - 256) return FW_ERR_UNSUPPORTED;
    if (!aligned(Qw, 16) || !aligned(K, 16)) return FW_ERR_INVALID_ARG;
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < window_score_workspace(cells, T))
        return FW_ERR_WORKSPACE;
    return window_score(Qw, K, cells, T, d, w, scale, pool, scores, workspace, status, (cudaStream_t)stream);
}

size_t fw_selector_audit_workspace(const fw_rows *rows, int32_t nb)
{
    RowsDev R;
    if (check_rows(rows, R) != FW_OK || nb < 1 || nb > 4) return 0;
    return selector_audit_workspace(R, nb);
}

fw_status fw_selector_audit(const fw_rows *rows, const int32_t *s, int32_t nb, const fw_gap_out *topk, float *es,
                            uint32_t *bits, int32_t words, void *workspace, size_t workspace_bytes, void *stream)
{
    RowsDev R;
    fw_status st = check_rows(rows, R);
    if (st != FW_OK) return st;
    if (nb < 1 || nb > 4 || !s || !topk || !es) return FW_ERR_INVALID_ARG;
    for (int b = 0; b < nb; ++b)
        if (s[b] < 1 || s[b] > 4096) return FW_ERR_INVALID_ARG;
    if (!topk->o || !topk->row_max || !topk->row_sum) return FW_ERR_INVALID_ARG;
    if (bits && words != (R.max_n + 31) / 32) return FW_ERR_INVALID_ARG;
    if (R.max_n > 65536) return FW_ERR_UNSUPPORTED;
    if (R.rows == 0) return FW_OK;
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < selector_audit_workspace(R, nb))
        return FW_ERR_WORKSPACE;
    return selector_audit(R, s, nb, *topk, es, bits, words, workspace, (cudaStream_t)stream);
}

}  // extern "C"
