/*
 * fw.h -- C ABI of the forced-weight subset evaluation library (libfw.so).
 *
 * Implements, for batches of attention rows, the quantities of "Trust the
 * Mass: Forced Weights in KV-Cache Eviction":
 *   - Definition 2.1: an instance is a softmax row p over N keys with value
 *     points v_j; the dense output mu = sum_j p_j v_j; a kept set A with kept
 *     mass p(A), dropped mass 1 - p(A) and forced-weight output
 *     m_A = sum_{j in A} (p_j / p(A)) v_j; the top-mass set A*_s.
 *   - Sec. 2.1: the gap es(A) = ||mu - m_A||, its minimum ES(s) over |A| = s,
 *     and the balancing selector (greedy one-for-one swaps from A*_s that most
 *     decrease es, stopping when none does).
 *   - Lemma 2.1: g_A = sum_{j in A} p_j (v_j - mu) and es(A) = ||g_A|| / p(A);
 *     Phi = ||g_{A*_s}|| is the one-pass certificate.
 *   - Definition 2.2: the candidate set (top-mass set plus the keys of largest
 *     single-key error p_j ||v_j - mu||).
 *   - Sec. 2.1: the group vote (one kept set per KV head, by the mass summed
 *     over the head's query rows).
 *   - Sec. 4: ContourKV (one score, one global threshold, a recency floor of
 *     the last 32 positions per cell) and ragged per-head storage.
 *
 * Conventions for every entry point:
 *   - All array arguments are DEVICE pointers unless stated otherwise; the
 *     structs themselves (fw_rows, fw_gap_out, fw_swap_params) live in HOST
 *     memory and are read during the call only.
 *   - The caller owns every buffer, including the workspace; the library
 *     never allocates or frees device memory.  Size workspaces with the
 *     matching *_workspace() call; a workspace must be 256-byte aligned.
 *   - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) and the call returns without synchronising.  Outputs are valid
 *     once the stream has reached that point.
 *   - Arguments are validated on the host before any launch; on any error the
 *     call returns a status other than FW_OK and enqueues nothing.
 *   - Conditions only the device can see (non-finite logits, an out-of-range
 *     budget, a bounded wait that gave up) are reported per row in
 *     `row_status`.  The library never traps or asserts on the device, and
 *     every device-side wait (an mbarrier of a bulk copy or of the tensor
 *     core) gives up after a fixed number of polls instead of spinning.
 *   - Kept sets are stated by threshold: key j of a row is in the top-k set iff
 *     key(l_j) > thr_key or (key(l_j) == thr_key and j <= thr_idx), where key()
 *     maps a float to an unsigned integer of the same order after folding -0
 *     onto +0 (equal logits: the lower index is kept first).
 */
#ifndef FW_H
#define FW_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    FW_OK = 0,
    FW_ERR_INVALID_ARG = 1,   /* a size, budget or pointer is out of range     */
    FW_ERR_UNSUPPORTED = 2,   /* valid but not implemented (e.g. d not in 32k) */
    FW_ERR_CUDA = 3,          /* a CUDA launch or query failed                */
    FW_ERR_TIMEOUT = 4,       /* per-row: a bounded device-side wait gave up  */
    FW_ERR_WORKSPACE = 5,     /* workspace missing, too small or misaligned   */
    FW_ERR_NONFINITE = 6      /* per-row: a logit is NaN or infinite          */
} fw_status;

typedef enum { FW_F32 = 0, FW_BF16 = 1 } fw_dtype;

/* A batch of attention rows (instances of Definition 2.1).
 * Rows come in groups of `rows_per_group` consecutive rows that share one
 * value block and one length: a KV head's query rows, a GQA group, or a single
 * row (rows_per_group = 1).  Group g has n[g] keys (1 <= n[g] <= max_n); row
 * r = g * rows_per_group + i has its n[g] fp32 logits at
 * logits + logit_off[g] + i * n[g]; the group's values are the n[g] x d
 * row-major block at v + v_off[g] (elements of type v_dtype).  The softmax of
 * a row's logits is its mass vector p.
 * One batch has one value width d and one value dtype: a cache whose heads
 * differ in width (say d = 64 and d = 128 layers) is issued as one call per
 * width, each call a ragged batch over n. */
typedef struct {
    int64_t num_groups;
    int32_t rows_per_group;
    int32_t d;              /* value width: a multiple of 32, at most 256     */
    int32_t max_n;          /* host-side bound on every n[g]                   */
    int32_t v_dtype;        /* fw_dtype                                        */
    const float *logits;    /* device                                          */
    const int64_t *logit_off; /* device [num_groups], element offsets          */
    const int32_t *n;       /* device [num_groups]                             */
    const void *v;          /* device, 16-byte aligned                         */
    const int64_t *v_off;   /* device [num_groups], element offsets, multiples of 8 */
} fw_rows;

/* Outputs of fw_dense_and_topk_gap.  rows = num_groups * rows_per_group.
 * Every pointer except gap and dropped may be NULL (not written). */
typedef struct {
    float *o;            /* [rows][d]      dense output mu                         */
    float *o_kept;       /* [rows][nb][d]  forced-weight output m_A                */
    float *gap;          /* [rows][nb]     es(A) = ||m_A - mu||                    */
    float *dropped;      /* [rows][nb]     dropped mass, summed over keys not in A */
    float *phi;          /* [rows][nb]     ||g_A|| = p(A) es(A)                    */
    float *row_max;      /* [rows]         M = max_j l_j                           */
    float *row_sum;      /* [rows]         Z = sum_j exp(l_j - M)                  */
    uint32_t *thr_key;   /* [rows][nb]     order key of the k-th kept logit        */
    int32_t *thr_idx;    /* [rows][nb]     largest kept index carrying thr_key     */
    uint32_t *kept_bits; /* [rows][nb][kept_words] bit j%32 of word j/32 = (j in A) */
    int32_t kept_words;  /* words per (row, budget); >= ceil(max_n/32) if kept_bits */
    int32_t *row_status; /* [rows]         FW_OK, FW_ERR_NONFINITE, FW_ERR_INVALID_ARG
                                           (budget out of range) or FW_ERR_TIMEOUT */
} fw_gap_out;

/* Dense output, top-k kept sets, forced-weight outputs, gaps and dropped mass
 * (Definition 2.1, Sec. 2.1, Lemma 2.1) for every row and each of nb nested or
 * independent budgets.
 *   rows : host pointer to the batch description.
 *   k    : device [rows][nb] int32 budgets, 1 <= k <= n of the row (checked on
 *          the device: an out-of-range budget sets row_status to
 *          FW_ERR_INVALID_ARG and leaves that row's outputs unspecified).
 *   nb   : 1..4.
 * The kept set of budget b is the k largest logits, equal logits kept in
 * ascending index order.  The dropped mass is the sum of p_j over the keys
 * not kept.  Non-finite logits set row_status[r] = FW_ERR_NONFINITE. */
fw_status fw_dense_and_topk_gap(const fw_rows *rows, const int32_t *k, int32_t nb,
                                const fw_gap_out *out, void *workspace, size_t workspace_bytes,
                                void *stream);
/* Workspace bytes (0 for max_n <= 32): per-row softmax statistics, thresholds
 * and status, and a list of the rows whose threshold search falls back to the
 * radix select (rows with heavy ties). */
size_t fw_dense_and_topk_gap_workspace(const fw_rows *rows, int32_t nb);

/* Parameters of the balancing selector. */
typedef struct {
    int32_t E;          /* extras: the E dropped keys of largest single-key error
                           p_j ||v_j - mu|| (Definition 2.2) join the candidate
                           set; 0 <= E.  E >= n - k puts every key in the pool. */
    int32_t max_swaps;  /* cap on swaps per (row, budget), >= 1                 */
} fw_swap_params;

/* The balancing selector (Sec. 2.1) inside the candidate set (Definition 2.2).
 * Starts from the top-k set described by `topk` (a fw_gap_out filled by
 * fw_dense_and_topk_gap for the same rows, k and nb; its thr_key, thr_idx, o,
 * row_max and row_sum must be non-NULL).  Each round scores every swap of one
 * kept key for one pool key outside the set and takes the one with the
 * smallest es (ties: smallest kept index, then smallest added index) if it is
 * strictly below the current es; otherwise it stops.
 * Outputs (device): n_swaps [rows][nb]; swap_out / swap_in
 * [rows][nb][max_swaps] (removed / added key of each swap in the order taken;
 * entries past n_swaps are -1); refined_gap [rows][nb]; topk_gap [rows][nb]
 * (may be NULL); capped [rows][nb] = 1 if max_swaps stopped the search (may be
 * NULL).  Rows with max_n > 32 accept E <= 96 (FW_ERR_UNSUPPORTED above). */
fw_status fw_swap_refine(const fw_rows *rows, const int32_t *k, int32_t nb, const fw_gap_out *topk,
                         const fw_swap_params *prm, int32_t *n_swaps, int32_t *swap_out,
                         int32_t *swap_in, float *refined_gap, float *topk_gap, int32_t *capped,
                         void *workspace, size_t workspace_bytes, void *stream);
/* Workspace bytes (0 for max_n <= 32): for up to 3 x 152 persistent blocks,
 * per-key arrays of max_n entries and a table of kept x pool cross products
 * (fp32, max_n x round_up(E, 32) entries per block: 1.9 GB for max_n = 32,768
 * and E = 32). */
size_t fw_swap_refine_workspace(const fw_rows *rows, int32_t nb, const fw_swap_params *prm);

/* Exact ES(k) (Sec. 2.1) by exhaustive search over all C(n, k) subsets, for
 * rows with n <= 32.  k: device [rows] int32, 1 <= k <= n.
 * Outputs (device): best_rank [rows] colex rank sum_i C(c_i, i) of the
 * minimising set c_1 < ... < c_k (0-based; exact ties -> smallest rank);
 * best_gap [rows] = ES(k); best_idx [rows][k_max] ascending members (entries
 * past k are -1); topk_gap [rows] = es of the top-k set (may be NULL);
 * row_status [rows] (may be NULL).  k_max >= every k. */
fw_status fw_best_subset(const fw_rows *rows, const int32_t *k, uint64_t *best_rank,
                         float *best_gap, int32_t *best_idx, int32_t k_max, float *topk_gap,
                         int32_t *row_status, void *workspace, size_t workspace_bytes,
                         void *stream);
size_t fw_best_subset_workspace(const fw_rows *rows);

/* What the last fw_best_subset call made with `workspace` spent: the search
 * covers all C(n, k) subsets, but evaluates only those no bound excludes.
 * The paper has no counterpart; these are the search's own work counters. */
typedef struct {
    int64_t rows_exhaustive;  /* rows whose candidates overflowed and that went to the
                                 exhaustive fp64 path (every subset screened in fp32) */
    int64_t candidates;       /* subsets re-scored in double-float after the walk     */
    uint64_t inner_nodes;     /* inner-set enumerations the walk ran                  */
    uint64_t inner_leaves;    /* subsets those enumerations visited                   */
    uint64_t inner_ops;       /* fp32 add/min operations of those enumerations        */
    uint64_t skipped;         /* walk nodes and removal classes excluded by a bound   */
} fw_best_subset_stats;
/* Waits for `stream` (on which that call ran) and fills *stats.  rows must
 * describe the same batch.  Returns FW_ERR_UNSUPPORTED for max_n > 32. */
fw_status fw_best_subset_read_stats(const fw_rows *rows, const void *workspace, fw_best_subset_stats *stats,
                                    void *stream);

/* The group vote (Sec. 2.1).  Deployment keeps one set per KV head and
 * applies it to every query row that shares the head.  For each group of
 * rows_per_group rows (one value block) the vote keeps the s keys of largest
 * summed mass G_j = sum over the group's rows of p_j (equal G: the lower index
 * is kept first), and every row of the group is scored against that set with
 * its own masses.  With rows_per_group = 1 the vote is each row's own top-mass
 * set.  The sets of one group for its nb budgets are nested (prefixes of one
 * order).
 *   s    : device [num_groups][nb] int32 budgets, 1 <= s <= n[g] (checked on
 *          the device: a group with an out-of-range budget gets row_status
 *          FW_ERR_INVALID_ARG on all its rows, its outputs unspecified).
 *   nb   : 1..4.
 *   topk : a fw_gap_out filled by fw_dense_and_topk_gap for the same rows; its
 *          o, row_max and row_sum must be non-NULL.
 * Outputs (device): vote_gap [rows][nb] es of the group's set for the row;
 * vote_dropped [rows][nb] the row's mass outside the set, summed over those
 * keys (may be NULL); vote_bits [num_groups][nb][kept_words] bit j%32 of word
 * j/32 = (j in the set) (may be NULL; kept_words >= ceil(max_n/32));
 * row_status [rows] FW_OK, FW_ERR_INVALID_ARG, or FW_ERR_NONFINITE when a logit
 * of the row's group is not finite (may be NULL). */
fw_status fw_group_vote(const fw_rows *rows, const int32_t *s, int32_t nb, const fw_gap_out *topk,
                        float *vote_gap, float *vote_dropped, uint32_t *vote_bits, int32_t kept_words,
                        int32_t *row_status, void *workspace, size_t workspace_bytes, void *stream);
/* Workspace bytes: the summed mass of every group (num_groups x max_n fp32)
 * and the threshold of every (group, budget). */
size_t fw_group_vote_workspace(const fw_rows *rows, int32_t nb);

/* ES_pool (Definition 2.2): the exact minimum of es over the size-s subsets
 * of the candidate set -- the top-mass set A*_s plus the E[b] dropped keys of
 * largest single-key error p_j ||v_j - mu|| (equal errors: lower index first)
 * -- by exhaustive search of the pool, for every row and budget slot b.
 *   k    : device [rows][nb] budgets, 1 <= s <= min(n, 32, k_max); a slot with
 *          s + min(E[b], n - s) > 64 pool keys, or more than 2^32 subsets on
 *          the pool's smaller side, is refused (row_status FW_ERR_UNSUPPORTED,
 *          its gap NaN); an out-of-range s gives FW_ERR_INVALID_ARG.
 *   E    : HOST [nb] extras per budget slot, >= 0 (the paper's schedule is
 *          24/12/6/4 at s = 4/8/16/32).
 *   topk : a fw_gap_out filled by fw_dense_and_topk_gap for the same rows, k
 *          and nb; its thr_key, thr_idx, o, row_max and row_sum must be
 *          non-NULL.  mu is taken as its dense output o.
 * Outputs (device): best_gap [rows][nb] = ES_pool; best_idx [rows][nb][k_max]
 * the minimising set's keys ascending (entries past s are -1; exact ties go
 * to the smallest colex rank of the members' positions in the pool, the pool
 * in ascending key order); topk_gap [rows][nb] es(A*_s) (may be NULL); n_cand
 * [rows][nb] the subsets re-scored in fp64 after the fp32 screen (may be
 * NULL); row_status [rows] (may be NULL).  Rows up to 49,152 keys
 * (FW_ERR_UNSUPPORTED above). */
fw_status fw_pool_best_subset(const fw_rows *rows, const int32_t *k, int32_t nb, const int32_t *E,
                              const fw_gap_out *topk, float *best_gap, int32_t *best_idx, int32_t k_max,
                              float *topk_gap, int64_t *n_cand, int32_t *row_status, void *workspace,
                              size_t workspace_bytes, void *stream);
/* Workspace bytes: the pool of every (row, budget), 64 int32 each, and its
 * size; then, for each warp of the enumeration launch (4 blocks of 4 warps
 * per SM of the current device, fewer for small batches), a buffer of 4,096
 * re-scoring candidates and an fp64 Gram matrix of the pool (64 KB). */
size_t fw_pool_best_subset_workspace(const fw_rows *rows, int32_t nb);

/* The deployed selectors audited in Sec. 2.3 (App. C settings), as kept sets
 * scored with Definition 2.1's es.  For budget s:
 *   FW_SEL_STREAMING  the first min(4, s/2) positions and the last
 *                     s - min(4, s/2) (StreamingLLM: sinks plus recency);
 *   FW_SEL_H2O        the last s/2 positions and, of the others, the s - s/2
 *                     of largest mass accumulated over the group's rows (the
 *                     query rows sharing the KV head, i.e. one cache serving
 *                     them all);
 *   FW_SEL_SNAPKV     window w = max(1, min(32, s/2)): the last w positions and,
 *                     of the others, the s - w of largest pooled vote (a key's
 *                     mass summed over the group's last w rows, then the
 *                     maximum over the 7 positions around it, clipped to the
 *                     candidates);
 *   FW_SEL_QUEST      pages of P = max(2, s/4) keys, the floor(s/P) pages of
 *                     largest maximum logit (Quest's page bound, taken exact
 *                     since the logits are given);
 *   FW_SEL_QUEST16    the same with P = 16 (s >= 16; NaN below).
 * Equal scores keep lower positions (pages) first. */
typedef enum {
    FW_SEL_STREAMING = 0,
    FW_SEL_H2O = 1,
    FW_SEL_SNAPKV = 2,
    FW_SEL_QUEST = 3,
    FW_SEL_QUEST16 = 4
} fw_selector;
#define FW_NUM_SELECTORS 5

/* For every row, rule and budget: es [rows][FW_NUM_SELECTORS][nb] (NaN where
 * the rule keeps nothing: s > n, or Quest-16 with s < 16); bits (may be NULL)
 * [rows][FW_NUM_SELECTORS][nb][words] the kept sets, words = ceil(max_n/32)
 * exactly.  s: HOST [nb] budgets, 1 <= s <= 4096, nb 1..4.  topk: a fw_gap_out
 * filled by fw_dense_and_topk_gap for the same rows (o, row_max, row_sum used).
 * Rows up to 65,536 keys (FW_ERR_UNSUPPORTED above). */
fw_status fw_selector_audit(const fw_rows *rows, const int32_t *s, int32_t nb, const fw_gap_out *topk, float *es,
                            uint32_t *bits, int32_t words, void *workspace, size_t workspace_bytes, void *stream);
/* Workspace bytes: the accumulated masses (groups x max_n fp32), the window
 * votes (groups x nb x max_n fp32) and the group-level sets. */
size_t fw_selector_audit_workspace(const fw_rows *rows, int32_t nb);

/* ContourKV allocation (Sec. 4).  scores: device [cells][T] fp32, finite and
 * >= 0.  Every cell keeps its recency floor (the last min(floor, T) positions)
 * plus the non-floor positions among the K = total_budget - cells*min(floor,T)
 * best non-floor entries of the whole cache, ranked by (score desc, cell asc,
 * position asc); *tau is the score of the K-th (+inf if K = 0).
 * Outputs (device): counts [cells]; offsets [cells+1] exclusive prefix sum
 * (offsets[cells] = total_budget); kept_pos [total_budget] positions of each
 * cell in ascending order, cells in order; tau [1]; dropped_uniform [cells] and
 * dropped_alloc [cells]: the mass of the cell's normalised scores outside the
 * cell's own top-uniform_s set (ties -> lower position) and outside the
 * allocated set (either may be NULL).
 * Requires cells*min(floor,T) <= total_budget <= cells*T. */
fw_status fw_contour_alloc(const float *scores, int32_t cells, int32_t T, int32_t floor,
                           int64_t total_budget, int32_t uniform_s, int32_t *counts,
                           int64_t *offsets, int32_t *kept_pos, float *tau,
                           float *dropped_uniform, float *dropped_alloc, void *workspace,
                           size_t workspace_bytes, void *stream);
size_t fw_contour_alloc_workspace(int32_t cells, int32_t T);

/* ContourKV with its budget enforced per cell (Sec. 4: enforcement caps
 * every head at a uniform method's per-head count).  The allocation of
 * fw_contour_alloc -- same floor, same global ranking and tau -- truncated
 * per cell: a cell whose allocation exceeds `cap` keeps its recency floor
 * plus its best cap - min(floor, T) non-floor entries (score desc, position
 * asc), so counts[h] = min(allocated count, cap) and the total
 * offsets[cells] = sum_h counts[h] <= total_budget (kept_pos needs room for
 * total_budget entries; the positions past offsets[cells] are not written).
 * dropped_alloc is the mass outside the truncated set; tau and
 * dropped_uniform are those of fw_contour_alloc.  Requires
 * cap >= min(floor, T) (the floor is always kept); other rules as
 * fw_contour_alloc. */
fw_status fw_contour_alloc_capped(const float *scores, int32_t cells, int32_t T, int32_t floor, int64_t total_budget,
                                  int32_t uniform_s, int32_t cap, int32_t *counts, int64_t *offsets, int32_t *kept_pos,
                                  float *tau, float *dropped_uniform, float *dropped_alloc, void *workspace,
                                  size_t workspace_bytes, void *stream);
size_t fw_contour_alloc_capped_workspace(int32_t cells, int32_t T);

/* Ragged per-head storage (Sec. 4): copy the kept rows of K and V
 * ([cells][T][row_bytes] each) into packed [offsets[cells]][row_bytes] outputs,
 * cell by cell, positions in the order of kept_pos.  row_bytes must be a
 * positive multiple of 16; K, V, K_out, V_out 16-byte aligned.  `total` is
 * offsets[cells] as known to the host (the size of the packed outputs). */
fw_status fw_ragged_compact(const void *K, const void *V, int32_t cells, int32_t T,
                            int32_t row_bytes, const int64_t *offsets, const int32_t *kept_pos,
                            int64_t total, void *K_out, void *V_out, void *stream);

/* The observation-window importance score (Sec. 4 runs ContourKV with
 * SnapKV's window score as well as with a reconstruction score): the last w
 * query rows of a cell vote for the keys they attend to.  For cell c, keys
 * K[c][j] (j < T) and window queries Qw[c][i] (i < w; query i sits at
 * position T - w + i and sees the keys j <= T - w + i):
 *   a_ij   = softmax over the visible keys of scale * q_i . k_j,
 *   vote_j = sum_i a_ij,
 *   scores[c][j] = max of vote over positions [j - pool/2, j + pool/2]
 *                  clipped to the prefix [0, T - w), for prefix positions;
 *                  vote_j itself for the w window positions (which a
 *                  ContourKV floor of at least w keeps anyway).
 * The output feeds fw_contour_alloc as its importance score.
 *   Qw : bf16 [cells][w][d];  K : bf16 [cells][T][d] (the cache's keys);
 *        both 16-byte aligned.  d in {64, 128}; 1 <= w <= min(32, T);
 *        pool odd >= 1 (SnapKV: 7); scale > 0 (1 / sqrt(d) for attention).
 *   scores : fp32 [cells][T]; status [cells] (may be NULL): FW_OK, or
 *        FW_ERR_TIMEOUT if a bounded wait of the cell's CTA gave up.
 * Workspace: the votes, cells x T fp32.  The products run on the tensor
 * cores (bf16 inputs, fp32 accumulation), the key tiles arrive by TMA;
 * cells x T must stay below 2^31. */
fw_status fw_window_score(const void *Qw, const void *K, int32_t cells, int32_t T, int32_t d, int32_t w, float scale,
                          int32_t pool, float *scores, int32_t *status, void *workspace, size_t workspace_bytes,
                          void *stream);
size_t fw_window_score_workspace(int32_t cells, int32_t T);

/* Ragged per-head storage with room to grow (Sec. 4's ragged storage for the
 * multi-turn case of Sec. 1, where one compressed cache serves every later
 * query while decode keeps appending to it).  Cell h owns rows
 * [base[h], base[h] + capacity[h]) of K_store and V_store ([rows][row_bytes]
 * each, device).
 * fw_ragged_compact_to: as fw_ragged_compact, but cell h's kept rows go to
 *   its own rows from base[h] on; a cell whose count (offsets[h+1] -
 *   offsets[h]) exceeds capacity[h] is not copied and gets status[h] =
 *   FW_ERR_WORKSPACE (status [cells] may be NULL).
 * fw_ragged_append: appends m new rows per cell (new_K, new_V: [cells][m]
 *   [row_bytes], device) behind its counts[h] filled rows and adds m to
 *   counts[h] (device, in/out); a cell without room for all m rows takes none
 *   and gets status[h] = FW_ERR_WORKSPACE, its count unchanged.  A decode step
 *   is m = 1; a prefill chunk appends several.  Calls on one stream see each
 *   other's counts in order.
 * row_bytes: a positive multiple of 16; all row pointers 16-byte aligned. */
fw_status fw_ragged_compact_to(const void *K, const void *V, int32_t cells, int32_t T, int32_t row_bytes,
                               const int64_t *offsets, const int32_t *kept_pos, const int64_t *base,
                               const int32_t *capacity, void *K_store, void *V_store, int32_t *status, void *stream);
fw_status fw_ragged_append(void *K_store, void *V_store, const int64_t *base, const int32_t *capacity, int32_t *counts,
                           const void *new_K, const void *new_V, int32_t cells, int32_t m, int32_t row_bytes,
                           int32_t *status, void *stream);

/* Largest cells accepted by fw_contour_alloc_noalloc. */
#define FW_CONTOUR_NOALLOC_MAX_CELLS 4096

/* fw_contour_alloc for callers that cannot allocate device memory.
 * The paper has no counterpart: this is a deployment convenience.  Some
 * callers may not call cudaMalloc at all -- a plugin living inside another
 * framework's device-memory pool, or a latency-critical path where a
 * cudaMalloc would synchronise the device -- and cannot provide the
 * workspace fw_contour_alloc asks for.  This variant takes the same
 * arguments minus the workspace and uses a scratch area compiled into the
 * library instead: 333,568 bytes (80 bytes per cell of the maximum: four
 * per-cell words, a 48-byte cell record and a 16-byte slice record, no call
 * using more than max(cells, 2048) slices; plus 5,888 bytes of histograms,
 * radix state and alignment), held by every GPU that loads the library
 * until the process exits.
 *   - cells must be <= FW_CONTOUR_NOALLOC_MAX_CELLS, otherwise the call
 *     returns FW_ERR_WORKSPACE and launches nothing; the other argument
 *     rules and all outputs are exactly those of fw_contour_alloc.
 *   - It never allocates or frees device memory.
 *   - Every call looks up the scratch area's address in the current
 *     device's context (a host-side query), so the address stays right after
 *     a device reset.  The first call on a device may load the library's
 *     module there; make that first call before any stream capture on the
 *     device.
 *   - All calls share the one scratch area and every call re-initialises
 *     what it reads, so consecutive calls are independent; calls that
 *     overlap on the GPU (concurrent streams, several host threads) race on
 *     the scratch and must be serialised by the caller. */
fw_status fw_contour_alloc_noalloc(const float *scores, int32_t cells, int32_t T, int32_t floor,
                                   int64_t total_budget, int32_t uniform_s, int32_t *counts,
                                   int64_t *offsets, int32_t *kept_pos, float *tau,
                                   float *dropped_uniform, float *dropped_alloc, void *stream);

/* Waits for `stream` and reports the device-side outcome of the work queued
 * on it: FW_ERR_CUDA if the stream holds a failed launch or a device fault,
 * otherwise the first status other than FW_OK in row_status[0 .. rows) (a
 * per-row status array that an entry point above filled on that stream),
 * with its row in *first_row (-1, and FW_OK, when every row is fine;
 * first_row may be NULL).  row_status is device memory; it is read through
 * a host buffer on the stack, so the call allocates nothing. */
fw_status fw_sync_status(const int32_t *row_status, int64_t rows, int64_t *first_row, void *stream);

/* Measurement aid, not part of the path: `blocks` CTAs of 256 threads each
 * run `iters` iterations of 16 independent fp32 FMA chains (so 256 * 16 *
 * iters FMAs per CTA, 2 flops each) and write one float per thread to
 * out [blocks * 256] (device) so the work is kept.  Timed by the caller, it
 * measures the fp32 FMA throughput that the exact search's ALU roofline is
 * stated against.  FW_ERR_INVALID_ARG for blocks < 1 or iters < 1. */
fw_status fw_fp32_fma_probe(int32_t blocks, int32_t iters, float *out, void *stream);

/* Human-readable name of a status. */
const char *fw_status_string(fw_status s);

/* Number of kernels this library has launched since it was loaded. */
uint64_t fw_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* FW_H */
