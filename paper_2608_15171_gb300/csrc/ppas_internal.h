// Internal structures shared by the host launchers and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stddef.h>
#include <stdint.h>

#include <vector>

#include "ppas.h"

namespace ppas {

constexpr int kPage = PPAS_PAGE_TOKENS;        // tokens per KV block
constexpr int kHeadDim = 128;                  // the only head size with kernels
constexpr int kRowBytes = kHeadDim * 2;        // one bf16 K or V row
constexpr int kPageBytes = kPage * kRowBytes;  // one (block, kv-head) page: 4 KB

// ------------------------------------------------------------------ prefill
// Rows with q_len > 1.  One CTA computes one 128-token query tile of
// heads_per_cta q-heads of one kv-head over a range of its causal KV tiles.
// Long ranges are split over several CTAs (split-KV); each split writes a
// partial (m, l, O) and the last CTA of the tile merges them.
constexpr int kTileQ = 128;            // query tokens per tile (tcgen05 M)
constexpr int kPrefillKT = 128;        // keys per KV tile
constexpr int kMaxPrefillSeqs = 128;
constexpr int kMaxPrefillWork = 1024;  // work items per launch
// split-KV sizing: a step is cut into about this many CTAs, with at least
// kPrefillMinSplitTiles KV tiles per CTA and at most kPrefillMaxSplits per tile
constexpr int64_t kPrefillTargetCtas = 304;
constexpr int kPrefillMinSplitTiles = 16;
constexpr int kPrefillMaxSplits = 64;

struct PrefillSeq {
    int32_t q_start;   // first row of the sequence in packed q / out
    int32_t q_len;
    int32_t ctx_len;
    int32_t table_row; // row of d_block_tables
};

struct PrefillWork {
    uint32_t seq_qt;    // (launch-local sequence << 16) | q tile
    uint32_t kt_range;  // (first KV tile << 16) | end KV tile (exclusive)
    int32_t part;       // first partial slot of this tile's splits; -1: not split
    uint32_t split;     // (number of splits << 16) | this split
};

struct PrefillParams {
    const int32_t *block_tables;
    int32_t table_stride;
    int32_t num_blocks;
    void *out;
    int32_t out_fp32;
    int32_t n_q_heads;
    int32_t n_kv_heads;
    int32_t group;          // n_q_heads / n_kv_heads
    int32_t heads_per_cta;  // 2 when the group has >= 2 heads, else 1
    float scale_log2;       // scale * log2(e)
    int32_t *err;
    float *part_o;          // [n_part, slots, heads_per_cta, 4 chunks, 128 rows, 32]
    float *part_ml;         // [n_part, slots, heads_per_cta, 128 rows, 2]
    int32_t *tickets;       // [n_part, slots] (first slot of each split tile)
    int32_t n_work;         // work items in this launch; grid = n_work * slots
    PrefillWork work[kMaxPrefillWork];  // heaviest first
    PrefillSeq seqs[kMaxPrefillSeqs];
};

struct PrefillItem {
    int32_t seq, qt, kt0, kt1, part, split, n_splits;
};

struct PrefillPlan {
    std::vector<PrefillItem> items;  // sorted heaviest first
    int64_t n_part = 0;
    int32_t slots = 0, heads_per_cta = 1;
    size_t o_bytes = 0, ml_bytes = 0, ticket_bytes = 0;
    size_t total_bytes() const { return o_bytes + ml_bytes + ticket_bytes; }
};

PrefillPlan plan_prefill(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                         int32_t n_kv_heads, bool allow_split);

// ------------------------------------------------------------------ decode
// Rows with q_len == 1.  One CTA handles one (row, kv-head, split): the
// split's pages are spread over the CTA's warps; partial (m, l, o) go to the
// workspace and the last CTA of a (row, kv-head) combines them.
constexpr int kDecodeWarps = 8;        // each warp streams its own pages (8 TMA issuers per SM)
constexpr int kDecodeStages = 3;       // pages in flight per warp
constexpr int kDecodeMaxPagesPerSplit = 1024;  // page ids of a split are staged in shared memory
constexpr int kMaxDecodeRows = 256;
constexpr int kDecodeMinPagesPerSplit = 16;

struct DecodeRow {
    int32_t q_row;       // row of packed q / out
    int32_t ctx_len;
    int32_t table_row;
    int32_t n_splits;
    int32_t pages_per_split;
    int32_t cta_base;    // first CTA of this row (all kv-heads)
    int32_t part_base;   // first partial slot (units of splits) of this row
};

struct DecodeParams {
    const __nv_bfloat16 *q;
    const int32_t *block_tables;
    int32_t table_stride;
    int32_t num_blocks;
    void *out;
    int32_t out_fp32;
    int32_t n_q_heads;
    int32_t n_kv_heads;
    int32_t group;
    float scale_log2;
    float *part_ml;      // [n_part, n_q_heads, 2]   (m, l)
    float *part_o;       // [n_part, n_q_heads, 128] unnormalised
    int32_t *counters;   // [n_rows, n_kv_heads]
    int32_t *err;
    int32_t n_rows;
    int32_t n_ctas;
    DecodeRow rows[kMaxDecodeRows];
};

struct DecodePlan {
    std::vector<int32_t> rows;       // indices of q_len == 1 rows
    std::vector<int32_t> n_splits;   // per decode row
    std::vector<int32_t> pages_per_split;  // per decode row
    int64_t n_part = 0;              // sum of splits
    int64_t n_ctas = 0;
    size_t ml_bytes = 0, o_bytes = 0, counter_bytes = 0;
    size_t total_bytes() const { return ml_bytes + o_bytes + counter_bytes; }
};

// workspace the step needs without prefill splits (decode partials only)
size_t workspace_min_size(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                          int32_t n_kv_heads);

DecodePlan plan_decode(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                       int32_t n_kv_heads, int32_t num_sms);

int32_t device_sm_count();

// launchers (return a cudaError_t of the launch)
cudaError_t launch_wait_timeout(int32_t *err, unsigned long long limit_ns, cudaStream_t st);

cudaError_t launch_kv_append(const void *k_new, const void *v_new, const int32_t *slots, int32_t n_tokens,
                             void *k_cache, void *v_cache, int32_t num_blocks, int32_t n_kv_heads,
                             int32_t head_dim, int32_t *err, cudaStream_t st);

cudaError_t launch_prefill(const CUtensorMap &tm_q, const CUtensorMap &tm_k, const CUtensorMap &tm_v,
                           const PrefillParams &p, cudaStream_t st);

cudaError_t launch_decode(const CUtensorMap &tm_k, const CUtensorMap &tm_v, const DecodeParams &p,
                          cudaStream_t st);

// tensor maps (driver entry point fetched at run time)
bool encode_kv_map(CUtensorMap *map, const void *cache, int32_t num_blocks, int32_t n_kv_heads);
bool encode_q_map(CUtensorMap *map, const void *q, int32_t total_q, int32_t n_q_heads);

}  // namespace ppas
