// Internal structures shared by the host launchers and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stddef.h>
#include <stdint.h>

#include <atomic>
#include <memory>
#include <vector>

#include "ppas.h"

namespace ppas {

constexpr int kPage = PPAS_PAGE_TOKENS;        // tokens per KV block
constexpr int kHeadDim = 128;                  // the only head size with kernels
constexpr int kRowBytes = kHeadDim * 2;        // one bf16 K or V row
constexpr int kPageBytes = kPage * kRowBytes;  // one (block, kv-head) page: 4 KB
// SMs the step plans assume when no device can be queried (GB300); with a
// device the plans are made for its SM count (plan_sms()).
constexpr int32_t kDefaultPlanSms = 152;

// ------------------------------------------------------------------ prefill
// Rows with q_len > 1.  The kernel is persistent: one CTA per SM works
// through a list of items, each one 128-token query tile of heads_per_cta
// q-heads of one kv-head (a "head slot") over a range of its causal KV
// tiles.  The host lays the (tile, head slot) units end to end, longest
// first, and cuts the line into one equal segment per CTA (stream-K style),
// so a unit is split only where a segment ends.  Each piece of a split unit
// writes a partial (m, l, O) and a merge kernel launched after the prefill
// (or mixed) launch combines them.
constexpr int kTileQ = 128;             // query tokens per tile (tcgen05 M)
constexpr int kPrefillKT = 128;         // keys per KV tile
constexpr int kMaxPrefillSeqs = 128;    // per launch
constexpr int kMaxPrefillWork = 2200;   // items per launch (bounded by the 32 KB parameter space)
constexpr int kMaxPrefillCtas = 256;    // CTAs per launch (one per SM)
constexpr int kPrefillItemCost = 3;     // per-item overhead (Q load, pipeline fill, epilogue), in KV tiles
constexpr int kPrefillMinPiece = 4;     // shortest piece of a split unit, in KV tiles
// longest piece, in KV tiles: the tensor core's fp32 accumulation of O in
// TMEM loses ~7e-7 of |O| per tile, so pieces are capped and the merge
// (ordinary fp32) combines them
constexpr int kPrefillMaxPiece = 512;
constexpr int kPrefillMergeCost = 6;    // partial writes and the merge launch, in KV tiles
constexpr uint16_t kNoPart = 0xFFFF;    // an item of an unsplit unit

struct PrefillSeq {
    int32_t q_start;   // first row of the sequence in packed q / out
    int32_t q_len;
    int32_t ctx_len;
    int32_t table_row; // row of d_block_tables
};

struct PrefillWork {     // one item: (sequence, q tile, head slot, KV range)
    uint16_t qt;         // q tile within the sequence
    uint8_t seq;         // launch-local sequence
    uint8_t slot;        // q-heads slot * heads_per_cta ... + heads_per_cta - 1
    uint16_t kt0, kt1;   // KV tiles [kt0, kt1)
    uint16_t part;       // partial slot (launch-relative); kNoPart: unsplit
    uint16_t pad;
};
static_assert(sizeof(PrefillWork) == 12, "compact work item");

template <int kWork>
struct PrefillParamsT {
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
    float *part_o;          // [n_part, heads_per_cta, 4 chunks, 128 rows, 32]
    float *part_ml;         // [n_part, heads_per_cta, 128 rows, 2]
    int32_t n_ctas;         // CTAs running prefill items
    uint16_t cta_begin[kMaxPrefillCtas + 1];  // CTA c runs work[cta_begin[c] .. cta_begin[c + 1])
    PrefillWork work[kWork];
    PrefillSeq seqs[kMaxPrefillSeqs];
};
using PrefillParams = PrefillParamsT<kMaxPrefillWork>;
static_assert(sizeof(PrefillParams) + 3 * 128 <= 32764, "kernel parameter space");

// Merge of the split units' partials, launched after the prefill (or mixed)
// launch: one thread per (split unit, head of the slot, query row, 4 columns).
constexpr int kMaxMergeUnits = 1024;  // split units per merge launch

struct MergeUnit {
    int32_t out_row0;     // packed row of the tile's first query token
    int32_t part;         // first partial slot of the unit's pieces
    uint16_t rows_valid;  // query tokens of the tile
    uint16_t n_splits;    // pieces
    uint16_t head0;       // first q-head of the slot
    uint16_t pad;
};

struct MergeParams {
    const float *part_o;  // layouts as in PrefillParams
    const float *part_ml;
    void *out;
    int32_t out_fp32;
    int32_t n_q_heads;
    int32_t heads_per_cta;
    int32_t n_units;
    MergeUnit units[kMaxMergeUnits];
};

struct PrefillSplitUnit {
    int32_t seq, qt, slot, n_splits, part;
};

// one launch of the prefill kernel, as planned on the host
struct PrefillLaunchPlan {
    std::vector<int32_t> seqs;          // global sequence index per launch-local sequence
    std::vector<PrefillWork> work;      // grouped by CTA, in each CTA's order
    std::vector<uint16_t> cta_begin;    // n_ctas + 1 entries
    std::vector<PrefillSplitUnit> split_units;  // units of this launch cut into several pieces
    int32_t n_part = 0;                 // partial slots of this launch
};

struct PrefillPlan {
    std::vector<PrefillLaunchPlan> launches;
    int64_t n_part = 0;                 // most partial slots of one launch (the merge follows each launch)
    int32_t slots = 0, heads_per_cta = 1;
    size_t o_bytes = 0, ml_bytes = 0;
    bool empty() const { return launches.empty(); }
    size_t total_bytes() const { return o_bytes + ml_bytes; }
};

// SMs the persistent prefill kernel leaves to the decode launch of the same
// step on a device of num_sms SMs (0 without decode rows or without prefill
// chunks)
int32_t decode_reserve_sms(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                           int32_t n_kv_heads, int32_t num_sms);

// n_ctas: CTAs (SMs) the persistent kernel may occupy; allow_split == false
// keeps every unit whole (no workspace); max_work: items a launch may take
// (kMaxMixedWork for a step that may run as one mixed launch)
PrefillPlan plan_prefill(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                         int32_t n_kv_heads, bool allow_split, int32_t n_ctas, int32_t max_work = kMaxPrefillWork);

// ------------------------------------------------------------------ decode
// Rows with q_len == 1.  One CTA handles one (row, kv-head, split): the
// split's pages are spread over the CTA's warps; partial (m, l, o) go to the
// workspace and the last CTA of a (row, kv-head) combines them.
constexpr int kDecodeWarps = 8;        // each warp streams its own pages (8 TMA issuers per SM)
constexpr int kDecodeStages = 3;       // pages in flight per warp
constexpr int kDecodeMaxPagesPerSplit = 1024;  // page ids of a split are staged in shared memory
constexpr int kMaxDecodeSplitsPerRow = 2048;   // the merge keeps every split's weights in shared memory
// longest decode context: kMaxDecodeSplitsPerRow splits of kDecodeMaxPagesPerSplit pages
constexpr int64_t kMaxDecodeCtx = int64_t{kMaxDecodeSplitsPerRow} * kDecodeMaxPagesPerSplit * 16;
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

template <int kRows>
struct DecodeParamsT {
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
    // [n_rows, n_kv_heads] split tickets: (launch tag << 16) | arrivals; a
    // word with an older tag counts as no arrival, and the last arriver
    // resets its word to 0, so no call has to clear them
    unsigned long long *counters;
    unsigned long long launch_tag;  // 47 bits, never 0, larger for every launch
    int32_t *err;
    int32_t n_rows;
    int32_t n_ctas;
    DecodeRow rows[kRows];
};
using DecodeParams = DecodeParamsT<kMaxDecodeRows>;

// ------------------------------------------------------------------ mixed step
// A step with both kinds of rows runs as one launch when its plan fits these
// tables (the prefill items of one launch and up to kMaxMixedRows decode
// rows): CTAs [0, pf.n_ctas) run prefill items, the rest decode splits.
constexpr int kMaxMixedWork = kMaxPrefillWork;  // prefill items of a mixed launch
constexpr int kMaxMixedRows = 112;              // decode rows of a mixed launch (the rest of the 32 KB)
struct MixedParams {
    PrefillParamsT<kMaxMixedWork> pf;
    DecodeParamsT<kMaxMixedRows> dc;
};
static_assert(sizeof(MixedParams) + 3 * 128 <= 32764, "kernel parameter space");

struct DecodePlan {
    std::vector<int32_t> rows;       // indices of q_len == 1 rows
    std::vector<int32_t> n_splits;   // per decode row (a multiple of cluster)
    std::vector<int32_t> pages_per_split;  // per decode row
    // CTAs per thread-block cluster of the decode launch: the splits of a
    // (row, kv-head) come in groups of `cluster` consecutive CTAs that merge
    // their partials through distributed shared memory, so one partial slot
    // per group reaches the workspace (1: no clusters)
    int32_t cluster = 1;
    int64_t n_part = 0;              // partial slots: sum of splits / cluster
    int64_t n_ctas = 0;
    size_t ml_bytes = 0, o_bytes = 0, counter_bytes = 0;
    size_t total_bytes() const { return ml_bytes + o_bytes + counter_bytes; }
};

struct StepPlan {
    DecodePlan dp;
    PrefillPlan pf;
    int32_t n_ctas = 0;   // SMs the prefill launches may occupy
    bool mixed = false;   // prefill and decode rows in one launch
    size_t total_bytes() const { return dp.total_bytes() + pf.total_bytes(); }
};
// the plan of a step given the caller's workspace (SIZE_MAX: as large as it needs)
StepPlan plan_step(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                   int32_t n_kv_heads, size_t workspace_bytes);
// the same, from a small per-thread cache of the last plans (a step is
// planned once for all the layers that run it)
std::shared_ptr<const StepPlan> plan_step_cached(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens,
                                                 int32_t n_q_heads, int32_t n_kv_heads, size_t workspace_bytes);

// workspace the step needs without prefill splits (decode partials only)
size_t workspace_min_size(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                          int32_t n_kv_heads);

// How many decode CTAs can be co-resident in clusters of 2 and of 4 (0: no
// clusters, e.g. without a device).
struct DecodeClusterCaps {
    int32_t ctas2 = 0, ctas4 = 0;
};
DecodeClusterCaps decode_cluster_caps();  // the current device's, cached

// decode splits for a device of num_sms SMs: one wave of CTAs where the
// split-size limits allow it.  A step of decode rows only may run its
// splits in clusters (caps: what the device holds co-resident).
DecodePlan plan_decode(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                       int32_t n_kv_heads, int32_t num_sms, const DecodeClusterCaps &caps = {});

int32_t device_sm_count();
// SMs the current device's step plans are made for: its SM count, at most
// kMaxPrefillCtas (one persistent prefill CTA per SM); kDefaultPlanSms
// without a device
int32_t plan_sms();

// ------------------------------------------------------------------ gate-up projection
struct GateUpParams {
    __nv_bfloat16 *y;  // [n_tokens, inter]
    int32_t n_tokens;
    int32_t hidden;    // multiple of 64
    int32_t inter;     // multiple of 128
    int32_t *err;
};

// 2D bf16 row-major tensor [outer, inner] with a (box_inner x box_outer) box,
// 128-byte swizzle (box_inner * 2 bytes must be 128)
bool encode_bf16_2d(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer, uint32_t box_inner,
                    uint32_t box_outer);

cudaError_t launch_gateup(const CUtensorMap &tm_x, const CUtensorMap &tm_w, const GateUpParams &p, int grid,
                          cudaStream_t st);
cudaError_t launch_gateup_pack(const void *w, void *wp, int hidden, int inter, cudaStream_t st);

// launch configuration with programmatic stream serialization: the kernel
// may launch before its predecessor in the stream completes and orders its
// own global accesses after it with grid_dep_wait()
// Raises a kernel's dynamic shared memory limit, once per device (the
// attribute belongs to the device's context); safe from several threads.
template <typename Kernel>
cudaError_t ensure_smem_limit(Kernel *kernel, int bytes, std::atomic<uint64_t> &done) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = dev >= 0 && dev < 64 ? uint64_t{1} << dev : 0;
    if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_release);
    return e;
}

struct PdlLaunch {
    cudaLaunchAttribute attr[1];
    cudaLaunchConfig_t cfg;
    PdlLaunch(dim3 grid, dim3 block, size_t smem, cudaStream_t st) {
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg = cudaLaunchConfig_t{};
        cfg.gridDim = grid;
        cfg.blockDim = block;
        cfg.dynamicSmemBytes = smem;
        cfg.stream = st;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
    }
};

// launchers (return a cudaError_t of the launch)
cudaError_t launch_wait_timeout(int32_t *err, unsigned long long limit_ns, cudaStream_t st);

cudaError_t launch_kv_append(const void *k_new, const void *v_new, const int32_t *slots, int32_t n_tokens,
                             void *k_cache, void *v_cache, int32_t num_blocks, int32_t n_kv_heads,
                             int32_t head_dim, int32_t *err, cudaStream_t st);

cudaError_t launch_prefill_merge(const MergeParams &p, cudaStream_t st);
cudaError_t launch_prefill(const CUtensorMap &tm_q, const CUtensorMap &tm_k, const CUtensorMap &tm_v,
                           const PrefillParams &p, cudaStream_t st);
// one launch of a mixed step: p.pf.n_ctas prefill CTAs, then p.dc.n_ctas decode CTAs
cudaError_t launch_mixed(const CUtensorMap &tm_q, const CUtensorMap &tm_k, const CUtensorMap &tm_v,
                         const MixedParams &p, cudaStream_t st);

// cluster: CTAs per thread-block cluster (the plan's DecodePlan::cluster)
cudaError_t launch_decode(const CUtensorMap &tm_k, const CUtensorMap &tm_v, const DecodeParams &p,
                          int32_t cluster, cudaStream_t st);

// One-time per-device set-up the launchers otherwise do lazily on first use:
// the kernels' shared-memory limits and the side stream and events of mixed
// steps (for the current device).
cudaError_t prepare_prefill();
cudaError_t prepare_decode();
cudaError_t prepare_mixed();
cudaError_t prepare_current_device();

// tensor maps (driver entry point fetched at run time)
bool encode_kv_map(CUtensorMap *map, const void *cache, int32_t num_blocks, int32_t n_kv_heads);
bool encode_q_map(CUtensorMap *map, const void *q, int32_t total_q, int32_t n_q_heads);

}  // namespace ppas
