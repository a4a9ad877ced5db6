#pragma once

// Decode-row attention (one query token per sequence), split over the context:
// the body of one decode CTA, shared by the decode kernel and the single
// launch of a mixed step.
//
// A decode row is bandwidth-bound: every K/V byte is read once and used by
// the group's q-heads only.  One CTA takes one (row, kv-head, split): its
// pages are fetched by TMA (two 16x64 boxes per page and matrix, 128-byte
// swizzle) into a 3-stage ring per warp (eight warps, so eight threads issue
// copies; one issuing thread alone moves only ~7 B/clk); the split's page ids
// are staged in shared memory first.  Each warp computes
//   S^T[heads x 16 keys] = Q[heads x 128] . K_page^T     (mma.sync m16n8k16)
//   online softmax per head (fp32, exp2 domain)
//   O[heads x 128] += P[heads x 16 keys] . V_page         (mma.sync m16n8k16)
// with the group's q-heads as the MMA rows (rows >= group are zero).  The
// warps merge their (m, l, O) in shared memory; with several splits the
// partial goes to the workspace and the last CTA of the (row, kv-head) to
// finish merges all splits:
//   o = sum_i 2^(m_i - M) o_i / sum_i 2^(m_i - M) l_i,  M = max_i m_i.
// The splits count their arrivals in a 64-bit ticket per (row, kv-head)
// that carries the launch's tag (tags increase from launch to launch), so
// tickets never need clearing before a launch; the kernel is launched with
// programmatic stream serialization and touches global memory only after
// grid_dep_wait().
#include <math.h>

#include "ppas_device.cuh"
#include "ppas_internal.h"

namespace ppas {
namespace decode_detail {

constexpr uint32_t kBox = 2048;                     // 16 rows x 128 B
constexpr uint32_t kStageBytes = 4 * kBox;          // K lo, K hi, V lo, V hi
constexpr uint32_t kRingBytes = kDecodeStages * kStageBytes;
constexpr uint32_t kOffBar = kDecodeWarps * kRingBytes;
constexpr uint32_t kOffFlag = kOffBar + kDecodeWarps * kDecodeStages * 8;
constexpr uint32_t kOffIds = kOffFlag + 16;   // page ids of this split
// a cluster's merge: rank 0's slots for the cluster's CTA partials
// ([rank][group][128] O, then [rank][group][2] (m, l)), outside the rings,
// which a slower CTA of the cluster may still be streaming through when a
// faster one writes its partial
constexpr int kMaxCluster = 4;
constexpr uint32_t kOffClusterRecv = kOffIds + kDecodeMaxPagesPerSplit * 4;
constexpr uint32_t kClusterRecvBytes = kMaxCluster * 8 * (kHeadDim + 2) * 4;
constexpr uint32_t kSmemBytes = kOffClusterRecv + kClusterRecvBytes + 1024;
static_assert(kSmemBytes <= 232448, "shared memory per CTA");
// merge scratch (aliases the rings once every warp is done)
constexpr int kMaxGroup = 8;
static_assert(kDecodeWarps * kMaxGroup * (2 + kHeadDim) * 4 <= static_cast<int>(kOffBar), "merge scratch");
static_assert(2 * kMaxDecodeSplitsPerRow * kMaxGroup * 4 <= static_cast<int>(kOffBar), "split weights");
static_assert(kDecodeWarps >= kMaxGroup, "the split merge gives each head of a group one warp");
static_assert(kClusterRecvBytes == kMaxCluster * kMaxGroup * (kHeadDim + 2) * 4, "cluster slots");

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// byte offset of 16-byte chunk `chunk` (0..15 over 128 columns) of `row` in
// a page stored as two 16-row x 128 B halves with the 128-byte swizzle
__device__ __forceinline__ uint32_t swz(int row, int chunk) {
    return static_cast<uint32_t>((chunk >> 3) * kBox + row * 128 + (((chunk & 7) ^ (row & 7)) << 4));
}

}  // namespace decode_detail

constexpr int kDecodeThreads = kDecodeWarps * 32;
constexpr uint32_t kDecodeSmemBytes = decode_detail::kSmemBytes;

// The CTA-wide barrier of the decode body: all threads of a decode launch,
// or the kDecodeThreads threads that run it inside a larger CTA (named
// barrier 1).
template <bool kPartial>
__device__ __forceinline__ void decode_cta_sync() {
    if constexpr (kPartial)
        nbar_sync(1, kDecodeThreads);
    else
        __syncthreads();
}

// One (row, kv-head, split) of a step's decode rows: CTA `bid` of the decode
// plan in p, run by threads 0 .. kDecodeThreads - 1 of the CTA (kPartial:
// the CTA has more threads, which do not take part).
template <bool kPartial, class P>
__device__ __forceinline__ void decode_cta(const CUtensorMap &tm_k, const CUtensorMap &tm_v, const P &p, int bid) {
    // in a cluster launch every CTA announces that it has started; the
    // matching wait comes before the first store into another CTA's shared
    // memory (the barrier phases of every CTA: this one, then one after
    // the stores, on every path)
    if constexpr (!kPartial)
        if (cluster_nctarank() > 1) cluster_arrive_relaxed();
    using namespace decode_detail;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_s = smem_u32(smem_raw);
    const uint32_t sb = (raw_s + 1023u) & ~1023u;
    uint8_t *const sg = smem_raw + (sb - raw_s);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    // ---- which (row, kv-head, split)
    int lo = 0, hi = p.n_rows - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.rows[mid].cta_base <= bid) lo = mid; else hi = mid - 1;
    }
    const DecodeRow row = p.rows[lo];
    const int local = bid - row.cta_base;
    const int kvh = local / row.n_splits, sp = local % row.n_splits;
    const int g = p.group;
    const int n_pages = (row.ctx_len + kPage - 1) / kPage;
    const int pg0 = sp * row.pages_per_split;
    const int pg1 = min(pg0 + row.pages_per_split, n_pages);
    const int my_count = max(0, (pg1 - pg0 - warp + kDecodeWarps - 1) / kDecodeWarps);
    const int32_t *table = p.block_tables + static_cast<int64_t>(row.table_row) * p.table_stride;
    volatile int *abort_flag = reinterpret_cast<volatile int *>(sg + kOffFlag);

    const uint32_t ring = sb + warp * kRingBytes;
    auto bar = [&](int st) { return sb + kOffBar + (warp * kDecodeStages + st) * 8u; };
    int32_t *ids = reinterpret_cast<int32_t *>(sg + kOffIds);
    if (lane == 0) {
        for (int st = 0; st < kDecodeStages; ++st) mbar_init(bar(st), 1);
        fence_mbar_init();
    }
    if (tid == 0) *abort_flag = 0;
    // the set-up above overlaps the kernel before this one on the stream;
    // global memory (page ids, Q, pages, workspace, output) only after it
    grid_dep_wait();
    // the split's page ids, loaded once by every thread in parallel
    for (int i = tid; i < pg1 - pg0; i += kDecodeThreads) ids[i] = __ldg(table + pg0 + i);
    decode_cta_sync<kPartial>();

    auto issue = [&](int i) {
        const int st = i % kDecodeStages;
        const int pg = pg0 + warp + kDecodeWarps * i;
        int blk = ids[pg - pg0];
        if (blk < 0 || blk >= p.num_blocks) {
            report_error(p.err, PPAS_DEVERR_BAD_INDEX);
            blk = 0;
        }
        const int r = (blk * p.n_kv_heads + kvh) * kPage;
        const uint32_t dst = ring + st * kStageBytes, b = bar(st);
        mbar_expect_tx(b, kStageBytes);
        tma_load_2d(dst, &tm_k, 0, r, b);
        tma_load_2d(dst + kBox, &tm_k, 64, r, b);
        tma_load_2d(dst + 2 * kBox, &tm_v, 0, r, b);
        tma_load_2d(dst + 3 * kBox, &tm_v, 64, r, b);
    };
    if (lane == 0)
        for (int i = 0; i < min(kDecodeStages, my_count); ++i) issue(i);

    // ---- Q as the A operand: rows = the group's heads, k = head dims
    const int hr = lane >> 2, c = lane & 3;
    uint32_t qa[8][4];
    {
        const bool valid = hr < g;
        const uint32_t *qrow = reinterpret_cast<const uint32_t *>(
            p.q + (static_cast<int64_t>(row.q_row) * p.n_q_heads + kvh * g + (valid ? hr : 0)) * kHeadDim);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
            qa[kk][0] = valid ? __ldg(qrow + kk * 8 + c) : 0u;
            qa[kk][1] = 0u;
            qa[kk][2] = valid ? __ldg(qrow + kk * 8 + 4 + c) : 0u;
            qa[kk][3] = 0u;
        }
    }

    float m_run = -INFINITY, l_run = 0.f;
    float o[16][4];
#pragma unroll
    for (int n = 0; n < 16; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
    const float sl2 = p.scale_log2;
    int consumed = 0;

    for (int i = 0; i < my_count; ++i) {
        const int st = i % kDecodeStages;
        const bool ok = __all_sync(0xffffffffu, mbar_wait(bar(st), (i / kDecodeStages) & 1, p.err));
        if (!ok) {
            *abort_flag = 1;
            break;
        }
        consumed = i + 1;
        const int pg = pg0 + warp + kDecodeWarps * i;
        const int valid = min(kPage, row.ctx_len - pg * kPage);
        const uint32_t kb = ring + st * kStageBytes, vb = kb + 2 * kBox;
        if (valid < kPage) {
            // tokens past the context: zero their V rows so that 0 * V stays 0
            uint8_t *vg = sg + (vb - sb);
            const int n = (kPage - valid) * 8;
            for (int x = lane; x < 2 * n; x += 32) {
                const int half = x / n, rr = valid + (x % n) / 8, ch = x % 8;
                *reinterpret_cast<uint4 *>(vg + half * kBox + rr * 128 + ch * 16) = make_uint4(0, 0, 0, 0);
            }
            fence_proxy_async_smem();
            __syncwarp();
        }
        // S = Q K^T for the 16 tokens of the page (two n-tiles of 8 tokens)
        float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
        {
            const int mi = lane >> 3, ri = lane & 7;
            const int tok = (mi >> 1) * 8 + ri;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4(kb + swz(tok, kk * 2 + (mi & 1)), b0, b1, b2, b3);
                mma_bf16_16816(s0, qa[kk], b0, b1);
                mma_bf16_16816(s1, qa[kk], b2, b3);
            }
        }
        const float x0 = (2 * c < valid) ? s0[0] * sl2 : -INFINITY;
        const float x1 = (2 * c + 1 < valid) ? s0[1] * sl2 : -INFINITY;
        const float x2 = (8 + 2 * c < valid) ? s1[0] * sl2 : -INFINITY;
        const float x3 = (9 + 2 * c < valid) ? s1[1] * sl2 : -INFINITY;
        float mx = fmaxf(fmaxf(x0, x1), fmaxf(x2, x3));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        const float m_new = fmaxf(m_run, mx);
        const float alpha = ex2(m_run - m_new);
        m_run = m_new;
        const float e0 = ex2(x0 - m_new), e1 = ex2(x1 - m_new), e2 = ex2(x2 - m_new), e3 = ex2(x3 - m_new);
        l_run = l_run * alpha + (e0 + e1) + (e2 + e3);
#pragma unroll
        for (int n = 0; n < 16; ++n) {
            o[n][0] *= alpha;
            o[n][1] *= alpha;
        }
        const uint32_t pa[4] = {pack_bf16x2(e0, e1), 0u, pack_bf16x2(e2, e3), 0u};
        {
            const int mi = lane >> 3, ri = lane & 7;
            const int tok = (mi & 1) * 8 + ri;
#pragma unroll
            for (int n2 = 0; n2 < 8; ++n2) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(vb + swz(tok, n2 * 2 + (mi >> 1)), b0, b1, b2, b3);
                mma_bf16_16816(o[2 * n2], pa, b0, b1);
                mma_bf16_16816(o[2 * n2 + 1], pa, b2, b3);
            }
        }
        __syncwarp();
        if (lane == 0 && i + kDecodeStages < my_count) issue(i + kDecodeStages);
    }
    // copies still in flight (only after an abort)
    if (lane == 0)
        for (int i = consumed; i < min(consumed + kDecodeStages, my_count); ++i)
            mbar_wait(bar(i % kDecodeStages), (i / kDecodeStages) & 1, nullptr);

    l_run += __shfl_xor_sync(0xffffffffu, l_run, 1);
    l_run += __shfl_xor_sync(0xffffffffu, l_run, 2);

    decode_cta_sync<kPartial>();  // rings are free from here on
    float *cm = reinterpret_cast<float *>(sg);
    float *cl = cm + kDecodeWarps * kMaxGroup;
    float *co = cl + kDecodeWarps * kMaxGroup;
    if (hr < g) {
        if (c == 0) {
            cm[warp * kMaxGroup + hr] = m_run;
            cl[warp * kMaxGroup + hr] = l_run;
        }
        float *dst = co + (warp * kMaxGroup + hr) * kHeadDim;
#pragma unroll
        for (int n = 0; n < 16; ++n) *reinterpret_cast<float2 *>(dst + n * 8 + 2 * c) = make_float2(o[n][0], o[n][1]);
    }
    decode_cta_sync<kPartial>();
    // CTAs per thread-block cluster: 1 unless the launch groups the splits of
    // a (row, kv-head) into clusters (steps of decode rows only)
    const uint32_t nct = kPartial ? 1u : cluster_nctarank();
    // (in a cluster an aborted CTA carries on to the cluster barrier below)
    if (nct == 1 && *abort_flag) return;
    // rank 0's slot for this CTA's partial (cluster launches only)
    const uint32_t crank = nct > 1 ? cluster_ctarank() : 0u;
    const uint32_t recv = sb + kOffClusterRecv;
    const uint32_t slot_o = nct > 1 ? dsmem_addr(recv + crank * (kMaxGroup * kHeadDim * 4), 0) : 0u;
    const uint32_t slot_ml =
        nct > 1 ? dsmem_addr(recv + kMaxCluster * kMaxGroup * kHeadDim * 4 + crank * (kMaxGroup * 2 * 4), 0) : 0u;
    if (nct > 1) cluster_wait();  // every CTA of the cluster has started (its arrive at entry)

    // thread -> (head-dim column, first head); the CTA's threads cover
    // kDecodeThreads / 128 heads at a time
    const int t = tid & (kHeadDim - 1);
    const int hstep = kDecodeThreads / kHeadDim;
    for (int hh = tid / kHeadDim; hh < g; hh += hstep) {
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kDecodeWarps; ++w) M = fmaxf(M, cm[w * kMaxGroup + hh]);
        float L = 0.f, O = 0.f;
#pragma unroll
        for (int w = 0; w < kDecodeWarps; ++w) {
            // a warp without keys (or a split past its row's pages, which a
            // cluster plan may hold) has m = -inf and weight 0
            const float m = cm[w * kMaxGroup + hh];
            const float f = m == -INFINITY ? 0.f : ex2(m - M);
            L += f * cl[w * kMaxGroup + hh];
            O += f * co[(w * kMaxGroup + hh) * kHeadDim + t];
        }
        const int head = kvh * g + hh;
        if (row.n_splits == 1) {
            const int64_t oi = (static_cast<int64_t>(row.q_row) * p.n_q_heads + head) * kHeadDim + t;
            if (p.out_fp32) static_cast<float *>(p.out)[oi] = O / L;
            else static_cast<__nv_bfloat16 *>(p.out)[oi] = __float2bfloat16_rn(O / L);
        } else if (nct > 1) {
            dsmem_st_f32(slot_o + static_cast<uint32_t>(hh * kHeadDim + t) * 4u, O);
            if (t == 0) {
                dsmem_st_f32(slot_ml + static_cast<uint32_t>(hh * 2) * 4u, M);
                dsmem_st_f32(slot_ml + static_cast<uint32_t>(hh * 2 + 1) * 4u, L);
            }
        } else {
            const int64_t pi = static_cast<int64_t>(row.part_base + sp) * p.n_q_heads + head;
            p.part_o[pi * kHeadDim + t] = O;
            if (t == 0) {
                p.part_ml[pi * 2] = M;
                p.part_ml[pi * 2 + 1] = L;
            }
        }
    }
    if (row.n_splits == 1) return;
    int n_parts = row.n_splits;  // partial slots of this (row, kv-head)
    if constexpr (!kPartial) {
        if (nct > 1) {
            // The cluster's CTAs are consecutive splits sp0 .. sp0 + nct - 1
            // of this (row, kv-head) (sp0 a multiple of nct, rank = sp -
            // sp0).  Each has stored its partial into rank 0's slots above;
            // after the barrier (every CTA reaches it, an aborted one too)
            // rank 0 merges them from its own shared memory into partial
            // slot sp0 / nct, and the others are done.
            cluster_sync_all();
            if (crank != 0) return;
            const float *ro = reinterpret_cast<const float *>(sg + kOffClusterRecv);
            const float *rml = ro + kMaxCluster * kMaxGroup * kHeadDim;
            for (int hh = tid / kHeadDim; hh < g; hh += hstep) {
                float M = -INFINITY;
                for (uint32_t r = 0; r < nct; ++r) M = fmaxf(M, rml[(r * kMaxGroup + hh) * 2]);
                float L = 0.f, O = 0.f;
                for (uint32_t r = 0; r < nct; ++r) {
                    const float m = rml[(r * kMaxGroup + hh) * 2];
                    const float f = m == -INFINITY ? 0.f : ex2(m - M);
                    L += f * rml[(r * kMaxGroup + hh) * 2 + 1];
                    O += f * ro[(r * kMaxGroup + hh) * kHeadDim + t];
                }
                const int64_t pi =
                    static_cast<int64_t>(row.part_base + sp / static_cast<int>(nct)) * p.n_q_heads + kvh * g + hh;
                p.part_o[pi * kHeadDim + t] = O;
                if (t == 0) {
                    p.part_ml[pi * 2] = M;
                    p.part_ml[pi * 2 + 1] = L;
                }
            }
            n_parts = row.n_splits / static_cast<int>(nct);
        }
    }

    // ---- the last CTA of this (row, kv-head) merges every split
    __threadfence();
    decode_cta_sync<kPartial>();
    __shared__ int s_last;
    if (tid == 0) {
        // ticket = (tag << 16) | arrivals.  Tags grow from launch to launch, so
        // atomicMax turns a word left by an earlier launch (or reset to 0)
        // into this launch's tag with no arrivals, and leaves a word this
        // launch already owns alone; only a word with a larger tag (memory
        // nothing of this process wrote) is claimed by compare-and-swap.
        // Then every split adds its arrival: two atomics, no retries.
        unsigned long long *ctr = p.counters + lo * p.n_kv_heads + kvh;
        const unsigned long long mine = p.launch_tag << 16;
        unsigned long long cur = atomicMax(ctr, mine);
        for (int it = 0; (cur >> 16) > p.launch_tag && it < (1 << 20); ++it) {
            const unsigned long long got = atomicCAS(ctr, cur, mine);
            cur = got == cur ? mine : got;
        }
        const unsigned long long old = atomicAdd(ctr, 1ull);
        const int prev = (old >> 16) == p.launch_tag ? static_cast<int>(old & 0xFFFFull) : -1;
        if (prev < 0) report_error(p.err, PPAS_DEVERR_TIMEOUT);  // the word was never claimed
        s_last = (prev == n_parts - 1);
        if (s_last) *ctr = 0;  // also ready for a replay with the same tag (a captured graph)
    }
    decode_cta_sync<kPartial>();
    if (!s_last) return;
    __threadfence();
    // Warp hh merges head hh on its own (lane: 4 columns).  The first 16
    // splits' O go out before the weights are known, so their latency hides
    // that of the (m, l) round; the weights w = 2^(m - M) stay in a
    // shared-memory row of the warp (the rings are free), 1 / L is applied
    // at the end.
    const int ns = n_parts;
    const int hh = warp, c4 = lane;
    if (hh >= g) return;
    const int head = kvh * g + hh;
    const float4 *po = reinterpret_cast<const float4 *>(p.part_o) + c4;
    auto part_index = [&](int s_) { return static_cast<int64_t>(row.part_base + s_) * p.n_q_heads + head; };
    float4 ov[16];
#pragma unroll
    for (int k = 0; k < 16; ++k)
        ov[k] = k < ns ? __ldcg(po + part_index(k) * (kHeadDim / 4)) : make_float4(0.f, 0.f, 0.f, 0.f);
    float *wm = reinterpret_cast<float *>(sg) + hh * 2 * kMaxDecodeSplitsPerRow;  // [ns] m, then w
    float *wl = wm + kMaxDecodeSplitsPerRow;                                     // [ns] l
    float M = -INFINITY;
    for (int s_ = lane; s_ < ns; s_ += 32) {
        const float2 ml = __ldcg(reinterpret_cast<const float2 *>(p.part_ml + part_index(s_) * 2));
        wm[s_] = ml.x;
        wl[s_] = ml.y;
        M = fmaxf(M, ml.x);
    }
#pragma unroll
    for (int o_ = 16; o_ >= 1; o_ >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o_));
    float L = 0.f;
    for (int s_ = lane; s_ < ns; s_ += 32) {
        const float m = wm[s_];
        const float f = m == -INFINITY ? 0.f : ex2(m - M);
        wm[s_] = f;
        L += f * wl[s_];
    }
#pragma unroll
    for (int o_ = 16; o_ >= 1; o_ >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o_);
    __syncwarp();
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s0 = 0; s0 < ns; s0 += 16) {
        if (s0 > 0) {
#pragma unroll
            for (int k = 0; k < 16; ++k)
                ov[k] = s0 + k < ns ? __ldcg(po + part_index(s0 + k) * (kHeadDim / 4)) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int k = 0; k < 16; ++k) {
            const float f = s0 + k < ns ? wm[s0 + k] : 0.f;
            acc = make_float4(acc.x + f * ov[k].x, acc.y + f * ov[k].y, acc.z + f * ov[k].z, acc.w + f * ov[k].w);
        }
    }
    const float inv_l = 1.f / L;
    acc = make_float4(acc.x * inv_l, acc.y * inv_l, acc.z * inv_l, acc.w * inv_l);
    const int64_t oi = (static_cast<int64_t>(row.q_row) * p.n_q_heads + head) * kHeadDim + 4 * c4;
    if (p.out_fp32) {
        *reinterpret_cast<float4 *>(static_cast<float *>(p.out) + oi) = acc;
    } else {
        *reinterpret_cast<uint2 *>(static_cast<__nv_bfloat16 *>(p.out) + oi) =
            make_uint2(pack_bf16x2(acc.x, acc.y), pack_bf16x2(acc.z, acc.w));
    }
}

}  // namespace ppas
