// Prefill-chunk attention on the 5th-generation tensor cores (tcgen05),
// as a persistent kernel.
//
// One CTA runs on each SM and works through a list of items, each one
// 128-token query tile of two q-heads of the same kv-head (one head when the
// group size is 1) over a range of 128-key KV tiles; both Q tiles share every
// K/V tile the CTA loads.  Per Q tile t the work is a chain
// S_t = Q_t K^T -> softmax -> P_t (bf16, written over S_t in TMEM) ->
// O_t += P_t V, and the two tiles' chains interleave on the tensor core.
// TMEM, the barriers and the K/V rings live across items, so an item's
// epilogue overlaps the next item's first Q K^T and its K/V loads.
// Warp roles (512 threads, four warpgroups):
//   warps 0-3   TMA producers: warps 0/1 fetch pages 0-3 / 4-7 of each K
//               tile (3-stage ring), warps 2/3 those of each V tile (2
//               stages), through the block table.  One issuing thread moves
//               only ~7 B/clk of small TMA boxes on GB300, so every tile is
//               fetched by two threads.
//   warps 4, 5  MMA issuers, one thread per Q tile: S_t = Q_t K^T (A = Q in
//               shared memory) and O_t += P_t V (A = P in TMEM); Q K^T for the
//               next tile is issued once P V has consumed P.
//   warp 6      Q loader: Q_t of the next item once the last Q K^T of the
//               current item on tile t has completed.
//   warps 8-11  softmax for tile 0, warps 12-15 for tile 1: each thread owns
//               one query row (its TMEM lane), loads its S row, masks by
//               absolute position, runs the online softmax in fp32 (exp2
//               domain) and stores P back to TMEM; at the end of an item it
//               writes O (or a piece's partial).  The two warpgroups take
//               turns, tile 0 then tile 1, so that one tile's softmax runs
//               under the other tile's MMAs.
// Registers move from the producer/MMA warpgroups to the softmax warpgroups
// with setmaxnreg.  The running max is only raised (and O rescaled in TMEM)
// when it grows by more than 2^8; until then the stale max keeps every
// exponent <= 2^8, and the final O / l is exact either way.
// The host plan may cut a long (query tile, head slot) unit into pieces on
// consecutive CTAs (stream-K): each piece writes its partial (m, l, O) to the
// workspace, and prefill_merge_kernel, launched after this kernel, combines
// the pieces of every cut unit.
// The same CTA body serves the mixed step's single launch (mixed_attn_kernel
// below), whose CTAs past the prefill ones run decode splits
// (attn_decode_body.cuh).
// The kernel is launched with programmatic stream serialization: its set-up
// (TMEM allocation, barriers, tensor-map prefetch) overlaps the kernel before
// it on the stream, and global memory is touched only after grid_dep_wait().
#include <math.h>

#include "attn_decode_body.cuh"
#include "ppas_device.cuh"
#include "ppas_internal.h"

namespace ppas {
namespace {

constexpr int kKT = kPrefillKT;              // keys per KV tile (128)
constexpr int kPagesPerTile = kKT / kPage;   // 8
constexpr int kNK = 3;                       // K ring depth
constexpr int kNV = 2;                       // V ring depth
constexpr uint32_t kBox = 2048;              // one TMA box: 16 rows x 128 B
constexpr uint32_t kHalf = 16384;            // 128 rows x 128 B (64 columns)
constexpr uint32_t kTileBytes = 2 * kHalf;   // a Q, K or V tile: 128 rows x 256 B

constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kOffQ + 2 * kTileBytes;
constexpr uint32_t kOffV = kOffK + kNK * kTileBytes;
constexpr uint32_t kOffBar = kOffV + kNV * kTileBytes;
enum : int {
    B_Q = 0,                   // [tile]
    B_QEMPTY = B_Q + 2,        // [tile]
    B_KFULL = B_QEMPTY + 2,
    B_KEMPTY = B_KFULL + kNK,
    B_VFULL = B_KEMPTY + kNK,
    B_VEMPTY = B_VFULL + kNV,
    B_SFULL = B_VEMPTY + kNV,  // [tile]
    B_PFULL = B_SFULL + 2,     // [tile]
    B_ODONE = B_PFULL + 2,     // [tile]
    B_TURN = B_ODONE + 2,      // [tile]: the softmax warpgroups take turns
    B_DRAIN = B_TURN + 2,
    B_COUNT = B_DRAIN + 1
};
constexpr uint32_t kOffTmem = kOffBar + B_COUNT * 8;
constexpr uint32_t kOffAbort = kOffTmem + 4;
static_assert(kOffAbort + 4 <= kOffBar + 256, "barrier area");
constexpr uint32_t kSmemBytes = kOffBar + 256 + 1024;  // + alignment slack
static_assert(kSmemBytes <= 232448, "shared memory per CTA");
constexpr uint32_t kTmemCols = 512;  // tile t: S/P at t*256, O at t*256 + 128
constexpr float kRescaleThreshold = 8.0f;  // log2 units
constexpr int kThreads = 512;
constexpr int kMmaWarp = 4;       // warps 4..7 form the MMA warpgroup
constexpr int kQWarp = 6;         // loads Q (warps 4, 5 issue MMAs)
constexpr int kSoftmaxWarp0 = 8;  // warps 8..11 tile 0, 12..15 tile 1
// register split: 8 warps x 56 + 8 warps x 200 = 512 threads x 128 at launch
constexpr int kRegsSmall = 56;
constexpr int kRegsLarge = 200;
static_assert(8 * 32 * kRegsSmall + 8 * 32 * kRegsLarge <= kThreads * 128, "register split");

constexpr uint32_t kIdescQK = idesc_bf16_f32(128, kKT, false, false);  // B = K rows (K-major)
constexpr uint32_t kIdescPV = idesc_bf16_f32(128, 128, false, true);   // B = V rows (MN-major)

__device__ __forceinline__ void tmem_ld32_sync(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
          "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
          "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// 64 TMEM columns of this warp's lanes (one S row per thread), waiting for
// completion before the registers are used.
__device__ __forceinline__ void tmem_ld64_sync(uint32_t taddr, float (&v)[64]) {
    uint32_t r[64];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x64.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,"
        "%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,"
        "%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%64];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
          "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
          "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]),
          "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]),
          "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]),
          "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]),
          "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 64; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_st32_f(uint32_t taddr, const float (&v)[32]) {
    uint32_t r[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(v[i]);
    tmem_st32(taddr, r);
}

// two fp32 lanes at once (Blackwell packed FP32 pipe)
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
    float2 r;
    asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
        "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return r;
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
    float2 r;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

// 32 consecutive output columns of one row, scaled by inv_l
template <class P>
__device__ __forceinline__ void store_row32(const P &p, int64_t orow, int c4, const float (&v)[32], float inv_l) {
    if (p.out_fp32) {
        float4 *dst = reinterpret_cast<float4 *>(static_cast<float *>(p.out) + orow * kHeadDim + c4 * 32);
#pragma unroll
        for (int i = 0; i < 8; ++i)
            dst[i] = make_float4(v[4 * i] * inv_l, v[4 * i + 1] * inv_l, v[4 * i + 2] * inv_l, v[4 * i + 3] * inv_l);
    } else {
        uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(p.out) + orow * kHeadDim + c4 * 32);
#pragma unroll
        for (int i = 0; i < 4; ++i)
            dst[i] = make_uint4(pack_bf16x2(v[8 * i] * inv_l, v[8 * i + 1] * inv_l),
                                pack_bf16x2(v[8 * i + 2] * inv_l, v[8 * i + 3] * inv_l),
                                pack_bf16x2(v[8 * i + 4] * inv_l, v[8 * i + 5] * inv_l),
                                pack_bf16x2(v[8 * i + 6] * inv_l, v[8 * i + 7] * inv_l));
    }
}

// The parts of a work item each role needs (read from the kernel parameters).
struct ItemView {
    const int32_t *table;  // the sequence's block-table row
    int ctx_len;
    int kvh;               // kv-head of the item's head slot
    int kt0, n_kt;         // KV tiles [kt0, kt0 + n_kt)
};

template <class P>
__device__ __forceinline__ ItemView item_view(const P &p, int w) {
    const PrefillWork wk = p.work[w];
    const PrefillSeq sq = p.seqs[wk.seq];
    ItemView v;
    v.table = p.block_tables + static_cast<int64_t>(sq.table_row) * p.table_stride;
    v.ctx_len = sq.ctx_len;
    v.kvh = wk.slot * p.heads_per_cta / p.group;
    v.kt0 = wk.kt0;
    v.n_kt = wk.kt1 - wk.kt0;
    return v;
}

// pages of KV tile j that hold at least one context key
__device__ __forceinline__ int pages_in(int ctx_len, int j) {
    return min(kPagesPerTile, (ctx_len - j * kKT + kPage - 1) / kPage);
}

}  // namespace

// The work of prefill CTA `cta` of the plan in p (all 512 threads).
template <class P>
__device__ __forceinline__ void prefill_cta(const CUtensorMap &tm_q, const CUtensorMap &tm_k,
                                            const CUtensorMap &tm_v, const P &p, int cta) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_s = smem_u32(smem_raw);
    const uint32_t sb = (raw_s + 1023u) & ~1023u;  // 1024-aligned for the 128-byte swizzle
    uint8_t *const sg = smem_raw + (sb - raw_s);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int hpc = p.heads_per_cta;
    // this CTA's items, in order
    const int w_beg = p.cta_begin[cta], w_end = p.cta_begin[cta + 1];

    auto bar = [&](int i) { return sb + kOffBar + 8u * static_cast<uint32_t>(i); };
    volatile int *abort_flag = reinterpret_cast<volatile int *>(sg + kOffAbort);

    if (warp == kMmaWarp) {
        tmem_alloc(sb + kOffTmem, kTmemCols);
        tmem_relinquish();
    }
    if (tid == 0) {
        for (int t = 0; t < 2; ++t) {
            mbar_init(bar(B_Q + t), 1);
            mbar_init(bar(B_QEMPTY + t), 1);
        }
        for (int s = 0; s < kNK; ++s) {
            mbar_init(bar(B_KFULL + s), 2);      // two producer threads per tile
            mbar_init(bar(B_KEMPTY + s), hpc);   // one release per tile's MMA thread
        }
        for (int s = 0; s < kNV; ++s) {
            mbar_init(bar(B_VFULL + s), 2);
            mbar_init(bar(B_VEMPTY + s), hpc);
        }
        for (int t = 0; t < 2; ++t) {
            mbar_init(bar(B_SFULL + t), 1);
            mbar_init(bar(B_PFULL + t), 4);
            mbar_init(bar(B_ODONE + t), 1);
            mbar_init(bar(B_TURN + t), 4);
        }
        mbar_init(bar(B_DRAIN), hpc);
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tm_q);
        prefetch_tmap(&tm_k);
        prefetch_tmap(&tm_v);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(sg + kOffTmem);
    // the set-up above overlaps the previous kernel of the stream; global
    // memory (KV pages, Q, block tables, outputs) only after it has completed
    grid_dep_wait();

    if (warp < 4) {
        // ------------------------------------------------------------ K/V producers
        // The rings run on across item boundaries: tile g of this CTA (over
        // all its items) goes to stage g % depth.
        asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsSmall));
        if (lane == 0 && w_beg < w_end) {
            const bool is_v = warp >= 2;
            const int pg_lo = (warp & 1) * (kPagesPerTile / 2);  // this thread's pages of each tile
            const int ns = is_v ? kNV : kNK;
            const CUtensorMap *tm = is_v ? &tm_v : &tm_k;
            const uint32_t ring = sb + (is_v ? kOffV : kOffK);
            const int full0 = is_v ? B_VFULL : B_KFULL, empty0 = is_v ? B_VEMPTY : B_KEMPTY;
            // page ids of the next tile are loaded while the current one is issued
            int ids[kPagesPerTile / 2];
            auto load_ids = [&](const ItemView &v, int jj) {
                const int j = v.kt0 + jj;
                const int np = pages_in(v.ctx_len, j);
#pragma unroll
                for (int i = 0; i < kPagesPerTile / 2; ++i)
                    ids[i] = (pg_lo + i < np) ? __ldg(v.table + j * kPagesPerTile + pg_lo + i) : 0;
            };
            int w = w_beg, jj = 0;
            ItemView cur = item_view(p, w);
            load_ids(cur, 0);
            for (int g = 0;; ++g) {
                const int j = cur.kt0 + jj;
                const int s = g % ns;
                const int np = max(0, min(kPagesPerTile / 2, pages_in(cur.ctx_len, j) - pg_lo));
                int rows[kPagesPerTile / 2];
#pragma unroll
                for (int i = 0; i < kPagesPerTile / 2; ++i) {
                    int blk = ids[i];
                    if (i < np && (blk < 0 || blk >= p.num_blocks)) {
                        report_error(p.err, PPAS_DEVERR_BAD_INDEX);
                        blk = 0;  // keep the barrier's byte count consistent
                    }
                    rows[i] = (blk * p.n_kv_heads + cur.kvh) * kPage;
                }
                // the next tile: this item's, else the next item's first
                int jn = jj + 1, wn = w;
                if (jn == cur.n_kt) {
                    jn = 0;
                    ++wn;
                }
                const bool more = wn < w_end;
                const ItemView nxt = (more && wn != w) ? item_view(p, wn) : cur;
                if (more) load_ids(nxt, jn);
                if (g >= ns && !mbar_wait(bar(empty0 + s), ((g / ns) & 1) ^ 1, p.err)) {
                    *abort_flag = 1;
                    break;
                }
                const uint32_t b = bar(full0 + s);
                mbar_expect_tx(b, static_cast<uint32_t>(np) * 2 * kBox);
                const uint32_t dst = ring + s * kTileBytes + pg_lo * kBox;
                for (int i = 0; i < np; ++i) {
                    tma_load_2d(dst + i * kBox, tm, 0, rows[i], b);
                    tma_load_2d(dst + kHalf + i * kBox, tm, 64, rows[i], b);
                }
                if (!more) break;
                w = wn;
                jj = jn;
                cur = nxt;
            }
        }
    } else if (warp < kSoftmaxWarp0) {
        asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsSmall));
        const int t = warp - kMmaWarp;
        if (t < hpc && lane == 0 && w_beg < w_end) {
            // -------------------------------------------------------- MMA issuer of Q tile t
            // descriptors are built once; advancing one operand by b bytes
            // adds b >> 4 to the start-address field (no carry: < 256 KB)
            const uint64_t dq = smem_desc_sw128(sb + kOffQ + t * kTileBytes, 16, 1024);
            const uint64_t dk0 = smem_desc_sw128(sb + kOffK, 16, 1024);
            const uint64_t dv0 = smem_desc_sw128(sb + kOffV, kHalf, 1024);
            const uint32_t d_s = tmem + t * 256, d_o = tmem + t * 256 + 128;
            bool ok = true;
            int g = 0;  // KV tiles of this CTA so far
            for (int w = w_beg, i = 0; ok && w < w_end; ++w, ++i) {
                const ItemView v = item_view(p, w);
                if (!mbar_wait(bar(B_Q + t), i & 1, p.err)) {
                    ok = false;
                    break;
                }
                for (int jj = 0; jj < v.n_kt; ++jj, ++g) {
                    const int j = v.kt0 + jj;
                    // ---- S_t = Q_t K(j)^T, once P V (g-1) has read P out of S's columns
                    const int sk = g % kNK;
                    if (!mbar_wait(bar(B_KFULL + sk), (g / kNK) & 1, p.err)) { ok = false; break; }
                    if (g >= 1 && !mbar_wait(bar(B_ODONE + t), (g - 1) & 1, p.err)) { ok = false; break; }
                    tc_fence_after();
                    const uint64_t dk = dk0 + ((sk * kTileBytes) >> 4);
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        const uint32_t o = (kk >> 2) * kHalf + (kk & 3) * 32;
                        umma_bf16(d_s, dq + (o >> 4), dk + (o >> 4), kIdescQK, kk > 0 ? 1u : 0u);
                    }
                    umma_commit(bar(B_SFULL + t));
                    umma_commit(bar(B_KEMPTY + sk));
                    // the item's last Q K^T frees Q_t for the next item
                    if (jj == v.n_kt - 1) umma_commit(bar(B_QEMPTY + t));
                    // ---- O_t += P_t V(j), P_t from TMEM; the item's first tile overwrites O_t
                    const int sv = g % kNV;
                    if (!mbar_wait(bar(B_VFULL + sv), (g / kNV) & 1, p.err)) { ok = false; break; }
                    if (!mbar_wait(bar(B_PFULL + t), g & 1, p.err)) { ok = false; break; }
                    tc_fence_after();
                    const uint64_t dv = dv0 + ((sv * kTileBytes) >> 4);
                    const int chunks = pages_in(v.ctx_len, j);
                    if (chunks == kPagesPerTile) {
#pragma unroll
                        for (int kk = 0; kk < kPagesPerTile; ++kk)
                            umma_bf16_ts(d_o, d_s + kk * 8, dv + ((kk * 2048) >> 4), kIdescPV,
                                         (jj > 0 || kk > 0) ? 1u : 0u);
                    } else {
                        for (int kk = 0; kk < chunks; ++kk)
                            umma_bf16_ts(d_o, d_s + kk * 8, dv + ((kk * 2048) >> 4), kIdescPV,
                                         (jj > 0 || kk > 0) ? 1u : 0u);
                    }
                    umma_commit(bar(B_ODONE + t));
                    umma_commit(bar(B_VEMPTY + sv));
                }
            }
            if (!ok) *abort_flag = 1;
            // every MMA issued so far completes before TMEM is released
            umma_commit(bar(B_DRAIN));
            mbar_wait(bar(B_DRAIN), 0, p.err);
        } else if (warp == kQWarp && lane == 0) {
            // -------------------------------------------------------- Q loader
            // Q tile t of item i is loaded once the last Q K^T of item i-1 on
            // that tile has completed.
            for (int w = w_beg, i = 0; w < w_end; ++w, ++i) {
                const PrefillWork wk = p.work[w];
                const int qrow = p.seqs[wk.seq].q_start + wk.qt * kTileQ;
                const int h0 = wk.slot * hpc;
                bool ok = true;
                for (int t = 0; t < hpc; ++t) {
                    if (i > 0 && !mbar_wait(bar(B_QEMPTY + t), (i - 1) & 1, p.err)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(bar(B_Q + t), kTileBytes);
                    tma_load_3d(sb + kOffQ + t * kTileBytes, &tm_q, 0, h0 + t, qrow, bar(B_Q + t));
                    tma_load_3d(sb + kOffQ + t * kTileBytes + kHalf, &tm_q, 64, h0 + t, qrow, bar(B_Q + t));
                }
                if (!ok) {
                    *abort_flag = 1;
                    break;
                }
            }
        }
    } else {
        // ------------------------------------------------------------ softmax warpgroups
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsLarge));
      if ((warp - kSoftmaxWarp0) / 4 < hpc) {
        const int t = (warp - kSoftmaxWarp0) / 4;
        const int wq = warp & 3;
        const int r = wq * 32 + lane;  // query row == TMEM lane
        const uint32_t t_lane = tmem + (static_cast<uint32_t>(wq * 32) << 16);
        const uint32_t t_s = t_lane + t * 256, t_o = t_lane + t * 256 + 128;
        const float sl2 = p.scale_log2;
        bool ok = true;
        int g = 0;  // KV tiles of this CTA so far

        for (int w = w_beg; w < w_end; ++w) {
            // what the KV loop needs (the epilogue reads the rest again)
            int pos, min_pos, kt0, n_kt, last_j, ctx_len;
            {
                const PrefillWork wk = p.work[w];
                const PrefillSeq sq = p.seqs[wk.seq];
                const int t0 = wk.qt * kTileQ;
                const int prefix = sq.ctx_len - sq.q_len;
                ctx_len = sq.ctx_len;
                pos = min(prefix + t0 + r, ctx_len - 1);  // last key this row may see
                min_pos = prefix + t0;
                last_j = (prefix + t0 + min(kTileQ, sq.q_len - t0) - 1) / kKT;  // last KV tile of the causal range
                kt0 = wk.kt0;
                n_kt = wk.kt1 - wk.kt0;
            }
            float m_used = -INFINITY, l_run = 0.f;

            for (int jj = 0; ok && jj < n_kt; ++jj, ++g) {
                const int j = kt0 + jj;  // absolute KV tile
                // S_t(g) ready; it was issued after P V (g-1) completed, so O_t is stable
                ok = __all_sync(0xffffffffu, !*abort_flag && mbar_wait(bar(B_SFULL + t), g & 1, p.err));
                // the two tiles' softmax phases alternate (tile 0 first), so one
                // tile's softmax overlaps the other tile's MMAs instead of both
                // competing for the exponential and FP32 pipes at once
                if (ok && hpc == 2 && (t == 1 || g > 0))
                    ok = __all_sync(0xffffffffu, mbar_wait(bar(B_TURN + t), (t == 0 ? g - 1 : g) & 1, p.err));
                if (!ok) break;
                tc_fence_after();
                float s[kKT];
                {
                    float h[64];
                    tmem_ld64_sync(t_s, h);
#pragma unroll
                    for (int i = 0; i < 64; ++i) s[i] = h[i];
                    tmem_ld64_sync(t_s + 64, h);
#pragma unroll
                    for (int i = 0; i < 64; ++i) s[64 + i] = h[i];
                }
                const int first_key = j * kKT;
                if (first_key + kKT - 1 > min_pos) {
#pragma unroll
                    for (int i = 0; i < kKT; ++i)
                        if (first_key + i > pos) s[i] = -INFINITY;
                }
                // four independent chains over the 128 scores, two new ones per max3
                float mx0 = fmaxf(s[0], s[4]), mx1 = fmaxf(s[1], s[5]);
                float mx2 = fmaxf(s[2], s[6]), mx3 = fmaxf(s[3], s[7]);
#pragma unroll
                for (int i = 8; i < kKT; i += 8) {
                    mx0 = max3(mx0, s[i], s[i + 4]);
                    mx1 = max3(mx1, s[i + 1], s[i + 5]);
                    mx2 = max3(mx2, s[i + 2], s[i + 6]);
                    mx3 = max3(mx3, s[i + 3], s[i + 7]);
                }
                const float m_cand = max3(fmaxf(mx0, mx1), mx2, mx3) * sl2;
                const bool need = m_cand > m_used + kRescaleThreshold;
                float alpha = 1.f;
                if (need) {
                    alpha = ex2(m_used - m_cand);
                    m_used = m_cand;
                }
                // a row whose keys in this range are all masked keeps m = -inf and p = 0
                const float neg_m = m_used == -INFINITY ? 0.f : -m_used;
                const float2 sl2x2 = make_float2(sl2, sl2), negx2 = make_float2(neg_m, neg_m);
                float2 ra = make_float2(0.f, 0.f), rb = make_float2(0.f, 0.f);
#pragma unroll
                for (int i = 0; i < kKT; i += 4) {
                    const float2 xa = fma2(make_float2(s[i], s[i + 1]), sl2x2, negx2);
                    const float2 xb = fma2(make_float2(s[i + 2], s[i + 3]), sl2x2, negx2);
                    s[i] = ex2(xa.x);
                    s[i + 1] = ex2(xa.y);
                    s[i + 2] = ex2(xb.x);
                    s[i + 3] = ex2(xb.y);
                    ra = add2(ra, make_float2(s[i], s[i + 1]));
                    rb = add2(rb, make_float2(s[i + 2], s[i + 3]));
                }
                l_run = l_run * alpha + ((ra.x + ra.y) + (rb.x + rb.y));
                if (j == last_j) {
                    // rows of the last page past the context may hold anything:
                    // zero them in V so that P = 0 times V stays 0.  Each tile's
                    // warpgroup does it before releasing its own P, so both P V
                    // products are ordered after it (the second writes the same
                    // zeros again)
                    const int keys_here = min(kKT, ctx_len - first_key);
                    if (keys_here & (kPage - 1)) {
                        const int s_idx = g % kNV;
                        ok = __all_sync(0xffffffffu, mbar_wait(bar(B_VFULL + s_idx), (g / kNV) & 1, p.err));
                        if (!ok) break;
                        const int pg = keys_here / kPage, from = keys_here & (kPage - 1);
                        const int n = (kPage - from) * 8;  // 16-byte chunks per half
                        uint8_t *vb = sg + kOffV + s_idx * kTileBytes + pg * kBox + from * 128;
                        for (int c = r; c < 2 * n; c += 128)
                            *reinterpret_cast<uint4 *>(vb + (c / n) * kHalf + (c % n) * 16) = make_uint4(0, 0, 0, 0);
                        fence_proxy_async_smem();
                    }
                }
                // P (bf16 pairs, lower key in the low half) over the first 64 columns of S
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    uint32_t pk[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) pk[i] = pack_bf16x2(s[64 * h + 2 * i], s[64 * h + 2 * i + 1]);
                    tmem_st32(t_s + 32 * h, pk);
                }
                if (jj >= 1 && __any_sync(0xffffffffu, need)) {
#pragma unroll
                    for (int c4 = 0; c4 < 4; ++c4) {
                        float v[32];
                        tmem_ld32_sync(t_o + c4 * 32, v);
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] *= alpha;
                        tmem_st32_f(t_o + c4 * 32, v);
                    }
                }
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(bar(B_PFULL + t));
                    if (hpc == 2) mbar_arrive(bar(B_TURN + (t ^ 1)));  // the other tile's turn
                }
            }

            // ---- epilogue of the item: O_t after its last P V
            if (ok) ok = __all_sync(0xffffffffu, mbar_wait(bar(B_ODONE + t), (g - 1) & 1, p.err));
            const PrefillWork wk = p.work[w];
            const PrefillSeq sq = p.seqs[wk.seq];
            const int t0 = wk.qt * kTileQ;
            const int rows_valid = min(kTileQ, sq.q_len - t0);
            const int64_t orow = static_cast<int64_t>(sq.q_start + t0 + r) * p.n_q_heads + wk.slot * hpc + t;
            if (wk.part == kNoPart) {
                if (ok) {
                    tc_fence_after();
                    const float inv_l = 1.f / l_run;
#pragma unroll
                    for (int c4 = 0; c4 < 4; ++c4) {
                        float v[32];
                        tmem_ld32_sync(t_o + c4 * 32, v);
                        if (r < rows_valid) store_row32(p, orow, c4, v, inv_l);
                    }
                }
            } else if (ok) {
                // a piece of a split unit: this range's (m, l, O) for the row;
                // the merge kernel combines the unit's pieces after this
                // launch.  Partial O of one (piece, head) is stored as 4 column
                // chunks of [128 rows][32 floats], so a warp writes 4 KB
                // contiguous per chunk.
                tc_fence_after();
                const int64_t b = static_cast<int64_t>(wk.part) * hpc + t;
#pragma unroll
                for (int c4 = 0; c4 < 4; ++c4) {
                    float v[32];
                    tmem_ld32_sync(t_o + c4 * 32, v);
                    float4 *dst = reinterpret_cast<float4 *>(p.part_o + ((b * 4 + c4) * kTileQ + r) * 32);
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        __stcg(dst + i, make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]));
                }
                // two scalar stores: the paired float2 store costs the softmax loop
                // register spills at its 200-register budget
                __stcg(p.part_ml + (b * kTileQ + r) * 2, m_used);
                __stcg(p.part_ml + (b * kTileQ + r) * 2 + 1, l_run);
            }
        }
        if (!ok) *abort_flag = 1;
      }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

__global__ void __launch_bounds__(kThreads, 1)
    prefill_attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                        const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ PrefillParams p) {
    prefill_cta(tm_q, tm_k, tm_v, p, blockIdx.x);
}

// A whole mixed step in one launch: CTAs [0, p.pf.n_ctas) run the prefill
// items, the CTAs after them the decode splits (one (row, kv-head, split)
// each, on warps 0-7; warps 8-15 hand their registers to them and leave).
// The block scheduler starts CTAs in index order, so the first wave holds
// every prefill CTA and fills the SMs left to the decode rows.
__global__ void __launch_bounds__(kThreads, 1)
    mixed_attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                      const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ MixedParams p) {
    if (static_cast<int>(blockIdx.x) < p.pf.n_ctas) {
        prefill_cta(tm_q, tm_k, tm_v, p.pf, blockIdx.x);
        return;
    }
    if ((threadIdx.x >> 5) >= kDecodeWarps) {
        asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsSmall));
        return;
    }
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsLarge));
    decode_cta<true>(tm_k, tm_v, p.dc, static_cast<int>(blockIdx.x) - p.pf.n_ctas);
}
static_assert(kDecodeThreads == 8 * 32 && kDecodeSmemBytes <= kSmemBytes,
              "decode CTAs of a mixed launch: warps 0-7 of the CTA, within its shared memory");

// Combines the pieces of a split unit:
//   o = sum_i 2^(m_i - M) o_i / sum_i 2^(m_i - M) l_i,  M = max_i m_i
// (m in log2 units), taking the pieces four at a time with the running
// maximum (exact up to rounding).  One thread per (query row, 4 columns):
// CTA (unit, head t, chunk c4, quarter) covers 32 rows x 32 columns, so a
// warp reads 512 contiguous bytes of a partial chunk.
__global__ void __launch_bounds__(256) prefill_merge_kernel(const __grid_constant__ MergeParams p) {
    grid_dep_wait();  // the partials come from the prefill launch before this one
    const int hpc = p.heads_per_cta;
    const int lin = (blockIdx.x & 3) * 256 + threadIdx.x;  // 0..1023 within (unit, head, chunk)
    const int r = lin >> 3, j4 = lin & 7;
    int rest = blockIdx.x >> 2;
    const int c4 = rest & 3;
    rest >>= 2;
    const int t = rest % hpc;
    const MergeUnit mu = p.units[rest / hpc];
    const int ns = mu.n_splits;
    auto pblk = [&](int i) { return (static_cast<int64_t>(mu.part) + i) * hpc + t; };
    float M = -INFINITY, L = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int i0 = 0; i0 < ns; i0 += 4) {
        float2 ml[4];
        float4 o[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            if (i0 + k < ns) {
                const int64_t b = pblk(i0 + k);
                ml[k] = __ldcg(reinterpret_cast<const float2 *>(p.part_ml + (b * kTileQ + r) * 2));
                o[k] = __ldcg(reinterpret_cast<const float4 *>(p.part_o + ((b * 4 + c4) * kTileQ + r) * 32) + j4);
            } else {
                ml[k] = make_float2(-INFINITY, 0.f);
                o[k] = make_float4(0.f, 0.f, 0.f, 0.f);
            }
        }
        const float mn = fmaxf(fmaxf(M, fmaxf(ml[0].x, ml[1].x)), fmaxf(ml[2].x, ml[3].x));
        if (mn == -INFINITY) continue;  // every key of these pieces is masked for this row
        const float sc = M == -INFINITY ? 0.f : ex2(M - mn);
        L *= sc;
        acc = make_float4(acc.x * sc, acc.y * sc, acc.z * sc, acc.w * sc);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float f = ml[k].x == -INFINITY ? 0.f : ex2(ml[k].x - mn);
            L += f * ml[k].y;
            acc = make_float4(acc.x + f * o[k].x, acc.y + f * o[k].y, acc.z + f * o[k].z, acc.w + f * o[k].w);
        }
        M = mn;
    }
    if (r >= mu.rows_valid) return;
    const float inv_l = 1.f / L;
    const int64_t orow = static_cast<int64_t>(mu.out_row0 + r) * p.n_q_heads + mu.head0 + t;
    const int64_t col = orow * kHeadDim + c4 * 32 + j4 * 4;
    if (p.out_fp32) {
        *reinterpret_cast<float4 *>(static_cast<float *>(p.out) + col) =
            make_float4(acc.x * inv_l, acc.y * inv_l, acc.z * inv_l, acc.w * inv_l);
    } else {
        *reinterpret_cast<uint2 *>(static_cast<__nv_bfloat16 *>(p.out) + col) =
            make_uint2(pack_bf16x2(acc.x * inv_l, acc.y * inv_l), pack_bf16x2(acc.z * inv_l, acc.w * inv_l));
    }
}

cudaError_t launch_prefill_merge(const MergeParams &p, cudaStream_t st) {
    if (p.n_units <= 0) return cudaSuccess;
    PdlLaunch l(dim3(p.n_units * p.heads_per_cta * 16), dim3(256), 0, st);
    return cudaLaunchKernelEx(&l.cfg, prefill_merge_kernel, p);
}

static std::atomic<uint64_t> g_prefill_smem_set{0};
static std::atomic<uint64_t> g_mixed_smem_set{0};

cudaError_t prepare_prefill() {
    return ensure_smem_limit(prefill_attn_kernel, static_cast<int>(kSmemBytes), g_prefill_smem_set);
}

cudaError_t prepare_mixed() {
    return ensure_smem_limit(mixed_attn_kernel, static_cast<int>(kSmemBytes), g_mixed_smem_set);
}

cudaError_t launch_prefill(const CUtensorMap &tm_q, const CUtensorMap &tm_k, const CUtensorMap &tm_v,
                           const PrefillParams &p, cudaStream_t st) {
    const cudaError_t e = prepare_prefill();
    if (e != cudaSuccess) return e;
    if (p.n_ctas <= 0) return cudaSuccess;
    PdlLaunch l(dim3(p.n_ctas), dim3(kThreads), kSmemBytes, st);
    return cudaLaunchKernelEx(&l.cfg, prefill_attn_kernel, tm_q, tm_k, tm_v, p);
}

cudaError_t launch_mixed(const CUtensorMap &tm_q, const CUtensorMap &tm_k, const CUtensorMap &tm_v,
                         const MixedParams &p, cudaStream_t st) {
    const cudaError_t e = prepare_mixed();
    if (e != cudaSuccess) return e;
    const int grid = p.pf.n_ctas + p.dc.n_ctas;
    if (grid <= 0) return cudaSuccess;
    PdlLaunch l(dim3(grid), dim3(kThreads), kSmemBytes, st);
    return cudaLaunchKernelEx(&l.cfg, mixed_attn_kernel, tm_q, tm_k, tm_v, p);
}

}  // namespace ppas
