// Prefill-chunk attention on the 5th-generation tensor cores (tcgen05).
//
// One CTA computes O for one 128-token query tile of one q-head:
//   S = Q K^T            tcgen05.mma, Q and K tiles in shared memory (TMA),
//                        S accumulated in TMEM (128 lanes x 128 fp32 columns)
//   online softmax       each thread owns one query row (its TMEM lane),
//                        fp32, exp2 domain, causal mask by absolute position
//   O += P V             P written to shared memory as bf16, V via TMA,
//                        O accumulated in TMEM
// K/V tiles are 128 keys = eight 16-token pages, fetched page by page through
// the block table with 2D TMA boxes of 16 rows x 64 columns (128-byte swizzle).
#include <math.h>

#include "ppas_device.cuh"
#include "ppas_internal.h"

namespace ppas {
namespace {

constexpr uint32_t kHalf = 16384;                       // 128 rows x 128 B (64 bf16 columns)
constexpr uint32_t kTileBytes = 2 * kHalf;              // 128 rows x 256 B
constexpr uint32_t kBoxBytes = kPage * 128;             // 16 rows x 128 B = one TMA box
constexpr int kStages = 2;
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kOffQ + kTileBytes;
constexpr uint32_t kOffV = kOffK + kStages * kTileBytes;
constexpr uint32_t kOffP = kOffV + kStages * kTileBytes;
constexpr uint32_t kOffBar = kOffP + kTileBytes;
// barriers: q, kv[2], s, o (8 B each), then TMEM base address and abort word
constexpr uint32_t kBarQ = 0, kBarKV = 8, kBarS = 24, kBarO = 32, kTmemSlot = 64;
constexpr uint32_t kSmemBytes = kOffBar + 128 + 1024;   // + alignment slack
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kColS = 0, kColO = 128;

constexpr uint32_t kIdescQK = idesc_bf16_f32(128, 128, false, false);  // B = K rows, K-major
constexpr uint32_t kIdescPV = idesc_bf16_f32(128, 128, false, true);   // B = V rows, MN-major

// 32 TMEM columns of this warp's lanes, waiting for completion before the
// registers are used.
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

__device__ __forceinline__ void tmem_st32_f(uint32_t taddr, const float (&v)[32]) {
    uint32_t r[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(v[i]);
    tmem_st32(taddr, r);
}

}  // namespace

__global__ void __launch_bounds__(128, 1)
    prefill_attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                        const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ PrefillParams p) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_s = smem_u32(smem_raw);
    const uint32_t sb = (raw_s + 1023u) & ~1023u;  // 1024-aligned for the 128-byte swizzle
    uint8_t *const sg = smem_raw + (sb - raw_s);   // generic pointer to the same place

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int h = blockIdx.x % p.n_q_heads;
    const uint32_t tile = p.tiles[blockIdx.x / p.n_q_heads];
    const PrefillSeq sq = p.seqs[tile >> 16];
    const int t0 = static_cast<int>(tile & 0xFFFFu) * kTileQ;
    const int rows_valid = min(kTileQ, sq.q_len - t0);
    const int prefix = sq.ctx_len - sq.q_len;
    const int kvh = h / p.group;
    const int last_pos = prefix + t0 + rows_valid - 1;
    const int n_kt = last_pos / kTileK + 1;
    const int32_t *table = p.block_tables + static_cast<int64_t>(sq.table_row) * p.table_stride;

    const uint32_t bar_q = sb + kOffBar + kBarQ, bar_s = sb + kOffBar + kBarS, bar_o = sb + kOffBar + kBarO;
    auto bar_kv = [&](int st) { return sb + kOffBar + kBarKV + 8u * st; };
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(sg + kOffBar + kTmemSlot);

    if (warp == 0) {
        tmem_alloc(sb + kOffBar + kTmemSlot, kTmemCols);
        tmem_relinquish();
    }
    if (tid == 32) {
        mbar_init(bar_q, 1);
        mbar_init(bar_kv(0), 1);
        mbar_init(bar_kv(1), 1);
        mbar_init(bar_s, 1);
        mbar_init(bar_o, 1);
        fence_mbar_init();
        prefetch_tmap(&tm_q);
        prefetch_tmap(&tm_k);
        prefetch_tmap(&tm_v);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    // ---- producer (thread 0): one KV tile = up to 8 pages of K and V
    auto issue_kv = [&](int j) {
        const int st = j & 1;
        const uint32_t bar = bar_kv(st);
        const int first_key = j * kTileK;
        const int n_pages = min(8, (sq.ctx_len - first_key + kPage - 1) / kPage);
        mbar_expect_tx(bar, static_cast<uint32_t>(n_pages) * 4u * kBoxBytes);
        const uint32_t dk = sb + kOffK + st * kTileBytes, dv = sb + kOffV + st * kTileBytes;
        for (int pg = 0; pg < n_pages; ++pg) {
            int blk = __ldg(table + j * 8 + pg);
            if (blk < 0 || blk >= p.num_blocks) {
                report_error(p.err, PPAS_DEVERR_BAD_INDEX);
                blk = 0;  // keep the byte count of the barrier consistent
            }
            const int row = (blk * p.n_kv_heads + kvh) * kPage;
            tma_load_2d(dk + pg * kBoxBytes, &tm_k, 0, row, bar);
            tma_load_2d(dk + kHalf + pg * kBoxBytes, &tm_k, 64, row, bar);
            tma_load_2d(dv + pg * kBoxBytes, &tm_v, 0, row, bar);
            tma_load_2d(dv + kHalf + pg * kBoxBytes, &tm_v, 64, row, bar);
        }
    };

    if (tid == 0) {
        mbar_expect_tx(bar_q, kTileBytes);
        const int qrow = sq.q_start + t0;
        tma_load_3d(sb + kOffQ, &tm_q, 0, h, qrow, bar_q);
        tma_load_3d(sb + kOffQ + kHalf, &tm_q, 64, h, qrow, bar_q);
        issue_kv(0);
        if (n_kt > 1) issue_kv(1);
    }

    const int r = warp * 32 + lane;                       // query row of the tile == TMEM lane
    const int pos = min(prefix + t0 + r, sq.ctx_len - 1); // last key this row may see
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    int j = 0;

    for (; j < n_kt; ++j) {
        const int st = j & 1;
        bool w_ok = mbar_wait(bar_kv(st), (j >> 1) & 1, p.err);
        if (j == 0) w_ok = w_ok && mbar_wait(bar_q, 0, p.err);
        // rows of the last page past the context may hold anything; zero the
        // V rows there so that P = 0 times V stays 0
        const int first_key = j * kTileK;
        const int keys_here = min(kTileK, sq.ctx_len - first_key);
        if (w_ok && (keys_here & (kPage - 1))) {
            const int pg = keys_here / kPage;
            const int from = keys_here & (kPage - 1);
            const int n_chunks = (kPage - from) * 8;  // 16-byte chunks per half
            uint8_t *vbase = sg + kOffV + st * kTileBytes + pg * kBoxBytes + from * 128;
            for (int c = tid; c < 2 * n_chunks; c += blockDim.x) {
                const int half = c / n_chunks, cc = c % n_chunks;
                *reinterpret_cast<uint4 *>(vbase + half * kHalf + cc * 16) = make_uint4(0, 0, 0, 0);
            }
            fence_proxy_async_smem();
        }
        tc_fence_before();
        if (__syncthreads_or(!w_ok)) { ok = false; break; }

        if (tid == 0) {
            tc_fence_after();
            const uint32_t q0 = sb + kOffQ, k0 = sb + kOffK + st * kTileBytes;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                const uint32_t off = (kk >> 2) * kHalf + (kk & 3) * 32;
                umma_bf16(tmem + kColS, smem_desc_sw128(q0 + off, 16, 1024), smem_desc_sw128(k0 + off, 16, 1024),
                          kIdescQK, kk > 0);
            }
            umma_commit(bar_s);
        }
        w_ok = __all_sync(0xffffffffu, mbar_wait(bar_s, j & 1, p.err));
        tc_fence_after();

        if (w_ok) {
            // ---- softmax of this row over the 128 keys of tile j
            float s[128];
#pragma unroll
            for (int c4 = 0; c4 < 4; ++c4) {
                float v[32];
                tmem_ld32_sync(t_lane + kColS + c4 * 32, v);
#pragma unroll
                for (int i = 0; i < 32; ++i) s[c4 * 32 + i] = v[i];
            }
            float mx = -INFINITY;
#pragma unroll
            for (int i = 0; i < 128; ++i) {
                s[i] = (first_key + i <= pos) ? s[i] * p.scale_log2 : -INFINITY;
                mx = fmaxf(mx, s[i]);
            }
            const float m_new = fmaxf(m_run, mx);
            const float alpha = ex2(m_run - m_new);
            m_run = m_new;
            float rs = 0.f;
#pragma unroll
            for (int i = 0; i < 128; ++i) {
                s[i] = ex2(s[i] - m_new);
                rs += s[i];
            }
            l_run = l_run * alpha + rs;
            if (j > 0) {
#pragma unroll
                for (int c4 = 0; c4 < 4; ++c4) {
                    float v[32];
                    tmem_ld32_sync(t_lane + kColO + c4 * 32, v);
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] *= alpha;
                    tmem_st32_f(t_lane + kColO + c4 * 32, v);
                }
                tmem_wait_st();
            }
            // P (bf16) into the K-major, 128-byte-swizzled A-operand layout
            uint8_t *prow = sg + kOffP + (r >> 3) * 1024 + (r & 7) * 128;
#pragma unroll
            for (int c = 0; c < 16; ++c) {
                uint4 v;
                v.x = pack_bf16x2(s[8 * c + 0], s[8 * c + 1]);
                v.y = pack_bf16x2(s[8 * c + 2], s[8 * c + 3]);
                v.z = pack_bf16x2(s[8 * c + 4], s[8 * c + 5]);
                v.w = pack_bf16x2(s[8 * c + 6], s[8 * c + 7]);
                *reinterpret_cast<uint4 *>(prow + (c >> 3) * kHalf + (((c & 7) ^ (r & 7)) << 4)) = v;
            }
            fence_proxy_async_smem();
        }
        tc_fence_before();
        if (__syncthreads_or(!w_ok)) { ok = false; break; }

        if (tid == 0) {
            tc_fence_after();
            const uint32_t p0 = sb + kOffP, v0 = sb + kOffV + st * kTileBytes;
            const int n_chunks = (keys_here + kPage - 1) / kPage;  // 16-key chunks with a valid key
            for (int kk = 0; kk < n_chunks; ++kk) {
                const uint64_t da = smem_desc_sw128(p0 + (kk >> 2) * kHalf + (kk & 3) * 32, 16, 1024);
                const uint64_t db = smem_desc_sw128(v0 + kk * 2048, kHalf, 1024);
                umma_bf16(tmem + kColO, da, db, kIdescPV, (j > 0 || kk > 0) ? 1u : 0u);
            }
            umma_commit(bar_o);
        }
        w_ok = mbar_wait(bar_o, j & 1, p.err);
        tc_fence_after();
        if (__syncthreads_or(!w_ok)) { ok = false; break; }
        if (tid == 0 && j + 2 < n_kt) issue_kv(j + 2);
    }

    if (ok) {
        // ---- epilogue: O / l for valid rows
        const float inv_l = 1.f / l_run;
        const int64_t orow = static_cast<int64_t>(sq.q_start + t0 + r) * p.n_q_heads + h;
#pragma unroll
        for (int c4 = 0; c4 < 4; ++c4) {
            float v[32];
            tmem_ld32_sync(t_lane + kColO + c4 * 32, v);
            if (r < rows_valid) {
                if (p.out_fp32) {
                    float4 *dst = reinterpret_cast<float4 *>(static_cast<float *>(p.out) + orow * kHeadDim + c4 * 32);
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        dst[i] = make_float4(v[4 * i] * inv_l, v[4 * i + 1] * inv_l, v[4 * i + 2] * inv_l,
                                             v[4 * i + 3] * inv_l);
                } else {
                    uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(p.out) + orow * kHeadDim +
                                                           c4 * 32);
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        dst[i] = make_uint4(pack_bf16x2(v[8 * i] * inv_l, v[8 * i + 1] * inv_l),
                                            pack_bf16x2(v[8 * i + 2] * inv_l, v[8 * i + 3] * inv_l),
                                            pack_bf16x2(v[8 * i + 4] * inv_l, v[8 * i + 5] * inv_l),
                                            pack_bf16x2(v[8 * i + 6] * inv_l, v[8 * i + 7] * inv_l));
                }
            }
        }
    } else if (tid == 0) {
        // drain: copies of tiles j+1, j+2 (issued, never consumed) and the MMAs in flight
        for (int jj = j; jj < min(j + 2, n_kt); ++jj) mbar_wait(bar_kv(jj & 1), (jj >> 1) & 1, nullptr);
        mbar_wait(bar_s, j & 1, nullptr);
        mbar_wait(bar_o, j & 1, nullptr);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

cudaError_t launch_prefill(const CUtensorMap &tm_q, const CUtensorMap &tm_k, const CUtensorMap &tm_v,
                           const PrefillParams &p, cudaStream_t st) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(prefill_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(kSmemBytes));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    if (p.n_tiles <= 0) return cudaSuccess;
    prefill_attn_kernel<<<p.n_tiles * p.n_q_heads, 128, kSmemBytes, st>>>(tm_q, tm_k, tm_v, p);
    return cudaGetLastError();
}

}  // namespace ppas
