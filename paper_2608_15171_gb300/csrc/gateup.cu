// Gate-up projection of the decoder MLP with the gated activation fused in:
//   Y[t, i] = silu(X[t] . W_gate[i]) * (X[t] . W_up[i])
// (the GEMM profiled beside attention in Section 6.1), on the tcgen05 tensor
// cores.
//
// The weights are packed once (gateup_pack_kernel) so that every 256-row
// block holds 128 gate rows followed by the 128 up rows of the same
// features.  One output tile is 128 tokens x 128 features: a single
// M128 x N256 accumulator whose left half is the gate product and right half
// the up product, so the epilogue combines them without leaving the SM and
// the [T, 2I] intermediate never reaches HBM.
//
// Persistent kernel, one CTA per SM, 192 threads:
//   warp 0      TMA producer: X tile (128 x 64) and W tile (256 x 64) per
//               64-wide K block, 128-byte swizzle, 4-stage ring
//   warp 1      allocates TMEM, issues the MMAs (4 x K16 per K block) into one
//               of two 256-column accumulators
//   warps 2-5   epilogue: each thread owns one token row (its TMEM lane),
//               reads 32 gate and 32 up columns at a time, writes bf16
// Tiles are visited in groups of 32 M blocks with the M block fastest, so
// the CTAs running at one time share a few weight tiles and keep a few MB of
// X tiles hot in L2.
#include <algorithm>

#include "ppas_device.cuh"
#include "ppas_internal.h"

namespace ppas {
namespace {

constexpr int kGM = 128;   // tokens per tile
constexpr int kGN = 256;   // accumulator columns: 128 gate + 128 up
constexpr int kGK = 64;    // K per stage (128 bytes of bf16: one swizzle row)
constexpr int kGStages = 4;
constexpr int kGroupM = 32;  // M blocks per raster group
constexpr uint32_t kABytes = kGM * kGK * 2;  // 16 KB
constexpr uint32_t kBBytes = kGN * kGK * 2;  // 32 KB
constexpr uint32_t kStage = kABytes + kBBytes;
constexpr uint32_t kOffBarG = kGStages * kStage;
enum : int {
    G_FULL = 0,
    G_EMPTY = G_FULL + kGStages,
    G_ACCFULL = G_EMPTY + kGStages,  // [2]
    G_ACCEMPTY = G_ACCFULL + 2,      // [2]
    G_DRAIN = G_ACCEMPTY + 2,
    G_COUNT = G_DRAIN + 1
};
constexpr uint32_t kOffTmemG = kOffBarG + G_COUNT * 8;
constexpr uint32_t kOffAbortG = kOffTmemG + 4;
constexpr uint32_t kSmemG = kOffBarG + 256 + 1024;  // + alignment slack
static_assert(kOffAbortG + 4 <= kOffBarG + 256, "barrier area");
static_assert(kSmemG <= 232448, "shared memory per CTA");
constexpr int kGThreads = 192;
constexpr uint32_t kIdescG = idesc_bf16_f32(kGM, kGN, false, false);  // A, B both K-major

// tile index -> (m block, n block), M fastest within groups of kGroupM
__device__ __forceinline__ void tile_mn(int t, int m_blocks, int n_blocks, int &mb, int &nb) {
    const int per_group = kGroupM * n_blocks;
    const int grp = t / per_group, rem = t - grp * per_group;
    const int gm = min(kGroupM, m_blocks - grp * kGroupM);
    nb = rem / gm;
    mb = grp * kGroupM + rem % gm;
}

__device__ __forceinline__ void tmem_ld32_wait(uint32_t taddr, float (&v)[32]) {
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

}  // namespace

__global__ void __launch_bounds__(kGThreads, 1)
    gateup_swiglu_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
                         const __grid_constant__ GateUpParams p) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_s = smem_u32(smem_raw);
    const uint32_t sb = (raw_s + 1023u) & ~1023u;
    uint8_t *const sg = smem_raw + (sb - raw_s);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto bar = [&](int i) { return sb + kOffBarG + 8u * static_cast<uint32_t>(i); };
    volatile int *abort_flag = reinterpret_cast<volatile int *>(sg + kOffAbortG);

    const int m_blocks = (p.n_tokens + kGM - 1) / kGM;
    const int n_blocks = p.inter / (kGN / 2);
    const int n_tiles = m_blocks * n_blocks;
    const int k_blocks = p.hidden / kGK;

    if (warp == 1) {
        tmem_alloc(sb + kOffTmemG, 512);
        tmem_relinquish();
    }
    if (tid == 0) {
        for (int s = 0; s < kGStages; ++s) {
            mbar_init(bar(G_FULL + s), 1);
            mbar_init(bar(G_EMPTY + s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(bar(G_ACCFULL + b), 1);
            mbar_init(bar(G_ACCEMPTY + b), 4);  // one arrive per epilogue warp
        }
        mbar_init(bar(G_DRAIN), 1);
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tm_x);
        prefetch_tmap(&tm_w);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(sg + kOffTmemG);

    if (warp == 0) {
        // ---------------------------------------------------------------- TMA producer
        if (lane == 0) {
            int q = 0;  // K blocks issued by this CTA
            for (int t = blockIdx.x; t < n_tiles; t += gridDim.x) {
                int mb, nb;
                tile_mn(t, m_blocks, n_blocks, mb, nb);
                bool ok = true;
                for (int kb = 0; kb < k_blocks; ++kb, ++q) {
                    const int s = q % kGStages;
                    if (q >= kGStages && !mbar_wait(bar(G_EMPTY + s), ((q / kGStages) & 1) ^ 1, p.err)) {
                        ok = false;
                        break;
                    }
                    const uint32_t dst = sb + s * kStage;
                    mbar_expect_tx(bar(G_FULL + s), kStage);
                    tma_load_2d(dst, &tm_x, kb * kGK, mb * kGM, bar(G_FULL + s));
                    tma_load_2d(dst + kABytes, &tm_w, kb * kGK, nb * kGN, bar(G_FULL + s));
                }
                if (!ok || *abort_flag) {
                    *abort_flag = 1;
                    break;
                }
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint64_t da0 = smem_desc_sw128(sb, 16, 1024);
            const uint64_t db0 = smem_desc_sw128(sb + kABytes, 16, 1024);
            int q = 0, it = 0;
            bool ok = true;
            for (int t = blockIdx.x; ok && t < n_tiles; t += gridDim.x, ++it) {
                const int buf = it & 1;
                const uint32_t d = tmem + buf * kGN;
                // the epilogue has drained this accumulator (two tiles ago)
                if (it >= 2 && !mbar_wait(bar(G_ACCEMPTY + buf), ((it >> 1) & 1) ^ 1, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int kb = 0; kb < k_blocks; ++kb, ++q) {
                    const int s = q % kGStages;
                    if (!mbar_wait(bar(G_FULL + s), (q / kGStages) & 1, p.err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t da = da0 + ((s * kStage) >> 4), db = db0 + ((s * kStage) >> 4);
#pragma unroll
                    for (int kk = 0; kk < kGK / 16; ++kk)
                        umma_bf16(d, da + (kk * 2), db + (kk * 2), kIdescG, (kb > 0 || kk > 0) ? 1u : 0u);
                    umma_commit(bar(G_EMPTY + s));
                }
                if (ok) umma_commit(bar(G_ACCFULL + buf));
            }
            if (!ok) *abort_flag = 1;
            umma_commit(bar(G_DRAIN));
            mbar_wait(bar(G_DRAIN), 0, p.err);
        }
    } else {
        // ---------------------------------------------------------------- epilogue
        const int wq = warp & 3;  // TMEM lane quarter of this warp
        const int r = wq * 32 + lane;
        const uint32_t t_lane = tmem + (static_cast<uint32_t>(wq * 32) << 16);
        int it = 0;
        for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++it) {
            const int buf = it & 1;
            const bool ok = __all_sync(0xffffffffu, !*abort_flag &&
                                                        mbar_wait(bar(G_ACCFULL + buf), (it >> 1) & 1, p.err));
            if (!ok) {
                *abort_flag = 1;
                break;
            }
            tc_fence_after();
            int mb, nb;
            tile_mn(t, m_blocks, n_blocks, mb, nb);
            const int row = mb * kGM + r;
            __nv_bfloat16 *out = p.y + static_cast<int64_t>(row) * p.inter + nb * (kGN / 2);
#pragma unroll 1
            for (int c = 0; c < 4; ++c) {
                float gv[32], uv[32];
                tmem_ld32_wait(t_lane + buf * kGN + c * 32, gv);
                tmem_ld32_wait(t_lane + buf * kGN + 128 + c * 32, uv);
                if (row < p.n_tokens) {
                    uint4 *dst = reinterpret_cast<uint4 *>(out + c * 32);
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        uint32_t w4[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const int e = 8 * i + 2 * k;
                            const float y0 = __fdividef(gv[e], 1.f + __expf(-gv[e])) * uv[e];
                            const float y1 = __fdividef(gv[e + 1], 1.f + __expf(-gv[e + 1])) * uv[e + 1];
                            w4[k] = pack_bf16x2(y0, y1);
                        }
                        dst[i] = make_uint4(w4[0], w4[1], w4[2], w4[3]);
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(G_ACCEMPTY + buf));
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// W [2I, H] (gate rows, then up rows) -> packed: block j of 256 rows holds
// gate rows 128j .. 128j+127 then up rows I+128j .. I+128j+127.
__global__ void gateup_pack_kernel(const uint4 *__restrict__ w, uint4 *__restrict__ wp, int hidden, int inter) {
    const int vec_per_row = hidden / 8;
    const int64_t total = static_cast<int64_t>(2 * inter) * vec_per_row;
    for (int64_t v = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; v < total;
         v += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t prow = v / vec_per_row;
        const int col = static_cast<int>(v - prow * vec_per_row);
        const int64_t blk = prow / 256, within = prow % 256;
        const int64_t src_row = within < 128 ? blk * 128 + within : inter + blk * 128 + (within - 128);
        wp[v] = w[src_row * vec_per_row + col];
    }
}

cudaError_t launch_gateup(const CUtensorMap &tm_x, const CUtensorMap &tm_w, const GateUpParams &p, int grid,
                          cudaStream_t st) {
    static std::atomic<uint64_t> smem_set{0};
    const cudaError_t e = ensure_smem_limit(gateup_swiglu_kernel, static_cast<int>(kSmemG), smem_set);
    if (e != cudaSuccess) return e;
    gateup_swiglu_kernel<<<grid, kGThreads, kSmemG, st>>>(tm_x, tm_w, p);
    return cudaGetLastError();
}

cudaError_t launch_gateup_pack(const void *w, void *wp, int hidden, int inter, cudaStream_t st) {
    const int64_t total = static_cast<int64_t>(2 * inter) * (hidden / 8);
    const int grid = static_cast<int>(std::min<int64_t>((total + 255) / 256, 152 * 16));
    gateup_pack_kernel<<<grid, 256, 0, st>>>(static_cast<const uint4 *>(w), static_cast<uint4 *>(wp), hidden,
                                             inter);
    return cudaGetLastError();
}

}  // namespace ppas
