// The split-K decode kernel: one CTA per (row, kv-head, split) of a step's
// decode rows (the CTA's work is decode_cta in attn_decode_body.cuh).
#include <algorithm>
#include <atomic>

#include "attn_decode_body.cuh"

namespace ppas {

__global__ void __launch_bounds__(kDecodeThreads, 1)
    decode_attn_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                       const __grid_constant__ DecodeParams p) {
    decode_cta<false>(tm_k, tm_v, p, blockIdx.x);
}

static std::atomic<uint64_t> g_decode_smem_set{0};

cudaError_t prepare_decode() {
    return ensure_smem_limit(decode_attn_kernel, static_cast<int>(kDecodeSmemBytes), g_decode_smem_set);
}

// CTAs of this kernel the current device holds co-resident in clusters of
// c (0 when it cannot say), from the occupancy calculator
static int32_t cluster_ctas(int c) {
    if (prepare_decode() != cudaSuccess) return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(c);
    cfg.blockDim = dim3(kDecodeThreads);
    cfg.dynamicSmemBytes = kDecodeSmemBytes;
    cudaLaunchAttribute a[1];
    a[0].id = cudaLaunchAttributeClusterDimension;
    a[0].val.clusterDim.x = c;
    a[0].val.clusterDim.y = 1;
    a[0].val.clusterDim.z = 1;
    cfg.attrs = a;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, decode_attn_kernel, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return n * c;
}

DecodeClusterCaps decode_cluster_caps() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
        cudaGetLastError();
        return {};
    }
    // per device: (1 << 62) | ctas4 << 16 | ctas2 once known
    static std::atomic<uint64_t> cached[64] = {};
    uint64_t v = cached[dev].load(std::memory_order_relaxed);
    if (!v) {
        const uint64_t c2 = static_cast<uint64_t>(std::max(0, cluster_ctas(2))) & 0xFFFF;
        const uint64_t c4 = static_cast<uint64_t>(std::max(0, cluster_ctas(4))) & 0xFFFF;
        v = (uint64_t{1} << 62) | (c4 << 16) | c2;
        cached[dev].store(v, std::memory_order_relaxed);
    }
    DecodeClusterCaps caps;
    caps.ctas2 = static_cast<int32_t>(v & 0xFFFF);
    caps.ctas4 = static_cast<int32_t>((v >> 16) & 0xFFFF);
    return caps;
}

cudaError_t launch_decode(const CUtensorMap &tm_k, const CUtensorMap &tm_v, const DecodeParams &p,
                          int32_t cluster, cudaStream_t st) {
    const cudaError_t e = prepare_decode();
    if (e != cudaSuccess) return e;
    if (p.n_ctas <= 0) return cudaSuccess;
    // rank 0 of a cluster has slots for decode_detail::kMaxCluster partials
    if (cluster < 1 || cluster > decode_detail::kMaxCluster || p.n_ctas % cluster != 0) return cudaErrorInvalidValue;
    PdlLaunch l(dim3(p.n_ctas), dim3(kDecodeThreads), kDecodeSmemBytes, st);
    cudaLaunchAttribute attrs[2] = {l.attr[0], {}};
    if (cluster > 1) {
        // the splits of a (row, kv-head) in groups of `cluster` CTAs that
        // merge through distributed shared memory (decode_cta)
        attrs[1].id = cudaLaunchAttributeClusterDimension;
        attrs[1].val.clusterDim.x = static_cast<unsigned>(cluster);
        attrs[1].val.clusterDim.y = 1;
        attrs[1].val.clusterDim.z = 1;
        l.cfg.attrs = attrs;
        l.cfg.numAttrs = 2;
    }
    return cudaLaunchKernelEx(&l.cfg, decode_attn_kernel, tm_k, tm_v, p);
}

}  // namespace ppas
