// The split-K decode kernel: one CTA per (row, kv-head, split) of a step's
// decode rows (the CTA's work is decode_cta in attn_decode_body.cuh).
#include "attn_decode_body.cuh"

namespace ppas {

__global__ void __launch_bounds__(kDecodeThreads)
    decode_attn_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                       const __grid_constant__ DecodeParams p) {
    decode_cta<false>(tm_k, tm_v, p, blockIdx.x);
}

static std::atomic<uint64_t> g_decode_smem_set{0};

cudaError_t prepare_decode() {
    return ensure_smem_limit(decode_attn_kernel, static_cast<int>(kDecodeSmemBytes), g_decode_smem_set);
}

cudaError_t launch_decode(const CUtensorMap &tm_k, const CUtensorMap &tm_v, const DecodeParams &p,
                          cudaStream_t st) {
    const cudaError_t e = prepare_decode();
    if (e != cudaSuccess) return e;
    if (p.n_ctas <= 0) return cudaSuccess;
    PdlLaunch l(dim3(p.n_ctas), dim3(kDecodeThreads), kDecodeSmemBytes, st);
    return cudaLaunchKernelEx(&l.cfg, decode_attn_kernel, tm_k, tm_v, p);
}

}  // namespace ppas
