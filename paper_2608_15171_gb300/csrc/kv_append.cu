// KV append: scatter the new tokens' keys and values into their 16-token
// pages (the KV-cache write every scheduled prefill or decode token makes,
// Section 2 of the paper).  Pure data movement with 16-byte accesses.
#include "ppas_device.cuh"
#include "ppas_internal.h"

namespace ppas {

// One thread moves one 16-byte chunk (8 bf16) of one (token, kv-head) row of
// K and the same chunk of V.  The launcher guarantees n_tokens * n_kv_heads *
// chunks_per_row < 2^31, so the element index is 32-bit.
__global__ void __launch_bounds__(256) kv_append_kernel(const uint4 *__restrict__ k_new, const uint4 *__restrict__ v_new,
                                                        const int32_t *__restrict__ slots, int32_t n_tokens,
                                                        uint4 *__restrict__ k_cache, uint4 *__restrict__ v_cache,
                                                        int32_t num_blocks, int32_t n_kv_heads, int32_t chunks_per_row,
                                                        int32_t *err) {
    // the attention launch that follows may start its set-up now
    grid_dep_launch();
    grid_dep_wait();
    const int32_t per_token = n_kv_heads * chunks_per_row;
    const int32_t total = per_token * n_tokens;
    for (int32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
        const int32_t t = i / per_token;
        const int32_t rem = i - t * per_token;
        const int32_t h = rem / chunks_per_row;
        const int32_t c = rem - h * chunks_per_row;
        const int32_t slot = __ldg(slots + t);
        if (slot < 0) continue;
        const int32_t blk = slot / kPage;
        const int32_t off = slot % kPage;
        if (blk >= num_blocks) {
            report_error(err, PPAS_DEVERR_BAD_INDEX);
            continue;
        }
        // cache layout [block][kv_head][16][head_dim]
        const int64_t dst = ((static_cast<int64_t>(blk) * n_kv_heads + h) * kPage + off) * chunks_per_row + c;
        k_cache[dst] = __ldg(k_new + i);
        v_cache[dst] = __ldg(v_new + i);
    }
}

// One thread waits on an mbarrier that nothing arrives on; the bounded wait
// gives up after limit_ns and records PPAS_DEVERR_TIMEOUT.  Exercises the
// failure path every kernel wait shares, without faulting or hanging.
__global__ void wait_timeout_kernel(int32_t *err, unsigned long long limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    const uint32_t b = smem_u32(&bar);
    mbar_init(b, 1);
    fence_mbar_init();
    mbar_wait(b, 0, err, limit_ns);
}

cudaError_t launch_wait_timeout(int32_t *err, unsigned long long limit_ns, cudaStream_t st) {
    wait_timeout_kernel<<<1, 1, 0, st>>>(err, limit_ns);
    return cudaGetLastError();
}

cudaError_t launch_kv_append(const void *k_new, const void *v_new, const int32_t *slots, int32_t n_tokens,
                             void *k_cache, void *v_cache, int32_t num_blocks, int32_t n_kv_heads,
                             int32_t head_dim, int32_t *err, cudaStream_t st) {
    const int32_t chunks = head_dim / 8;
    const int64_t total = static_cast<int64_t>(n_tokens) * n_kv_heads * chunks;
    if (total >= (int64_t{1} << 31)) return cudaErrorInvalidValue;
    const int threads = 256;
    int64_t blocks = (total + threads - 1) / threads;
    const int64_t cap = static_cast<int64_t>(device_sm_count()) * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    PdlLaunch l(dim3(static_cast<unsigned>(blocks)), dim3(threads), 0, st);
    return cudaLaunchKernelEx(&l.cfg, kv_append_kernel, static_cast<const uint4 *>(k_new),
                              static_cast<const uint4 *>(v_new), slots, n_tokens, static_cast<uint4 *>(k_cache),
                              static_cast<uint4 *>(v_cache), num_blocks, n_kv_heads, chunks, err);
}

}  // namespace ppas
