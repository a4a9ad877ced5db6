// An attention-step entry point for callers that cannot allocate device
// memory.
//
// Some callers of this library may not call cudaMalloc at all: a serving
// loop that has handed every byte of HBM to its KV-cache pool at start-up and
// must not allocate afterwards (cudaMalloc can synchronise the device, stall
// the loop or fail under memory pressure), or a host program whose memory is
// owned by someone else's allocator and that only passes in the tensors it
// was given.  For them this file keeps the step's scratch (the decode
// splits' partials and, when they fit beside them, the prefill pieces'
// partials) in a fixed-size array in the library's own device memory, so a
// call needs only the inputs and outputs.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds it (PPAS_NOALLOC_SCRATCH_BYTES) until the process exits.
// Host code may not use the array's name as a device address, so the first
// call on each device looks the address up with cudaGetSymbolAddress while
// that device is current, and later calls reuse it.  That first call also
// does the library's other one-time set-up for the device (the kernels'
// shared-memory limits, the decode cluster capacity, the side stream and
// events of mixed steps), so that no later call creates anything.
#include <mutex>

#include "ppas_internal.h"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[PPAS_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
void *g_scratch_ptr[kMaxDevices] = {nullptr};

// Device address of the scratch array on the current device (looked up once
// per device).  Returns nullptr when the lookup fails.
void *scratch_on_current_device() {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!g_scratch_ptr[dev]) {
        void *ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) return nullptr;
        if (ppas::prepare_current_device() != cudaSuccess) return nullptr;
        g_scratch_ptr[dev] = ptr;
    }
    return g_scratch_ptr[dev];
}

}  // namespace

extern "C" ppas_status ppas_attention_step_noalloc(const void *q, const void *k_cache, const void *v_cache,
                                                   int32_t num_blocks, const int32_t *d_block_tables,
                                                   int32_t max_blocks_per_seq, const int32_t *h_q_lens,
                                                   const int32_t *h_ctx_lens, int32_t n_seqs, int32_t n_q_heads,
                                                   int32_t n_kv_heads, int32_t head_dim, float scale, void *out,
                                                   int32_t out_is_fp32, int32_t *d_err_flag, void *stream) {
    // the decode scratch this step needs must fit the fixed array (checked
    // before any launch; on a device's first call the plan queries its
    // cluster capacity); the prefill tiles' split partials are used when
    // they fit beside it, else the prefill tiles run unsplit
    const size_t need = ppas::workspace_min_size(n_seqs, h_q_lens, h_ctx_lens, n_q_heads, n_kv_heads);
    if (need > static_cast<size_t>(PPAS_NOALLOC_SCRATCH_BYTES)) return PPAS_ERR_CAPACITY;
    void *scratch = nullptr;
    if (n_seqs > 0) {
        scratch = scratch_on_current_device();
        if (!scratch) return PPAS_ERR_CUDA;
    }
    // the step itself is the ordinary one, with the fixed array as its workspace
    return ppas_attention_step(q, k_cache, v_cache, num_blocks, d_block_tables, max_blocks_per_seq, h_q_lens,
                               h_ctx_lens, n_seqs, n_q_heads, n_kv_heads, head_dim, scale, out, out_is_fp32, scratch,
                               scratch ? static_cast<size_t>(PPAS_NOALLOC_SCRATCH_BYTES) : 0, d_err_flag, stream);
}
