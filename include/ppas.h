/*
 * ppas.h -- C ABI of the GB300 (sm_103a) mixed prefill+decode attention step
 * behind P-PAS (Prefill-Pressure Adaptive Scheduling).
 *
 * The library is a plain shared object (libppas.so).  Every entry point takes
 * plain host or device pointers and sizes; nothing here mentions a framework
 * type.  The library keeps no global state apart from per-device caches
 * (driver entry points, the SM count, the kernels' shared-memory limits, how
 * many decode thread-block clusters the device holds co-resident, one
 * side stream with two events for steps too large for one launch, all created
 * on first use and thread-safe)
 * and the fixed scratch array of ppas_attention_step_noalloc; the only
 * stateful object is the opaque planner ppas_sched, which owns the free list
 * of KV blocks.
 *
 * Ownership: the caller owns every buffer passed in (inputs, caches,
 * outputs, workspace, error flag, plan arrays).  No call allocates device
 * memory.  Device calls are asynchronous on the given stream
 * (a cudaStream_t passed as void*; NULL is the legacy default stream).
 *
 * Errors: every call returns a ppas_status.  Argument errors are detected on
 * the host before anything is enqueued.  Failures inside a kernel (a bounded
 * wait that ran out, an index outside its buffer) never trap: the kernel
 * writes a nonzero PPAS_DEVERR_* code to *d_err_flag (when given) and
 * returns; the caller reads the flag after synchronising.
 */
#ifndef PPAS_H_
#define PPAS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t ppas_status;

#define PPAS_OK 0
#define PPAS_ERR_INVALID_ARG (-1)   /* a length, pointer or parameter is invalid      */
#define PPAS_ERR_CAPACITY (-2)      /* an output array or workspace is too small      */
#define PPAS_ERR_OUT_OF_BLOCKS (-3) /* the KV block pool cannot hold this step        */
#define PPAS_ERR_UNSUPPORTED (-4)   /* a shape this build has no kernel for           */
#define PPAS_ERR_CUDA (-5)          /* a CUDA runtime or driver call failed           */

/* codes a kernel writes to *d_err_flag (0 = no error) */
#define PPAS_DEVERR_TIMEOUT 1       /* a bounded wait on a barrier ran out            */
#define PPAS_DEVERR_BAD_INDEX 2     /* a slot or block id outside the cache           */

/* page geometry of the KV cache: 16 tokens per block */
#define PPAS_PAGE_TOKENS 16

/* request states (ppas_request.state) */
#define PPAS_REQ_PENDING 0   /* not arrived yet (arrival_us > now)               */
#define PPAS_REQ_WAITING 1   /* arrived, never scheduled                          */
#define PPAS_REQ_RUNNING 2   /* scheduled at least once, not finished             */
#define PPAS_REQ_FINISHED 3  /* all output tokens produced                        */

/* One request as the planner sees it (host memory, caller-owned array).
 * The caller fills arrival_us, prompt_len >= 1, output_len >= 1 and zeroes
 * the rest; the planner updates num_computed, num_generated, state and
 * n_blocks in place. */
typedef struct ppas_request {
    int64_t arrival_us;
    int32_t prompt_len;
    int32_t output_len;
    int32_t num_computed;  /* prompt tokens whose K/V have been scheduled     */
    int32_t num_generated; /* output tokens emitted so far                     */
    int32_t state;         /* PPAS_REQ_*                                        */
    int32_t n_blocks;      /* KV blocks the request holds (read-only)           */
} ppas_request;

/* The plan of one scheduler iteration.  The caller sets the three cap_*
 * fields and the five array pointers (host memory it owns); the planner
 * writes everything else.  Rows are listed decodes first (arrival order),
 * then prefill chunks (arrival order). */
typedef struct ppas_step {
    int32_t cap_rows;           /* capacity of req_idx / q_len / ctx_len         */
    int32_t cap_blocks_per_seq; /* row width of block_table                      */
    int32_t cap_tokens;         /* capacity of slot_mapping                      */
    int32_t n_rows;             /* rows scheduled this iteration                 */
    int32_t n_decode;           /* of which decode rows (q_len == 1)             */
    int32_t n_prefill;          /* of which prefill chunks                       */
    int32_t b_prefill;          /* prefill budget chosen by Algorithm 1          */
    int32_t pressure;           /* 1 when the cap B_cap applied                   */
    int32_t n_p;                /* running + waiting prefills (Algorithm 1)      */
    int32_t n_d;                /* running decodes (Algorithm 1)                 */
    int32_t prefill_tokens;     /* sum of prefill chunk lengths                   */
    int32_t total_tokens;       /* prefill_tokens + n_decode                      */
    int32_t *req_idx;           /* [cap_rows] request index of each row           */
    int32_t *q_len;             /* [cap_rows] new tokens of each row              */
    int32_t *ctx_len;           /* [cap_rows] context after the row (incl. new)   */
    int32_t *block_table;       /* [cap_rows * cap_blocks_per_seq], pad = -1      */
    int32_t *slot_mapping;      /* [cap_tokens] block*16+offset per new token     */
} ppas_step;

typedef struct ppas_sched ppas_sched;

/* ---------------------------------------------------------------------------
 * Planner (host only, integer work).
 * Follows Algorithm 1 of the paper (Section 3): N_p = running + waiting
 * prefills, N_d = running decodes; when N_p >= threshold and N_d > 0 the
 * aggregate prefill tokens of the iteration are limited to mbt_lo (B_cap),
 * otherwise to mbt_hi (B_max).  The global budget mbt_hi (vLLM's MBT) stays
 * in force for decode + prefill tokens together (Section 3, Section 2).
 * Decodes are scheduled first, then prefill chunks first-come-first-served.
 * ------------------------------------------------------------------------- */

/* Create a planner over a pool of num_blocks KV blocks whose free list starts
 * in the order initial_free_order[0..num_blocks) (a permutation of
 * 0..num_blocks-1; NULL means 0,1,2,...).  *out receives the handle.
 * Errors: PPAS_ERR_INVALID_ARG for num_blocks < 1, a NULL out, or an order
 * that is not a permutation. */
ppas_status ppas_sched_create(int32_t num_blocks, const int32_t *initial_free_order,
                              ppas_sched **out);

/* Destroy a planner (NULL is ignored). */
void ppas_sched_destroy(ppas_sched *sched);

/* Number of blocks on the free list. */
int32_t ppas_sched_free_blocks(const ppas_sched *sched);

/* Plan one iteration at time now_us over reqs[0..n_reqs) (the same array,
 * same order, on every call; requests may only be appended).  Steps:
 *  1. blocks of requests that finished in an earlier iteration return to the
 *     tail of the free list (queue order, table order);
 *  2. requests with arrival_us <= now_us are admitted;
 *  3. Algorithm 1 picks b_prefill from (threshold, mbt_hi, mbt_lo);
 *  4. every running decode gets one row (up to mbt_hi rows), then prefill
 *     chunks q = min(remaining prompt, b_prefill - used prefill,
 *     mbt_hi - used total) in queue order while q > 0;
 *  5. each row's request grows to ceil(ctx/16) blocks taken from the head of
 *     the free list; block tables and the slot mapping are written;
 *  6. request state advances (the final prefill chunk emits the first output
 *     token; a request finishes when num_generated == output_len).
 * Queue order is ascending (arrival_us, index).
 * Errors (nothing is modified): PPAS_ERR_INVALID_ARG for NULL pointers,
 * threshold < 1, mbt_lo < 1, mbt_hi < mbt_lo or a malformed request;
 * PPAS_ERR_CAPACITY when rows, table width or tokens exceed the caps;
 * PPAS_ERR_OUT_OF_BLOCKS when the free list is too short. */
ppas_status ppas_plan_step(ppas_sched *sched, ppas_request *reqs, int32_t n_reqs, int64_t now_us,
                           int32_t threshold, int32_t mbt_hi, int32_t mbt_lo, ppas_step *out);

/* ---------------------------------------------------------------------------
 * KV append (device).  Stores the keys and values of the step's new tokens
 * in the paged cache, the KV-cache write that prefill and decode perform for
 * every scheduled token (Section 2).
 *   k_new, v_new   : device bf16 [n_tokens, n_kv_heads, head_dim], contiguous
 *   d_slot_mapping : device int32 [n_tokens], slot = block*16 + offset;
 *                    a negative slot skips that token
 *   k_cache,v_cache: device bf16 [num_blocks, n_kv_heads, 16, head_dim]
 *   d_err_flag     : device int32 or NULL; PPAS_DEVERR_BAD_INDEX is written
 *                    when a slot is >= num_blocks*16 (that token is skipped)
 * head_dim must be a multiple of 8.  n_tokens == 0 is a no-op.
 * PPAS_ERR_UNSUPPORTED when n_tokens * n_kv_heads * head_dim / 8 >= 2^31.
 * The kernel is launched with programmatic stream serialization and lets the
 * next kernel of the stream start its set-up early; an attention step that
 * follows on the same stream still reads the cache only after it completes.
 * ------------------------------------------------------------------------- */
ppas_status ppas_kv_append(const void *k_new, const void *v_new, const int32_t *d_slot_mapping,
                           int32_t n_tokens, void *k_cache, void *v_cache, int32_t num_blocks,
                           int32_t n_kv_heads, int32_t head_dim, int32_t *d_err_flag, void *stream);

/* ---------------------------------------------------------------------------
 * Mixed-batch attention step (device).
 * One scheduler iteration's attention: prefill chunks attend causally to
 * their own paged KV prefix and decode rows attend to their whole context,
 * all in one call (Section 6.2: prefill and decode tokens of one iteration
 * run together).  For sequence s with q_s = h_q_lens[s] new tokens and
 * context ctx_s = h_ctx_lens[s] (the new tokens are the last q_s positions,
 * already appended to the cache), query token t sits at position
 * ctx_s - q_s + t and sees keys 0..ctx_s-q_s+t; q-head h reads kv-head
 * h / (n_q_heads / n_kv_heads):
 *   out[s,t,h,:] = sum_j softmax_j(scale * q[s,t,h,:] . K_s[j,:]) V_s[j,:].
 *
 *   q             : device bf16 [sum(q_lens), n_q_heads, head_dim], sequences
 *                   packed in order, 16-byte aligned
 *   k_cache,v_cache: device bf16 [num_blocks, n_kv_heads, 16, head_dim],
 *                   16-byte aligned
 *   d_block_tables: device int32 [n_seqs, max_blocks_per_seq]; entry j of row
 *                   s is the physical block of positions 16j..16j+15
 *   h_q_lens, h_ctx_lens : HOST int32 [n_seqs], 1 <= q_len <= ctx_len <=
 *                   16*max_blocks_per_seq
 *   out           : device [sum(q_lens), n_q_heads, head_dim], bf16
 *                   (out_is_fp32 == 0) or fp32 (out_is_fp32 != 0)
 *   workspace     : device scratch of at least
 *                   ppas_attention_workspace_size(...) bytes, 256-byte aligned
 *                   (may be NULL when that size is 0)
 *   d_err_flag    : device int32 or NULL (see PPAS_DEVERR_*)
 * Supported shapes: head_dim == 128, n_q_heads a multiple of n_kv_heads with
 * group size n_q_heads/n_kv_heads in {1, 2, 4, 8}, at most 256 q-heads
 * (512 with group >= 2), ctx_len <= 65535*128 for rows with q_len > 1 and
 * ctx_len <= 2^25 for rows with q_len == 1; otherwise PPAS_ERR_UNSUPPORTED.  n_seqs == 0 is a no-op.  Block ids in the tables
 * must lie in [0, num_blocks) for every position below ctx_len.
 * Rows with q_len == 1 run as split-K decode work; longer rows run on the
 * tcgen05 prefill path, whose long (query tile, head) units may be cut into
 * pieces on several CTAs (when the workspace holds their partials) and
 * merged by a short merge launch right after.
 * Launches: a step with only decode rows is one decode launch (for a few
 * rows on a device that holds enough of them co-resident, in thread-block
 * clusters of 4 CTAs whose split partials merge through distributed shared
 * memory before reaching the workspace); a step with
 * prefill chunks is one launch of the prefill kernel, or, with decode rows
 * as well, one mixed launch whose first CTAs run the prefill items and whose
 * remaining CTAs run the decode splits; either is followed by the merge
 * launch when its plan cuts units.  Only a step whose prefill items exceed
 * one launch's tables (over 2200 items, 128 sequences, or with more than 112
 * decode rows beside the chunks) takes several prefill launches; then the
 * decode launch runs on a library-owned side stream forked from `stream`
 * (an event) and joined back into it (a second event).
 * Stream semantics: all work is ordered after the work already on `stream`
 * and everything later on `stream` is ordered after it, as for one kernel.
 * The kernels are launched with programmatic stream serialization (their
 * set-up may overlap the kernel before them on their stream; every
 * global-memory access waits for that kernel to complete).  The workspace
 * needs no initialisation: the decode splits' arrival tickets in it carry a
 * per-launch tag.  Plans, and so
 * ppas_attention_workspace_size, follow the current device's SM count (and,
 * for steps of decode rows only, its cluster capacity).
 * ------------------------------------------------------------------------- */
size_t ppas_attention_workspace_size(int32_t n_seqs, const int32_t *h_q_lens,
                                     const int32_t *h_ctx_lens, int32_t n_q_heads,
                                     int32_t n_kv_heads);

/* ---------------------------------------------------------------------------
 * Number of kernels ppas_attention_step launches for this step when given a
 * workspace of workspace_bytes (host only), for the current device's plan:
 * its prefill (or mixed) launches, the merge launch after each one whose
 * plan cuts units, and its decode launches unless they are part of a mixed
 * launch (see ppas_attention_step; the call enqueues nothing else: no
 * memset, no copy).  Returns -1 for arguments
 * ppas_attention_step would reject (see there); 0 for n_seqs == 0.
 * ------------------------------------------------------------------------- */
int32_t ppas_attention_kernel_count(int32_t n_seqs, const int32_t *h_q_lens, const int32_t *h_ctx_lens,
                                    int32_t n_q_heads, int32_t n_kv_heads, size_t workspace_bytes);

ppas_status ppas_attention_step(const void *q, const void *k_cache, const void *v_cache,
                                int32_t num_blocks, const int32_t *d_block_tables,
                                int32_t max_blocks_per_seq, const int32_t *h_q_lens,
                                const int32_t *h_ctx_lens, int32_t n_seqs, int32_t n_q_heads,
                                int32_t n_kv_heads, int32_t head_dim, float scale, void *out,
                                int32_t out_is_fp32, void *workspace, size_t workspace_bytes,
                                int32_t *d_err_flag, void *stream);

/* ---------------------------------------------------------------------------
 * Gate-up projection of the decoder MLP with the gated activation fused in
 * (the GEMM Section 6.1 profiles beside attention):
 *   y[t, i] = silu(x[t] . w[i]) * (x[t] . w[inter + i]),  silu(a) = a / (1 + e^-a)
 * for the stacked weight w = [w_gate; w_up] of shape [2*inter, hidden].
 *
 * ppas_gateup_pack (device, async on `stream`): rearranges w (device bf16
 *   [2*inter, hidden], gate rows then up rows) into w_packed (device bf16,
 *   same size, caller-owned): block j of 256 rows holds gate rows
 *   128j..128j+127 then up rows inter+128j..inter+128j+127.  Done once per
 *   weight.
 * ppas_gateup_swiglu (device, async on `stream`): x device bf16
 *   [n_tokens, hidden] row-major, w_packed as produced above, y device bf16
 *   [n_tokens, inter] row-major (caller-owned).  fp32 accumulation.
 * Both: hidden a multiple of 64 and inter a multiple of 128, else
 * PPAS_ERR_UNSUPPORTED; pointers 16-byte aligned, else PPAS_ERR_INVALID_ARG;
 * n_tokens == 0 is a no-op.  d_err_flag (device int32 or NULL) records
 * PPAS_DEVERR_TIMEOUT if a bounded wait runs out.
 * ------------------------------------------------------------------------- */
ppas_status ppas_gateup_pack(const void *w, void *w_packed, int32_t hidden, int32_t inter, void *stream);
ppas_status ppas_gateup_swiglu(const void *x, const void *w_packed, void *y, int32_t n_tokens, int32_t hidden,
                               int32_t inter, int32_t *d_err_flag, void *stream);

/* ---------------------------------------------------------------------------
 * Attention step without a caller-provided workspace.  The paper has no
 * counterpart to this entry point: it exists for callers that may not
 * allocate device memory at all (a serving loop that gave all of HBM to its
 * KV-cache pool at start-up and cannot call cudaMalloc afterwards, or a host
 * program whose device memory belongs to another allocator).
 *
 * Same arguments, layouts and results as ppas_attention_step, minus the
 * workspace: the scratch lives in a fixed array of
 * PPAS_NOALLOC_SCRATCH_BYTES (64 MiB) inside the library's device memory,
 * which every GPU that loads the library holds until the process exits.
 * The call makes no cudaMalloc, cudaFree or other allocating call.
 *  - The split-K decode scratch of the step must fit the array, else the
 *    step is rejected with PPAS_ERR_CAPACITY before any device work.
 *  - When the prefill tiles' split partials also fit beside it
 *    (ppas_attention_workspace_size <= PPAS_NOALLOC_SCRATCH_BYTES, true for
 *    every workload of the paper's configurations) the step runs exactly as
 *    ppas_attention_step with a full workspace.  Otherwise the prefill
 *    tiles run unsplit: same results up to rounding, except that a query
 *    tile over a context longer than 65,536 keys then accumulates in one
 *    piece, whose fp32 tensor-core accumulation drifts towards smaller
 *    magnitude (~4e-4 relative at 110k keys, ~5e-3 at 880k).
 *  - The first call on a device (with rows to run) does the library's
 *    one-time set-up for that device with it current: it looks up the
 *    array's device address, sets the kernels' shared-memory limits,
 *    queries how many decode clusters the device holds co-resident and
 *    creates the side stream and two events that steps too large for one
 *    launch use.  Make that first
 *    call before any stream capture and before a phase in which nothing may
 *    be created.  PPAS_ERR_CUDA if the set-up fails.
 *  - All calls share one array, which keeps the last call's contents (the
 *    decode split tickets in it carry a per-launch tag, so nothing in it has
 *    to start at zero).
 *    Calls whose work overlaps on the GPU (other streams, other host threads)
 *    race on it: serialise them.
 * ------------------------------------------------------------------------- */
#define PPAS_NOALLOC_SCRATCH_BYTES (64 * 1024 * 1024)

ppas_status ppas_attention_step_noalloc(const void *q, const void *k_cache, const void *v_cache,
                                        int32_t num_blocks, const int32_t *d_block_tables,
                                        int32_t max_blocks_per_seq, const int32_t *h_q_lens,
                                        const int32_t *h_ctx_lens, int32_t n_seqs, int32_t n_q_heads,
                                        int32_t n_kv_heads, int32_t head_dim, float scale, void *out,
                                        int32_t out_is_fp32, int32_t *d_err_flag, void *stream);

/* Failure-path check (device).  Launches one thread that waits, with a
 * limit of limit_us microseconds (1 .. 2,000,000), on a barrier nothing
 * arrives on -- the same bounded wait every kernel of this library uses --
 * so that the wait runs out and PPAS_DEVERR_TIMEOUT is written to
 * *d_err_flag (device int32, required).  The GPU context stays usable. */
ppas_status ppas_debug_wait_timeout(int32_t *d_err_flag, uint32_t limit_us, void *stream);

/* Static description of a status code (never NULL). */
const char *ppas_status_string(ppas_status status);

/* ABI version of this header (bumped on any signature change). */
int32_t ppas_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* PPAS_H_ */
