// P-PAS step planner: Algorithm 1 (Section 3) on top of chunked prefill with a
// shared token budget (Section 2), plus the FIFO KV block pool, block tables
// and slot mapping of the step.  Host-only integer work.
#include <algorithm>
#include <cstdint>
#include <deque>
#include <numeric>
#include <vector>

#include "ppas.h"

struct ppas_sched {
    int32_t num_blocks = 0;
    std::deque<int32_t> free_list;               // head = next block handed out
    std::vector<std::vector<int32_t>> blocks;    // per request index, table order
};

namespace {

inline int32_t ceil_div16(int64_t x) { return static_cast<int32_t>((x + PPAS_PAGE_TOKENS - 1) / PPAS_PAGE_TOKENS); }

struct Row {
    int32_t req;
    int32_t q;
    int32_t ctx;
    bool prefill;
};

}  // namespace

extern "C" ppas_status ppas_sched_create(int32_t num_blocks, const int32_t *order, ppas_sched **out) {
    if (!out || num_blocks < 1) return PPAS_ERR_INVALID_ARG;
    *out = nullptr;
    std::vector<int32_t> seen(num_blocks, 0);
    auto *s = new ppas_sched();
    s->num_blocks = num_blocks;
    for (int32_t i = 0; i < num_blocks; ++i) {
        int32_t b = order ? order[i] : i;
        if (b < 0 || b >= num_blocks || seen[b]) {
            delete s;
            return PPAS_ERR_INVALID_ARG;
        }
        seen[b] = 1;
        s->free_list.push_back(b);
    }
    *out = s;
    return PPAS_OK;
}

extern "C" void ppas_sched_destroy(ppas_sched *s) { delete s; }

extern "C" int32_t ppas_sched_free_blocks(const ppas_sched *s) {
    return s ? static_cast<int32_t>(s->free_list.size()) : 0;
}

extern "C" ppas_status ppas_plan_step(ppas_sched *s, ppas_request *reqs, int32_t n_reqs, int64_t now_us,
                                      int32_t threshold, int32_t mbt_hi, int32_t mbt_lo, ppas_step *out) {
    if (!s || !out || n_reqs < 0 || (n_reqs > 0 && !reqs)) return PPAS_ERR_INVALID_ARG;
    if (threshold < 1 || mbt_lo < 1 || mbt_hi < mbt_lo) return PPAS_ERR_INVALID_ARG;
    if (out->cap_rows < 0 || out->cap_blocks_per_seq < 0 || out->cap_tokens < 0) return PPAS_ERR_INVALID_ARG;
    if ((out->cap_rows > 0 && (!out->req_idx || !out->q_len || !out->ctx_len)) ||
        (out->cap_rows > 0 && out->cap_blocks_per_seq > 0 && !out->block_table) ||
        (out->cap_tokens > 0 && !out->slot_mapping))
        return PPAS_ERR_INVALID_ARG;
    for (int32_t i = 0; i < n_reqs; ++i) {
        const ppas_request &r = reqs[i];
        if (r.prompt_len < 1 || r.output_len < 1 || r.num_computed < 0 || r.num_computed > r.prompt_len ||
            r.num_generated < 0 || r.state < PPAS_REQ_PENDING || r.state > PPAS_REQ_FINISHED)
            return PPAS_ERR_INVALID_ARG;
    }
    if (static_cast<int32_t>(s->blocks.size()) > n_reqs) return PPAS_ERR_INVALID_ARG;  // requests only grow
    s->blocks.resize(n_reqs);

    // queue order: ascending (arrival_us, index)
    std::vector<int32_t> order(n_reqs);
    std::iota(order.begin(), order.end(), 0);
    std::stable_sort(order.begin(), order.end(),
                     [&](int32_t a, int32_t b) { return reqs[a].arrival_us < reqs[b].arrival_us; });

    // --- everything below is computed first and committed only on success ---
    // 1. blocks of finished requests go back to the tail (queue order, table order)
    std::vector<int32_t> released;
    for (int32_t i : order)
        if (reqs[i].state == PPAS_REQ_FINISHED && !s->blocks[i].empty())
            released.insert(released.end(), s->blocks[i].begin(), s->blocks[i].end());

    // 2. admission, 3. Algorithm 1
    auto admitted = [&](int32_t i) {
        const ppas_request &r = reqs[i];
        return r.state == PPAS_REQ_WAITING || r.state == PPAS_REQ_RUNNING ||
               (r.state == PPAS_REQ_PENDING && r.arrival_us <= now_us);
    };
    std::vector<int32_t> prefills, decodes;
    for (int32_t i : order) {
        if (!admitted(i)) continue;
        if (reqs[i].num_computed < reqs[i].prompt_len)
            prefills.push_back(i);
        else
            decodes.push_back(i);
    }
    const int32_t n_p = static_cast<int32_t>(prefills.size());
    const int32_t n_d = static_cast<int32_t>(decodes.size());
    const bool pressure = (n_p >= threshold) && (n_d > 0);
    const int32_t b_prefill = pressure ? mbt_lo : mbt_hi;

    // 4. decodes first under the global budget, then FCFS prefill chunks
    std::vector<Row> rows;
    int64_t used_total = 0, used_prefill = 0;
    for (int32_t i : decodes) {
        if (used_total >= mbt_hi) break;
        rows.push_back({i, 1, reqs[i].prompt_len + reqs[i].num_generated, false});
        used_total += 1;
    }
    const int32_t n_decode = static_cast<int32_t>(rows.size());
    for (int32_t i : prefills) {
        int64_t q = std::min<int64_t>({static_cast<int64_t>(reqs[i].prompt_len - reqs[i].num_computed),
                                       b_prefill - used_prefill, mbt_hi - used_total});
        if (q <= 0) break;
        rows.push_back({i, static_cast<int32_t>(q), reqs[i].num_computed + static_cast<int32_t>(q), true});
        used_prefill += q;
        used_total += q;
    }

    // capacity checks
    const int32_t n_rows = static_cast<int32_t>(rows.size());
    if (n_rows > out->cap_rows || used_total > out->cap_tokens) return PPAS_ERR_CAPACITY;
    int64_t need = 0;
    for (const Row &w : rows) {
        int32_t want = ceil_div16(w.ctx);
        if (want > out->cap_blocks_per_seq) return PPAS_ERR_CAPACITY;
        need += std::max<int64_t>(0, want - static_cast<int64_t>(s->blocks[w.req].size()));
    }
    if (need > static_cast<int64_t>(s->free_list.size() + released.size())) return PPAS_ERR_OUT_OF_BLOCKS;

    // ---- commit ----
    for (int32_t i : order)
        if (reqs[i].state == PPAS_REQ_FINISHED && !s->blocks[i].empty()) {
            for (int32_t b : s->blocks[i]) s->free_list.push_back(b);
            s->blocks[i].clear();
            reqs[i].n_blocks = 0;
        }
    for (int32_t i : order)
        if (reqs[i].state == PPAS_REQ_PENDING && reqs[i].arrival_us <= now_us) reqs[i].state = PPAS_REQ_WAITING;

    // 5. allocation, tables, slots
    const int32_t width = out->cap_blocks_per_seq;
    int32_t tok = 0;
    for (int32_t r = 0; r < n_rows; ++r) {
        const Row &w = rows[r];
        std::vector<int32_t> &bl = s->blocks[w.req];
        const int32_t want = ceil_div16(w.ctx);
        while (static_cast<int32_t>(bl.size()) < want) {
            bl.push_back(s->free_list.front());
            s->free_list.pop_front();
        }
        reqs[w.req].n_blocks = static_cast<int32_t>(bl.size());
        out->req_idx[r] = w.req;
        out->q_len[r] = w.q;
        out->ctx_len[r] = w.ctx;
        int32_t *trow = out->block_table + static_cast<int64_t>(r) * width;
        for (int32_t j = 0; j < width; ++j) trow[j] = j < static_cast<int32_t>(bl.size()) ? bl[j] : -1;
        for (int32_t pos = w.ctx - w.q; pos < w.ctx; ++pos)
            out->slot_mapping[tok++] = bl[pos / PPAS_PAGE_TOKENS] * PPAS_PAGE_TOKENS + pos % PPAS_PAGE_TOKENS;
    }

    // 6. state update
    for (const Row &w : rows) {
        ppas_request &q = reqs[w.req];
        q.state = PPAS_REQ_RUNNING;
        if (w.prefill) {
            q.num_computed += w.q;
            if (q.num_computed == q.prompt_len) q.num_generated = 1;
        } else {
            q.num_generated += 1;
        }
        if (q.num_computed == q.prompt_len && q.num_generated >= q.output_len) q.state = PPAS_REQ_FINISHED;
    }

    out->n_rows = n_rows;
    out->n_decode = n_decode;
    out->n_prefill = n_rows - n_decode;
    out->b_prefill = b_prefill;
    out->pressure = pressure ? 1 : 0;
    out->n_p = n_p;
    out->n_d = n_d;
    out->prefill_tokens = static_cast<int32_t>(used_prefill);
    out->total_tokens = static_cast<int32_t>(used_total);
    return PPAS_OK;
}
