// Checks the host plan of the split-K decode kernel against what the kernel
// indexes: for every case read from stdin
//   <sms> <n_q_heads> <n_kv_heads> <n_seqs> <q_len>... <ctx_len>...
// it plans the step's decode rows the way the attention call does on a
// device of <sms> SMs and verifies that
//  * the decode rows are exactly the rows with q_len == 1, in order;
//  * split sp of a row covers pages [sp * pps, min((sp + 1) * pps, pages)),
//    every split holds at least one page and the splits cover the row's
//    pages exactly once;
//  * pages per split lie in [min(pages, kDecodeMinPagesPerSplit),
//    kDecodeMaxPagesPerSplit] and a row has at most kMaxDecodeSplitsPerRow
//    splits (the merge keeps their weights in shared memory);
//  * the partial and CTA counts add up and the workspace sizes hold every
//    partial (m, l), partial O and ticket, in 256-byte multiples.
// It prints one line per case: "ok <ctas> <parts>" or "FAIL <reason>".
#include <algorithm>
#include <cstdio>
#include <iostream>
#include <string>
#include <vector>

#include "ppas_internal.h"

using namespace ppas;

static std::string check(int sms, int hq, int hk, const std::vector<int32_t> &q, const std::vector<int32_t> &c,
                         long long *ctas, long long *parts) {
    const int n = static_cast<int>(q.size());
    DecodePlan d = plan_decode(n, q.data(), c.data(), hq, hk, sms);
    std::vector<int32_t> want;
    for (int s = 0; s < n; ++s)
        if (q[s] == 1) want.push_back(s);
    if (d.rows != want) return "decode rows";
    if (d.n_splits.size() != d.rows.size() || d.pages_per_split.size() != d.rows.size()) return "plan sizes";
    long long np = 0, nc = 0;
    for (size_t k = 0; k < d.rows.size(); ++k) {
        const long long pages = (c[d.rows[k]] + kPage - 1) / kPage;
        const long long ns = d.n_splits[k], pps = d.pages_per_split[k];
        if (ns < 1 || ns > kMaxDecodeSplitsPerRow) return "split count";
        if (pps < 1 || pps > kDecodeMaxPagesPerSplit) return "pages per split";
        if (pps < std::min<long long>(pages, kDecodeMinPagesPerSplit)) return "split shorter than the minimum";
        // every split non-empty, the last one ending at the row's last page
        if ((ns - 1) * pps >= pages || ns * pps < pages) return "split coverage";
        np += ns;
        nc += ns * hk;
    }
    if (np != d.n_part || nc != d.n_ctas) return "totals";
    if (d.ml_bytes % 256 || d.o_bytes % 256 || d.counter_bytes % 256) return "alignment";
    if (d.ml_bytes < static_cast<size_t>(np) * hq * 2 * sizeof(float)) return "partial m/l bytes";
    if (d.o_bytes < static_cast<size_t>(np) * hq * kHeadDim * sizeof(float)) return "partial O bytes";
    if (d.counter_bytes < d.rows.size() * hk * sizeof(unsigned long long)) return "ticket bytes";
    *ctas = nc;
    *parts = np;
    return "";
}

int main() {
    int sms, hq, hk, n;
    while (std::cin >> sms >> hq >> hk >> n) {
        std::vector<int32_t> q(n), c(n);
        for (auto &x : q) std::cin >> x;
        for (auto &x : c) std::cin >> x;
        long long ctas = 0, parts = 0;
        const std::string err = check(sms, hq, hk, q, c, &ctas, &parts);
        if (!err.empty())
            std::printf("FAIL %s\n", err.c_str());
        else
            std::printf("ok %lld %lld\n", ctas, parts);
    }
    return 0;
}
