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
//  * with clusters (a step of decode rows only, on a device that holds
//    clusters of 4 co-resident), every row's split count is a multiple
//    of the cluster size, at most cluster - 1 of a row's splits lie past
//    its pages, the CTAs fit the clusters the device holds and fill at least
//    15/16 of its SMs, and a cluster writes one partial slot;
//  * the partial and CTA counts add up and the workspace sizes hold every
//    partial (m, l), partial O and ticket, in 256-byte multiples.
// Each case is planned without clusters (the line printed) and with the
// cluster capacities of a GB300-like device scaled to <sms> (checked).
// It prints one line per case: "ok <ctas> <parts> <cluster>" or
// "FAIL <reason>".
#include <algorithm>
#include <cstdio>
#include <iostream>
#include <string>
#include <vector>

#include "ppas_internal.h"

using namespace ppas;

static std::string check(int sms, int hq, int hk, const std::vector<int32_t> &q, const std::vector<int32_t> &c,
                         const DecodeClusterCaps &caps, long long *ctas, long long *parts, int *cluster) {
    const int n = static_cast<int>(q.size());
    DecodePlan d = plan_decode(n, q.data(), c.data(), hq, hk, sms, caps);
    std::vector<int32_t> want;
    for (int s = 0; s < n; ++s)
        if (q[s] == 1) want.push_back(s);
    if (d.rows != want) return "decode rows";
    if (d.n_splits.size() != d.rows.size() || d.pages_per_split.size() != d.rows.size()) return "plan sizes";
    const long long cl = d.cluster;
    if (cl != 1 && cl != 2 && cl != 4) return "cluster size";
    if (cl > 1 && static_cast<int>(d.rows.size()) != n) return "clusters beside prefill rows";
    long long np = 0, nc = 0;
    for (size_t k = 0; k < d.rows.size(); ++k) {
        const long long pages = (c[d.rows[k]] + kPage - 1) / kPage;
        const long long ns = d.n_splits[k], pps = d.pages_per_split[k];
        if (ns < 1 || ns > kMaxDecodeSplitsPerRow) return "split count";
        if (ns % cl) return "splits not a whole number of clusters";
        if (pps < 1 || pps > kDecodeMaxPagesPerSplit) return "pages per split";
        if (pps < std::min<long long>(pages, kDecodeMinPagesPerSplit)) return "split shorter than the minimum";
        // the splits cover the row's pages; without clusters every split
        // holds a page, with them at most cl - 1 splits lie past the pages
        const long long used = (pages + pps - 1) / pps;
        if (ns * pps < pages || used > ns || used <= ns - cl) return "split coverage";
        np += ns / cl;
        nc += ns * hk;
    }
    if (np != d.n_part || nc != d.n_ctas) return "totals";
    if (cl == 2 && (nc > caps.ctas2 || nc * 16 < 15LL * sms)) return "clusters of 2 beyond one wave";
    if (cl == 4 && (nc > caps.ctas4 || nc * 16 < 15LL * sms)) return "clusters of 4 beyond one wave";
    if (d.ml_bytes % 256 || d.o_bytes % 256 || d.counter_bytes % 256) return "alignment";
    if (d.ml_bytes < static_cast<size_t>(np) * hq * 2 * sizeof(float)) return "partial m/l bytes";
    if (d.o_bytes < static_cast<size_t>(np) * hq * kHeadDim * sizeof(float)) return "partial O bytes";
    if (d.counter_bytes < d.rows.size() * hk * sizeof(unsigned long long)) return "ticket bytes";
    *ctas = nc;
    *parts = np;
    *cluster = d.cluster;
    return "";
}

int main() {
    int sms, hq, hk, n;
    while (std::cin >> sms >> hq >> hk >> n) {
        std::vector<int32_t> q(n), c(n);
        for (auto &x : q) std::cin >> x;
        for (auto &x : c) std::cin >> x;
        long long ctas = 0, parts = 0;
        int cluster = 1;
        std::string err = check(sms, hq, hk, q, c, DecodeClusterCaps{}, &ctas, &parts, &cluster);
        if (err.empty()) {
            // a GB300 holds 76 clusters of 2 and 36 of 4 of the decode kernel (152 SMs)
            DecodeClusterCaps caps;
            caps.ctas2 = sms / 2 * 2;
            caps.ctas4 = sms * 36 / 38 / 4 * 4;
            long long c2 = 0, p2 = 0;
            int cl2 = 1;
            err = check(sms, hq, hk, q, c, caps, &c2, &p2, &cl2);
            if (err.empty() && cl2 > 1) cluster = cl2;
        }
        if (!err.empty())
            std::printf("FAIL %s\n", err.c_str());
        else
            std::printf("ok %lld %lld %d\n", ctas, parts, cluster);
    }
    return 0;
}
