// Checks the host plan of the persistent prefill kernel against what the
// kernel indexes: for every case read from stdin
//   <sms> <n_q_heads> <n_kv_heads> <n_seqs> <q_len>... <ctx_len>...
// it plans the step the way the attention call does on a device of <sms>
// SMs and verifies that
//  * each launch's tables (items, sequences, CTAs) fit their capacities and
//    every CTA has at least one item;
//  * every item's sequence, query tile, head slot and KV range are valid,
//    and every page it reads lies inside the sequence's context;
//  * the items of each (query tile, head slot) unit cover its causal KV
//    tiles exactly once;
//  * each piece of a split unit owns one partial slot inside the workspace,
//    and the unit's merge entry lists exactly its pieces;
//  * with splits allowed no item spans more than kPrefillMaxPiece KV tiles
//    (the accumulation depth of one fp32 partial in TMEM);
//  * without splits (a small workspace) the same coverage holds.
// It prints one line per case: "ok <launches> <ctas> <items> <parts>
// <max_load> <mean_load>" or "FAIL <reason>".
#include <algorithm>
#include <cstdio>
#include <iostream>
#include <map>
#include <string>
#include <tuple>
#include <vector>

#include "ppas_internal.h"

using namespace ppas;

static std::string check(int sms, int hq, int hk, const std::vector<int32_t> &q, const std::vector<int32_t> &c, bool split,
                         double *max_load, double *mean_load, size_t *n_launch, size_t *n_ctas, size_t *n_items,
                         long long *n_part) {
    const int n = static_cast<int>(q.size());
    const int reserve = decode_reserve_sms(n, q.data(), c.data(), hq, hk, sms);
    if (reserve < 0 || reserve > sms / 2) return "reserve out of range";
    const int avail = sms - reserve;
    PrefillPlan pf = plan_prefill(n, q.data(), c.data(), hq, hk, split, avail);
    const int hpc = hq / hk >= 2 ? 2 : 1, slots = hq / hpc;
    if (pf.slots != slots || pf.heads_per_cta != hpc) return "head slots";
    std::map<std::tuple<int, int, int>, std::vector<int>> cover;
    double sum = 0, mx = 0;
    size_t ctas = 0, items = 0;
    for (const PrefillLaunchPlan &lp : pf.launches) {
        const size_t nc = lp.cta_begin.size() - 1;
        if (nc < 1 || nc > static_cast<size_t>(avail) || nc > static_cast<size_t>(kMaxPrefillCtas)) return "CTA count";
        if (lp.work.size() > static_cast<size_t>(kMaxPrefillWork)) return "item capacity";
        if (lp.seqs.size() > static_cast<size_t>(kMaxPrefillSeqs)) return "sequence capacity";
        if (lp.cta_begin[0] != 0 || lp.cta_begin[nc] != lp.work.size()) return "CTA ranges";
        if (lp.n_part > pf.n_part || (!split && lp.n_part)) return "partial count";
        for (size_t k = 0; k < nc; ++k) {
            if (lp.cta_begin[k] >= lp.cta_begin[k + 1]) return "CTA without items";
            double load = 0;
            for (int w = lp.cta_begin[k]; w < lp.cta_begin[k + 1]; ++w)
                load += lp.work[w].kt1 - lp.work[w].kt0 + kPrefillItemCost;
            mx = std::max(mx, load);
            sum += load;
        }
        ctas += nc;
        items += lp.work.size();
        std::vector<int> part_owner(lp.n_part, 0);
        std::map<std::tuple<int, int, int>, int> pieces;
        for (const PrefillWork &wk : lp.work) {
            if (wk.seq >= lp.seqs.size()) return "sequence index";
            const int s = lp.seqs[wk.seq];
            if (s < 0 || s >= n || q[s] == 1) return "sequence of an item";
            if (wk.slot >= slots) return "head slot";
            const int t0 = wk.qt * kTileQ;
            if (t0 >= q[s]) return "query tile";
            const int last = c[s] - q[s] + std::min(q[s], t0 + kTileQ) - 1;
            if (wk.kt0 >= wk.kt1 || wk.kt1 > last / kPrefillKT + 1) return "KV range";
            if (split && wk.kt1 - wk.kt0 > kPrefillMaxPiece) return "piece longer than the cap";
            if (wk.part != kNoPart && wk.kt1 - wk.kt0 < std::min(kPrefillMinPiece, last / kPrefillKT + 1))
                return "piece shorter than the minimum";
            for (int j = wk.kt0; j < wk.kt1; ++j) {
                const int pages = std::min(kPrefillKT / kPage, (c[s] - j * kPrefillKT + kPage - 1) / kPage);
                if (pages < 1 || j * (kPrefillKT / kPage) + pages > (c[s] + kPage - 1) / kPage) return "page read";
            }
            auto key = std::make_tuple(s, static_cast<int>(wk.qt), static_cast<int>(wk.slot));
            for (int j = wk.kt0; j < wk.kt1; ++j) cover[key].push_back(j);
            if (wk.part != kNoPart) {
                if (wk.part >= lp.n_part) return "partial slot";
                part_owner[wk.part]++;
                const long long blk = static_cast<long long>(wk.part) * hpc + hpc - 1;
                if ((blk + 1) * 4LL * kTileQ * 32 * 4 > static_cast<long long>(pf.o_bytes)) return "partial O bound";
                if ((blk + 1) * kTileQ * 2LL * 4 > static_cast<long long>(pf.ml_bytes)) return "partial m/l bound";
                pieces[key]++;
            }
        }
        for (int o : part_owner)
            if (o != 1) return "partial slot not owned by exactly one piece";
        for (const PrefillSplitUnit &su : lp.split_units) {
            if (su.part < 0 || su.part + su.n_splits > lp.n_part) return "merge entry parts";
            if (pieces[std::make_tuple(su.seq, su.qt, su.slot)] != su.n_splits) return "merge entry pieces";
        }
        if (lp.split_units.size() != pieces.size()) return "units with pieces but no merge entry";
    }
    size_t units = 0;
    for (int s = 0; s < n; ++s) {
        if (q[s] == 1) continue;
        for (int t = 0; t * kTileQ < q[s]; ++t) {
            const int nk = (c[s] - q[s] + std::min(q[s], (t + 1) * kTileQ) - 1) / kPrefillKT + 1;
            for (int sl = 0; sl < slots; ++sl) {
                ++units;
                auto it = cover.find(std::make_tuple(s, t, sl));
                if (it == cover.end()) return "unit without items";
                std::vector<int> v = it->second;
                std::sort(v.begin(), v.end());
                if (static_cast<int>(v.size()) != nk) return "unit coverage";
                for (int j = 0; j < nk; ++j)
                    if (v[j] != j) return "unit coverage";
            }
        }
    }
    if (cover.size() != units) return "items outside the step";
    *max_load = mx;
    *mean_load = ctas ? sum / ctas : 0;
    *n_launch = pf.launches.size();
    *n_ctas = ctas;
    *n_items = items;
    *n_part = pf.n_part;
    return "";
}

int main() {
    int sms, hq, hk, n;
    while (std::cin >> sms >> hq >> hk >> n) {
        std::vector<int32_t> q(n), c(n);
        for (auto &x : q) std::cin >> x;
        for (auto &x : c) std::cin >> x;
        for (int split = 1; split >= 0; --split) {
            double mx = 0, mean = 0;
            size_t nl = 0, nc = 0, ni = 0;
            long long np = 0;
            const std::string err = check(sms, hq, hk, q, c, split, &mx, &mean, &nl, &nc, &ni, &np);
            if (!err.empty())
                std::printf("FAIL %s%s\n", split ? "" : "(unsplit) ", err.c_str());
            else
                std::printf("ok %zu %zu %zu %lld %.1f %.2f\n", nl, nc, ni, np, mx, mean);
        }
    }
    return 0;
}
