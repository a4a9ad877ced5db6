// Host side of the C ABI: argument checks, TMA descriptors, the split of one
// attention step into prefill tiles and decode splits, and the launches.
#include <algorithm>
#include <chrono>
#include <cmath>
#include <cstring>
#include <memory>
#include <mutex>
#include <vector>

#include <cudaTypedefs.h>

#include "ppas_internal.h"

namespace ppas {

namespace {

// Throughput model behind the SMs the prefill kernel leaves to the decode
// launch (measured on GB300): one item's KV tile (two q-heads x 128 queries x
// 128 keys) takes about 2.06 us of one SM; next to a running prefill kernel
// the decode kernel streams 65-80 GB/s per SM (the upper figure is used, so
// that a wrong estimate leaves decode rows rather than prefill items as the
// tail: the slower side of the balance), and at most kDecodeBytesPerUs on
// the GPU.
constexpr double kPrefillTileUs = 2.06;
constexpr double kDecodeBytesPerSmUs = 8.0e4;
constexpr double kDecodeBytesPerUs = 4.35e6;

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    });
    return fn;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// A side stream per device for the decode launch of a mixed step: the
// prefill kernel goes first on the caller's stream, the decode kernel is
// forked after it, so decode CTAs fill SMs as prefill CTAs retire.  Events
// join it back before the call returns.  The mutex serialises the enqueue
// (the events are shared per device).
struct SideStream {
    cudaStream_t stream = nullptr;
    cudaEvent_t fork = nullptr, join = nullptr;
};
std::mutex g_side_mutex;
SideStream g_side[64];

SideStream *side_stream() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    SideStream &ss = g_side[dev];
    if (!ss.stream && cudaStreamCreateWithFlags(&ss.stream, cudaStreamNonBlocking) != cudaSuccess) {
        ss.stream = nullptr;
        return nullptr;
    }
    if (!ss.fork && cudaEventCreateWithFlags(&ss.fork, cudaEventDisableTiming) != cudaSuccess) {
        ss.fork = nullptr;
        return nullptr;
    }
    if (!ss.join && cudaEventCreateWithFlags(&ss.join, cudaEventDisableTiming) != cudaSuccess) {
        ss.join = nullptr;
        return nullptr;
    }
    return &ss;
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// Tags of the decode launches' split tickets: never 0 and larger for every
// launch of the process (the kernel relies on the order: a ticket word
// holding a smaller tag is stale).  47 bits, so (tag << 16) | arrivals stays
// below 2^63; the start is drawn from the clock so that tickets another
// process left in recycled memory rarely match.
unsigned long long next_launch_tag() {
    static std::atomic<unsigned long long> next{
        1 + ((static_cast<unsigned long long>(std::chrono::steady_clock::now().time_since_epoch().count()) *
              0x9E3779B97F4A7C15ull) >> 24)};
    return next.fetch_add(1, std::memory_order_relaxed) & ((1ull << 47) - 1);
}

}  // namespace

cudaError_t prepare_current_device() {
    {
        std::lock_guard<std::mutex> lock(g_side_mutex);
        if (!side_stream()) return cudaErrorInitializationError;
    }
    cudaError_t e = prepare_prefill();
    if (e == cudaSuccess) e = prepare_decode();
    if (e == cudaSuccess) e = prepare_mixed();
    if (e == cudaSuccess) decode_cluster_caps();  // the occupancy queries, once per device
    return e;
}

int32_t device_sm_count() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return kDefaultPlanSms;
    static std::atomic<int> cached[64] = {};
    if (dev >= 0 && dev < 64) {
        const int c = cached[dev].load(std::memory_order_relaxed);
        if (c) return c;
    }
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = kDefaultPlanSms;
    if (dev >= 0 && dev < 64) cached[dev].store(n, std::memory_order_relaxed);
    return n;
}

int32_t plan_sms() { return std::max(1, std::min(device_sm_count(), kMaxPrefillCtas)); }

// K or V cache [num_blocks, n_kv_heads, 16, 128] bf16 viewed as rows of 128
// elements; one TMA box = 16 rows (one page) x 64 columns.
bool encode_kv_map(CUtensorMap *map, const void *cache, int32_t num_blocks, int32_t n_kv_heads) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(kHeadDim),
                          static_cast<cuuint64_t>(num_blocks) * n_kv_heads * kPage};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(kRowBytes)};
    cuuint32_t box[2] = {64, static_cast<cuuint32_t>(kPage)};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(cache), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_bf16_2d(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer, uint32_t box_inner,
                    uint32_t box_outer) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {inner * 2};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Q [total_q, n_q_heads, 128] bf16: dims (column, head, token); one box =
// 128 tokens of one head x 64 columns.
bool encode_q_map(CUtensorMap *map, const void *q, int32_t total_q, int32_t n_q_heads) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(n_q_heads),
                          static_cast<cuuint64_t>(total_q)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(kRowBytes),
                             static_cast<cuuint64_t>(kRowBytes) * n_q_heads};
    cuuint32_t box[3] = {64, 1, static_cast<cuuint32_t>(kTileQ)};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(q), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

DecodePlan plan_decode(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                       int32_t n_kv_heads, int32_t num_sms, const DecodeClusterCaps &caps) {
    DecodePlan d;
    int64_t total_pages = 0;  // over (row, kv-head) pairs
    for (int32_t s = 0; s < n_seqs; ++s)
        if (q_lens[s] == 1) {
            d.rows.push_back(s);
            total_pages += static_cast<int64_t>((ctx_lens[s] + kPage - 1) / kPage) * n_kv_heads;
        }
    if (d.rows.empty()) return d;
    const size_t nr = d.rows.size();
    // Splits of every row for target_ctas CTAs in clusters of c: each
    // (row, kv-head) gets a share of them in proportion to its pages
    // (largest remainders first), so one step fills one wave; with c > 1
    // the shares are whole numbers of clusters.  False when c does not fit.
    auto splits = [&](int64_t target_ctas, int32_t c, std::vector<int32_t> &ns_out, std::vector<int32_t> &pps_out) {
        std::vector<int64_t> shares(nr);
        const int64_t per_head = std::max<int64_t>(1, target_ctas / n_kv_heads);
        int64_t given = 0;
        std::vector<std::pair<int64_t, size_t>> rem(nr);  // (remainder, row)
        for (size_t k = 0; k < nr; ++k) {
            const int64_t pages = (ctx_lens[d.rows[k]] + kPage - 1) / kPage;
            const int64_t num = per_head * pages * n_kv_heads;  // share = num / total_pages
            shares[k] = num / total_pages;
            rem[k] = {num % total_pages, k};
            given += shares[k];
        }
        std::stable_sort(rem.begin(), rem.end(),
                         [](const std::pair<int64_t, size_t> &a, const std::pair<int64_t, size_t> &b) {
                             return a.first > b.first;
                         });
        for (size_t k = 0; k < nr && given < per_head; ++k, ++given) ++shares[rem[k].second];
        ns_out.assign(nr, 0);
        pps_out.assign(nr, 0);
        for (size_t k = 0; k < nr; ++k) {
            const int64_t pages = (ctx_lens[d.rows[k]] + kPage - 1) / kPage;
            const int64_t share = c > 1 ? shares[k] / c * c : std::max<int64_t>(shares[k], 1);
            if (share < 1) return false;
            // even splits (the last one short by fewer than n_splits pages)
            int64_t pps = (pages + share - 1) / share;
            pps = std::max<int64_t>(pps, kDecodeMinPagesPerSplit);
            pps = std::min<int64_t>(pps, kDecodeMaxPagesPerSplit);
            int64_t ns = (pages + pps - 1) / pps;
            if (c > 1) {
                // a whole number of clusters; at most c - 1 of the splits are
                // empty (past the row's pages), and the share is not exceeded
                if (ns > share || ns <= share - c) return false;
                ns = share;
            }
            ns_out[k] = static_cast<int32_t>(ns);
            pps_out[k] = static_cast<int32_t>(pps);
        }
        return true;
    };
    std::vector<int32_t> ns1, pps1;
    splits(std::max(1, num_sms), 1, ns1, pps1);
    d.n_splits = ns1;
    d.pages_per_split = pps1;
    // Clusters of 4, for steps of decode rows only (a mixed launch keeps its
    // grid free of them), when that plan still fills 15/16 of the SMs and
    // streams at most 6 % more pages in its longest split than the plan
    // without clusters.  The split merge's last CTA then reads a quarter of
    // the partials, which is what bounds steps of a few rows.  (Clusters of
    // 2, on a 4-row step, measured no faster and are not used.)
    if (static_cast<int32_t>(nr) == n_seqs) {
        int64_t max1 = 0;
        for (size_t k = 0; k < nr; ++k) max1 = std::max<int64_t>(max1, pps1[k]);
        const int32_t cs[1] = {4};
        const int32_t cap[1] = {caps.ctas4};
        for (int i = 0; i < 1; ++i) {
            if (cap[i] < cs[i] || cap[i] > num_sms) continue;
            std::vector<int32_t> ns, pps;
            if (!splits(cap[i], cs[i], ns, pps)) continue;
            int64_t ctas = 0, maxc = 0;
            for (size_t k = 0; k < nr; ++k) {
                ctas += static_cast<int64_t>(ns[k]) * n_kv_heads;
                maxc = std::max<int64_t>(maxc, pps[k]);
            }
            if (ctas > cap[i] || ctas * 16 < static_cast<int64_t>(num_sms) * 15 || maxc * 100 > max1 * 106) continue;
            d.n_splits = ns;
            d.pages_per_split = pps;
            d.cluster = cs[i];
            break;
        }
    }
    for (size_t k = 0; k < nr; ++k) {
        d.n_part += d.n_splits[k] / d.cluster;
        d.n_ctas += static_cast<int64_t>(d.n_splits[k]) * n_kv_heads;
    }
    d.ml_bytes = align256(static_cast<size_t>(d.n_part) * n_q_heads * 2 * sizeof(float));
    d.o_bytes = align256(static_cast<size_t>(d.n_part) * n_q_heads * kHeadDim * sizeof(float));
    d.counter_bytes = align256(d.rows.size() * n_kv_heads * sizeof(unsigned long long));
    return d;
}

PrefillPlan plan_prefill(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                         int32_t n_kv_heads, bool allow_split, int32_t n_ctas, int32_t max_work) {
    PrefillPlan pf;
    max_work = std::max(1, std::min(max_work, kMaxPrefillWork));
    const int32_t g = n_q_heads / n_kv_heads;
    pf.heads_per_cta = g >= 2 ? 2 : 1;
    pf.slots = n_q_heads / pf.heads_per_cta;
    n_ctas = std::max(1, std::min(n_ctas, kMaxPrefillCtas));
    struct Unit {
        int32_t seq, qt, slot, n_kt;
    };
    std::vector<Unit> units;
    for (int32_t s = 0; s < n_seqs; ++s) {
        if (q_lens[s] == 1) continue;
        const int32_t prefix = ctx_lens[s] - q_lens[s];
        const int32_t n_qt = (q_lens[s] + kTileQ - 1) / kTileQ;
        for (int32_t t = 0; t < n_qt; ++t) {
            const int32_t last = prefix + std::min(q_lens[s], (t + 1) * kTileQ) - 1;
            for (int32_t sl = 0; sl < pf.slots; ++sl) units.push_back({s, t, sl, last / kPrefillKT + 1});
        }
    }
    if (units.empty()) return pf;
    // longest first
    std::stable_sort(units.begin(), units.end(), [](const Unit &a, const Unit &b) { return a.n_kt > b.n_kt; });

    size_t u0 = 0;
    while (u0 < units.size()) {
        // a launch takes consecutive units while its tables have room (a unit
        // is at least ceil(n_kt / kPrefillMaxPiece) items, and every CTA
        // boundary adds at most one more)
        PrefillLaunchPlan lp;
        std::vector<int32_t> local(n_seqs, -1);
        size_t u1 = u0;
        int64_t min_items = 0;
        bool needs_cut = false;  // a unit longer than a piece may be
        for (; u1 < units.size(); ++u1) {
            const bool new_seq = local[units[u1].seq] < 0;
            const int64_t pieces = (units[u1].n_kt + kPrefillMaxPiece - 1) / kPrefillMaxPiece;
            if (min_items + pieces + n_ctas > max_work) break;
            if (new_seq && lp.seqs.size() == static_cast<size_t>(kMaxPrefillSeqs)) break;
            if (new_seq) {
                local[units[u1].seq] = static_cast<int32_t>(lp.seqs.size());
                lp.seqs.push_back(units[u1].seq);
            }
            min_items += pieces;
            needs_cut = needs_cut || units[u1].n_kt > kPrefillMaxPiece;
        }
        int64_t total = 0, tiles = 0;
        for (size_t u = u0; u < u1; ++u) {
            total += units[u].n_kt + kPrefillItemCost;
            tiles += units[u].n_kt;
        }
        auto item = [&](const Unit &u, int32_t kt0, int32_t kt1) {
            return PrefillWork{static_cast<uint16_t>(u.qt), static_cast<uint8_t>(local[u.seq]),
                               static_cast<uint8_t>(u.slot), static_cast<uint16_t>(kt0), static_cast<uint16_t>(kt1),
                               kNoPart, 0};
        };
        // whole units, longest first, each to the least loaded CTA
        const int32_t nc_whole = static_cast<int32_t>(std::min<int64_t>(n_ctas, u1 - u0));
        std::vector<std::vector<PrefillWork>> whole(nc_whole);
        int64_t whole_span = 0;
        {
            std::vector<std::pair<int64_t, int32_t>> heap;  // (load, cta), min-heap
            for (int32_t c = 0; c < nc_whole; ++c) heap.push_back({0, c});
            auto later = [](const std::pair<int64_t, int32_t> &a, const std::pair<int64_t, int32_t> &b) {
                return a.first != b.first ? a.first > b.first : a.second > b.second;
            };
            std::make_heap(heap.begin(), heap.end(), later);
            for (size_t u = u0; u < u1; ++u) {
                std::pop_heap(heap.begin(), heap.end(), later);
                auto &top = heap.back();
                whole[top.second].push_back(item(units[u], 0, units[u].n_kt));
                top.first += units[u].n_kt + kPrefillItemCost;
                whole_span = std::max(whole_span, top.first);
                std::push_heap(heap.begin(), heap.end(), later);
            }
        }
        // cutting units evens the CTAs out at the cost of partials and a
        // merge; it is taken when it shortens the launch by more than that
        const int32_t nc = static_cast<int32_t>(std::min<int64_t>(n_ctas, tiles));
        std::vector<std::vector<PrefillWork>> per_cta;
        if (allow_split) {
            // stream-K with an even target: the units laid end to end in
            // order are filled into CTAs up to a load T (tiles plus an item's
            // cost per item), a unit cut where a CTA reaches T (no piece
            // shorter than kPrefillMinPiece); T is the smallest load whose
            // fill needs at most nc CTAs
            auto fill = [&](int64_t T, std::vector<std::vector<std::pair<int32_t, PrefillWork>>> *out) -> int32_t {
                int32_t cta = 0;
                int64_t load = 0;
                for (size_t u = u0; u < u1; ++u) {
                    const Unit &un = units[u];
                    int32_t a = 0;
                    while (a < un.n_kt) {
                        const int32_t left = un.n_kt - a;
                        const int64_t room = T - load - kPrefillItemCost;
                        int32_t take;
                        if (left <= room) {
                            take = left;
                        } else if (room >= kPrefillMaxPiece) {
                            take = left;  // capped below, the CTA still has room
                        } else {
                            int64_t t = std::max<int64_t>(room, 0);
                            if (left - t < kPrefillMinPiece) t = left - kPrefillMinPiece;
                            if (t >= kPrefillMinPiece) {
                                take = static_cast<int32_t>(t);
                            } else if (load == 0) {
                                // an empty CTA too small for a legal cut: the
                                // remainder goes whole (or leaves a legal piece)
                                take = left >= 2 * kPrefillMinPiece ? kPrefillMinPiece : left;
                            } else {
                                ++cta;  // nothing of this unit fits here
                                load = 0;
                                continue;
                            }
                        }
                        // no piece longer than kPrefillMaxPiece (nor a remainder
                        // shorter than kPrefillMinPiece after one)
                        bool capped = false;
                        if (take > kPrefillMaxPiece) {
                            take = kPrefillMaxPiece;
                            if (left - take < kPrefillMinPiece) take = left - kPrefillMinPiece;
                            capped = true;
                        }
                        if (out) {
                            if (static_cast<size_t>(cta) >= out->size()) out->resize(cta + 1);
                            (*out)[cta].push_back({static_cast<int32_t>(u - u0), item(un, a, a + take)});
                        }
                        load += take + kPrefillItemCost;
                        a += take;
                        if (a < un.n_kt && !capped) {  // the unit goes on in the next CTA
                            ++cta;
                            load = 0;
                        }
                    }
                }
                return cta + (load > 0 ? 1 : 0);
            };
            int64_t lo = (total + nc - 1) / nc, hi = total;
            while (lo < hi) {
                const int64_t mid = lo + (hi - lo) / 2;
                if (fill(mid, nullptr) <= nc) hi = mid; else lo = mid + 1;
            }
            std::vector<std::vector<std::pair<int32_t, PrefillWork>>> filled;
            fill(lo, &filled);
            // pieces of a unit get consecutive partial slots
            std::vector<int32_t> n_pieces(u1 - u0, 0);
            for (const auto &v : filled)
                for (const auto &pc : v) ++n_pieces[pc.first];
            std::vector<int32_t> first_part(u1 - u0, -1), next_part(u1 - u0, 0);
            for (size_t u = u0; u < u1; ++u) {
                const int32_t k = static_cast<int32_t>(u - u0);
                if (n_pieces[k] > 1) {
                    first_part[k] = static_cast<int32_t>(lp.n_part);
                    lp.split_units.push_back({units[u].seq, units[u].qt, units[u].slot, n_pieces[k], lp.n_part});
                    lp.n_part += n_pieces[k];
                }
            }
            per_cta.resize(filled.size());
            for (size_t c = 0; c < filled.size(); ++c)
                for (auto &pc : filled[c]) {
                    if (first_part[pc.first] >= 0)
                        pc.second.part = static_cast<uint16_t>(first_part[pc.first] + next_part[pc.first]++);
                    per_cta[c].push_back(pc.second);
                }
            int64_t cut_span = 0;
            for (const auto &v : per_cta) {
                int64_t load = 0;
                for (const PrefillWork &w : v) load += w.kt1 - w.kt0 + kPrefillItemCost;
                cut_span = std::max(cut_span, load);
            }
            if (lp.n_part == 0 || (!needs_cut && cut_span + kPrefillMergeCost >= whole_span)) {
                per_cta = std::move(whole);  // not worth the partials
                lp.split_units.clear();
                lp.n_part = 0;
            }
        } else {
            per_cta = std::move(whole);
        }
        lp.cta_begin.push_back(0);
        for (size_t c = 0; c < per_cta.size(); ++c) {
            if (per_cta[c].empty()) continue;  // (a CTA with nothing is left out)
            lp.work.insert(lp.work.end(), per_cta[c].begin(), per_cta[c].end());
            lp.cta_begin.push_back(static_cast<uint16_t>(lp.work.size()));
        }
        pf.n_part = std::max<int64_t>(pf.n_part, lp.n_part);
        pf.launches.push_back(std::move(lp));
        u0 = u1;
    }
    const size_t per_part = static_cast<size_t>(pf.heads_per_cta) * kTileQ;
    pf.o_bytes = align256(static_cast<size_t>(pf.n_part) * per_part * kHeadDim * sizeof(float));
    pf.ml_bytes = align256(static_cast<size_t>(pf.n_part) * per_part * 2 * sizeof(float));
    return pf;
}

int32_t decode_reserve_sms(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                           int32_t n_kv_heads, int32_t num_sms) {
    const int32_t hpc = n_q_heads / n_kv_heads >= 2 ? 2 : 1;
    const int64_t slots = n_q_heads / hpc;
    double units = 0.0, bytes = 0.0;  // prefill KV tiles x head slots, decode K/V bytes
    for (int32_t s = 0; s < n_seqs; ++s) {
        if (q_lens[s] == 1) {
            bytes += static_cast<double>((ctx_lens[s] + kPage - 1) / kPage) * kPageBytes * 2 * n_kv_heads;
            continue;
        }
        const int32_t prefix = ctx_lens[s] - q_lens[s];
        const int32_t n_qt = (q_lens[s] + kTileQ - 1) / kTileQ;
        for (int32_t t = 0; t < n_qt; ++t) {
            const int32_t last = prefix + std::min(q_lens[s], (t + 1) * kTileQ) - 1;
            units += static_cast<double>(last / kPrefillKT + 1) * slots;
        }
    }
    if (units == 0.0 || bytes == 0.0) return 0;
    // the decode launch streams on k SMs while the prefill kernel runs on
    // the rest; the smallest k that finishes the decode rows by the time the
    // prefill items are done:  k r T(k) >= bytes,  T(k) = units tau / (S - k)
    const double sm_time = units * kPrefillTileUs;
    int32_t k = static_cast<int32_t>(std::ceil(bytes * num_sms / (kDecodeBytesPerSmUs * sm_time + bytes)));
    k = std::min(k, static_cast<int32_t>(kDecodeBytesPerUs / kDecodeBytesPerSmUs));
    return std::max(0, std::min(k, num_sms / 2));
}

size_t workspace_min_size(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                          int32_t n_kv_heads) {
    if (n_seqs <= 0 || !q_lens || !ctx_lens || n_q_heads < 1 || n_kv_heads < 1 || n_q_heads % n_kv_heads) return 0;
    for (int32_t s = 0; s < n_seqs; ++s)
        if (q_lens[s] < 1 || ctx_lens[s] < q_lens[s]) return 0;
    return plan_decode(n_seqs, q_lens, ctx_lens, n_q_heads, n_kv_heads, plan_sms(), decode_cluster_caps())
        .total_bytes();
}


// The plan of one step, shared by the workspace query, the launch count and
// the step itself so that the three always agree: the decode splits, the
// SMs left to the prefill kernel, and the prefill launches (with stream-K
// cuts when the workspace holds their partials).  A step with both kinds of
// rows whose prefill items fit one mixed launch runs as that single launch.
StepPlan plan_step(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens, int32_t n_q_heads,
                   int32_t n_kv_heads, size_t workspace_bytes) {
    StepPlan sp;
    const int32_t sms = plan_sms();
    sp.dp = plan_decode(n_seqs, q_lens, ctx_lens, n_q_heads, n_kv_heads, sms, decode_cluster_caps());
    sp.n_ctas = sms - decode_reserve_sms(n_seqs, q_lens, ctx_lens, n_q_heads, n_kv_heads, sms);
    const bool may_mix = !sp.dp.rows.empty() && sp.dp.rows.size() <= static_cast<size_t>(kMaxMixedRows);
    auto plan = [&](int32_t max_work) {
        PrefillPlan pf = plan_prefill(n_seqs, q_lens, ctx_lens, n_q_heads, n_kv_heads, true, sp.n_ctas, max_work);
        // a workspace too small for the pieces' partials runs every unit whole
        if (workspace_bytes < sp.dp.total_bytes() + pf.total_bytes())
            pf = plan_prefill(n_seqs, q_lens, ctx_lens, n_q_heads, n_kv_heads, false, sp.n_ctas, max_work);
        return pf;
    };
    sp.pf = plan(may_mix ? kMaxMixedWork : kMaxPrefillWork);
    sp.mixed = may_mix && sp.pf.launches.size() == 1;
    if (may_mix && !sp.mixed) sp.pf = plan(kMaxPrefillWork);  // several prefill launches anyway
    return sp;
}

namespace {

// The last few plans made on this thread: every layer of a scheduler
// iteration has the same step, so a serving loop plans it once per
// iteration instead of once per layer (the stream-K search of a step like
// MBT 2k takes ~70 us of host time).
struct CachedPlan {
    int32_t n = -1, hq = 0, hk = 0, sms = 0, clusters4 = 0;  // the device's SMs and cluster capacity
    size_t ws = 0;
    std::vector<int32_t> q, c;
    std::shared_ptr<const StepPlan> plan;
};
constexpr int kPlanCache = 4;
thread_local CachedPlan t_plans[kPlanCache];
thread_local int t_plan_next = 0;

}  // namespace

std::shared_ptr<const StepPlan> plan_step_cached(int32_t n_seqs, const int32_t *q_lens, const int32_t *ctx_lens,
                                                 int32_t n_q_heads, int32_t n_kv_heads, size_t workspace_bytes) {
    const int32_t sms = plan_sms();
    const int32_t clusters4 = decode_cluster_caps().ctas4;
    for (const CachedPlan &e : t_plans)
        if (e.plan && e.n == n_seqs && e.hq == n_q_heads && e.hk == n_kv_heads && e.sms == sms &&
            e.clusters4 == clusters4 && e.ws == workspace_bytes && std::equal(q_lens, q_lens + n_seqs, e.q.begin()) &&
            std::equal(ctx_lens, ctx_lens + n_seqs, e.c.begin()))
            return e.plan;
    auto sp = std::make_shared<const StepPlan>(
        plan_step(n_seqs, q_lens, ctx_lens, n_q_heads, n_kv_heads, workspace_bytes));
    CachedPlan &e = t_plans[t_plan_next];
    t_plan_next = (t_plan_next + 1) % kPlanCache;
    e.n = n_seqs;
    e.hq = n_q_heads;
    e.hk = n_kv_heads;
    e.sms = sms;
    e.clusters4 = clusters4;
    e.ws = workspace_bytes;
    e.q.assign(q_lens, q_lens + n_seqs);
    e.c.assign(ctx_lens, ctx_lens + n_seqs);
    e.plan = sp;
    return sp;
}

}  // namespace ppas

using namespace ppas;

namespace {

ppas_status check_step(const void *q, const void *k_cache, const void *v_cache, int32_t num_blocks,
                       const int32_t *d_block_tables, int32_t max_blocks_per_seq, const int32_t *h_q_lens,
                       const int32_t *h_ctx_lens, int32_t n_seqs, int32_t n_q_heads, int32_t n_kv_heads,
                       int32_t head_dim, const void *out, int64_t *total_q) {
    if (n_seqs < 0) return PPAS_ERR_INVALID_ARG;
    if (n_seqs > 0 && (!h_q_lens || !h_ctx_lens)) return PPAS_ERR_INVALID_ARG;
    if (n_q_heads < 1 || n_kv_heads < 1 || head_dim < 1) return PPAS_ERR_INVALID_ARG;
    if (head_dim != kHeadDim) return PPAS_ERR_UNSUPPORTED;
    if (n_q_heads % n_kv_heads != 0) return PPAS_ERR_INVALID_ARG;
    const int32_t g = n_q_heads / n_kv_heads;
    if (g != 1 && g != 2 && g != 4 && g != 8) return PPAS_ERR_UNSUPPORTED;
    if (n_q_heads / (g >= 2 ? 2 : 1) > 256) return PPAS_ERR_UNSUPPORTED;  // head slots of the prefill items
    int64_t tq = 0;
    for (int32_t s = 0; s < n_seqs; ++s) {
        if (h_q_lens[s] < 1 || h_ctx_lens[s] < h_q_lens[s]) return PPAS_ERR_INVALID_ARG;
        // KV tile indices of the prefill items are 16-bit
        if (h_q_lens[s] > 1 && h_ctx_lens[s] > 65535 * kPrefillKT) return PPAS_ERR_UNSUPPORTED;
        if (h_q_lens[s] == 1 && h_ctx_lens[s] > kMaxDecodeCtx) return PPAS_ERR_UNSUPPORTED;
        if (static_cast<int64_t>(h_ctx_lens[s]) > static_cast<int64_t>(max_blocks_per_seq) * kPage)
            return PPAS_ERR_INVALID_ARG;
        tq += h_q_lens[s];
    }
    *total_q = tq;
    if (n_seqs == 0) return PPAS_OK;
    if (!q || !k_cache || !v_cache || !d_block_tables || !out) return PPAS_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(out))
        return PPAS_ERR_INVALID_ARG;
    if (num_blocks < 1 || max_blocks_per_seq < 1) return PPAS_ERR_INVALID_ARG;
    if (tq * n_q_heads > INT32_MAX || static_cast<int64_t>(num_blocks) * n_kv_heads * kPage > INT32_MAX)
        return PPAS_ERR_UNSUPPORTED;
    return PPAS_OK;
}

}  // namespace

extern "C" const char *ppas_status_string(ppas_status s) {
    switch (s) {
        case PPAS_OK: return "ok";
        case PPAS_ERR_INVALID_ARG: return "invalid argument";
        case PPAS_ERR_CAPACITY: return "capacity exceeded";
        case PPAS_ERR_OUT_OF_BLOCKS: return "out of KV blocks";
        case PPAS_ERR_UNSUPPORTED: return "unsupported shape";
        case PPAS_ERR_CUDA: return "CUDA error";
        default: return "unknown status";
    }
}

extern "C" int32_t ppas_abi_version(void) { return 1; }

extern "C" ppas_status ppas_debug_wait_timeout(int32_t *d_err_flag, uint32_t limit_us, void *stream) {
    if (!d_err_flag || limit_us < 1 || limit_us > 2000000) return PPAS_ERR_INVALID_ARG;
    return launch_wait_timeout(d_err_flag, static_cast<unsigned long long>(limit_us) * 1000ull,
                               static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? PPAS_OK
               : PPAS_ERR_CUDA;
}

extern "C" ppas_status ppas_kv_append(const void *k_new, const void *v_new, const int32_t *d_slot_mapping,
                                      int32_t n_tokens, void *k_cache, void *v_cache, int32_t num_blocks,
                                      int32_t n_kv_heads, int32_t head_dim, int32_t *d_err_flag, void *stream) {
    if (n_tokens < 0 || n_kv_heads < 1 || head_dim < 8 || head_dim % 8 != 0 || num_blocks < 1)
        return PPAS_ERR_INVALID_ARG;
    if (n_tokens == 0) return PPAS_OK;
    if (!k_new || !v_new || !d_slot_mapping || !k_cache || !v_cache) return PPAS_ERR_INVALID_ARG;
    if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(k_cache) || !aligned16(v_cache))
        return PPAS_ERR_INVALID_ARG;
    if (static_cast<int64_t>(n_tokens) * n_kv_heads * (head_dim / 8) >= (int64_t{1} << 31))
        return PPAS_ERR_UNSUPPORTED;
    cudaError_t e = launch_kv_append(k_new, v_new, d_slot_mapping, n_tokens, k_cache, v_cache, num_blocks,
                                     n_kv_heads, head_dim, d_err_flag, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? PPAS_OK : PPAS_ERR_CUDA;
}

extern "C" size_t ppas_attention_workspace_size(int32_t n_seqs, const int32_t *h_q_lens, const int32_t *h_ctx_lens,
                                                int32_t n_q_heads, int32_t n_kv_heads) {
    if (n_seqs <= 0 || !h_q_lens || !h_ctx_lens || n_q_heads < 1 || n_kv_heads < 1 || n_q_heads % n_kv_heads)
        return 0;
    for (int32_t s = 0; s < n_seqs; ++s)
        if (h_q_lens[s] < 1 || h_ctx_lens[s] < h_q_lens[s]) return 0;
    return plan_step_cached(n_seqs, h_q_lens, h_ctx_lens, n_q_heads, n_kv_heads, SIZE_MAX)->total_bytes();
}

extern "C" int32_t ppas_attention_kernel_count(int32_t n_seqs, const int32_t *h_q_lens, const int32_t *h_ctx_lens,
                                               int32_t n_q_heads, int32_t n_kv_heads, size_t workspace_bytes) {
    if (n_seqs < 0 || (n_seqs > 0 && (!h_q_lens || !h_ctx_lens))) return -1;
    if (n_q_heads < 1 || n_kv_heads < 1 || n_q_heads % n_kv_heads) return -1;
    const int32_t g = n_q_heads / n_kv_heads;
    if (g != 1 && g != 2 && g != 4 && g != 8) return -1;
    for (int32_t s = 0; s < n_seqs; ++s) {
        if (h_q_lens[s] < 1 || h_ctx_lens[s] < h_q_lens[s]) return -1;
        if (h_q_lens[s] > 1 && h_ctx_lens[s] > 65535 * kPrefillKT) return -1;
        if (h_q_lens[s] == 1 && h_ctx_lens[s] > kMaxDecodeCtx) return -1;
    }
    if (n_seqs == 0) return 0;
    // the same plan as ppas_attention_step
    const auto spp = plan_step_cached(n_seqs, h_q_lens, h_ctx_lens, n_q_heads, n_kv_heads, workspace_bytes);
    const StepPlan &sp = *spp;
    // the prefill (or mixed) launches, each followed by its merge launches
    // when its plan cuts units, and the decode launches unless mixed in
    int32_t n = sp.mixed ? 0 : static_cast<int32_t>((sp.dp.rows.size() + kMaxDecodeRows - 1) / kMaxDecodeRows);
    for (const PrefillLaunchPlan &lp : sp.pf.launches)
        n += 1 + static_cast<int32_t>((lp.split_units.size() + kMaxMergeUnits - 1) / kMaxMergeUnits);
    return n;
}

namespace {

// The prefill launch parameters of one planned launch (prefill or mixed).
template <class P>
void fill_prefill_params(P &pp, const PrefillPlan &pf, const PrefillLaunchPlan &lp, const std::vector<int32_t> &q_start,
                         const int32_t *h_q_lens, const int32_t *h_ctx_lens, uint8_t *pws) {
    for (size_t i = 0; i < lp.seqs.size(); ++i) {
        const int32_t sq = lp.seqs[i];
        pp.seqs[i] = {q_start[sq], h_q_lens[sq], h_ctx_lens[sq], sq};
    }
    std::memcpy(pp.work, lp.work.data(), lp.work.size() * sizeof(PrefillWork));
    std::memcpy(pp.cta_begin, lp.cta_begin.data(), lp.cta_begin.size() * sizeof(uint16_t));
    pp.n_ctas = static_cast<int32_t>(lp.cta_begin.size()) - 1;
    if (pf.n_part > 0) {
        pp.part_o = reinterpret_cast<float *>(pws);
        pp.part_ml = reinterpret_cast<float *>(pws + pf.o_bytes);
    }
}

// The merge launches of one prefill launch's cut units (none when it cuts none).
bool launch_merges(const PrefillPlan &pf, const PrefillLaunchPlan &lp, const std::vector<int32_t> &q_start,
                   const int32_t *h_q_lens, const float *part_o, const float *part_ml, void *out, int32_t out_fp32,
                   int32_t n_q_heads, cudaStream_t st) {
    static thread_local MergeParams mp;
    for (size_t i0 = 0; i0 < lp.split_units.size(); i0 += kMaxMergeUnits) {
        const size_t i1 = std::min(lp.split_units.size(), i0 + kMaxMergeUnits);
        mp.part_o = part_o;
        mp.part_ml = part_ml;
        mp.out = out;
        mp.out_fp32 = out_fp32;
        mp.n_q_heads = n_q_heads;
        mp.heads_per_cta = pf.heads_per_cta;
        mp.n_units = static_cast<int32_t>(i1 - i0);
        for (size_t i = i0; i < i1; ++i) {
            const PrefillSplitUnit &su = lp.split_units[i];
            MergeUnit &mu = mp.units[i - i0];
            mu.out_row0 = q_start[su.seq] + su.qt * kTileQ;
            mu.part = su.part;
            mu.rows_valid = static_cast<uint16_t>(std::min(kTileQ, h_q_lens[su.seq] - su.qt * kTileQ));
            mu.n_splits = static_cast<uint16_t>(su.n_splits);
            mu.head0 = static_cast<uint16_t>(su.slot * pf.heads_per_cta);
            mu.pad = 0;
        }
        if (launch_prefill_merge(mp, st) != cudaSuccess) return false;
    }
    return true;
}

}  // namespace

extern "C" ppas_status ppas_attention_step(const void *q, const void *k_cache, const void *v_cache,
                                           int32_t num_blocks, const int32_t *d_block_tables,
                                           int32_t max_blocks_per_seq, const int32_t *h_q_lens,
                                           const int32_t *h_ctx_lens, int32_t n_seqs, int32_t n_q_heads,
                                           int32_t n_kv_heads, int32_t head_dim, float scale, void *out,
                                           int32_t out_is_fp32, void *workspace, size_t workspace_bytes,
                                           int32_t *d_err_flag, void *stream) {
    int64_t total_q = 0;
    ppas_status st = check_step(q, k_cache, v_cache, num_blocks, d_block_tables, max_blocks_per_seq, h_q_lens,
                                h_ctx_lens, n_seqs, n_q_heads, n_kv_heads, head_dim, out, &total_q);
    if (st != PPAS_OK || n_seqs == 0) return st;
    if (!(scale > 0.f) || !std::isfinite(scale)) return PPAS_ERR_INVALID_ARG;
    const cudaStream_t cs = static_cast<cudaStream_t>(stream);
    const int32_t g = n_q_heads / n_kv_heads;
    const float scale_log2 = scale * 1.4426950408889634f;

    // packed row offsets
    std::vector<int32_t> q_start(n_seqs);
    {
        int32_t acc = 0;
        for (int32_t s = 0; s < n_seqs; ++s) {
            q_start[s] = acc;
            acc += h_q_lens[s];
        }
    }

    const auto spp = plan_step_cached(n_seqs, h_q_lens, h_ctx_lens, n_q_heads, n_kv_heads, workspace_bytes);
    const StepPlan &sp = *spp;
    const DecodePlan &dp = sp.dp;
    const PrefillPlan &pf = sp.pf;
    const size_t need = sp.total_bytes();
    if (need > 0) {
        if (!workspace || workspace_bytes < need) return PPAS_ERR_CAPACITY;
        if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return PPAS_ERR_INVALID_ARG;
    }

    CUtensorMap tm_k, tm_v;
    if (!encode_kv_map(&tm_k, k_cache, num_blocks, n_kv_heads) ||
        !encode_kv_map(&tm_v, v_cache, num_blocks, n_kv_heads))
        return PPAS_ERR_CUDA;

    uint8_t *const ws = static_cast<uint8_t *>(workspace);
    // the decode rows [b0, b1) of the plan as launch parameters
    auto fill_decode = [&](auto &dprm, size_t b0, size_t b1, int32_t part_base) {
        dprm.q = static_cast<const __nv_bfloat16 *>(q);
        dprm.block_tables = d_block_tables;
        dprm.table_stride = max_blocks_per_seq;
        dprm.num_blocks = num_blocks;
        dprm.out = out;
        dprm.out_fp32 = out_is_fp32 ? 1 : 0;
        dprm.n_q_heads = n_q_heads;
        dprm.n_kv_heads = n_kv_heads;
        dprm.group = g;
        dprm.scale_log2 = scale_log2;
        dprm.part_ml = reinterpret_cast<float *>(ws);
        dprm.part_o = reinterpret_cast<float *>(ws + dp.ml_bytes);
        dprm.err = d_err_flag;
        dprm.n_rows = static_cast<int32_t>(b1 - b0);
        dprm.counters = reinterpret_cast<unsigned long long *>(ws + dp.ml_bytes + dp.o_bytes) + b0 * n_kv_heads;
        int32_t cta = 0;
        for (size_t i = b0; i < b1; ++i) {
            const int32_t s = dp.rows[i];
            DecodeRow &r = dprm.rows[i - b0];
            r.q_row = q_start[s];
            r.ctx_len = h_ctx_lens[s];
            r.table_row = s;
            r.n_splits = dp.n_splits[i];
            r.pages_per_split = dp.pages_per_split[i];
            r.cta_base = cta;
            r.part_base = part_base;
            cta += r.n_splits * n_kv_heads;
            part_base += r.n_splits / dp.cluster;
        }
        dprm.n_ctas = cta;
        dprm.launch_tag = next_launch_tag();
        return part_base;
    };
    auto fill_prefill_common = [&](auto &pp) {
        pp.block_tables = d_block_tables;
        pp.table_stride = max_blocks_per_seq;
        pp.num_blocks = num_blocks;
        pp.out = out;
        pp.out_fp32 = out_is_fp32 ? 1 : 0;
        pp.n_q_heads = n_q_heads;
        pp.n_kv_heads = n_kv_heads;
        pp.group = g;
        pp.heads_per_cta = pf.heads_per_cta;
        pp.scale_log2 = scale_log2;
        pp.err = d_err_flag;
    };
    uint8_t *const pws = ws + dp.total_bytes();
    auto q_map = [&](CUtensorMap *tm) { return encode_q_map(tm, q, static_cast<int32_t>(total_q), n_q_heads); };

    // ---------------- both kinds of rows in one launch
    if (sp.mixed) {
        CUtensorMap tm_q;
        if (!q_map(&tm_q)) return PPAS_ERR_CUDA;
        static thread_local MixedParams mp;  // ~32 KB: kept off the stack
        std::memset(&mp, 0, sizeof(mp));
        fill_prefill_common(mp.pf);
        fill_prefill_params(mp.pf, pf, pf.launches[0], q_start, h_q_lens, h_ctx_lens, pws);
        fill_decode(mp.dc, 0, dp.rows.size(), 0);
        if (launch_mixed(tm_q, tm_k, tm_v, mp, cs) != cudaSuccess) return PPAS_ERR_CUDA;
        return launch_merges(pf, pf.launches[0], q_start, h_q_lens, mp.pf.part_o, mp.pf.part_ml, out, mp.pf.out_fp32,
                             n_q_heads, cs)
                   ? PPAS_OK
                   : PPAS_ERR_CUDA;
    }

    auto run_decode = [&](cudaStream_t ds) -> ppas_status {
        static thread_local DecodeParams dprm;
        int32_t part_base = 0;
        for (size_t b0 = 0; b0 < dp.rows.size(); b0 += kMaxDecodeRows) {
            const size_t b1 = std::min(dp.rows.size(), b0 + kMaxDecodeRows);
            std::memset(&dprm, 0, sizeof(dprm));
            part_base = fill_decode(dprm, b0, b1, part_base);
            if (launch_decode(tm_k, tm_v, dprm, dp.cluster, ds) != cudaSuccess) return PPAS_ERR_CUDA;
        }
        return PPAS_OK;
    };

    // decode rows alone: launch on the caller's stream
    if (pf.empty()) return run_decode(cs);

    // prefill chunks over several launches (more items than one launch
    // holds) with decode rows: the decode launch is forked onto a side
    // stream after the first prefill launch is queued and joined back
    // (the side stream and its events are created, and used, under the lock)
    std::unique_lock<std::mutex> side_lock(g_side_mutex, std::defer_lock);
    if (!dp.rows.empty()) side_lock.lock();
    SideStream *side = dp.rows.empty() ? nullptr : side_stream();
    if (side) {
        if (cudaEventRecord(side->fork, cs) != cudaSuccess ||
            cudaStreamWaitEvent(side->stream, side->fork, 0) != cudaSuccess)
            return PPAS_ERR_CUDA;
    } else if (!dp.rows.empty()) {
        const ppas_status ds = run_decode(cs);
        if (ds != PPAS_OK) return ds;
    }
    // ---------------- prefill chunks
    {
        CUtensorMap tm_q;
        if (!q_map(&tm_q)) return PPAS_ERR_CUDA;
        static thread_local PrefillParams pp;  // ~31 KB: kept off the stack
        for (const PrefillLaunchPlan &lp : pf.launches) {
            std::memset(&pp, 0, sizeof(pp));
            fill_prefill_common(pp);
            fill_prefill_params(pp, pf, lp, q_start, h_q_lens, h_ctx_lens, pws);
            if (launch_prefill(tm_q, tm_k, tm_v, pp, cs) != cudaSuccess) return PPAS_ERR_CUDA;
            // the launch's cut units are merged once it is done
            if (!launch_merges(pf, lp, q_start, h_q_lens, pp.part_o, pp.part_ml, out, pp.out_fp32, n_q_heads, cs))
                return PPAS_ERR_CUDA;
        }
    }
    if (side) {
        const ppas_status ds = run_decode(side->stream);
        if (ds != PPAS_OK) return ds;
        if (cudaEventRecord(side->join, side->stream) != cudaSuccess ||
            cudaStreamWaitEvent(cs, side->join, 0) != cudaSuccess)
            return PPAS_ERR_CUDA;
    }
    return PPAS_OK;
}

extern "C" ppas_status ppas_gateup_pack(const void *w, void *w_packed, int32_t hidden, int32_t inter, void *stream) {
    if (hidden < 64 || hidden % 64 || inter < 128 || inter % 128) return PPAS_ERR_UNSUPPORTED;
    if (!w || !w_packed || !aligned16(w) || !aligned16(w_packed)) return PPAS_ERR_INVALID_ARG;
    return launch_gateup_pack(w, w_packed, hidden, inter, static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? PPAS_OK
               : PPAS_ERR_CUDA;
}

extern "C" ppas_status ppas_gateup_swiglu(const void *x, const void *w_packed, void *y, int32_t n_tokens,
                                          int32_t hidden, int32_t inter, int32_t *d_err_flag, void *stream) {
    if (n_tokens < 0) return PPAS_ERR_INVALID_ARG;
    if (hidden < 64 || hidden % 64 || inter < 128 || inter % 128) return PPAS_ERR_UNSUPPORTED;
    if (n_tokens == 0) return PPAS_OK;
    if (!x || !w_packed || !y || !aligned16(x) || !aligned16(w_packed) || !aligned16(y)) return PPAS_ERR_INVALID_ARG;
    CUtensorMap tm_x, tm_w;
    if (!encode_bf16_2d(&tm_x, x, static_cast<uint64_t>(hidden), static_cast<uint64_t>(n_tokens), 64, 128) ||
        !encode_bf16_2d(&tm_w, w_packed, static_cast<uint64_t>(hidden), 2ull * inter, 64, 256))
        return PPAS_ERR_CUDA;
    GateUpParams gp;
    gp.y = static_cast<__nv_bfloat16 *>(y);
    gp.n_tokens = n_tokens;
    gp.hidden = hidden;
    gp.inter = inter;
    gp.err = d_err_flag;
    const int64_t tiles = static_cast<int64_t>((n_tokens + 127) / 128) * (inter / 128);
    const int grid = static_cast<int>(std::min<int64_t>(tiles, device_sm_count()));
    return launch_gateup(tm_x, tm_w, gp, grid, static_cast<cudaStream_t>(stream)) == cudaSuccess ? PPAS_OK
                                                                                                  : PPAS_ERR_CUDA;
}
