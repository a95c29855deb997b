// frt_plan.cu — host-side work split of an attention launch.
//
// A launch runs one CTA per work item; the hardware hands items to SMs in launch order as
// SMs free up (list scheduling). Query groups (stream, head, 256 query rows) cost their
// KV tiles, so with G equal groups on P SMs the last wave holds only G mod P of them and
// the other SMs idle. Cutting every group's KV range into s parts (split-KV) fills that
// wave but makes every group pay for writing and merging partials. The plan here cuts
// only the tail: groups [0, n_full) run whole and each later group is cut into n_split
// parts, with n_full and n_split chosen by simulating the list schedule of the launch
// under a cost model of the kernel (in units of one KV step of a two-tile group).
#include <algorithm>
#include <functional>
#include <queue>
#include <vector>

#include "frt_internal.h"

namespace frt {

namespace {

// Cost model, in KV steps of a two-tile query group (~3300 cycles on the GB300):
constexpr double kItemFixed = 7.0;    // per item: prologue (Q load, RoPE-Q), epilogue, launch
constexpr double kPartExtra = 1.0;    // per split item: its partial's write and merge share
constexpr double kSingleStep = 0.6;   // a KV step of a group with one 128-row query tile

double simulate(const int* tiles, const unsigned char* single, int groups, int n_full,
                int n_split, int sms) {
    std::priority_queue<double, std::vector<double>, std::greater<double>> free_at;
    for (int i = 0; i < sms; ++i) free_at.push(0.0);
    double makespan = 0.0;
    auto run = [&](double cost) {
        const double t = free_at.top() + cost;
        free_at.pop();
        free_at.push(t);
        makespan = std::max(makespan, t);
    };
    for (int g = 0; g < groups; ++g) {
        const double w = single[g] ? kSingleStep : 1.0;
        if (g < n_full) {
            run(kItemFixed + tiles[g] * w);
            continue;
        }
        for (int s = 0; s < n_split; ++s) {
            const int t = (s + 1) * tiles[g] / n_split - s * tiles[g] / n_split;
            run(kItemFixed + kPartExtra + t * w);
        }
    }
    return makespan;
}

}  // namespace

SplitPlan plan_attention(const int* tiles, const unsigned char* single, int groups, int sms,
                         int max_split, long long max_rows, long long max_tails) {
    SplitPlan best;
    best.n_full = groups;
    best.n_split = 1;
    if (groups <= 0 || sms <= 0) return best;
    double best_t = simulate(tiles, single, groups, groups, 1, sms);
    // tail sizes: what is left after whole waves, plus up to three more waves, or all
    const int r = groups % sms == 0 ? sms : groups % sms;
    std::vector<int> tails;
    for (int m = 0; m < 4; ++m)
        if (r + m * sms <= groups) tails.push_back(r + m * sms);
    if (tails.empty() || tails.back() != groups) tails.push_back(groups);
    for (int sp = 2; sp <= max_split && sp <= kMaxSplit; ++sp)
        for (int tail : tails) {
            const int n_full = groups - tail;
            int min_tiles = 1 << 30;
            for (int g = n_full; g < groups; ++g) min_tiles = std::min(min_tiles, tiles[g]);
            if (min_tiles < 2 * sp) continue;   // every part keeps at least two KV tiles
            if (max_rows >= 0 && (long long)tail * sp * 256 > max_rows) continue;
            if (max_tails >= 0 && tail > max_tails) continue;
            const double t = simulate(tiles, single, groups, n_full, sp, sms);
            if (t < best_t * (1.0 - 1e-9)) {
                best_t = t;
                best.n_full = n_full;
                best.n_split = sp;
            }
        }
    return best;
}

}  // namespace frt
