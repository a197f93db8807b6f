// Host planner: resolves the splice rule of §3 / Algorithm 1 for a whole
// decode batch into per-(epoch, layer class) tables.
//
// Layer l at decode step t reads the donor span of the sequence's slot iff
// l >= L and t >= W (the patched layers are {l >= L}; the replacement made at
// t = W persists).  Because the rule only compares l with the L values and t
// with the W values present in the batch, the (layer, step) plane splits into
// rectangles -- layer classes between consecutive distinct L, epochs between
// consecutive distinct W -- inside which every sequence reads one source.
// One table per rectangle lists that source per sequence and groups the
// sequences that read the same stored (prompt, source) span, so the prefix
// pass can read each span once for all its readers.  In delta mode the
// readers of a delta-encoded donor slot share the clean span's groups (with
// a row mask) and read the slot's encoded rows as a group of their own.
#include <algorithm>
#include <cstdio>
#include <numeric>
#include <string>
#include <tuple>

#include "splice_internal.h"

namespace splice {

int Plan::table_of(int layer, int step) const {
    const int e = int(std::upper_bound(epoch_bounds.begin(), epoch_bounds.end(), step) -
                      epoch_bounds.begin()) - 1;
    const int c = int(std::upper_bound(class_bounds.begin(), class_bounds.end(), layer) -
                      class_bounds.begin()) - 1;
    return e * int(class_bounds.size()) + c;
}

static std::string fmt(const char* f, long a = 0, long b = 0) {
    char buf[256];
    std::snprintf(buf, sizeof buf, f, a, b);
    return buf;
}

std::string build_plan(const splice_model_shape& sh, int P, int Tp, int Dslots, const splice_donor_kind* kinds,
                       int B, const splice_seq* seqs, int T, const uint8_t* slot_delta, Plan& plan) {
    const int N = sh.num_layers;
    const int G = sh.num_q_heads / sh.num_kv_heads;

    std::vector<int> eb{0}, cb{0};
    for (int s = 0; s < B; ++s) {
        if (seqs[s].W <= T) eb.push_back(seqs[s].W);
        if (seqs[s].L < N) cb.push_back(seqs[s].L);
    }
    std::sort(eb.begin(), eb.end());
    eb.erase(std::unique(eb.begin(), eb.end()), eb.end());
    std::sort(cb.begin(), cb.end());
    cb.erase(std::unique(cb.begin(), cb.end()), cb.end());
    plan.epoch_bounds = eb;
    plan.class_bounds = cb;
    plan.num_tables = int(eb.size() * cb.size());
    plan.seqs_per_tile = std::max(1, kTileRows / G);

    // stored-donor index of every slot (the non-ZERO slots in slot order)
    std::vector<int> stored(Dslots, -1);
    int n_stored = 0;
    for (int k = 0; k < Dslots; ++k)
        if (kinds[k] != SPLICE_DONOR_ZERO) stored[k] = n_stored++;

    plan.src.assign(size_t(plan.num_tables) * B, 0);
    plan.table_group_off.assign(plan.num_tables + 1, 0);
    plan.table_tile_off.assign(plan.num_tables + 1, 0);
    plan.table_span_tiles.assign(plan.num_tables, 0);
    plan.group_prompt.clear();
    plan.group_src.clear();
    plan.group_first.clear();
    plan.group_count.clear();
    plan.group_seqs.clear();
    plan.group_mask.clear();
    plan.tiles.clear();

    // (delta group?, prompt, group source, row mask, sequence): sorting puts
    // the stored-span groups first and, inside a group, rows without a mask
    // first and the rows of each masked slot together.
    using Key = std::tuple<int, int, int, int, int>;
    std::vector<Key> keyed;
    keyed.reserve(2 * size_t(B));
    for (int e = 0; e < int(eb.size()); ++e) {
        for (int c = 0; c < int(cb.size()); ++c) {
            const int tab = e * int(cb.size()) + c;
            const int t_rep = eb[e], l_rep = cb[c];
            uint8_t* src = &plan.src[size_t(tab) * B];
            keyed.clear();
            for (int s = 0; s < B; ++s) {
                const splice_seq& q = seqs[s];
                uint8_t code = SPLICE_SRC_CLEAN;
                if (l_rep >= q.L && t_rep >= q.W)
                    code = kinds[q.donor_slot] == SPLICE_DONOR_ZERO
                               ? uint8_t(SPLICE_SRC_ZERO)
                               : uint8_t(SPLICE_SRC_DONOR0 + q.donor_slot);
                src[s] = code;
                if (code == SPLICE_SRC_ZERO) continue;
                if (code >= SPLICE_SRC_DONOR0 && slot_delta && slot_delta[q.donor_slot]) {
                    keyed.emplace_back(0, q.prompt_id, int(SPLICE_SRC_CLEAN), stored[q.donor_slot] + 1, s);
                    keyed.emplace_back(1, q.prompt_id, kGroupDelta | int(code), 0, s);
                } else {
                    keyed.emplace_back(0, q.prompt_id, int(code), 0, s);
                }
            }
            std::sort(keyed.begin(), keyed.end());
            plan.table_group_off[tab] = int(plan.group_prompt.size());
            plan.table_tile_off[tab] = int(plan.tiles.size() / 4);
            int span_tiles = 0;
            size_t i = 0;
            while (i < keyed.size()) {
                size_t j = i;
                while (j < keyed.size() && std::get<0>(keyed[j]) == std::get<0>(keyed[i]) &&
                       std::get<1>(keyed[j]) == std::get<1>(keyed[i]) && std::get<2>(keyed[j]) == std::get<2>(keyed[i]))
                    ++j;
                const int gid = int(plan.group_prompt.size());
                const int first = int(plan.group_seqs.size());
                plan.group_prompt.push_back(std::get<1>(keyed[i]));
                plan.group_src.push_back(std::get<2>(keyed[i]));
                plan.group_first.push_back(first);
                plan.group_count.push_back(int(j - i));
                for (size_t k = i; k < j; ++k) {
                    plan.group_seqs.push_back(std::get<4>(keyed[k]));
                    plan.group_mask.push_back(std::get<3>(keyed[k]));
                }
                // the tile's store and its span base index: kind 0 = clean
                // span (base = prompt), 1 = stored donor span, 2 = a donor's
                // delta rows (base = prompt * stored slots + stored index);
                // the span of (layer l, kv head h) is (base * N + l) * Hkv + h
                const int gsrc = std::get<2>(keyed[i]);
                const int gprompt = std::get<1>(keyed[i]);
                int kind = 0, base = gprompt;
                if (gsrc != int(SPLICE_SRC_CLEAN)) {
                    kind = (gsrc & kGroupDelta) ? 2 : 1;
                    base = gprompt * n_stored + stored[(gsrc & 0xff) - int(SPLICE_SRC_DONOR0)];
                }
                for (int off = 0; off < int(j - i); off += plan.seqs_per_tile) {
                    plan.tiles.push_back(gid);
                    plan.tiles.push_back(first + off);
                    plan.tiles.push_back(std::min(plan.seqs_per_tile, int(j - i) - off));
                    plan.tiles.push_back((base << 2) | kind);
                    if (std::get<0>(keyed[i]) == 0) ++span_tiles;
                }
                i = j;
            }
            plan.table_span_tiles[tab] = span_tiles;
        }
    }
    plan.table_group_off[plan.num_tables] = int(plan.group_prompt.size());
    plan.table_tile_off[plan.num_tables] = int(plan.tiles.size() / 4);
    (void)P;
    (void)Tp;
    return std::string();
}

Visible visible_keys(const splice_model_shape& sh, int Tp, int layer, int step) {
    // The step-t query sits at absolute position Tp + t - 1; on a local layer
    // key j is visible iff (Tp + t - 1) - j < window.
    Visible v{0, Tp, 0, step};
    const bool global = sh.sliding_window <= 0 ||
                        (sh.global_every > 0 && (layer + 1) % sh.global_every == 0);
    if (!global) {
        const long lo = long(Tp) + step - sh.sliding_window;   // first visible absolute position
        if (lo > 0) {
            v.p_lo = int(std::min<long>(lo, Tp));
            v.s_lo = int(std::max<long>(0, std::min<long>(lo - Tp, step)));
        }
    }
    return v;
}

}  // namespace splice
