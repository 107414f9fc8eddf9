// Provenance-graph queries of Alg. 1 (lines 1-3) on the host: the runtime's
// artifact DAG (Sec. 3.4(a): id, type, parents, source ids, token span, turn,
// committed) and the three reachability queries that produce tau for pe_crop.
//   LocateSource(z)  the artifact through which z entered: a carrier of z none
//                    of whose parents carries z; the earliest (token_begin,
//                    then id) if several
//   TaintClosure(s)  I(z): artifacts reachable from s along parent -> child
//                    edges, s included (Lemma 2)
//   FirstEntry(s)    tau = 1-based position of the closure's first token
#include <algorithm>
#include <cstdint>
#include <new>
#include <unordered_map>
#include <unordered_set>
#include <vector>

#include "pe.h"
#include "pe_internal.h"

struct pe_prov {
    struct Art {
        int64_t id;
        int32_t type, turn, committed;
        int64_t begin, end;
        std::vector<int32_t> parents;   // indices
        std::vector<int32_t> children;  // indices
        std::vector<int64_t> sources;
    };
    std::vector<Art> arts;
    std::unordered_map<int64_t, int32_t> index;                 // id -> position
    std::unordered_map<int64_t, std::vector<int32_t>> carriers; // source id -> artifacts carrying it
};

namespace {

bool carries(const pe_prov::Art &a, int64_t z)
{
    return std::find(a.sources.begin(), a.sources.end(), z) != a.sources.end();
}

pe_status closure_of(const pe_prov *g, int64_t source, std::vector<int32_t> &out)
{
    auto it = g->index.find(source);
    if (it == g->index.end()) return pe::report_error(PE_ERR_RANGE, "unknown artifact");
    std::vector<uint8_t> seen(g->arts.size(), 0);
    std::vector<int32_t> frontier{it->second};
    seen[it->second] = 1;
    out.assign(1, it->second);
    while (!frontier.empty()) {
        std::vector<int32_t> next;
        for (int32_t a : frontier)
            for (int32_t c : g->arts[a].children)
                if (!seen[c]) {
                    seen[c] = 1;
                    next.push_back(c);
                    out.push_back(c);
                }
        frontier.swap(next);
    }
    return PE_OK;
}

}  // namespace

extern "C" {

pe_status pe_prov_create(pe_prov **out)
{
    if (!out) return pe::report_error(PE_ERR_INVALID, "null argument");
    *out = new (std::nothrow) pe_prov();
    return *out ? PE_OK : pe::report_error(PE_ERR_OOM, "host allocation failed");
}

pe_status pe_prov_destroy(pe_prov *g)
{
    if (!g) return pe::report_error(PE_ERR_INVALID, "null graph");
    delete g;
    return PE_OK;
}

pe_status pe_prov_add(pe_prov *g, int64_t id, int32_t type, const int64_t *parents, int32_t n_parents,
                      const int64_t *source_ids, int32_t n_sources, int64_t token_begin, int64_t token_end,
                      int32_t turn, int32_t committed)
{
    if (!g) return pe::report_error(PE_ERR_INVALID, "null graph");
    if (n_parents < 0 || n_sources < 0 || (n_parents > 0 && !parents) || (n_sources > 0 && !source_ids))
        return pe::report_error(PE_ERR_INVALID, "bad parent or source arrays");
    if (g->index.count(id)) return pe::report_error(PE_ERR_INVALID, "duplicate artifact id");
    if (token_begin < 0 || token_end < token_begin) return pe::report_error(PE_ERR_INVALID, "bad token span");
    pe_prov::Art a;
    a.id = id;
    a.type = type;
    a.turn = turn;
    a.committed = committed ? 1 : 0;
    a.begin = token_begin;
    a.end = token_end;
    for (int32_t i = 0; i < n_parents; ++i) {
        auto it = g->index.find(parents[i]);
        if (it == g->index.end()) return pe::report_error(PE_ERR_INVALID, "unknown parent (add artifacts in execution order)");
        if (std::find(a.parents.begin(), a.parents.end(), it->second) == a.parents.end()) a.parents.push_back(it->second);
    }
    for (int32_t i = 0; i < n_sources; ++i)
        if (!carries(a, source_ids[i])) a.sources.push_back(source_ids[i]);
    const int32_t idx = static_cast<int32_t>(g->arts.size());
    for (int32_t p : a.parents) g->arts[p].children.push_back(idx);
    for (int64_t z : a.sources) g->carriers[z].push_back(idx);
    g->index.emplace(id, idx);
    g->arts.push_back(std::move(a));
    return PE_OK;
}

pe_status pe_prov_locate_source(const pe_prov *g, int64_t z, int64_t *source)
{
    if (!g || !source) return pe::report_error(PE_ERR_INVALID, "null argument");
    auto it = g->carriers.find(z);
    if (it == g->carriers.end() || it->second.empty()) return pe::report_error(PE_ERR_RANGE, "no artifact carries this source id");
    int32_t best = -1;
    for (int32_t a : it->second) {
        const pe_prov::Art &art = g->arts[a];
        bool root = true;
        for (int32_t p : art.parents)
            if (carries(g->arts[p], z)) { root = false; break; }
        if (!root) continue;
        if (best < 0 || art.begin < g->arts[best].begin ||
            (art.begin == g->arts[best].begin && art.id < g->arts[best].id))
            best = a;
    }
    *source = g->arts[best].id;
    return PE_OK;
}

pe_status pe_prov_taint_closure(const pe_prov *g, int64_t source, int64_t *out, int32_t cap, int32_t *n,
                                int32_t *n_committed)
{
    if (!g) return pe::report_error(PE_ERR_INVALID, "null graph");
    std::vector<int32_t> clo;
    pe_status s = closure_of(g, source, clo);
    if (s != PE_OK) return s;
    std::vector<int64_t> ids;
    ids.reserve(clo.size());
    int32_t nc = 0;
    for (int32_t a : clo) {
        ids.push_back(g->arts[a].id);
        nc += g->arts[a].committed;
    }
    std::sort(ids.begin(), ids.end());
    if (n) *n = static_cast<int32_t>(ids.size());
    if (n_committed) *n_committed = nc;
    if (out) {
        if (cap < static_cast<int32_t>(ids.size())) return pe::report_error(PE_ERR_RANGE, "output capacity too small");
        std::copy(ids.begin(), ids.end(), out);
    }
    return PE_OK;
}

pe_status pe_prov_first_entry(const pe_prov *g, int64_t source, int64_t *tau)
{
    if (!g || !tau) return pe::report_error(PE_ERR_INVALID, "null argument");
    std::vector<int32_t> clo;
    pe_status s = closure_of(g, source, clo);
    if (s != PE_OK) return s;
    int64_t first = g->arts[clo[0]].begin;
    for (int32_t a : clo) first = std::min(first, g->arts[a].begin);
    *tau = first + 1;
    return PE_OK;
}

}  // extern "C"
