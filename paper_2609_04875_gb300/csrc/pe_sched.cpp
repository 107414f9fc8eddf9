// Replay passes with the indep split (Sec. 4.5, the T - tau + 1 paragraph;
// Sec. 4.1 methods B7 and B5'): which suffix positions are re-prefilled and
// which are re-decoded, and the lockstep rounds that batch many agents.
//
// Host-only planning: a unit is a maximal run of consecutive positions whose
// content is known in the counterfactual world (one prefill pass), or a single
// position that must be generated again (one decode pass).  Round r runs
// every agent's r-th unit, so one batched append + one batched attention
// launch per layer serve all agents of a round.
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <vector>

#include "pe.h"
#include "pe_internal.h"

namespace {

pe_status sched_fail(pe_status code, const char *fmt, ...)
{
    char buf[256];
    va_list ap;
    va_start(ap, fmt);
    std::vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    return pe::report_error(code, buf);
}

// Positions of kind `kind` count as known (prefilled) under `policy`.
bool known(int32_t policy, int32_t kind)
{
    return kind == PE_TURN_INPUT || (policy == PE_POLICY_SELECTIVE && kind == PE_TURN_MODEL_INDEP);
}

}  // namespace

extern "C" pe_status pe_replay_schedule(int32_t n, const int32_t *cu_turns, const int32_t *turn_len,
                                        const int32_t *turn_kind, int32_t policy, int32_t *take, int64_t take_cap,
                                        int32_t *n_rounds, int64_t *decode_tokens)
{
    if (!n_rounds) return sched_fail(PE_ERR_INVALID, "null n_rounds");
    if (n < 0 || (n > 0 && !cu_turns)) return sched_fail(PE_ERR_INVALID, "bad agent arguments");
    if (policy != PE_POLICY_SELECTIVE && policy != PE_POLICY_PREFIX_CACHE)
        return sched_fail(PE_ERR_INVALID, "unknown policy %d", policy);
    if (take_cap < 0 || (take_cap > 0 && !take)) return sched_fail(PE_ERR_INVALID, "bad take buffer");
    if (n > 0 && cu_turns[0] != 0) return sched_fail(PE_ERR_INVALID, "cu_turns[0] must be 0");
    if (n > 0 && cu_turns[n] > 0 && (!turn_len || !turn_kind)) return sched_fail(PE_ERR_INVALID, "null turn arrays");

    // units of every agent, in session order
    std::vector<std::vector<int32_t>> units(n);
    int64_t decoded = 0;
    size_t rounds = 0;
    for (int32_t i = 0; i < n; ++i) {
        if (cu_turns[i + 1] < cu_turns[i]) return sched_fail(PE_ERR_INVALID, "cu_turns must be non-decreasing");
        int64_t run = 0, total = 0;
        std::vector<int32_t> &u = units[i];
        for (int32_t t = cu_turns[i]; t < cu_turns[i + 1]; ++t) {
            const int32_t len = turn_len[t], kind = turn_kind[t];
            if (kind != PE_TURN_INPUT && kind != PE_TURN_MODEL_INDEP && kind != PE_TURN_MODEL_DEP)
                return sched_fail(PE_ERR_INVALID, "turn %d: unknown kind %d", t, kind);
            if (len < 0) return sched_fail(PE_ERR_INVALID, "turn %d: negative length", t);
            total += len;
            if (total > INT32_MAX) return sched_fail(PE_ERR_INVALID, "agent %d: suffix exceeds int32", i);
            if (len == 0) continue;
            if (known(policy, kind)) {
                run += len;
            } else {
                if (run > 0) u.push_back(static_cast<int32_t>(run));
                run = 0;
                u.insert(u.end(), static_cast<size_t>(len), 1);
                decoded += len;
            }
        }
        if (run > 0) u.push_back(static_cast<int32_t>(run));
        rounds = std::max(rounds, u.size());
    }
    if (rounds > static_cast<size_t>(INT32_MAX)) return sched_fail(PE_ERR_INVALID, "too many rounds");
    *n_rounds = static_cast<int32_t>(rounds);
    if (decode_tokens) *decode_tokens = decoded;
    if (!take) return PE_OK;  // size query
    const int64_t cells = static_cast<int64_t>(rounds) * n;
    if (cells > take_cap)
        return sched_fail(PE_ERR_RANGE, "take needs %lld entries, capacity %lld", static_cast<long long>(cells),
                          static_cast<long long>(take_cap));
    for (int64_t k = 0; k < cells; ++k) take[k] = 0;
    for (int32_t i = 0; i < n; ++i)
        for (size_t r = 0; r < units[i].size(); ++r) take[static_cast<int64_t>(r) * n + i] = units[i][r];
    return PE_OK;
}
