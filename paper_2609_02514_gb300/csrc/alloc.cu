// Host-side tree budgeting and shape allocation (Sec. IV-B and IV-C).
//
//   aces_tree_budget   B* = min(B_max, largest B whose tree-draft latency fits
//                      in RTT + T_verify), the network-aware budget of
//                      Eq. (budget), from a tabulated latency profile.
//   aces_branch_alloc  F_k = B_alloc (1 - eta) / (1 - eta^gamma) eta^k with
//                      eta = alpha^(1/(beta+1)) (Eq. for F*_k after the
//                      Lagrangian condition), rounded to integers that sum to
//                      B_alloc: floor, then one more branch for the largest
//                      fractional parts, ties to the shallower depth.
#include <algorithm>
#include <cmath>
#include <vector>

#define ACES_FILE 2  // site numbers of the checked build
#include "common.cuh"

extern "C" {

aces_status aces_tree_budget(const double *draft_latency_s, int n, double rtt_s, double verify_s, int B_max,
                             int *B_star) {
    if (!draft_latency_s || !B_star || n < 1 || B_max < 0) return ACES_ERR_INVALID_ARG;
    if (!(rtt_s >= 0.0) || !(verify_s >= 0.0) || !std::isfinite(rtt_s) || !std::isfinite(verify_s))
        return ACES_ERR_INVALID_ARG;
    for (int i = 0; i < n; ++i) {
        const double t = draft_latency_s[i];
        if (!(t >= 0.0) || !std::isfinite(t)) return ACES_ERR_INVALID_ARG;
        if (i > 0 && t < draft_latency_s[i - 1]) return ACES_ERR_INVALID_ARG;  // must not decrease
    }
    const double window = rtt_s + verify_s;
    int b = 0;  // largest tree size whose drafting time is masked by the window
    while (b < n && draft_latency_s[b] <= window) ++b;
    *B_star = b < B_max ? b : B_max;
    return ACES_OK;
}

aces_status aces_branch_alloc(int B_alloc, int gamma, double alpha, double beta, int32_t *F_out) {
    if (!F_out || B_alloc < 0 || gamma < 1 || gamma > ACES_MAX_K) return ACES_ERR_INVALID_ARG;
    if (!(alpha > 0.0 && alpha <= 1.0) || !(beta > 0.0) || !std::isfinite(beta)) return ACES_ERR_INVALID_ARG;
    const double eta = std::pow(alpha, 1.0 / (beta + 1.0));
    std::vector<double> share(gamma);
    if (eta == 1.0) {
        for (int d = 0; d < gamma; ++d) share[d] = (double)B_alloc / gamma;
    } else {
        const double base = (double)B_alloc * (1.0 - eta) / (1.0 - std::pow(eta, (double)gamma));
        for (int d = 0; d < gamma; ++d) share[d] = base * std::pow(eta, (double)d);
    }
    long long given = 0;
    std::vector<int> order(gamma);
    for (int d = 0; d < gamma; ++d) {
        F_out[d] = (int32_t)std::floor(share[d]);
        given += F_out[d];
        order[d] = d;
    }
    std::stable_sort(order.begin(), order.end(), [&](int x, int y) {
        return (share[x] - F_out[x]) > (share[y] - F_out[y]);
    });
    for (long long i = 0; i < (long long)B_alloc - given && i < gamma; ++i) F_out[order[(size_t)i]] += 1;
    return ACES_OK;
}

}  // extern "C"
