// mc_pmq.cpp -- the pre-loading mixed-precision allocation of Sec. 2.2 (PMQ):
// expert significance from routing statistics (Sec. 2.2.1) and the bit-width
// integer program of Eq. 4 (Sec. 2.2.2), solved exactly by enumerating every
// assignment of {1, 2, 3} bits to the experts (3^E of them; E <= 16).  Host code:
// it runs once per layer before the experts are quantised.
#include <math.h>
#include <string.h>

#include <vector>

#include "mc_host.h"

using namespace mc;

extern "C" {

int mc_expert_significance_host(const int32_t *idx, const float *w, const uint8_t *pruned, int T, int E,
                                double *phi, double *wact)
{
    clear_error();
    if (T <= 0 || E < 2 || E > kMaxE) return set_error(MC_ERR_INVALID_ARG, "T=%d E=%d", T, E);
    if (!idx || !w || !phi || !wact) return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    for (int e = 0; e < E; ++e) phi[e] = wact[e] = 0.0;
    for (int t = 0; t < T; ++t)
        for (int s = 0; s < 2; ++s) {
            const int p = pruned ? pruned[t] : 0;
            if ((s == 1 && p) || p == 2) continue;  // not an activation of the expert
            const int e = idx[2 * t + s];
            if (e < 0 || e >= E) return set_error(MC_ERR_INVALID_ARG, "token %d slot %d: expert %d", t, s, e);
            phi[e] += 1.0;
            wact[e] += (double)w[2 * t + s];
        }
    for (int e = 0; e < E; ++e) {
        phi[e] /= (double)T;   // n_i / N
        wact[e] /= (double)T;  // sum of the routing weights / N
    }
    return MC_OK;
}

int mc_pmq_allocate(const double *phi, const double *wact, const double *eps, int E, int bits_total, double alpha,
                    double beta, double gamma, int8_t *bits_out, double *objective_out)
{
    clear_error();
    if (E < 2 || E > kMaxE) return set_error(MC_ERR_INVALID_ARG, "E=%d: need 2 <= E <= %d", E, kMaxE);
    if (!phi || !wact || !eps || !bits_out) return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    // cost of expert i at j bits: phi^alpha * w^beta * eps_ij^gamma (the x_ij = 0 terms vanish)
    std::vector<double> cost((size_t)E * 3);
    for (int i = 0; i < E; ++i) {
        const double sig = pow(phi[i], alpha) * pow(wact[i], beta);
        for (int j = 0; j < 3; ++j) {
            const double e = eps[3 * i + j];
            if (!(e >= 0.0) || !isfinite(e) || !(sig >= 0.0) || !isfinite(sig))
                return set_error(MC_ERR_INVALID_ARG, "expert %d: significance or eps[%d] not a finite value >= 0", i, j);
            cost[3 * i + j] = sig * pow(e, gamma);
        }
    }
    // every assignment in base-3 order (expert 0 the least significant digit);
    // the first strict minimum wins, so ties go to the earliest assignment
    std::vector<int> a(E, 0);
    double best = INFINITY;
    std::vector<int> best_a;
    for (;;) {
        int sum = 0, n3 = 0, n2 = 0;
        double c = 0.0;
        for (int i = 0; i < E; ++i) {
            sum += a[i] + 1;
            n3 += a[i] == 2;
            n2 += a[i] == 1;
            c += cost[3 * i + a[i]];
        }
        if (sum == bits_total && n3 >= 1 && n2 >= 1 && c < best) {
            best = c;
            best_a = a;
        }
        int i = 0;
        while (i < E && a[i] == 2) a[i++] = 0;
        if (i == E) break;
        ++a[i];
    }
    if (best_a.empty())
        return set_error(MC_ERR_INVALID_ARG, "no assignment of 1..3 bits to %d experts sums to %d with a 3-bit and a "
                                             "2-bit expert", E, bits_total);
    for (int i = 0; i < E; ++i) bits_out[i] = (int8_t)(best_a[i] + 1);
    if (objective_out) *objective_out = best;
    return MC_OK;
}

}  // extern "C"
