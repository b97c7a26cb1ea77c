// First-layer prefix caching (§5.1): Eq. (1), Eq. (2) and the per-layer
// load/compute pipeline they summarise. Host arithmetic only.
#include <cmath>
#include <cstdint>

#include "common.hpp"
#include "t2istore.h"

namespace {
bool finite_pos(double x) { return std::isfinite(x) && x > 0.0; }
bool finite_nonneg(double x) { return std::isfinite(x) && x >= 0.0; }
}  // namespace

extern "C" {

t2i_status t2i_e2e_latency(uint32_t L, uint32_t L_e, double t_load, double t_comp, double* out) {
    if (!out || L_e > L || !finite_nonneg(t_load) || !finite_nonneg(t_comp)) {
        t2i::set_thread_error("t2i_e2e_latency: need L_e <= L, finite non-negative times, out");
        return T2I_ERR_INVALID;
    }
    const double compute = double(L) * t_comp;
    const double exposed = double(L - L_e) * t_load + t_comp;
    *out = compute > exposed ? compute : exposed;
    return T2I_OK;
}

t2i_status t2i_prefix_layers(uint32_t L, double t_load, double t_comp, uint32_t* out) {
    if (!out || !finite_pos(t_load) || !finite_nonneg(t_comp)) {
        t2i::set_thread_error("t2i_prefix_layers: need t_load > 0, t_comp >= 0, finite, and out");
        return T2I_ERR_INVALID;
    }
    const double v = std::ceil((double(L) * (t_load - t_comp) + t_comp) / t_load);
    *out = v <= 0.0 ? 0u : (v >= double(L) ? L : static_cast<uint32_t>(v));
    return T2I_OK;
}

t2i_status t2i_pipeline_latency(const double* t_load, const double* t_comp, uint32_t L, uint32_t L_e,
                                double* out) {
    if (!out || (L && (!t_load || !t_comp)) || L_e > L) {
        t2i::set_thread_error("t2i_pipeline_latency: bad arguments");
        return T2I_ERR_INVALID;
    }
    double loads_done = 0.0;  // the loads run back to back from time 0
    double comp_end = 0.0;
    for (uint32_t l = 0; l < L; ++l) {
        if (!finite_nonneg(t_load[l]) || !finite_nonneg(t_comp[l])) {
            t2i::set_thread_error("t2i_pipeline_latency: times must be finite and non-negative");
            return T2I_ERR_INVALID;
        }
        double ready = 0.0;
        if (l >= L_e) {
            loads_done += t_load[l];
            ready = loads_done;
        }
        comp_end = (comp_end > ready ? comp_end : ready) + t_comp[l];
    }
    *out = comp_end;
    return T2I_OK;
}

t2i_status t2i_prefix_layers_pipeline(const double* t_load, const double* t_comp, uint32_t L, uint32_t* out) {
    if (!out || (L && (!t_load || !t_comp))) {
        t2i::set_thread_error("t2i_prefix_layers_pipeline: bad arguments");
        return T2I_ERR_INVALID;
    }
    double total = 0.0;
    for (uint32_t l = 0; l < L; ++l) total += t_comp[l];
    const double bound = total * (1.0 + 1e-12);
    // the latency never grows with the prefix: bisect for the smallest
    // prefix that leaves no loading exposed
    uint32_t lo = 0, hi = L;
    while (lo < hi) {
        const uint32_t mid = lo + (hi - lo) / 2;
        double t = 0.0;
        t2i_status st = t2i_pipeline_latency(t_load, t_comp, L, mid, &t);
        if (st != T2I_OK) return st;
        if (t <= bound)
            hi = mid;
        else
            lo = mid + 1;
    }
    *out = lo;
    return T2I_OK;
}

}  // extern "C"
