// Flexible resource scheduling (Sec. IV-D, Eq. 15-17): a controller that picks the split
// point of each frame inside the dynamic zone from the runtime state (co-tenant utilisation
// of GPU and CPU, pipeline backlog) and the per-block stage costs it has observed. The rule
// is stated in vla_cpu.h; it is host-only code and touches no device.
#include <algorithm>
#include <cstdlib>
#include <new>

#include "vla_cpu.h"

struct vla_scheduler {
    vla_sched_config cfg;
    int k = 0;                          // current split
    double g = -1.0, c = -1.0, x = -1.0;  // ms per GPU block, per CPU block, per transfer
};

namespace {

double ema(double old, double v, double a) { return old < 0.0 ? v : (1.0 - a) * old + a * v; }

double clamp_u(double u) { return std::min(std::max(u, 0.0), 0.95); }

}  // namespace

extern "C" {

vla_status vla_scheduler_create(const vla_sched_config* cfg, vla_scheduler** out) {
    if (!out) return VLA_ERR_INVALID_ARG;
    *out = nullptr;
    if (!cfg) return VLA_ERR_INVALID_ARG;
    const vla_sched_config& c = *cfg;
    if (c.n_layers < 1 || c.k_min < 0 || c.k_max > c.n_layers || c.k_min > c.k_max || c.k_init < c.k_min ||
        c.k_init > c.k_max || c.max_step < 1 || !(c.alpha > 0.0 && c.alpha <= 1.0) || c.backlog_limit < 1)
        return VLA_ERR_INVALID_ARG;
    vla_scheduler* s = new (std::nothrow) vla_scheduler();
    if (!s) return VLA_ERR_OOM;
    s->cfg = c;
    s->k = c.k_init;
    *out = s;
    return VLA_OK;
}

vla_status vla_scheduler_observe(vla_scheduler* s, const vla_frame_times* t) {
    if (!s || !t || t->split < 0 || t->split > s->cfg.n_layers) return VLA_ERR_INVALID_ARG;
    const double a = s->cfg.alpha;
    const int N = s->cfg.n_layers;
    if (t->split > 0) s->g = ema(s->g, t->t_gpu_ms / t->split, a);
    if (t->split < N) s->c = ema(s->c, t->t_cpu_ms / (N - t->split), a);
    s->x = ema(s->x, t->t_xfer_ms, a);
    return VLA_OK;
}

int vla_scheduler_next(vla_scheduler* s, const vla_sched_state* z) {
    if (!s || !z) return -1;
    const vla_sched_config& c = s->cfg;
    if (s->g < 0.0 || s->c < 0.0) return s->k;  // a side never observed: no basis to move
    const int N = c.n_layers;
    const double g = s->g / (1.0 - clamp_u(z->u_gpu));
    const double cc = s->c / (1.0 - clamp_u(z->u_cpu));
    const double x = std::max(s->x, 0.0);
    auto interval = [&](int p) { return std::max(p * g, x + (N - p) * cc); };
    int best = s->k;
    double best_t = interval(best);
    for (int p = c.k_min; p <= c.k_max; ++p) {
        const double tp = interval(p);
        if (tp < best_t || (tp == best_t && std::abs(p - s->k) < std::abs(best - s->k))) {
            best = p;
            best_t = tp;
        }
    }
    int step = std::min(std::max(best - s->k, -c.max_step), c.max_step);
    if (step == 0 && z->backlog >= c.backlog_limit) {
        // frames pile up: move one block off the stage predicted to be slower
        step = (x + (N - s->k) * cc > s->k * g) ? 1 : -1;
    }
    s->k = std::min(std::max(s->k + step, c.k_min), c.k_max);
    return s->k;
}

vla_status vla_scheduler_estimates(const vla_scheduler* s, double* g_ms, double* c_ms, double* x_ms) {
    if (!s) return VLA_ERR_INVALID_ARG;
    if (g_ms) *g_ms = s->g;
    if (c_ms) *c_ms = s->c;
    if (x_ms) *x_ms = s->x;
    return VLA_OK;
}

vla_status vla_scheduler_destroy(vla_scheduler* s) {
    delete s;
    return VLA_OK;
}

}  // extern "C"
