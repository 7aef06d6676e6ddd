// Offline plan: row-impact factors, lifetime weights, FP16 pivots, Lifetime-aware
// Bit Allocation and the packed page layout (Sec. 3.2, Sec. 4.3, App. A.3,
// App. C.2, App. D). Host code; the result is uploaded once as device tables.
//
// The allocation rules must give bit-identical maps to any other faithful
// implementation, so their tie-breaking is fixed: the multiple-choice DP runs
// over units in reverse index order in 2-bit steps and keeps the wider code on
// exact ties; the Lagrangian keeps the narrower code on ties, bisects 60 times
// for the smallest feasible multiplier and then spends leftover bits greedily
// on the best objective reduction per bit (ties: lower unit, narrower code).
#include <algorithm>
#include <cmath>
#include <cstring>
#include <limits>
#include <numeric>

#include "internal.h"

namespace stepq {

stepq_status validate_config(const stepq_config *cfg, bool quant) {
    if (!cfg) return STEPQ_ERR_ARG;
    if (cfg->dk != kD || cfg->dv != kD) return STEPQ_ERR_UNSUPPORTED;
    if (cfg->n_layers <= 0 || cfg->n_key_heads <= 0 || cfg->n_value_heads <= 0) return STEPQ_ERR_ARG;
    if (cfg->n_value_heads % cfg->n_key_heads) return STEPQ_ERR_ARG;
    if (cfg->gate_kind != STEPQ_GATE_SCALAR && cfg->gate_kind != STEPQ_GATE_CHANNEL) return STEPQ_ERR_ARG;
    if (!quant) return STEPQ_OK;
    if (cfg->nominal_bits != 4 && cfg->nominal_bits != 6 && cfg->nominal_bits != 8) return STEPQ_ERR_ARG;
    if (cfg->n_candidates < 1 || cfg->n_candidates > 4) return STEPQ_ERR_ARG;
    for (int a = 0; a < cfg->n_candidates; a++) {
        int b = cfg->candidates[a];
        if (b != 2 && b != 4 && b != 6 && b != 8) return STEPQ_ERR_ARG;
        for (int c = 0; c < a; c++)
            if (cfg->candidates[c] == b) return STEPQ_ERR_ARG;
    }
    if (cfg->horizon < 1 || cfg->fit_iters < 1 || cfg->n_pivots < 0) return STEPQ_ERR_ARG;
    return STEPQ_OK;
}

static size_t units_of(const stepq_config *cfg) {
    size_t heads = (size_t)cfg->n_layers * cfg->n_value_heads;
    return cfg->gate_kind == STEPQ_GATE_CHANNEL ? heads * kD : heads;
}

// ---- Eq. allocation solvers -------------------------------------------------

// Exact multiple-choice knapsack over `cost` ([U][K]) with weights cands[k]/2
// and integer capacity. Returns false when nothing fits.
static bool solve_dp(const std::vector<double> &cost, size_t U, const std::vector<int> &cands,
                     long long capacity, std::vector<int> &pick) {
    if (capacity < 0) return false;
    const size_t K = cands.size(), C = (size_t)capacity + 1;
    std::vector<int> by_width(K);
    std::iota(by_width.begin(), by_width.end(), 0);
    std::stable_sort(by_width.begin(), by_width.end(),
                     [&](int a, int b) { return cands[a] > cands[b]; });
    std::vector<double> next(C, 0.0), cur(C);
    std::vector<int8_t> arg(U * C);
    for (size_t u = U; u-- > 0;) {
        for (size_t c = 0; c < C; c++) {
            double best = std::numeric_limits<double>::infinity();
            int bk = -1;
            for (int k : by_width) {
                size_t a = (size_t)(cands[k] / 2);
                if (a > c) continue;
                double val = cost[u * K + k] + next[c - a];
                if (val < best) { best = val; bk = k; }
            }
            cur[c] = best;
            arg[u * C + c] = (int8_t)bk;
        }
        std::swap(next, cur);
    }
    if (!std::isfinite(next[C - 1])) return false;
    pick.assign(U, 0);
    size_t c = C - 1;
    for (size_t u = 0; u < U; u++) {
        int k = arg[u * C + c];
        if (k < 0) return false;
        pick[u] = k;
        c -= (size_t)(cands[k] / 2);
    }
    return true;
}

static long long lagrange_pick(const std::vector<double> &cost, size_t U,
                               const std::vector<int> &cands, const std::vector<int> &asc,
                               double lam, std::vector<int> &pick) {
    const size_t K = cands.size();
    long long total = 0;
    for (size_t u = 0; u < U; u++) {
        double best = std::numeric_limits<double>::infinity();
        int bk = asc[0];
        for (int k : asc) {
            double val = cost[u * K + k] + lam * cands[k];
            if (val < best) { best = val; bk = k; }
        }
        pick[u] = bk;
        total += cands[bk];
    }
    return total;
}

static bool solve_lagrangian(const std::vector<double> &cost, size_t U,
                             const std::vector<int> &cands, long long budget,
                             std::vector<int> &pick) {
    const size_t K = cands.size();
    std::vector<int> asc(K);
    std::iota(asc.begin(), asc.end(), 0);
    std::stable_sort(asc.begin(), asc.end(), [&](int a, int b) { return cands[a] < cands[b]; });
    if ((long long)cands[asc[0]] * (long long)U > budget) return false;
    pick.assign(U, 0);
    double lam = 0.0;
    if (lagrange_pick(cost, U, cands, asc, 0.0, pick) > budget) {
        double lo = 0.0, hi = 1.0;
        for (int guard = 0; lagrange_pick(cost, U, cands, asc, hi, pick) > budget; guard++) {
            hi *= 2.0;
            if (guard > 2000 || !std::isfinite(hi)) return false;
        }
        for (int it = 0; it < 60; it++) {
            double mid = 0.5 * (lo + hi);
            if (lagrange_pick(cost, U, cands, asc, mid, pick) <= budget) hi = mid;
            else lo = mid;
        }
        lam = hi;
    }
    long long slack = budget - lagrange_pick(cost, U, cands, asc, lam, pick);
    // discrete repair: spend the remaining bits where they buy the most
    while (true) {
        long long bu = -1;
        int bk = -1;
        double best_ratio = -1.0;
        for (size_t u = 0; u < U; u++) {
            const int cur = pick[u];
            for (int k : asc) {
                long long db = cands[k] - cands[cur];
                if (db <= 0 || db > slack) continue;
                double gain = cost[u * K + cur] - cost[u * K + k];
                if (gain < 0.0) continue;
                double ratio = gain / (double)db;
                if (ratio > best_ratio) { best_ratio = ratio; bu = (long long)u; bk = k; }
            }
        }
        if (bu < 0) break;
        slack -= cands[bk] - cands[pick[bu]];
        pick[bu] = bk;
    }
    return true;
}

static int index_of(const std::vector<int> &cands, int b) {
    for (size_t k = 0; k < cands.size(); k++)
        if (cands[k] == b) return (int)k;
    return -1;
}

static stepq_status pivots_impl(const stepq_config *cfg, const std::vector<double> &life,
                                const double *dist, std::vector<uint8_t> &mask) {
    const size_t U = units_of(cfg);
    const size_t K = (size_t)cfg->n_candidates;
    std::vector<int> cands(cfg->candidates, cfg->candidates + K);
    mask.assign(U, 0);
    if (cfg->n_pivots == 0) return STEPQ_OK;
    if ((size_t)cfg->n_pivots > U) return STEPQ_ERR_ARG;
    std::vector<double> risk(U);
    if (cfg->gate_kind == STEPQ_GATE_SCALAR) {
        // residual allocation risk: allocate without pivots, weigh the error left
        std::vector<double> cost(U * K);
        for (size_t u = 0; u < U; u++)
            for (size_t k = 0; k < K; k++) cost[u * K + k] = life[u] * dist[u * (K + 1) + k];
        std::vector<int> pick;
        if (!solve_dp(cost, U, cands, (long long)(cfg->nominal_bits / 2) * (long long)U, pick))
            return STEPQ_ERR_BUDGET;
        for (size_t u = 0; u < U; u++) risk[u] = life[u] * dist[u * (K + 1) + pick[u]];
    } else {
        int kn = index_of(cands, cfg->nominal_bits);
        if (kn < 0) return STEPQ_ERR_ARG;
        for (size_t u = 0; u < U; u++)
            risk[u] = life[u] * (dist[u * (K + 1) + kn] - dist[u * (K + 1) + K]);
    }
    std::vector<size_t> order(U);
    std::iota(order.begin(), order.end(), 0);
    std::stable_sort(order.begin(), order.end(),
                     [&](size_t a, size_t b) { return risk[a] > risk[b]; });
    for (int p = 0; p < cfg->n_pivots; p++) mask[order[p]] = 1;
    return STEPQ_OK;
}

}  // namespace stepq

using namespace stepq;

extern "C" size_t stepq_num_units(const stepq_config *cfg) {
    return validate_config(cfg, false) == STEPQ_OK ? units_of(cfg) : 0;
}

extern "C" stepq_status stepq_row_weights(const stepq_config *cfg, const float *omega, float *w) {
    stepq_status st = validate_config(cfg, false);
    if (st != STEPQ_OK) return st;
    if (!omega || !w) return STEPQ_ERR_ARG;
    const size_t heads = (size_t)cfg->n_layers * cfg->n_value_heads;
    const double half_gamma = 0.125;            // gamma = 0.25
    for (size_t h = 0; h < heads; h++) {
        double lw[kD], mean = 0.0;
        for (int i = 0; i < kD; i++) {
            double om = omega[h * kD + i];
            lw[i] = half_gamma * std::log(om > 1e-30 ? om : 1e-30);
            mean += lw[i];
        }
        mean /= kD;
        for (int i = 0; i < kD; i++) w[h * kD + i] = (float)std::exp(lw[i] - mean);
    }
    return STEPQ_OK;
}

extern "C" double stepq_lifetime_weight(double ell, int H) {
    double L = 0.0;
    for (int j = 0; j < H; j++) L += std::exp(2.0 * j * ell);
    return L;
}

extern "C" stepq_status stepq_select_pivots(const stepq_config *cfg, const double *mean_log_ret,
                                            const double *distortion, uint8_t *mask_out) {
    stepq_status st = validate_config(cfg, true);
    if (st != STEPQ_OK) return st;
    if (!mean_log_ret || !distortion || !mask_out) return STEPQ_ERR_ARG;
    const size_t U = units_of(cfg);
    std::vector<double> life(U);
    for (size_t u = 0; u < U; u++) life[u] = stepq_lifetime_weight(mean_log_ret[u], cfg->horizon);
    std::vector<uint8_t> mask;
    st = pivots_impl(cfg, life, distortion, mask);
    if (st == STEPQ_OK) std::memcpy(mask_out, mask.data(), U);
    return st;
}

extern "C" stepq_status stepq_fit_scales(const stepq_config *cfg, const stepq_calib *cal,
                                         stepq_plan **out) {
    if (!out) return STEPQ_ERR_ARG;
    *out = nullptr;
    stepq_status st = validate_config(cfg, true);
    if (st != STEPQ_OK) return st;
    if (!cal || !cal->omega || !cal->mean_log_ret || !cal->distortion) return STEPQ_ERR_ARG;
    auto *p = new stepq_plan();
    p->cfg = *cfg;
    const size_t U = units_of(cfg), K = (size_t)cfg->n_candidates;
    const size_t heads = (size_t)cfg->n_layers * cfg->n_value_heads;
    const bool rows = cfg->gate_kind == STEPQ_GATE_CHANNEL;
    p->n_units = U;
    p->w.resize(heads * kD);
    stepq_row_weights(cfg, cal->omega, p->w.data());
    p->life.resize(U);
    for (size_t u = 0; u < U; u++)
        p->life[u] = stepq_lifetime_weight(cal->mean_log_ret[u], cfg->horizon);
    if (cal->pivot_mask) {
        p->pivot.assign(cal->pivot_mask, cal->pivot_mask + U);
        for (auto &m : p->pivot) m = m ? 1 : 0;
    } else if ((st = pivots_impl(cfg, p->life, cal->distortion, p->pivot)) != STEPQ_OK) {
        delete p;
        return st;
    }
    // Lifetime-aware Bit Allocation over the integer units; pivots count as
    // 8-bit replacements against the nominal budget (App. D).
    std::vector<int> cands(cfg->candidates, cfg->candidates + K);
    std::vector<size_t> idx;
    for (size_t u = 0; u < U; u++)
        if (!p->pivot[u]) idx.push_back(u);
    const long long n_piv = (long long)(U - idx.size());
    std::vector<double> cost(idx.size() * K);
    for (size_t t = 0; t < idx.size(); t++)
        for (size_t k = 0; k < K; k++)
            cost[t * K + k] = p->life[idx[t]] * cal->distortion[idx[t] * (K + 1) + k];
    std::vector<int> pick;
    bool ok = rows ? solve_lagrangian(cost, idx.size(), cands,
                                      (long long)cfg->nominal_bits * (long long)U - 8 * n_piv, pick)
                   : solve_dp(cost, idx.size(), cands,
                              (long long)(cfg->nominal_bits / 2) * (long long)U - 4 * n_piv, pick);
    if (!ok) {
        delete p;
        return STEPQ_ERR_BUDGET;
    }
    p->unit_bits.assign(U, (int8_t)kPivot);
    for (size_t t = 0; t < idx.size(); t++) p->unit_bits[idx[t]] = (int8_t)cands[pick[t]];

    // Packed layout: head segments in (layer, head) order, stride rounded to 256 B.
    std::vector<uint8_t> head_bits(heads), row_bits(heads * kD);
    std::vector<uint32_t> row_off(heads * kD), row_slot(heads * kD, 0);
    p->head_off.resize(heads);
    p->head_bytes.resize(heads);
    uint64_t off = 0;
    for (size_t h = 0; h < heads; h++) {
        uint32_t bytes;
        if (!rows) {
            int b = p->unit_bits[h];
            head_bits[h] = (uint8_t)b;
            for (int i = 0; i < kD; i++) {
                row_bits[h * kD + i] = (uint8_t)b;
                row_off[h * kD + i] = b == kPivot ? 256u * i : 512u + 16u * b * i;
            }
            bytes = b == kPivot ? 256u * kD : 512u + 16u * b * kD;
        } else {
            // rows by decreasing width, equal widths in index order; slot s of
            // the head is the s-th row stored: offset | width << 16 | row << 24
            head_bits[h] = 0;
            int order[kD];
            for (int i = 0; i < kD; i++) {
                order[i] = i;
                row_bits[h * kD + i] = (uint8_t)p->unit_bits[h * kD + i];
            }
            std::stable_sort(order, order + kD,
                             [&](int x, int y) { return row_bits[h * kD + x] > row_bits[h * kD + y]; });
            bytes = 512;
            for (int s = 0; s < kD; s++) {
                const int i = order[s], b = row_bits[h * kD + i];
                row_off[h * kD + i] = bytes;
                row_slot[h * kD + s] = bytes | ((uint32_t)b << 16) | ((uint32_t)i << 24);
                bytes += 16u * b;
            }
        }
        p->head_off[h] = off;
        p->head_bytes[h] = bytes;
        p->max_head_bytes = std::max(p->max_head_bytes, bytes);
        off += bytes;
    }
    p->slot_stride = (size_t)((off + 255) / 256 * 256);

    // "Temporal only" layout: s[128] fp16, then row i (index order) in 16 b_i bytes.
    std::vector<uint32_t> t_row_off(heads * kD);
    p->t_head_off.resize(heads);
    uint64_t t_off = 0;
    for (size_t h = 0; h < heads; h++) {
        uint32_t bytes = 256;
        for (int i = 0; i < kD; i++) {
            t_row_off[h * kD + i] = bytes;
            bytes += 16u * row_bits[h * kD + i];
        }
        p->t_head_off[h] = t_off;
        t_off += bytes;
    }
    p->t_slot_stride = (size_t)((t_off + 255) / 256 * 256);

    // Device tables.
    std::vector<float> w2(heads * kD), wis(heads * kD);
    for (size_t t = 0; t < heads * kD; t++) {
        double wv = p->w[t];
        w2[t] = (float)(wv * wv);
        wis[t] = (float)(1.0 / std::sqrt(wv));
    }
    auto align = [](size_t x) { return (x + 255) / 256 * 256; };
    size_t o_w2 = 0, o_wis = align(o_w2 + heads * kD * 4), o_off = align(o_wis + heads * kD * 4),
           o_hb = align(o_off + heads * 8), o_hbits = align(o_hb + heads * 4),
           o_rbits = align(o_hbits + heads), o_roff = align(o_rbits + heads * kD),
           o_rslot = align(o_roff + heads * kD * 4), o_thoff = align(o_rslot + heads * kD * 4),
           o_troff = align(o_thoff + heads * 8), total = align(o_troff + heads * kD * 4);
    std::vector<uint8_t> host(total, 0);
    std::memcpy(host.data() + o_w2, w2.data(), heads * kD * 4);
    std::memcpy(host.data() + o_wis, wis.data(), heads * kD * 4);
    std::memcpy(host.data() + o_off, p->head_off.data(), heads * 8);
    std::memcpy(host.data() + o_hb, p->head_bytes.data(), heads * 4);
    std::memcpy(host.data() + o_hbits, head_bits.data(), heads);
    std::memcpy(host.data() + o_rbits, row_bits.data(), heads * kD);
    std::memcpy(host.data() + o_roff, row_off.data(), heads * kD * 4);
    std::memcpy(host.data() + o_rslot, row_slot.data(), heads * kD * 4);
    std::memcpy(host.data() + o_thoff, p->t_head_off.data(), heads * 8);
    std::memcpy(host.data() + o_troff, t_row_off.data(), heads * kD * 4);
    int n_dev = 0;
    if (cudaGetDeviceCount(&n_dev) != cudaSuccess || n_dev == 0) {
        cudaGetLastError();          // host-only plan: its device calls return STEPQ_ERR_CUDA
        p->device = -1;
        *out = p;
        return STEPQ_OK;
    }
    if (cudaGetDevice(&p->device) != cudaSuccess || cudaMalloc(&p->dev_mem, total) != cudaSuccess ||
        cudaMemcpy(p->dev_mem, host.data(), total, cudaMemcpyHostToDevice) != cudaSuccess) {
        if (p->dev_mem) cudaFree(p->dev_mem);
        delete p;
        return STEPQ_ERR_CUDA;
    }
    uint8_t *base = (uint8_t *)p->dev_mem;
    p->d_w2 = (float *)(base + o_w2);
    p->d_wis = (float *)(base + o_wis);
    p->d_head_off = (uint64_t *)(base + o_off);
    p->d_head_bytes = (uint32_t *)(base + o_hb);
    p->d_head_bits = base + o_hbits;
    p->d_row_bits = base + o_rbits;
    p->d_row_off = (uint32_t *)(base + o_roff);
    p->d_row_slot = (uint32_t *)(base + o_rslot);
    p->d_t_head_off = (uint64_t *)(base + o_thoff);
    p->d_t_row_off = (uint32_t *)(base + o_troff);
    *out = p;
    return STEPQ_OK;
}

extern "C" stepq_status stepq_plan_query(const stepq_plan *p, stepq_plan_info *info) {
    if (!p || !info) return STEPQ_ERR_ARG;
    info->slot_stride = p->slot_stride;
    info->n_units = p->n_units;
    info->unit_bits = p->unit_bits.data();
    info->pivot_mask = p->pivot.data();
    info->w = p->w.data();
    info->lifetime = p->life.data();
    info->head_offset = p->head_off.data();
    info->head_bytes = p->head_bytes.data();
    return STEPQ_OK;
}

extern "C" void stepq_plan_destroy(stepq_plan *p) {
    if (!p) return;
    if (p->dev_mem) {
        int cur = 0;
        cudaGetDevice(&cur);
        cudaSetDevice(p->device);
        cudaFree(p->dev_mem);
        cudaSetDevice(cur);
    }
    delete p;
}
