// plan.cpp -- residency planning on the host (no GPU needed).
//
// Single-device form of LOIP's allocation (Sec. III-B to III-E):
//   * memory-first fill (Algorithm 1, initial allocation): keep the largest R
//     layers resident such that fixed + KV + R layers + the streaming slots
//     fit the budget; slots take the place of the paper's "one stage of
//     offloaded layers" term of the Eq. 1 memory constraint;
//   * interleaving (Sec. III-A): offloaded layers spread evenly among the
//     resident ones so every load gets an equal window of resident compute
//     (Eq. 2's T_idle with one device);
//   * step time: Eq. 1 with one device and no network term, and a
//     discrete-event model of the copy and compute streams with K slots;
//   * online threshold (Eq. 6): tokens the memory left after the plan holds;
//     past it one more layer is demoted (the resident layer in the middle of
//     the longest run of resident layers);
//   * block granularity (Algorithm 1's fine-grained step and Eq. 7): a layer is
//     an MHA block and an MLP block; memory left after the fill keeps blocks of
//     offloaded layers resident, and online growth offloads the combination of
//     resident blocks that covers the shortfall with the fewest bytes.
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <vector>

#include "../../include/loip.h"
#include "plan.h"

namespace loip {

bool memory_first_fill(int L, uint64_t l_size, uint64_t budget, uint64_t fixed, uint64_t kv, int n_slots, int* R) {
    if (fixed + kv > budget) return false;
    uint64_t free_b = budget - fixed - kv;
    if (free_b / l_size >= (uint64_t)L) {
        *R = L;
        return true;
    }
    uint64_t slots = (uint64_t)n_slots * l_size;
    if (free_b < slots) return false;
    uint64_t r = (free_b - slots) / l_size;
    *R = (int)std::min<uint64_t>(r, (uint64_t)L);
    return true;
}

void evenly_spaced(int L, int m, uint8_t* offloaded) {
    for (int l = 0; l < L; ++l) offloaded[l] = ((int64_t)(l + 1) * m) / L > ((int64_t)l * m) / L ? 1 : 0;
}

double eq1_single_device(const std::vector<double>& comp, const std::vector<double>& load, const uint8_t* off) {
    double tc = 0, tl = 0, ti = 0;
    for (size_t l = 0; l < comp.size(); ++l) {
        tc += comp[l];
        if (off[l])
            tl += load[l];
        else
            ti += comp[l];
    }
    return tc + std::max(tl - ti, 0.0);
}

double simulate_step(const std::vector<double>& comp, const std::vector<double>& load, const uint8_t* off, int K,
                     int n_steps) {
    const int L = (int)comp.size();
    std::vector<int> offl;
    for (int l = 0; l < L; ++l)
        if (off[l]) offl.push_back(l);
    const int m = (int)offl.size();
    double total = 0;
    for (double c : comp) total += c;
    if (m == 0) return total;
    if (K < 1) K = 1;
    // copy j (global order over steps) -> layer offl[j % m] of step j / m
    std::vector<double> copy_end((size_t)m * n_steps), comp_end_off((size_t)m * n_steps);
    double prev_copy = 0, t = 0, last_end = 0, prev_end = 0;
    int next_copy = 0;
    for (int s = 0; s < n_steps; ++s) {
        int j_in_step = 0;
        for (int l = 0; l < L; ++l) {
            double start = t;
            if (off[l]) {
                int j = s * m + j_in_step;
                while (next_copy <= j) {
                    double st = prev_copy;
                    if (next_copy - K >= 0) st = std::max(st, comp_end_off[next_copy - K]);
                    prev_copy = st + load[offl[next_copy % m]];
                    copy_end[next_copy] = prev_copy;
                    ++next_copy;
                }
                start = std::max(start, copy_end[j]);
                t = start + comp[l];
                comp_end_off[j] = t;
                ++j_in_step;
            } else {
                t = start + comp[l];
            }
        }
        prev_end = last_end;
        last_end = t;
    }
    return last_end - prev_end;
}

int demote_one(int L, uint8_t* off) {
    int m = 0;
    for (int l = 0; l < L; ++l) m += off[l];
    if (m == L) return -1;
    if (m == 0) {
        off[L - 1] = 1;
        return L - 1;
    }
    int best_start = -1, best_len = -1;
    for (int l = 0; l < L; ++l) {
        if (!off[l]) continue;
        // run of resident layers after offloaded layer l (cyclic)
        int len = 0;
        while (len < L && !off[(l + 1 + len) % L]) ++len;
        if (len > best_len) {
            best_len = len;
            best_start = (l + 1) % L;
        }
    }
    if (best_len <= 0) return -1;
    int victim = (best_start + (best_len - 1) / 2) % L;
    off[victim] = 1;
    return victim;
}

uint64_t refine_blocks(uint64_t left, int L, const uint8_t* offloaded, uint64_t mha_bytes, uint64_t mlp_bytes,
                       uint8_t* masks) {
    for (int l = 0; l < L; ++l) masks[l] = offloaded[l] ? 0 : 3;
    for (int l = 0; l < L; ++l) {
        if (masks[l] != 0) continue;
        if (left >= mlp_bytes) {  // keep the MLP block; the layer streams its MHA block only
            masks[l] = 2;
            left -= mlp_bytes;
        } else if (left >= mha_bytes) {  // keep the MHA block; the MLP block streams
            masks[l] = 1;
            left -= mha_bytes;
        } else {
            break;
        }
    }
    return left;
}

bool eq7_choice(uint64_t need, int n_mha, int n_mlp, uint64_t mha_bytes, uint64_t mlp_bytes, int* alpha, int* beta) {
    bool found = false;
    uint64_t best_bytes = 0;
    int best_blocks = 0;
    for (int a = 0; a <= n_mha; ++a) {
        const uint64_t covered = (uint64_t)a * mha_bytes;
        const uint64_t rest = need > covered ? need - covered : 0;
        const uint64_t b = rest == 0 ? 0 : (rest + mlp_bytes - 1) / mlp_bytes;
        if (b > (uint64_t)n_mlp) continue;
        const uint64_t bytes = covered + b * mlp_bytes;
        const int blocks = a + (int)b;
        if (!found || bytes < best_bytes || (bytes == best_bytes && blocks < best_blocks)) {
            found = true;
            best_bytes = bytes;
            best_blocks = blocks;
            *alpha = a;
            *beta = (int)b;
        }
    }
    return found;
}

}  // namespace loip

using namespace loip;

extern "C" int loip_refine_blocks(const loip_model_desc* desc, uint64_t left_bytes, const uint8_t* offloaded,
                                  uint8_t* masks, uint64_t* left_out) {
    if (!desc || !offloaded || !masks || !left_out || desc->n_layers <= 0) return LOIP_ERR_INVALID;
    loip_layer_layout_t lay;
    int rc = loip_layer_layout(desc, &lay);
    if (rc) return rc;
    *left_out = refine_blocks(left_bytes, desc->n_layers, offloaded, lay.mha_bytes, lay.mlp_bytes, masks);
    return LOIP_OK;
}

extern "C" int loip_eq7_choice(const loip_model_desc* desc, uint64_t need_bytes, int32_t n_mha, int32_t n_mlp,
                               int32_t* alpha, int32_t* beta) {
    if (!desc || !alpha || !beta || n_mha < 0 || n_mlp < 0) return LOIP_ERR_INVALID;
    loip_layer_layout_t lay;
    int rc = loip_layer_layout(desc, &lay);
    if (rc) return rc;
    int a = 0, b = 0;
    if (!eq7_choice(need_bytes, n_mha, n_mlp, lay.mha_bytes, lay.mlp_bytes, &a, &b)) return LOIP_ERR_INFEASIBLE;
    *alpha = a;
    *beta = b;
    return LOIP_OK;
}

extern "C" int loip_plan_residency(const loip_model_desc* desc, const uint64_t* layer_bytes, uint64_t device_budget,
                                   uint64_t kv_bytes, uint64_t fixed_bytes, int32_t n_slots, double hbm_Bps,
                                   double link_Bps, loip_plan* out) {
    if (!desc || !layer_bytes || !out || !out->resident || desc->n_layers <= 0 || n_slots < 1 || n_slots > 3 ||
        !(hbm_Bps > 0) || !(link_Bps > 0))
        return LOIP_ERR_INVALID;
    const int L = desc->n_layers;
    uint64_t l_size = 0;
    for (int l = 0; l < L; ++l) l_size = std::max(l_size, layer_bytes[l]);
    if (l_size == 0) return LOIP_ERR_INVALID;
    int R = 0;
    if (!memory_first_fill(L, l_size, device_budget, fixed_bytes, kv_bytes, n_slots, &R)) return LOIP_ERR_INFEASIBLE;
    const int m = L - R;
    evenly_spaced(L, m, out->resident);
    std::vector<double> comp(L), load(L);
    double tcopy = 0, tcomp = 0;
    for (int l = 0; l < L; ++l) {
        comp[l] = (double)layer_bytes[l] / hbm_Bps;
        load[l] = (double)layer_bytes[l] / link_Bps;
        tcomp += comp[l];
        if (out->resident[l]) tcopy += load[l];
    }
    out->pred_step_s = simulate_step(comp, load, out->resident, n_slots, 4);
    out->eq1_step_s = eq1_single_device(comp, load, out->resident);
    for (int l = 0; l < L; ++l) out->resident[l] = out->resident[l] ? 0 : 1;  // offloaded -> resident flag
    out->n_layers = L;
    out->n_resident = R;
    out->n_offloaded = m;
    out->pred_copy_s = tcopy;
    out->pred_compute_s = tcomp;
    uint64_t used = fixed_bytes + kv_bytes + (uint64_t)R * l_size + (m > 0 ? (uint64_t)n_slots * l_size : 0);
    out->left_bytes = device_budget >= used ? device_budget - used : 0;
    return LOIP_OK;
}

extern "C" int loip_kv_threshold(uint64_t left_bytes, uint64_t kv_bytes_per_token, uint64_t* out_tokens) {
    if (!out_tokens || kv_bytes_per_token == 0) return LOIP_ERR_INVALID;
    *out_tokens = left_bytes / kv_bytes_per_token;
    return LOIP_OK;
}
