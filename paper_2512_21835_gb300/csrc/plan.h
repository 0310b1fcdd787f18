// plan.h -- host-side residency planning helpers (see plan.cpp).
#pragma once
#include <stdint.h>

#include <vector>

namespace loip {
// largest resident count R with fixed + kv + R*l + K*l <= budget (no slots
// when all layers fit); false if even the slots do not fit.
bool memory_first_fill(int L, uint64_t l_size, uint64_t budget, uint64_t fixed, uint64_t kv, int n_slots, int* R);
// offloaded[l] = 1 for m of L layers spread evenly
void evenly_spaced(int L, int m, uint8_t* offloaded);
double eq1_single_device(const std::vector<double>& comp, const std::vector<double>& load, const uint8_t* off);
double simulate_step(const std::vector<double>& comp, const std::vector<double>& load, const uint8_t* off, int K,
                     int n_steps);
// marks one more layer offloaded (middle of the longest resident run); returns it or -1
int demote_one(int L, uint8_t* off);
// Algorithm 1's block-level refinement on one device: masks[l] = resident blocks
// of layer l (bit 0 MHA, bit 1 MLP); returns the memory still left
uint64_t refine_blocks(uint64_t left, int L, const uint8_t* offloaded, uint64_t mha_bytes, uint64_t mlp_bytes,
                       uint8_t* masks);
// Eq. 7 on one device: alpha MHA and beta MLP blocks covering `need` with the
// fewest bytes (then the fewest blocks); false if the available blocks cannot
bool eq7_choice(uint64_t need, int n_mha, int n_mlp, uint64_t mha_bytes, uint64_t mlp_bytes, int* alpha, int* beta);
}  // namespace loip
