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
}  // namespace loip
