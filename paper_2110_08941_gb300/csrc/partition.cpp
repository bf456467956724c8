// Host-side sizing rule of Dynamic Partitioning (Section 4.1, Algorithm 1; Eq. 2).
//
// Algorithm 1 normalises the compute powers CP_m and sets |D^m_{t+1}| = CP_m * |D|.
// That product is real; the integer sizes here use largest-remainder rounding in
// fp64 with a fixed operation order (normalise, then multiply), equal remainders
// to the lower worker index, and a final pass that gives every empty worker one
// sample from the currently largest worker (lower index on ties), so that every
// worker has a defined mean loss (Eq. 1).  Compiled with -ffp-contract=off so the
// fp64 arithmetic is the same on every host ISA.
#include <cmath>
#include <cstdint>
#include <vector>

#include "../../include/hs.h"

namespace hs {

// Returns HS_OK and fills sizes[M] / quota_norm[M] (normalised CP), or an error.
hs_status partition_sizes_impl(int32_t M, int32_t N, const double* cp, int32_t* sizes,
                               double* cp_norm, const char** why) {
  if (M < 1) { *why = "M must be >= 1"; return HS_ERR_INVALID_ARG; }
  if (N < M) { *why = "global batch N must be >= M (every worker needs a sample)"; return HS_ERR_INVALID_ARG; }
  if (!cp || !sizes) { *why = "null pointer"; return HS_ERR_INVALID_ARG; }
  for (int32_t m = 0; m < M; ++m) {
    const double c = cp[m];
    if (!std::isfinite(c) || !(c > 0.0)) { *why = "compute power must be finite and > 0"; return HS_ERR_INVALID_ARG; }
  }
  double s = 0.0;
  for (int32_t m = 0; m < M; ++m) s = s + cp[m];
  if (!std::isfinite(s)) { *why = "sum of compute powers overflows"; return HS_ERR_INVALID_ARG; }
  std::vector<double> rem(M);
  int64_t floor_sum = 0;
  for (int32_t m = 0; m < M; ++m) {
    const double norm = cp[m] / s;
    if (cp_norm) cp_norm[m] = norm;
    const double q = norm * static_cast<double>(N);
    const double f = std::floor(q);
    sizes[m] = static_cast<int32_t>(f);
    rem[m] = q - f;
    floor_sum += static_cast<int64_t>(f);
  }
  const int64_t r = static_cast<int64_t>(N) - floor_sum;
  if (r < 0 || r > M) { *why = "rounding residue out of range"; return HS_ERR_INVALID_ARG; }
  // Hand out r extra samples: repeatedly pick the largest remainder not yet taken,
  // lowest index first among equals (a stable selection, O(M^2), M is small).
  std::vector<char> taken(M, 0);
  for (int64_t k = 0; k < r; ++k) {
    int32_t best = -1;
    for (int32_t m = 0; m < M; ++m) {
      if (taken[m]) continue;
      if (best < 0 || rem[m] > rem[best]) best = m;
    }
    taken[best] = 1;
    sizes[best] += 1;
  }
  for (int32_t m = 0; m < M; ++m) {
    if (sizes[m] != 0) continue;
    int32_t donor = 0;
    for (int32_t j = 1; j < M; ++j)
      if (sizes[j] > sizes[donor]) donor = j;
    sizes[donor] -= 1;
    sizes[m] += 1;
  }
  return HS_OK;
}

}  // namespace hs

extern "C" hs_status hs_partition_sizes(int32_t M, int32_t N, const double* cp, int32_t* counts_out) {
  const char* why = nullptr;
  if (M < 1 || M > (1 << 20)) return HS_ERR_INVALID_ARG;
  std::vector<double> norm(static_cast<size_t>(M));
  return hs::partition_sizes_impl(M, N, cp, counts_out, norm.data(), &why);
}
