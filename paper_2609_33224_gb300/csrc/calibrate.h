// Online calibration of the decode model (Section 5.3), host side: one multiplicative EMA factor
// per decode-batch segment scales the decode term of every TPOT prediction.  Plain C++ (no CUDA),
// compiled without floating-point contraction, so each operation below is one IEEE fp32 rounding.
#pragma once

#include <cstdint>

namespace pscal {

// Feeds n pure-decode samples in order.  Sample k: measured batch size batch[k], total context
// tokens ctx_tokens[k], measured forward duration measured_ms[k].  The base model's prediction at
// the same batch size and context is (b0 + b1 B) + b2 S; the measured-to-predicted ratio, clipped to
// [0.5, 2], pulls the factor of B's segment (the last segment whose lower bound is <= B) by the
// update weight: f <- f + weight (ratio - f), and the factor is clipped to [1, 2].
inline void ema_update(float b0, float b1, float b2, int nseg, const int32_t* seg_lo, float* factor, uint64_t n,
                       const int32_t* batch, const int64_t* ctx_tokens, const float* measured_ms, float weight) {
  for (uint64_t k = 0; k < n; ++k) {
    const int64_t B = batch[k];
    const float pred = (b0 + b1 * (float)B) + b2 * (float)ctx_tokens[k];
    float ratio = measured_ms[k] / pred;
    ratio = ratio < 0.5f ? 0.5f : (ratio > 2.0f ? 2.0f : ratio);
    int seg = 0;
    for (int s = 0; s < nseg; ++s)
      if ((int64_t)seg_lo[s] <= B) seg = s;
    float f = factor[seg] + weight * (ratio - factor[seg]);
    f = f < 1.0f ? 1.0f : (f > 2.0f ? 2.0f : f);
    factor[seg] = f;
  }
}

}  // namespace pscal
