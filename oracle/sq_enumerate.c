/*
 * sq_enumerate.c -- exhaustive-enumeration harness for the accept rule.
 *
 * TEST INFRASTRUCTURE ONLY.  It calls nothing but the public oq_accept of
 * the oracle: for one sequence it sweeps one uniform over every point of
 * the grid m * 2^-grid_bits (m = 0 .. 2^grid_bits - 1) and histograms the
 * outcome.  Tests combine such sweeps with the draft probabilities to get
 * the exact distribution of emitted tokens (Sec. III-D.4, Sec. I).
 */
#include "sq_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

int oq_enum_sweep(const float* p, const float* q, const int32_t* draft,
                  const float* u_fixed, int64_t K, int64_t V, int mode,
                  int pos, int grid_bits, uint64_t* hist) {
  if (pos < 0 || pos > K || grid_bits < 1 || grid_bits > 24) return OQ_BAD_ARG;
  const int64_t nbins = (K + 1) * V + 1;
  memset(hist, 0, (size_t)nbins * sizeof(uint64_t));
  const int64_t npts = (int64_t)1 << grid_bits;
  int status = OQ_OK;
#pragma omp parallel
  {
    uint64_t* local = (uint64_t*)calloc((size_t)nbins, sizeof(uint64_t));
    float* u = (float*)malloc((size_t)(K + 1) * sizeof(float));
    int32_t* tok = (int32_t*)malloc((size_t)(K + 1) * sizeof(int32_t));
    int32_t n;
    memcpy(u, u_fixed, (size_t)(K + 1) * sizeof(float));
#pragma omp for schedule(static)
    for (int64_t m = 0; m < npts; ++m) {
      u[pos] = (float)ldexp((double)m, -grid_bits);
      oq_accept(p, q, draft, u, 1, K, V, mode, &n, tok);
      if (n < 0) local[(K + 1) * V] += 1;
      else local[n * V + tok[n]] += 1;
    }
#pragma omp critical
    {
      for (int64_t i = 0; i < nbins; ++i) hist[i] += local[i];
    }
    free(local);
    free(u);
    free(tok);
  }
  return status;
}
