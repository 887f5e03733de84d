// Eq. 14's beta search (prep_beta.cu): the factors of Eq. 3 at one beta (W_d
// fp32 [E, r]; Q(W^u) codes and per-column scales), and the objective
// sum (Y - Q(C) Q(W^u))^2 over calibration tokens (partials: one fp64 per
// 64 x 64 tile, beta_objective_partials of them).
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace qsvd {

cudaError_t launch_beta_factors(const double *Wd_r, const double *Wu_r, const double *fd, const double *fu, int E,
                                int r, int n_out, int u_bits, float u_clip, float *W_d, void *u_codes, float *u_scale,
                                cudaStream_t s);
size_t beta_objective_partials(int64_t N, int n_out);
cudaError_t launch_beta_objective(const float *Y, int64_t N, int n_out, const void *lat_codes, const void *lat_scales,
                                  int lat_bits, int r, const void *u_codes, const float *u_scale, int u_bits,
                                  double *partial, double *objective, cudaStream_t s);

}  // namespace qsvd
