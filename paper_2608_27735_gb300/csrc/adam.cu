// K9: Adam on the active block only (Section 2: gradients reach theta_active only; frozen
// blocks are never touched).  torch semantics with bias correction, dense over every
// parameter of the block: m = b1 m + (1 - b1) g, v = b2 v + (1 - b2) g^2,
// theta -= (lr / (1 - b1^t)) m / (sqrt(v) / sqrt(1 - b2^t) + eps).
// HBM-bound: 4 reads and 3 writes of 4 bytes per parameter; one grid-stride pass over the
// five parameter arrays (the SH array carries two learning rates, degree 0 and the rest).
#include <cmath>

#include "abcd_internal.cuh"

namespace abcd {
namespace {

struct Seg {
  float* th;
  const float* g;
  float* m;
  float* v;
  long long n;
  int period;      // SH: 3 * D (degree-0 entries are the first 3 of each period); else 0
  float step_lr;   // lr / (1 - b1^t)
  float step_lr_rest;
};

struct AdamArgs {
  Seg s[5];
  long long start[6];
  float b1, b2, eps, inv_sqrt_bc2;
};

__global__ void __launch_bounds__(256) adam_kernel(const __grid_constant__ AdamArgs a) {
  pdl_prologue();
  const long long total = a.start[5];
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    int k = 0;
#pragma unroll
    for (int j = 1; j < 5; ++j) k += (e >= a.start[j]) ? 1 : 0;
    const Seg& s = a.s[k];
    const long long i = e - a.start[k];
    const float g = s.g[i];
    const float m = a.b1 * s.m[i] + (1.f - a.b1) * g;
    const float v = a.b2 * s.v[i] + (1.f - a.b2) * g * g;
    s.m[i] = m;
    s.v[i] = v;
    const float lr = (s.period > 0 && (i % s.period) >= 3) ? s.step_lr_rest : s.step_lr;
    s.th[i] -= lr * m / (sqrtf(v) * a.inv_sqrt_bc2 + a.eps);
  }
}

bool same_shape(const abcd_gaussians* a, const abcd_gaussians* b) {
  return a && b && a->n == b->n && a->sh_degree == b->sh_degree && a->means && b->means &&
         a->log_scales && b->log_scales && a->quats && b->quats && a->opacity_logits &&
         b->opacity_logits && a->sh && b->sh;
}

}  // namespace
}  // namespace abcd

using namespace abcd;

extern "C" abcd_status abcd_adam_active(abcd_ctx* ctx, abcd_gaussians* theta,
                                        const abcd_gaussians* grads, abcd_gaussians* m,
                                        abcd_gaussians* v, const float lr[6], float beta1,
                                        float beta2, float eps, int step) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!theta || theta->n < 0 || theta->sh_degree < 0 || theta->sh_degree > 3)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_adam_active: bad theta");
  if (theta->n == 0) return ABCD_OK;
  if (!same_shape(theta, grads) || !same_shape(theta, m) || !same_shape(theta, v) || !lr ||
      step < 1 || !(beta1 >= 0.f && beta1 < 1.f) || !(beta2 >= 0.f && beta2 < 1.f) || !(eps >= 0.f))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_adam_active: bad arguments");
  const double bc1 = 1.0 - std::pow((double)beta1, step);
  const double bc2 = 1.0 - std::pow((double)beta2, step);
  const long long n = theta->n;
  const int D = (theta->sh_degree + 1) * (theta->sh_degree + 1);
  AdamArgs a;
  float* th[5] = {theta->means, theta->log_scales, theta->quats, theta->opacity_logits, theta->sh};
  const float* gg[5] = {grads->means, grads->log_scales, grads->quats, grads->opacity_logits, grads->sh};
  float* mm[5] = {m->means, m->log_scales, m->quats, m->opacity_logits, m->sh};
  float* vv[5] = {v->means, v->log_scales, v->quats, v->opacity_logits, v->sh};
  const long long len[5] = {3 * n, 3 * n, 4 * n, n, 3LL * D * n};
  a.start[0] = 0;
  for (int k = 0; k < 5; ++k) {
    a.s[k] = Seg{th[k], gg[k], mm[k], vv[k], len[k], k == 4 ? 3 * D : 0,
                 (float)(lr[k] / bc1), (float)((k == 4 ? lr[5] : lr[k]) / bc1)};
    a.start[k + 1] = a.start[k] + len[k];
  }
  a.b1 = beta1;
  a.b2 = beta2;
  a.eps = eps;
  a.inv_sqrt_bc2 = (float)(1.0 / std::sqrt(bc2));
  const long long blocks = std::min<long long>((a.start[5] + 255) / 256, (long long)ctx->num_sms * 16);
  return check_launch(ctx, "adam_kernel",
                      launch_pdl(adam_kernel, dim3((unsigned)blocks), dim3(256), 0, ctx->stream, a));
}
