// K9: Adam on the active block only (Section 2: gradients reach theta_active only; frozen
// blocks are never touched).  torch semantics with bias correction, dense over every
// parameter of the block: m = b1 m + (1 - b1) g, v = b2 v + (1 - b2) g^2,
// theta -= (lr / (1 - b1^t)) m / (sqrt(v) / sqrt(1 - b2^t) + eps).
// HBM-bound: 4 reads and 3 writes of 4 bytes per parameter; one grid-stride pass over groups of
// four elements of the five parameter arrays (16-byte accesses; the SH array carries two
// learning rates, degree 0 and the rest).
#include <cmath>

#include "abcd_internal.cuh"

namespace abcd {
namespace {

struct Seg {
  float* th;
  const float* g;
  float* m;
  float* v;
  unsigned n;          // elements
  unsigned period;     // SH: 3 * D (degree-0 entries are the first 3 of each period); else 0
  float step_lr;       // lr / (1 - b1^t)
  float step_lr_rest;  // the SH coefficients of degree >= 1
  int vec;             // all four pointers 16-byte aligned: float4 groups
};

struct AdamArgs {
  Seg s[5];
  unsigned gstart[6];  // first group of each array (groups of 4 elements)
  float b1, b2, eps, inv_sqrt_bc2;
};

__device__ __forceinline__ float adam_one(float& th, float g, float& m, float& v, float lr,
                                          const AdamArgs& a) {
  m = a.b1 * m + (1.f - a.b1) * g;
  v = a.b2 * v + (1.f - a.b2) * g * g;
  th -= lr * m / (sqrtf(v) * a.inv_sqrt_bc2 + a.eps);
  return th;
}

// One thread per group of four consecutive elements of one array (float4 loads and stores when
// the array allows, else scalar), grid-stride over the groups of the five arrays.
__global__ void __launch_bounds__(256) adam_kernel(const __grid_constant__ AdamArgs a) {
  pdl_prologue();
  const unsigned total = a.gstart[5];
  for (unsigned q = blockIdx.x * blockDim.x + threadIdx.x; q < total; q += gridDim.x * blockDim.x) {
    int k = 0;
#pragma unroll
    for (int j = 1; j < 5; ++j) k += (q >= a.gstart[j]) ? 1 : 0;
    const Seg& s = a.s[k];
    const unsigned i0 = 4u * (q - a.gstart[k]);
    float lr[4];
    {
      unsigned r = s.period ? i0 % s.period : 0u;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        lr[c] = (s.period && r >= 3u) ? s.step_lr_rest : s.step_lr;
        if (s.period && ++r == s.period) r = 0u;
      }
    }
    if (s.vec && i0 + 4 <= s.n) {
      float4 th = *reinterpret_cast<const float4*>(s.th + i0);
      const float4 g = *reinterpret_cast<const float4*>(s.g + i0);
      float4 m = *reinterpret_cast<const float4*>(s.m + i0);
      float4 v = *reinterpret_cast<const float4*>(s.v + i0);
      adam_one(th.x, g.x, m.x, v.x, lr[0], a);
      adam_one(th.y, g.y, m.y, v.y, lr[1], a);
      adam_one(th.z, g.z, m.z, v.z, lr[2], a);
      adam_one(th.w, g.w, m.w, v.w, lr[3], a);
      *reinterpret_cast<float4*>(s.m + i0) = m;
      *reinterpret_cast<float4*>(s.v + i0) = v;
      *reinterpret_cast<float4*>(s.th + i0) = th;
    } else {
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const unsigned i = i0 + c;
        if (i < s.n) {
          float th = s.th[i], m = s.m[i], v = s.v[i];
          adam_one(th, s.g[i], m, v, lr[c], a);
          s.m[i] = m;
          s.v[i] = v;
          s.th[i] = th;
        }
      }
    }
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
  long long groups = 0;
  for (int k = 0; k < 5; ++k) groups += (len[k] + 3) / 4;
  if (len[4] >= (1LL << 32) || groups >= (1LL << 32))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_adam_active: too many parameters");
  a.gstart[0] = 0;
  for (int k = 0; k < 5; ++k) {
    const bool vec = (((uintptr_t)th[k] | (uintptr_t)gg[k] | (uintptr_t)mm[k] | (uintptr_t)vv[k]) & 15) == 0;
    a.s[k] = Seg{th[k], gg[k], mm[k], vv[k], (unsigned)len[k], k == 4 ? (unsigned)(3 * D) : 0u,
                 (float)(lr[k] / bc1), (float)((k == 4 ? lr[5] : lr[k]) / bc1), vec ? 1 : 0};
    a.gstart[k + 1] = a.gstart[k] + (unsigned)((len[k] + 3) / 4);
  }
  a.b1 = beta1;
  a.b2 = beta2;
  a.eps = eps;
  a.inv_sqrt_bc2 = (float)(1.0 / std::sqrt(bc2));
  const long long blocks = std::min<long long>((a.gstart[5] + 255) / 256, (long long)ctx->num_sms * 16);
  return check_launch(ctx, "adam_kernel",
                      launch_pdl(adam_kernel, dim3((unsigned)blocks), dim3(256), 0, ctx->stream, a));
}
