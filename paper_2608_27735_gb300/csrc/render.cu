// K5 (blend + composite forward, also the cache refresh K10) and K7 (its backward).
//
// Per pixel, front to back over its tile's list (3DGS blending): sigma = 1/2 d^T Q d with
// d = pixel centre - uv, alpha = min(alpha_max, o exp(-sigma)), skip alpha < alpha_min (and
// sigma < 0), stop before T (1 - alpha) < t_min; A = (sum T_i alpha_i c_i, 1 - T).  Then the
// frozen partitions enter through out = F over (A over B) (Section 2), over meaning
// X + (1 - X.a) Y on premultiplied RGBA, and out.rgb += (1 - out.a) bg.
//
// One CTA per 8x8 block of pixels (four per 16x16 binning tile), one thread per pixel, so the
// few heavily covered tiles of a small active block spread over four times as many CTAs and
// each CTA stops as soon as its own 64 pixels have terminated (__syncthreads_count).  List
// entries are staged 256 at a time in shared memory; while staging, an entry whose opacity
// cannot reach alpha_min anywhere on the CTA's pixel-centre box (analytic minimum of the
// quadratic form over the box, with a margin far above fp32 rounding) is dropped: every pixel
// would skip it, so results are unchanged.  Every quantity that decides a branch per pixel
// (sigma, alpha, T) is computed with explicit round-to-nearest intrinsics in one shared
// function, so the backward kernel retraces exactly the forward's contributors.
#include "abcd_internal.cuh"

namespace abcd {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kHalfLog2e = 0.7213475204444817f;
constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Conic scaled for base-2 exponentials: (a/2, b, c/2) * log2(e), opacity kept.
__device__ __forceinline__ float4 scaled_conic(float4 c) {
  return make_float4(__fmul_rn(kHalfLog2e, c.x), __fmul_rn(kLog2e, c.y), __fmul_rn(kHalfLog2e, c.z), c.w);
}

// sigma * log2(e) = dx (a/2 dx + b dy) + c/2 dy^2 in log2 units; dx, dy returned.
__device__ __forceinline__ float sigma2(float4 s, float2 m, float fx, float fy, float& dx, float& dy) {
  dx = __fsub_rn(fx, m.x);
  dy = __fsub_rn(fy, m.y);
  return __fmaf_rn(dx, __fmaf_rn(s.x, dx, __fmul_rn(s.y, dy)), __fmul_rn(__fmul_rn(s.z, dy), dy));
}

constexpr int kSub = 8;                          // CTA pixel block edge
constexpr int kSubThreads = kSub * kSub;         // 64
constexpr int kSubPerTile = (kTile / kSub) * (kTile / kSub);
constexpr int kRounds = 4;                       // list entries per thread per batch
constexpr int kBatch = kSubThreads * kRounds;    // 256

// Lower bound of sigma * log2(e) over the box [X0, X1] x [Y0, Y1] of offsets d = pixel - uv:
// 0 if the box contains d = 0, else the least value on its four edges (convex quadratic).
__device__ __forceinline__ float box_min_sigma2(float4 s, float X0, float X1, float Y0, float Y1) {
  if (X0 <= 0.f && X1 >= 0.f && Y0 <= 0.f && Y1 >= 0.f) return 0.f;
  float best = 3.0e38f;
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const float X = e ? X1 : X0;
    const float dy = fminf(fmaxf(-s.y * X / (2.f * s.z), Y0), Y1);
    best = fminf(best, X * (s.x * X + s.y * dy) + s.z * dy * dy);
    const float Y = e ? Y1 : Y0;
    const float dx = fminf(fmaxf(-s.y * Y / (2.f * s.x), X0), X1);
    best = fminf(best, dx * (s.x * dx + s.y * Y) + s.z * Y * Y);
  }
  return best;
}

// True when no pixel centre of the CTA's box can give alpha >= alpha_min: alpha = o 2^-sigma'
// < alpha_min needs sigma' > log2(o / alpha_min); the margin (0.02 + 0.2% in log2 units) is
// orders of magnitude above the fp32 error of either evaluation.
__device__ __forceinline__ bool cull(float4 s, float2 m, float bx0, float by0, float alpha_min) {
  if (!(s.w >= alpha_min)) return true;
  const float thr = __log2f(s.w / alpha_min);
  const float lo = box_min_sigma2(s, bx0 - m.x, bx0 + (kSub - 1) - m.x, by0 - m.y, by0 + (kSub - 1) - m.y);
  return lo * 0.998f > thr + 0.02f;
}

// Adds the warp-wide sums of v[0..9) to dst[0..9).  Transpose reduction: at each step a lane
// keeps half of its (padded to 16) partial sums and receives the partner's matching half, so
// 16 shuffles replace the 45 of a butterfly per value; afterwards lanes 2c, 2c + 1 hold the
// sum of component c = lane / 2 (bits 4..1), and lane 2c adds it to memory.
__device__ __forceinline__ void warp_sum9_atomic(const float v[9], float* dst, int lane) {
  float x[16];
#pragma unroll
  for (int k = 0; k < 16; ++k) x[k] = k < 9 ? v[k] : 0.f;
#pragma unroll
  for (int w = 8; w >= 1; w >>= 1) {       // halves of 16, 8, 4, 2 values; lane bits 4..1
    const bool up = (lane & (2 * w)) != 0;
#pragma unroll
    for (int k = 0; k < w; ++k) {
      const float send = up ? x[k] : x[k + w];
      const float keep = up ? x[k + w] : x[k];
      x[k] = keep + __shfl_xor_sync(0xffffffffu, send, 2 * w);
    }
  }
  x[0] += __shfl_xor_sync(0xffffffffu, x[0], 1);
  const int c = lane >> 1;
  if ((lane & 1) == 0 && c < 9) atomicAdd(&dst[c], x[0]);
}

__device__ __forceinline__ float4 load_px(const void* img, int dtype, long long p) {
  if (dtype == ABCD_F16) {
    const uint2 r = reinterpret_cast<const uint2*>(img)[p];
    const __half2 a = *reinterpret_cast<const __half2*>(&r.x);
    const __half2 b = *reinterpret_cast<const __half2*>(&r.y);
    const float2 fa = __half22float2(a), fb = __half22float2(b);
    return make_float4(fa.x, fa.y, fb.x, fb.y);
  }
  return reinterpret_cast<const float4*>(img)[p];
}

struct FwdArgs {
  Cam cam;
  Opts op;
  const float2* uv;
  const float4* co;
  const float* rgb;
  const unsigned* ids;
  const uint2* ranges;
  const void* F;
  const void* B;
  int fb_dtype;
  float bg[3];
  float4* out;
  float4* state_at;
  unsigned* n_last;
  uint2* refresh;      // fp16 x4 per pixel
};

// Stages one batch of list entries (positions base .. base + kBatch) and compacts the indices
// of the entries that survive the CTA-box cull into s_idx; returns the number of survivors.
template <bool WITH_ID>
__device__ __forceinline__ int stage_batch(const unsigned* ids, unsigned start, int n, int base,
                                           const float2* uv, const float4* co, const float* rgb,
                                           float bx0, float by0, float alpha_min, float2* s_uv,
                                           float4* s_co, float4* s_rgb, unsigned* s_id,
                                           unsigned short* s_idx, unsigned* s_ballot) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  bool keep[kRounds];
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const int q = threadIdx.x + r * kSubThreads;
    keep[r] = false;
    if (base + q < n) {
      const unsigned g = ids[start + base + q];
      const float2 m = uv[g];
      const float4 sc = scaled_conic(co[g]);
      keep[r] = !cull(sc, m, bx0, by0, alpha_min);
      if (keep[r]) {
        s_uv[q] = m;
        s_co[q] = sc;
        s_rgb[q] = make_float4(rgb[3 * g], rgb[3 * g + 1], rgb[3 * g + 2], 0.f);
        if (WITH_ID) s_id[q] = g;
      }
    }
    const unsigned b = __ballot_sync(0xffffffffu, keep[r]);
    if (lane == 0) s_ballot[r * 2 + w] = b;
  }
  __syncthreads();
  int total = 0, before_r = 0;
  const unsigned lt = (1u << lane) - 1u;
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const unsigned b0 = s_ballot[2 * r], b1 = s_ballot[2 * r + 1];
    const int at = before_r + (w ? __popc(b0) : 0) + __popc((w ? b1 : b0) & lt);
    if (keep[r]) s_idx[at] = (unsigned short)(threadIdx.x + r * kSubThreads);
    before_r += __popc(b0) + __popc(b1);
  }
  total = before_r;
  __syncthreads();
  return total;
}

__global__ void __launch_bounds__(kSubThreads) render_fwd_kernel(FwdArgs a) {
  __shared__ float2 s_uv[kBatch];
  __shared__ float4 s_co[kBatch];
  __shared__ float4 s_rgb[kBatch];
  __shared__ unsigned short s_idx[kBatch];
  __shared__ unsigned s_ballot[2 * kRounds];
  const int tile = blockIdx.x / kSubPerTile, sub = blockIdx.x % kSubPerTile;
  const int tx = tile % a.cam.tiles_x, ty = tile / a.cam.tiles_x;
  const int px0 = tx * kTile + (sub % (kTile / kSub)) * kSub;
  const int py0 = ty * kTile + (sub / (kTile / kSub)) * kSub;
  const int px = px0 + (threadIdx.x % kSub), py = py0 + (threadIdx.x / kSub);
  const bool inside = px < a.cam.width && py < a.cam.height;
  const uint2 rg = a.ranges[tile];
  const int n = rg.y > rg.x ? (int)(rg.y - rg.x) : 0;
  const float fx = (float)px + 0.5f, fy = (float)py + 0.5f;
  const float bx0 = (float)px0 + 0.5f, by0 = (float)py0 + 0.5f;
  float T = 1.f, c0 = 0.f, c1 = 0.f, c2 = 0.f;
  unsigned last = 0;
  bool done = !inside;
  for (int base = 0; base < n; base += kBatch) {
    if (__syncthreads_count(done) == kSubThreads) break;
    const int cnt = stage_batch<false>(a.ids, rg.x, n, base, a.uv, a.co, a.rgb, bx0, by0,
                                       a.op.alpha_min, s_uv, s_co, s_rgb, nullptr, s_idx, s_ballot);
    if (!done) {
      for (int j = 0; j < cnt; ++j) {
        const int q = s_idx[j];
        float dx, dy;
        const float4 s = s_co[q];
        const float sig = sigma2(s, s_uv[q], fx, fy, dx, dy);
        if (!(sig >= 0.f)) continue;
        const float alpha = fminf(a.op.alpha_max, __fmul_rn(s.w, ex2_approx(-sig)));
        if (alpha < a.op.alpha_min) continue;
        const float test = __fmul_rn(T, __fsub_rn(1.f, alpha));
        if (test < a.op.t_min) { done = true; break; }
        const float w = __fmul_rn(alpha, T);
        const float4 col = s_rgb[q];
        c0 = __fmaf_rn(w, col.x, c0);
        c1 = __fmaf_rn(w, col.y, c1);
        c2 = __fmaf_rn(w, col.z, c2);
        T = test;
        last = (unsigned)(base + q + 1);
      }
    }
  }
  if (!inside) return;
  const long long p = (long long)py * a.cam.width + px;
  const float Aa = 1.f - T;
  if (a.refresh) {
    const __half2 lo = __floats2half2_rn(c0, c1), hi = __floats2half2_rn(c2, Aa);
    uint2 r;
    r.x = *reinterpret_cast<const unsigned*>(&lo);
    r.y = *reinterpret_cast<const unsigned*>(&hi);
    a.refresh[p] = r;
  }
  if (a.state_at) {
    a.state_at[p] = make_float4(c0, c1, c2, T);
    a.n_last[p] = last;
  }
  if (a.out) {
    const float4 Bv = a.B ? load_px(a.B, a.fb_dtype, p) : make_float4(0.f, 0.f, 0.f, 0.f);
    const float4 Fv = a.F ? load_px(a.F, a.fb_dtype, p) : make_float4(0.f, 0.f, 0.f, 0.f);
    const float kb = 1.f - Aa;      // A over B
    const float m0 = c0 + kb * Bv.x, m1 = c1 + kb * Bv.y, m2 = c2 + kb * Bv.z, ma = Aa + kb * Bv.w;
    const float kf = 1.f - Fv.w;    // F over (A over B)
    float4 o = make_float4(Fv.x + kf * m0, Fv.y + kf * m1, Fv.z + kf * m2, Fv.w + kf * ma);
    const float kg = 1.f - o.w;
    o.x += kg * a.bg[0];
    o.y += kg * a.bg[1];
    o.z += kg * a.bg[2];
    a.out[p] = o;
  }
}

struct BwdArgs {
  Cam cam;
  Opts op;
  const float2* uv;
  const float4* co;
  const float* rgb;
  const unsigned* ids;
  const uint2* ranges;
  const void* F;
  const void* B;
  int fb_dtype;
  float bg[3];
  const float4* state_at;
  const unsigned* n_last;
  const float* dl_dout;
  float* grad2d;
};

__global__ void __launch_bounds__(kSubThreads) render_bwd_kernel(BwdArgs a) {
  __shared__ float2 s_uv[kBatch];
  __shared__ float4 s_co[kBatch];
  __shared__ float4 s_rgb[kBatch];
  __shared__ unsigned s_id[kBatch];
  __shared__ unsigned short s_idx[kBatch];
  __shared__ unsigned s_ballot[2 * kRounds];
  __shared__ unsigned s_max;
  const int tile = blockIdx.x / kSubPerTile, sub = blockIdx.x % kSubPerTile;
  const int tx = tile % a.cam.tiles_x, ty = tile / a.cam.tiles_x;
  const int px0 = tx * kTile + (sub % (kTile / kSub)) * kSub;
  const int py0 = ty * kTile + (sub / (kTile / kSub)) * kSub;
  const int px = px0 + (threadIdx.x % kSub), py = py0 + (threadIdx.x / kSub);
  const int lane = threadIdx.x & 31;
  const bool inside = px < a.cam.width && py < a.cam.height;
  const uint2 rg = a.ranges[tile];
  const int n = rg.y > rg.x ? (int)(rg.y - rg.x) : 0;
  const float fx = (float)px + 0.5f, fy = (float)py + 0.5f;
  const float bx0 = (float)px0 + 0.5f, by0 = (float)py0 + 0.5f;
  unsigned last = 0;
  float Gr = 0.f, Gg = 0.f, Gb = 0.f, Ga = 0.f, Tf = 1.f, A0 = 0.f, A1 = 0.f, A2 = 0.f;
  if (inside) {
    const long long p = (long long)py * a.cam.width + px;
    last = min(a.n_last[p], (unsigned)n);
    const float4 at = a.state_at[p];
    A0 = at.x; A1 = at.y; A2 = at.z; Tf = at.w;
    const float g0 = a.dl_dout[3 * p], g1 = a.dl_dout[3 * p + 1], g2 = a.dl_dout[3 * p + 2];
    const float4 Fv = a.F ? load_px(a.F, a.fb_dtype, p) : make_float4(0.f, 0.f, 0.f, 0.f);
    const float4 Bv = a.B ? load_px(a.B, a.fb_dtype, p) : make_float4(0.f, 0.f, 0.f, 0.f);
    const float kf = 1.f - Fv.w;
    Gr = kf * g0; Gg = kf * g1; Gb = kf * g2;
    // d final / d A.a = -(1 - F.a) (B.rgb + (1 - B.a) bg)
    Ga = -kf * (g0 * (Bv.x + (1.f - Bv.w) * a.bg[0]) + g1 * (Bv.y + (1.f - Bv.w) * a.bg[1]) +
                g2 * (Bv.z + (1.f - Bv.w) * a.bg[2]));
  }
  if (threadIdx.x == 0) s_max = 0;
  __syncthreads();
  const unsigned wmax = __reduce_max_sync(0xffffffffu, last);
  if (lane == 0) atomicMax(&s_max, wmax);
  __syncthreads();
  const int span = (int)s_max;
  float T = 1.f, c0 = 0.f, c1 = 0.f, c2 = 0.f;
  for (int base = 0; base < span; base += kBatch) {
    __syncthreads();
    const int cnt = stage_batch<true>(a.ids, rg.x, span, base, a.uv, a.co, a.rgb, bx0, by0,
                                      a.op.alpha_min, s_uv, s_co, s_rgb, s_id, s_idx, s_ballot);
    for (int j = 0; j < cnt; ++j) {
      const int q = s_idx[j];
      float v[9];
#pragma unroll
      for (int k = 0; k < 9; ++k) v[k] = 0.f;
      bool contrib = false;
      if ((unsigned)(base + q) < last) {
        float dx, dy;
        const float4 s = s_co[q];
        const float sig = sigma2(s, s_uv[q], fx, fy, dx, dy);
        if (sig >= 0.f) {
          const float G = ex2_approx(-sig);
          const float raw = __fmul_rn(s.w, G);
          const float alpha = fminf(a.op.alpha_max, raw);
          if (alpha >= a.op.alpha_min) {
            contrib = true;
            const float4 col = s_rgb[q];
            const float w = __fmul_rn(alpha, T);
            c0 = __fmaf_rn(w, col.x, c0);
            c1 = __fmaf_rn(w, col.y, c1);
            c2 = __fmaf_rn(w, col.z, c2);
            const float ioma = __fdividef(1.f, 1.f - alpha);   // gradient scale only
            // R = colour accumulated behind this Gaussian = A - (sum up to and including it)
            const float dalpha = Gr * (T * col.x - (A0 - c0) * ioma) +
                                 Gg * (T * col.y - (A1 - c1) * ioma) +
                                 Gb * (T * col.z - (A2 - c2) * ioma) + Ga * Tf * ioma;
            v[6] = Gr * w; v[7] = Gg * w; v[8] = Gb * w;
            if (raw <= a.op.alpha_max) {          // derivative of min() is 0 once clamped
              v[5] = dalpha * G;                   // d alpha / d opacity = exp(-sigma)
              const float dsig = -dalpha * raw;    // d alpha / d sigma = -alpha
              const float ca = 2.f * kLn2 * s.x, cb = kLn2 * s.y, cc = 2.f * kLn2 * s.z;
              v[0] = -dsig * (ca * dx + cb * dy);  // d = pixel - uv
              v[1] = -dsig * (cb * dx + cc * dy);
              v[2] = 0.5f * dsig * dx * dx;
              v[3] = dsig * dx * dy;
              v[4] = 0.5f * dsig * dy * dy;
            }
            T = __fmul_rn(T, __fsub_rn(1.f, alpha));
          }
        }
      }
      const unsigned who = __ballot_sync(0xffffffffu, contrib);
      if (who == 0) continue;
      float* dst = a.grad2d + 9 * (size_t)s_id[q];
      if (__popc(who) <= 2) {                   // one or two pixels: add directly
        if (contrib)
#pragma unroll
          for (int k = 0; k < 9; ++k) atomicAdd(&dst[k], v[k]);
      } else {
        warp_sum9_atomic(v, dst, lane);
      }
    }
  }
}

bool fb_ok(const void* F, const void* B, int dtype) {
  if (dtype != ABCD_F16 && dtype != ABCD_F32) return false;
  const uintptr_t al = dtype == ABCD_F16 ? 7 : 15;
  return (((uintptr_t)F & al) == 0) && (((uintptr_t)B & al) == 0);
}

bool proj_ok(const abcd_projected* p) {
  return p && p->uv && p->conic_opacity && p->rgb && ((uintptr_t)p->uv & 7) == 0 &&
         ((uintptr_t)p->conic_opacity & 15) == 0;
}

}  // namespace
}  // namespace abcd

using namespace abcd;

extern "C" abcd_status abcd_render_composite_fwd(abcd_ctx* ctx, const abcd_camera* cam,
                                                 const abcd_render_opts* opts,
                                                 const abcd_projected* proj,
                                                 const abcd_tiles* tiles, const void* F,
                                                 const void* B, int fb_dtype, const float* bg,
                                                 float* out_rgba, abcd_fwd_state* state,
                                                 void* refresh_f16) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!cam || cam->width <= 0 || cam->height <= 0 || !tiles || !tiles->ids || !tiles->ranges)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_composite_fwd: bad camera or tiles");
  if (!proj_ok(proj)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_composite_fwd: bad projected buffers");
  if (!fb_ok(F, B, fb_dtype)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_composite_fwd: bad F/B dtype or alignment");
  if (state && (!state->A_T || !state->n_last || ((uintptr_t)state->A_T & 15)))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_composite_fwd: bad state buffers");
  if (((uintptr_t)out_rgba & 15) || ((uintptr_t)refresh_f16 & 7))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_composite_fwd: misaligned output");
  FwdArgs a;
  a.cam = make_cam(cam, opts);
  a.op = make_opts(opts);
  a.uv = (const float2*)proj->uv;
  a.co = (const float4*)proj->conic_opacity;
  a.rgb = proj->rgb;
  a.ids = tiles->ids;
  a.ranges = (const uint2*)tiles->ranges;
  a.F = F; a.B = B; a.fb_dtype = fb_dtype;
  for (int c = 0; c < 3; ++c) a.bg[c] = bg ? bg[c] : 0.f;
  a.out = (float4*)out_rgba;
  a.state_at = state ? (float4*)state->A_T : nullptr;
  a.n_last = state ? state->n_last : nullptr;
  a.refresh = (uint2*)refresh_f16;
  const int n_tiles = a.cam.tiles_x * a.cam.tiles_y;
  render_fwd_kernel<<<n_tiles * kSubPerTile, kSubThreads, 0, ctx->stream>>>(a);
  return check_launch(ctx, "render_fwd_kernel");
}

extern "C" abcd_status abcd_render_backward(abcd_ctx* ctx, const abcd_camera* cam,
                                            const abcd_render_opts* opts,
                                            const abcd_projected* proj, const abcd_tiles* tiles,
                                            const void* F, const void* B, int fb_dtype,
                                            const float* bg, const abcd_fwd_state* state,
                                            const float* dL_dout, int n, float* grad2d) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!cam || cam->width <= 0 || cam->height <= 0 || !tiles || !tiles->ids || !tiles->ranges)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_backward: bad camera or tiles");
  if (!proj_ok(proj)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_backward: bad projected buffers");
  if (!fb_ok(F, B, fb_dtype)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_backward: bad F/B dtype or alignment");
  if (!state || !state->A_T || !state->n_last || !dL_dout || n < 0 || (n > 0 && !grad2d))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_backward: null state, gradient or output");
  if (n == 0) return ABCD_OK;
  cudaError_t e = cudaMemsetAsync(grad2d, 0, sizeof(float) * 9 * (size_t)n, ctx->stream);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "grad2d memset: %s", cudaGetErrorString(e));
  BwdArgs a;
  a.cam = make_cam(cam, opts);
  a.op = make_opts(opts);
  a.uv = (const float2*)proj->uv;
  a.co = (const float4*)proj->conic_opacity;
  a.rgb = proj->rgb;
  a.ids = tiles->ids;
  a.ranges = (const uint2*)tiles->ranges;
  a.F = F; a.B = B; a.fb_dtype = fb_dtype;
  for (int c = 0; c < 3; ++c) a.bg[c] = bg ? bg[c] : 0.f;
  a.state_at = (const float4*)state->A_T;
  a.n_last = state->n_last;
  a.dl_dout = dL_dout;
  a.grad2d = grad2d;
  const int n_tiles = a.cam.tiles_x * a.cam.tiles_y;
  render_bwd_kernel<<<n_tiles * kSubPerTile, kSubThreads, 0, ctx->stream>>>(a);
  return check_launch(ctx, "render_bwd_kernel");
}
