// K6: reconstruction loss of one step, L = (1 - lambda) mean|x - y| + lambda (1 - mean SSIM),
// and dL/dx, fused in one kernel (each step of Section 2 scores the composited image against
// the target; the L1 + D-SSIM form is that of 3D Gaussian Splatting).
//
// SSIM uses an 11x11 Gaussian window (sigma 1.5) with zero padding.  Per output tile of 32x32
// pixels and per channel, a CTA stages x, y over the tile plus a 10-pixel halo, computes the
// five windowed moments (separably) on the tile plus a 5-pixel halo, the per-pixel partials
// A = dS/dmu_x - 2 mu_x dS/dsigma_xx - mu_y dS/dsigma_xy, B = dS/dsigma_xx, C = dS/dsigma_xy,
// and windows them again: dSSIM_sum/dx(q) = (w*A)(q) + 2 x(q) (w*B)(q) + y(q) (w*C)(q).
// The scalar is reduced deterministically: per-CTA partial sums, then the last CTA to finish
// adds them in a fixed order (no waiting on other CTAs).
#include <mutex>

#include "abcd_internal.cuh"

namespace abcd {
namespace {

constexpr int T = kLossTile;      // 32
constexpr int R0 = T + 20;        // input region edge
constexpr int R1 = T + 10;        // moment region edge
constexpr int kThreads = 256;
constexpr int kSmemFloats = 2 * R0 * R0 + 5 * R0 * R1 + 5 * R1 * R1;

__global__ void __launch_bounds__(kThreads)
loss_kernel(const float* __restrict__ xin, const float* __restrict__ yin, int W, int H,
            float lam, float* __restrict__ grad, float* partials, unsigned* ticket,
            float* loss_out) {
  extern __shared__ float sm[];
  float* sX = sm;                       // [R0][R0]
  float* sY = sX + R0 * R0;             // [R0][R0]
  float* hq = sY + R0 * R0;             // 5 x [R0][R1]; later A, B, C [R1][R1]
  float* mq = hq + 5 * R0 * R1;         // 5 x [R1][R1]; later 3 x [R1][T]
  __shared__ float w[11];
  __shared__ float red[2][kThreads / 32];
  if (threadIdx.x < 11) {
    const float d = (float)threadIdx.x - 5.f;
    w[threadIdx.x] = expf(-d * d / (2.f * 1.5f * 1.5f));
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
    for (int k = 0; k < 11; ++k) s += w[k];
    for (int k = 0; k < 11; ++k) w[k] /= s;
  }
  __syncthreads();
  const int ox = blockIdx.x * T, oy = blockIdx.y * T;
  const float inv = 1.f / (3.f * (float)W * (float)H);
  float l1 = 0.f, ssim = 0.f;
  for (int ch = 0; ch < 3; ++ch) {
    for (int k = threadIdx.x; k < R0 * R0; k += kThreads) {
      const int r = k / R0, c = k % R0;
      const int gy = oy - 10 + r, gx = ox - 10 + c;
      float xv = 0.f, yv = 0.f;
      if (gx >= 0 && gx < W && gy >= 0 && gy < H) {
        const long long p = (long long)gy * W + gx;
        xv = xin[4 * p + ch];
        yv = yin[3 * p + ch];
      }
      sX[k] = xv;
      sY[k] = yv;
    }
    __syncthreads();
    // horizontal windows of x, y, x^2, y^2, xy: [R0][R1]
    for (int k = threadIdx.x; k < R0 * R1; k += kThreads) {
      const int r = k / R1, c = k % R1;
      const float* px = sX + r * R0 + c;
      const float* py = sY + r * R0 + c;
      float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f, a4 = 0.f;
#pragma unroll
      for (int t = 0; t < 11; ++t) {
        const float xv = px[t], yv = py[t], wt = w[t];
        a0 += wt * xv; a1 += wt * yv;
        a2 += wt * xv * xv; a3 += wt * yv * yv; a4 += wt * xv * yv;
      }
      hq[k] = a0; hq[R0 * R1 + k] = a1; hq[2 * R0 * R1 + k] = a2;
      hq[3 * R0 * R1 + k] = a3; hq[4 * R0 * R1 + k] = a4;
    }
    __syncthreads();
    // vertical windows: moments on [R1][R1]
    for (int k = threadIdx.x; k < R1 * R1; k += kThreads) {
      const int r = k / R1, c = k % R1;
      float a[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int t = 0; t < 11; ++t) {
        const float wt = w[t];
#pragma unroll
        for (int q = 0; q < 5; ++q) a[q] += wt * hq[q * R0 * R1 + (r + t) * R1 + c];
      }
#pragma unroll
      for (int q = 0; q < 5; ++q) mq[q * R1 * R1 + k] = a[q];
    }
    __syncthreads();
    // per-pixel SSIM and its partials A, B, C (zero outside the image)
    {
      const float C1 = 0.01f * 0.01f, C2 = 0.03f * 0.03f;
      float* A = hq;
      float* B = hq + R1 * R1;
      float* Cc = hq + 2 * R1 * R1;
      for (int k = threadIdx.x; k < R1 * R1; k += kThreads) {
        const int r = k / R1, c = k % R1;
        const int gy = oy - 5 + r, gx = ox - 5 + c;
        float av = 0.f, bv = 0.f, cv = 0.f;
        if (gx >= 0 && gx < W && gy >= 0 && gy < H) {
          const float mx = mq[k], my = mq[R1 * R1 + k];
          const float vx = mq[2 * R1 * R1 + k] - mx * mx;
          const float vy = mq[3 * R1 * R1 + k] - my * my;
          const float cxy = mq[4 * R1 * R1 + k] - mx * my;
          const float N1 = 2.f * mx * my + C1, N2 = 2.f * cxy + C2;
          const float D1 = mx * mx + my * my + C1, D2 = vx + vy + C2;
          const float iD = 1.f / (D1 * D2);
          const float S = N1 * N2 * iD;
          const float dmx = (2.f * my * N2 - S * 2.f * mx * D2) * iD;
          const float dvx = -S / D2;
          const float dcxy = 2.f * N1 * iD;
          av = dmx - 2.f * mx * dvx - my * dcxy;
          bv = dvx;
          cv = dcxy;
          if (r >= 5 && r < 5 + T && c >= 5 && c < 5 + T) ssim += S;
        }
        A[k] = av; B[k] = bv; Cc[k] = cv;
      }
    }
    __syncthreads();
    // horizontal windows of A, B, C: [R1][T]
    for (int k = threadIdx.x; k < R1 * T; k += kThreads) {
      const int r = k / T, c = k % T;
      float a0 = 0.f, a1 = 0.f, a2 = 0.f;
#pragma unroll
      for (int t = 0; t < 11; ++t) {
        const float wt = w[t];
        const int idx = r * R1 + c + t;
        a0 += wt * hq[idx]; a1 += wt * hq[R1 * R1 + idx]; a2 += wt * hq[2 * R1 * R1 + idx];
      }
      mq[k] = a0; mq[R1 * T + k] = a1; mq[2 * R1 * T + k] = a2;
    }
    __syncthreads();
    // vertical windows and the gradient on the output tile
    for (int k = threadIdx.x; k < T * T; k += kThreads) {
      const int r = k / T, c = k % T;
      const int gy = oy + r, gx = ox + c;
      if (gx >= W || gy >= H) continue;
      float a0 = 0.f, a1 = 0.f, a2 = 0.f;
#pragma unroll
      for (int t = 0; t < 11; ++t) {
        const float wt = w[t];
        const int idx = (r + t) * T + c;
        a0 += wt * mq[idx]; a1 += wt * mq[R1 * T + idx]; a2 += wt * mq[2 * R1 * T + idx];
      }
      const float xv = sX[(r + 10) * R0 + c + 10], yv = sY[(r + 10) * R0 + c + 10];
      const float d = xv - yv;
      l1 += fabsf(d);
      const float sgn = (d > 0.f) ? 1.f : ((d < 0.f) ? -1.f : 0.f);
      const float dS = a0 + 2.f * xv * a1 + yv * a2;
      if (grad) grad[3 * ((long long)gy * W + gx) + ch] = ((1.f - lam) * sgn - lam * dS) * inv;
    }
    __syncthreads();
  }
  // block partial sums -> last block finishes the scalar
  for (int o = 16; o > 0; o >>= 1) {
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
    ssim += __shfl_xor_sync(0xffffffffu, ssim, o);
  }
  if ((threadIdx.x & 31) == 0) { red[0][threadIdx.x >> 5] = l1; red[1][threadIdx.x >> 5] = ssim; }
  __syncthreads();
  const int nb = gridDim.x * gridDim.y;
  const int b = blockIdx.y * gridDim.x + blockIdx.x;
  __shared__ bool is_last;
  if (threadIdx.x == 0) {
    float s0 = 0.f, s1 = 0.f;
    for (int k = 0; k < kThreads / 32; ++k) { s0 += red[0][k]; s1 += red[1][k]; }
    partials[2 * b] = s0;
    partials[2 * b + 1] = s1;
    __threadfence();
    const unsigned t = atomicAdd(ticket, 1u);
    is_last = (t == (unsigned)(nb - 1));
  }
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  double s0 = 0.0, s1 = 0.0;
  for (int k = threadIdx.x; k < nb; k += kThreads) {
    s0 += (double)__ldcg(&partials[2 * k]);
    s1 += (double)__ldcg(&partials[2 * k + 1]);
  }
  __shared__ double dred[2][kThreads];
  dred[0][threadIdx.x] = s0;
  dred[1][threadIdx.x] = s1;
  __syncthreads();
  for (int st = kThreads / 2; st > 0; st >>= 1) {
    if ((int)threadIdx.x < st) {
      dred[0][threadIdx.x] += dred[0][threadIdx.x + st];
      dred[1][threadIdx.x] += dred[1][threadIdx.x + st];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const double n = 3.0 * (double)W * (double)H;
    if (loss_out) *loss_out = (float)((1.0 - lam) * dred[0][0] / n + lam * (1.0 - dred[1][0] / n));
    *ticket = 0u;
  }
}

}  // namespace

abcd_status loss_launch(abcd_ctx* ctx, const float* out_rgba, const float* gt_rgb, int width,
                        int height, float lambda_ssim, float* loss_out, float* dL_dout) {
  if (!has_workspace(ctx)) return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_loss: no workspace");
  if (!out_rgba || !gt_rgb || width <= 0 || height <= 0 || !(lambda_ssim >= 0.f && lambda_ssim <= 1.f))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_loss: bad arguments");
  const dim3 grid((width + T - 1) / T, (height + T - 1) / T);
  if ((long long)grid.x * grid.y > kMaxLossBlocks)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_loss: image too large (%d x %d)", width, height);
  const size_t smem = sizeof(float) * kSmemFloats;
  cudaError_t e = cudaFuncSetAttribute(loss_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "loss smem attribute: %s", cudaGetErrorString(e));
  loss_kernel<<<grid, kThreads, smem, ctx->stream>>>(out_rgba, gt_rgb, width, height, lambda_ssim,
                                                    dL_dout, ctx->ws.loss_partials,
                                                    ctx->ws.status + 1, loss_out);
  return check_launch(ctx, "loss_kernel");
}

}  // namespace abcd

extern "C" abcd_status abcd_loss(abcd_ctx* ctx, const float* out_rgba, const float* gt_rgb,
                                 int width, int height, float lambda_ssim, float* loss_out,
                                 float* dL_dout) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  return abcd::loss_launch(ctx, out_rgba, gt_rgb, width, height, lambda_ssim, loss_out, dL_dout);
}

// ---------------------------------------------------------------------------------------
// abcd_loss_static: the same loss kernel with its scratch in this file's static device array
// instead of the context workspace, for callers that cannot allocate device memory.

namespace abcd {
namespace {

constexpr int kStaticLossMaxBlocks = 16384;            // 32x32-pixel CTAs: up to 4096 x 4096
constexpr int kStaticLossWords = 2 * kStaticLossMaxBlocks + 64;   // partial sums, then the ticket

// Device scratch shared by every abcd_loss_static call on a device (held until exit).
static __device__ __align__(256) unsigned g_loss_static_scratch[kStaticLossWords];

constexpr int kMaxDevices = 256;
std::mutex g_static_mu;
unsigned* g_static_ptr[kMaxDevices] = {nullptr};

// Device address of the static scratch on the current device, looked up once per device.
cudaError_t static_scratch(int device, unsigned** out) {
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (!g_static_ptr[device]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_loss_static_scratch);
    if (e != cudaSuccess) return e;
    g_static_ptr[device] = static_cast<unsigned*>(p);
  }
  *out = g_static_ptr[device];
  return cudaSuccess;
}

}  // namespace
}  // namespace abcd

extern "C" abcd_status abcd_loss_static(void* cuda_stream, const float* out_rgba,
                                        const float* gt_rgb, int width, int height,
                                        float lambda_ssim, float* loss_out, float* dL_dout) {
  using namespace abcd;
  if (!out_rgba || !gt_rgb || width <= 0 || height <= 0 ||
      !(lambda_ssim >= 0.f && lambda_ssim <= 1.f))
    return ABCD_ERR_INVALID_ARG;
  const dim3 grid((width + T - 1) / T, (height + T - 1) / T);
  if ((long long)grid.x * grid.y > kStaticLossMaxBlocks) return ABCD_ERR_WORKSPACE;
  int device = 0;
  if (cudaGetDevice(&device) != cudaSuccess || device < 0 || device >= kMaxDevices)
    return ABCD_ERR_CUDA;
  unsigned* scratch = nullptr;
  if (static_scratch(device, &scratch) != cudaSuccess) return ABCD_ERR_CUDA;
  float* partials = reinterpret_cast<float*>(scratch);
  unsigned* ticket = scratch + 2 * kStaticLossMaxBlocks;
  cudaStream_t stream = (cudaStream_t)cuda_stream;
  // the ticket must start at zero whatever an earlier (possibly failed) call left there
  if (cudaMemsetAsync(ticket, 0, sizeof(unsigned), stream) != cudaSuccess) return ABCD_ERR_CUDA;
  const size_t smem = sizeof(float) * kSmemFloats;
  if (cudaFuncSetAttribute(loss_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
      cudaSuccess)
    return ABCD_ERR_CUDA;
  loss_kernel<<<grid, kThreads, smem, stream>>>(out_rgba, gt_rgb, width, height, lambda_ssim,
                                                dL_dout, partials, ticket, loss_out);
  return cudaGetLastError() == cudaSuccess ? ABCD_OK : ABCD_ERR_CUDA;
}
