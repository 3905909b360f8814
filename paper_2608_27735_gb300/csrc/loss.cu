// K6: reconstruction loss of one step, L = (1 - lambda) mean|x - y| + lambda (1 - mean SSIM),
// and dL/dx (each step of Section 2 scores the composited image against the target; the
// L1 + D-SSIM form is that of 3D Gaussian Splatting).  SSIM uses an 11x11 Gaussian window
// (sigma 1.5) with zero padding.  Per pixel q and channel, with the partials
// A = dS/dmu_x - 2 mu_x dS/dsigma_xx - mu_y dS/dsigma_xy, B = dS/dsigma_xx, C = dS/dsigma_xy
// of the SSIM S at each pixel, dSSIM_sum/dx(q) = (w*A)(q) + 2 x(q) (w*B)(q) + y(q) (w*C)(q).
//
// Two implementations:
//  * abcd_loss (and the step's backward) run two kernels, ssim_fwd_kernel and ssim_bwd_kernel,
//    that meet at A, B, C kept in the workspace (described below, before them).
//  * abcd_loss_static runs loss_kernel, one fused kernel that needs no per-pixel scratch: a CTA
//    takes one channel of an output tile of 64x28 pixels, stages x, y over the tile plus a
//    10-pixel halo, computes the five windowed moments (separably) on the tile plus a 5-pixel
//    halo, then A, B, C, and windows them again.  Every window pass is register-blocked: a
//    thread produces 8 consecutive outputs from a sliding run of 18 staged values, and the
//    windows of x and y (of x^2 and y^2, of A and B) share packed two-lane FMAs.  Shared
//    memory (about 105 KB) and registers (at most 64) are sized for two CTAs per SM.
// Both reduce the scalar deterministically: per-CTA partial sums, then the last CTA to finish
// adds them in a fixed order (no waiting on other CTAs).
#include <cmath>

#include "abcd_internal.cuh"

namespace abcd {
namespace {

constexpr int TW = 64;            // output tile (pixels)
constexpr int TH = 28;
// Outputs per thread in each window pass (a run reads RUN + 10 staged values), chosen so that
// every pass is one round over the CTA's 480 threads with few idle: 480, 444, 418 and 448 runs.
constexpr int RUN = 8;            // horizontal moments
constexpr int RUN_V = 7;          // vertical moments
constexpr int RUN_H3 = 6;         // horizontal windows of A, B, C
constexpr int RUN_V3 = 4;         // vertical windows of A, B, C
constexpr int IW = TW + 20, IH = TH + 20;    // inputs: tile + 10-pixel halo
constexpr int MW = TW + 10, MH = TH + 10;    // windowed moments: tile + 5-pixel halo
constexpr int HSEG = (MW + RUN - 1) / RUN;   // column runs of the horizontal moment pass
constexpr int VSEG = (MH + RUN_V - 1) / RUN_V;     // row runs of the vertical moment pass
constexpr int HSEG3 = (TW + RUN_H3 - 1) / RUN_H3;  // column runs of the horizontal A, B, C pass
constexpr int VSEG3 = (TH + RUN_V3 - 1) / RUN_V3;  // row runs of the vertical A, B, C pass
constexpr int kThreads = 480;                // 15 warps: one horizontal moment run per thread
static_assert(IH * HSEG <= kThreads && MW * VSEG <= kThreads && MH * HSEG3 <= kThreads &&
              TW * VSEG3 <= kThreads, "every window pass is one round");
static_assert(MH >= RUN_V && TW >= RUN_H3 && TH >= RUN_V3, "run tiling");
// Row pitches are odd (consecutive lanes take consecutive rows in the horizontal passes and
// consecutive columns in the vertical ones: no bank conflicts, also for the 8-byte pairs) and
// wide enough that a horizontal run never reads past its row (values read beyond the valid
// region only feed outputs that are discarded).  A vertical pass's last run starts early
// enough to stay inside its rows and skips the outputs the run before it made.
constexpr int IP = ((HSEG * RUN + 10) | 1);          // x|y row pitch (>= IW)
constexpr int MP = (MW | 1);                         // moment / A, B, C row pitch (>= MW)
constexpr int TP = (TW | 1);                         // pitch of the windows of A, B, C
// Shared memory, in floats, two regions:
//   R0: (x, y) pairs [IH][IP]; later (A, B) pairs and C [MH][MP]
//   R1: horizontal moment rows (mu_x, mu_y), (s_xx, s_yy) pairs and s_xy [IH][MP]; later the
//       horizontal windows of A, B, C: (A, B) pairs and C [MH][TP]
// The pairs go through the packed fp32 FMA (__ffma2_rn), two windows per instruction; each
// component is rounded exactly as a scalar fmaf.  The gradient pass reads x and y back from
// global memory (L2): R0 holds A, B, C by then.
constexpr int kR0 = 2 * IH * IP;
constexpr int kR1 = 5 * IH * MP;
constexpr int kSmemFloats = kR0 + kR1;
static_assert(IP >= IW && MP >= MW, "padded pitches");
static_assert(3 * MH * MP <= kR0, "A, B, C fit in the input region");
static_assert(3 * MH * TP <= kR1, "windows of A, B, C fit in the moment region");
static_assert(TW - RUN_H3 + RUN_H3 + 10 <= MW, "horizontal A, B, C runs stay in the valid columns");
static_assert(kR0 % 2 == 0 && (2 * MH * MP) % 2 == 0 && (2 * IH * MP) % 2 == 0, "pairs 8-byte aligned");
static_assert(sizeof(float) * kSmemFloats <= 110 * 1024, "two CTAs per SM");

struct Window {
  float w[11];      // normalised 11-tap Gaussian, sigma 1.5
};

// N outputs of an 11-tap window from N + 10 staged pairs / values.
template <int N>
__device__ __forceinline__ void window_pairs(const float2 (&v)[N + 10], const Window& win,
                                             float2 (&out)[N]) {
#pragma unroll
  for (int o = 0; o < N; ++o) {
    float2 a = make_float2(0.f, 0.f);
#pragma unroll
    for (int t = 0; t < 11; ++t) a = __ffma2_rn(make_float2(win.w[t], win.w[t]), v[o + t], a);
    out[o] = a;
  }
}

template <int N>
__device__ __forceinline__ void window_scalars(const float (&v)[N + 10], const Window& win,
                                               float (&out)[N]) {
#pragma unroll
  for (int o = 0; o < N; ++o) {
    float a = 0.f;
#pragma unroll
    for (int t = 0; t < 11; ++t) a = fmaf(win.w[t], v[o + t], a);
    out[o] = a;
  }
}

__global__ void __launch_bounds__(kThreads, 2)
loss_kernel(const float* __restrict__ xin, const float* __restrict__ yin, int W, int H,
            float lam, const Window win, float* __restrict__ grad, float* partials,
            unsigned* ticket, float* loss_out) {
  pdl_prologue();
  extern __shared__ __align__(16) float sm[];
  float2* sXY = reinterpret_cast<float2*>(sm);                        // [IH][IP]
  float2* aAB = reinterpret_cast<float2*>(sm);                        // [MH][MP]
  float* aC = reinterpret_cast<float*>(aAB + MH * MP);                // [MH][MP]
  float2* hM = reinterpret_cast<float2*>(sm + kR0);                   // [IH][MP]
  float2* hS = hM + IH * MP;                                          // [IH][MP]
  float* hC = reinterpret_cast<float*>(hS + IH * MP);                 // [IH][MP]
  float2* gAB = hM;                                                   // [MH][TP]
  float* gC = reinterpret_cast<float*>(gAB + MH * TP);                // [MH][TP]
  __shared__ float red[2][kThreads / 32];
  const int ox = blockIdx.x * TW, oy = blockIdx.y * TH, ch = blockIdx.z;
  const float inv = 1.f / (3.f * (float)W * (float)H);
  const float C1 = 0.01f * 0.01f, C2 = 0.03f * 0.03f;
  float l1 = 0.f, ssim = 0.f;
  // ---- inputs with a 10-pixel halo, zero outside the image (all loads issued before the
  // first store: one memory round trip)
  {
    constexpr int kLoads = (IH * IP + kThreads - 1) / kThreads;
    float xv[kLoads], yv[kLoads];
#pragma unroll
    for (int j = 0; j < kLoads; ++j) {
      const int k = threadIdx.x + j * kThreads;
      const int r = k / IP, c = k - r * IP;
      const int gy = oy - 10 + r, gx = ox - 10 + c;
      xv[j] = 0.f;
      yv[j] = 0.f;
      if (k < IH * IP && c < IW && gx >= 0 && gx < W && gy >= 0 && gy < H) {
        const long long p = (long long)gy * W + gx;
        xv[j] = __ldg(xin + 4 * p + ch);
        yv[j] = __ldg(yin + 3 * p + ch);
      }
    }
#pragma unroll
    for (int j = 0; j < kLoads; ++j) {
      const int k = threadIdx.x + j * kThreads;
      if (k < IH * IP) sXY[k] = make_float2(xv[j], yv[j]);
    }
  }
  __syncthreads();
  // ---- horizontal windows of (x, y), (x^2, y^2) and xy: RUN outputs per run
  for (int it = threadIdx.x; it < IH * HSEG; it += kThreads) {
    const int r = it % IH, c0 = (it / IH) * RUN;   // consecutive lanes: consecutive rows
    float2 v[RUN + 10], o2[RUN];
#pragma unroll
    for (int t = 0; t < RUN + 10; ++t) v[t] = sXY[r * IP + c0 + t];
    window_pairs<RUN>(v, win, o2);
#pragma unroll
    for (int o = 0; o < RUN; ++o) if (c0 + o < MW) hM[r * MP + c0 + o] = o2[o];
    float p[RUN + 10], o1[RUN];
#pragma unroll
    for (int t = 0; t < RUN + 10; ++t) {
      p[t] = v[t].x * v[t].y;
      v[t] = __fmul2_rn(v[t], v[t]);
    }
    window_pairs<RUN>(v, win, o2);
#pragma unroll
    for (int o = 0; o < RUN; ++o) if (c0 + o < MW) hS[r * MP + c0 + o] = o2[o];
    window_scalars<RUN>(p, win, o1);
#pragma unroll
    for (int o = 0; o < RUN; ++o) if (c0 + o < MW) hC[r * MP + c0 + o] = o1[o];
  }
  __syncthreads();
  // ---- vertical windows -> moments -> SSIM and its partials A, B, C (zero off-image)
  for (int it = threadIdx.x; it < MW * VSEG; it += kThreads) {
    const int c = it % MW, k0 = (it / MW) * RUN_V;
    const int r0 = min(k0, MH - RUN_V);            // the last run starts early ...
    const int o0 = k0 - r0;                        // ... and skips what the run before made
    float2 mm[RUN_V], ss[RUN_V];
    float mc[RUN_V];
    {
      float2 col[RUN_V + 10];
#pragma unroll
      for (int t = 0; t < RUN_V + 10; ++t) col[t] = hM[(r0 + t) * MP + c];
      window_pairs<RUN_V>(col, win, mm);
#pragma unroll
      for (int t = 0; t < RUN_V + 10; ++t) col[t] = hS[(r0 + t) * MP + c];
      window_pairs<RUN_V>(col, win, ss);
    }
    {
      float col[RUN_V + 10];
#pragma unroll
      for (int t = 0; t < RUN_V + 10; ++t) col[t] = hC[(r0 + t) * MP + c];
      window_scalars<RUN_V>(col, win, mc);
    }
#pragma unroll
    for (int o = 0; o < RUN_V; ++o) {
      if (o < o0) continue;
      const int r = r0 + o;
      const int gy = oy - 5 + r, gx = ox - 5 + c;
      float A = 0.f, B = 0.f, Cc = 0.f;
      if (gx >= 0 && gx < W && gy >= 0 && gy < H) {
        const float mx = mm[o].x, my = mm[o].y;
        const float vx = ss[o].x - mx * mx, vy = ss[o].y - my * my, cxy = mc[o] - mx * my;
        const float N1 = 2.f * mx * my + C1, N2 = 2.f * cxy + C2;
        const float D1 = mx * mx + my * my + C1, D2 = vx + vy + C2;
        const float iD = __fdividef(1.f, D1 * D2);   // fast reciprocal (about 2 ulp)
        const float S = N1 * N2 * iD;
        const float dvx = -S * (D1 * iD);           // -S / D2
        const float dcxy = 2.f * N1 * iD;
        A = (2.f * my * N2 - S * 2.f * mx * D2) * iD - 2.f * mx * dvx - my * dcxy;
        B = dvx;
        Cc = dcxy;
        if (r >= 5 && r < 5 + TH && c >= 5 && c < 5 + TW) ssim += S;
      }
      aAB[r * MP + c] = make_float2(A, B);
      aC[r * MP + c] = Cc;
    }
  }
  __syncthreads();
  // ---- horizontal windows of (A, B) and C: [MH][TW]
  for (int it = threadIdx.x; it < MH * HSEG3; it += kThreads) {
    const int r = it % MH, k0 = (it / MH) * RUN_H3;   // consecutive lanes: consecutive rows
    const int c0 = min(k0, TW - RUN_H3), o0 = k0 - c0;
    {
      float2 v[RUN_H3 + 10], o2[RUN_H3];
#pragma unroll
      for (int t = 0; t < RUN_H3 + 10; ++t) v[t] = aAB[r * MP + c0 + t];
      window_pairs<RUN_H3>(v, win, o2);
#pragma unroll
      for (int o = 0; o < RUN_H3; ++o) if (o >= o0) gAB[r * TP + c0 + o] = o2[o];
    }
    {
      float v[RUN_H3 + 10], o1[RUN_H3];
#pragma unroll
      for (int t = 0; t < RUN_H3 + 10; ++t) v[t] = aC[r * MP + c0 + t];
      window_scalars<RUN_H3>(v, win, o1);
#pragma unroll
      for (int o = 0; o < RUN_H3; ++o) if (o >= o0) gC[r * TP + c0 + o] = o1[o];
    }
  }
  __syncthreads();
  // ---- vertical windows and the gradient on the output tile
  for (int it = threadIdx.x; it < TW * VSEG3; it += kThreads) {
    const int c = it % TW, k0 = (it / TW) * RUN_V3;
    const int r0 = min(k0, TH - RUN_V3), o0 = k0 - r0;
    float2 gab[RUN_V3];
    float gc[RUN_V3];
    {
      float2 v[RUN_V3 + 10];
#pragma unroll
      for (int t = 0; t < RUN_V3 + 10; ++t) v[t] = gAB[(r0 + t) * TP + c];
      window_pairs<RUN_V3>(v, win, gab);
    }
    {
      float v[RUN_V3 + 10];
#pragma unroll
      for (int t = 0; t < RUN_V3 + 10; ++t) v[t] = gC[(r0 + t) * TP + c];
      window_scalars<RUN_V3>(v, win, gc);
    }
#pragma unroll
    for (int o = 0; o < RUN_V3; ++o) {
      const int gy = oy + r0 + o, gx = ox + c;
      if (o < o0 || gx >= W || gy >= H) continue;
      const long long q = (long long)gy * W + gx;
      const float xv = __ldg(xin + 4 * q + ch), yv = __ldg(yin + 3 * q + ch);
      const float d = xv - yv;
      l1 += fabsf(d);
      const float sgn = (d > 0.f) ? 1.f : ((d < 0.f) ? -1.f : 0.f);
      const float dS = gab[o].x + 2.f * xv * gab[o].y + yv * gc[o];
      if (grad) grad[3 * q + ch] = ((1.f - lam) * sgn - lam * dS) * inv;
    }
  }
  // block partial sums -> last block finishes the scalar
  for (int o = 16; o > 0; o >>= 1) {
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
    ssim += __shfl_xor_sync(0xffffffffu, ssim, o);
  }
  if ((threadIdx.x & 31) == 0) { red[0][threadIdx.x >> 5] = l1; red[1][threadIdx.x >> 5] = ssim; }
  __syncthreads();
  const int nb = gridDim.x * gridDim.y * gridDim.z;
  const int b = (blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
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
  for (int o = 16; o > 0; o >>= 1) {
    s0 += __shfl_xor_sync(0xffffffffu, s0, o);
    s1 += __shfl_xor_sync(0xffffffffu, s1, o);
  }
  __shared__ double dred[2][kThreads / 32];
  if ((threadIdx.x & 31) == 0) { dred[0][threadIdx.x >> 5] = s0; dred[1][threadIdx.x >> 5] = s1; }
  __syncthreads();
  if (threadIdx.x == 0) {
    double t0 = 0.0, t1 = 0.0;
    for (int k = 0; k < kThreads / 32; ++k) { t0 += dred[0][k]; t1 += dred[1][k]; }
    const double n = 3.0 * (double)W * (double)H;
    if (loss_out) *loss_out = (float)((1.0 - lam) * t0 / n + lam * (1.0 - t1 / n));
    *ticket = 0u;
  }
}

// ---------------------------------------------------------------------------------------
// The loss of a step as two kernels (the path abcd_loss and abcd_backward take).  Splitting
// the SSIM's forward windows from its backward windows at the per-pixel partials A, B, C
// (kept in the workspace, 36 bytes per pixel, L2-resident between the two launches) lets each
// kernel stage only a 5-pixel halo instead of the fused kernel's 10, and each runs its
// vertical windows first over the tile's long side: for a 118x16 output tile the windowed
// work is 1.085x the output area in the first pass and 1x in the second (the fused 64x28 tile
// computes its moments on 1.98x and 1.57x of its area).
//   ssim_fwd_kernel: x, y on the tile + 5 -> vertical windows of (x, y), (x^2, y^2), xy on
//     128 x 16 -> horizontal windows on 118 x 16 -> moments, SSIM, |x - y| and A, B, C per
//     pixel; per-CTA sums of SSIM and |x - y|, the last CTA adds them in a fixed order.
//   ssim_bwd_kernel: A, B, C on the tile + 5 -> vertical windows on 128 x 16 -> horizontal
//     windows on 118 x 16 -> dL/dx.
// Both use runs of 8 outputs from 18 staged values; 256 threads, about 66 KB of shared memory
// and at most 80 registers, so three CTAs share an SM.
constexpr int QW = 118, QH = 16;             // output tile
constexpr int QC = QW + 10, QR = QH + 10;    // staged columns and rows (5-pixel halo)
constexpr int QRUN = 8;                      // outputs per run
constexpr int QHSEG = (QW + QRUN - 1) / QRUN;      // horizontal runs per row (15)
constexpr int kQThreads = 256;
constexpr int QPM = QC | 1;                  // pitch of the vertical-window rows (odd)
constexpr int QPO = QW | 1;                  // pitch of the per-pixel results staged for the copy-out
static_assert(QC * (QH / QRUN) == kQThreads && QH % QRUN == 0, "one vertical run per thread");
static_assert(QH * QHSEG <= kQThreads, "one horizontal round");
static_assert(kQThreads == 2 * QC && QR % 2 == 0 && QH % 2 == 0, "a thread stages one column, every other row");
static_assert(QW - QRUN + QRUN + 10 <= QC, "horizontal runs stay in the staged columns");
constexpr int kQFwdFloats = 2 * QR * QC + 5 * QH * QPM;
constexpr int kQBwdFloats = 3 * QR * QC + 3 * QH * QPM;
static_assert(sizeof(float) * kQFwdFloats <= 72 * 1024 && sizeof(float) * kQBwdFloats <= 72 * 1024,
              "three CTAs per SM");
static_assert(3 * QH * QPO <= 2 * QR * QC && 2 * QH * QPO <= 2 * QR * QC && QH * QPO <= QR * QC,
              "the per-pixel results fit in the staging region");

__device__ __forceinline__ int q_block_index() {
  return (blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
}

__global__ void __launch_bounds__(kQThreads, 3)
ssim_fwd_kernel(const float* __restrict__ xin, const float* __restrict__ yin, int W, int H,
                float lam, const Window win, float2* __restrict__ abc_ab, float* __restrict__ abc_c,
                float* partials, unsigned* ticket, float* loss_out) {
  pdl_prologue();
  extern __shared__ __align__(16) float sm[];
  float2* sXY = reinterpret_cast<float2*>(sm);           // [QR][QC]
  float2* vM = sXY + QR * QC;                            // [QH][QPM] windows of (x, y)
  float2* vS = vM + QH * QPM;                            // [QH][QPM] windows of (x^2, y^2)
  float* vC = reinterpret_cast<float*>(vS + QH * QPM);   // [QH][QPM] windows of xy
  __shared__ float red[2][kQThreads / 32];
  const int ox = blockIdx.x * QW, oy = blockIdx.y * QH, ch = blockIdx.z;
  const float C1 = 0.01f * 0.01f, C2 = 0.03f * 0.03f;
  float l1 = 0.f, ssim = 0.f;
  // ---- x, y on the tile + 5, zero outside the image (all loads before the first store); a
  // thread stages one column, every other row
  {
    constexpr int kRows = QR / 2;
    const int c = threadIdx.x % QC, rb = threadIdx.x / QC;
    const int gx = ox - 5 + c;
    const bool col_in = gx >= 0 && gx < W;
    const bool col_own = c >= 5 && c < 5 + QW;     // a column of the tile itself
    float xv[kRows], yv[kRows];
#pragma unroll
    for (int j = 0; j < kRows; ++j) {
      const int gy = oy - 5 + rb + 2 * j;
      xv[j] = 0.f;
      yv[j] = 0.f;
      if (col_in && gy >= 0 && gy < H) {
        const int p = gy * W + gx;   // at most 65536 CTAs: about 41M pixels, 4p fits an int
        xv[j] = __ldg(xin + 4 * p + ch);
        yv[j] = __ldg(yin + 3 * p + ch);
      }
    }
#pragma unroll
    for (int j = 0; j < kRows; ++j) {
      const int r = rb + 2 * j;
      sXY[r * QC + c] = make_float2(xv[j], yv[j]);
      // |x - y| of the tile's own pixels (zero off the image, where both are zero)
      if (col_own && r >= 5 && r < 5 + QH) l1 += fabsf(xv[j] - yv[j]);
    }
  }
  __syncthreads();
  // ---- vertical windows: column c, rows r0 .. r0 + 7 (consecutive lanes: consecutive columns)
  {
    const int c = threadIdx.x % QC, r0 = (threadIdx.x / QC) * QRUN;
    float2 v[QRUN + 10], o2[QRUN];
#pragma unroll
    for (int t = 0; t < QRUN + 10; ++t) v[t] = sXY[(r0 + t) * QC + c];
    window_pairs<QRUN>(v, win, o2);
#pragma unroll
    for (int o = 0; o < QRUN; ++o) vM[(r0 + o) * QPM + c] = o2[o];
    float p[QRUN + 10], o1[QRUN];
#pragma unroll
    for (int t = 0; t < QRUN + 10; ++t) {
      p[t] = v[t].x * v[t].y;
      v[t] = __fmul2_rn(v[t], v[t]);
    }
    window_pairs<QRUN>(v, win, o2);
#pragma unroll
    for (int o = 0; o < QRUN; ++o) vS[(r0 + o) * QPM + c] = o2[o];
    window_scalars<QRUN>(p, win, o1);
#pragma unroll
    for (int o = 0; o < QRUN; ++o) vC[(r0 + o) * QPM + c] = o1[o];
  }
  __syncthreads();
  // ---- horizontal windows -> moments -> SSIM and A, B, C of the tile's pixels, staged in the
  // input region (free once the vertical pass is done) for a coalesced copy-out
  float* oA = sm;                   // [QH][QPO]
  float* oB = oA + QH * QPO;        // [QH][QPO]
  float* oC = oB + QH * QPO;        // [QH][QPO]
  if (threadIdx.x < QH * QHSEG) {
    const int r = threadIdx.x % QH, k0 = (threadIdx.x / QH) * QRUN;   // lanes: consecutive rows
    const int c0 = min(k0, QW - QRUN), o0 = k0 - c0;   // the last run starts early and skips
    float2 mm[QRUN], ss[QRUN];
    float mc[QRUN];
    {
      float2 v[QRUN + 10];
#pragma unroll
      for (int t = 0; t < QRUN + 10; ++t) v[t] = vM[r * QPM + c0 + t];
      window_pairs<QRUN>(v, win, mm);
#pragma unroll
      for (int t = 0; t < QRUN + 10; ++t) v[t] = vS[r * QPM + c0 + t];
      window_pairs<QRUN>(v, win, ss);
    }
    {
      float v[QRUN + 10];
#pragma unroll
      for (int t = 0; t < QRUN + 10; ++t) v[t] = vC[r * QPM + c0 + t];
      window_scalars<QRUN>(v, win, mc);
    }
    const int gy = oy + r;
#pragma unroll
    for (int o = 0; o < QRUN; ++o) {
      const int gx = ox + c0 + o;
      if (o < o0 || gx >= W || gy >= H) continue;
      const float mx = mm[o].x, my = mm[o].y;
      const float vx = ss[o].x - mx * mx, vy = ss[o].y - my * my, cxy = mc[o] - mx * my;
      const float N1 = 2.f * mx * my + C1, N2 = 2.f * cxy + C2;
      const float D1 = mx * mx + my * my + C1, D2 = vx + vy + C2;
      const float iD = __fdividef(1.f, D1 * D2);   // fast reciprocal (about 2 ulp)
      const float S = N1 * N2 * iD;
      const float dvx = -S * (D1 * iD);           // -S / D2
      const float dcxy = 2.f * N1 * iD;
      const float A = (2.f * my * N2 - S * 2.f * mx * D2) * iD - 2.f * mx * dvx - my * dcxy;
      ssim += S;
      oA[r * QPO + c0 + o] = A;
      oB[r * QPO + c0 + o] = dvx;
      oC[r * QPO + c0 + o] = dcxy;
    }
  }
  if (abc_ab) {
    __syncthreads();
    // a thread copies one column of the tile, every other row (coalesced along the rows)
    const int c = threadIdx.x % QC, rb = threadIdx.x / QC;
    const int gx = ox + c;
    if (c < QW && gx < W) {
#pragma unroll
      for (int j = 0; j < QH / 2; ++j) {
        const int r = rb + 2 * j, gy = oy + r;
        if (gy >= H) break;
        const int q = (ch * H + gy) * W + gx;
        abc_ab[q] = make_float2(oA[r * QPO + c], oB[r * QPO + c]);
        abc_c[q] = oC[r * QPO + c];
      }
    }
  }
  // block partial sums -> the last block finishes the scalar
  for (int o = 16; o > 0; o >>= 1) {
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
    ssim += __shfl_xor_sync(0xffffffffu, ssim, o);
  }
  if ((threadIdx.x & 31) == 0) { red[0][threadIdx.x >> 5] = l1; red[1][threadIdx.x >> 5] = ssim; }
  __syncthreads();
  const int nb = gridDim.x * gridDim.y * gridDim.z;
  const int b = q_block_index();
  __shared__ bool is_last;
  if (threadIdx.x == 0) {
    float s0 = 0.f, s1 = 0.f;
    for (int k = 0; k < kQThreads / 32; ++k) { s0 += red[0][k]; s1 += red[1][k]; }
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
  for (int k = threadIdx.x; k < nb; k += kQThreads) {
    s0 += (double)__ldcg(&partials[2 * k]);
    s1 += (double)__ldcg(&partials[2 * k + 1]);
  }
  for (int o = 16; o > 0; o >>= 1) {
    s0 += __shfl_xor_sync(0xffffffffu, s0, o);
    s1 += __shfl_xor_sync(0xffffffffu, s1, o);
  }
  __shared__ double dred[2][kQThreads / 32];
  if ((threadIdx.x & 31) == 0) { dred[0][threadIdx.x >> 5] = s0; dred[1][threadIdx.x >> 5] = s1; }
  __syncthreads();
  if (threadIdx.x == 0) {
    double t0 = 0.0, t1 = 0.0;
    for (int k = 0; k < kQThreads / 32; ++k) { t0 += dred[0][k]; t1 += dred[1][k]; }
    const double n = 3.0 * (double)W * (double)H;
    if (loss_out) *loss_out = (float)((1.0 - lam) * t0 / n + lam * (1.0 - t1 / n));
    *ticket = 0u;
  }
}

__global__ void __launch_bounds__(kQThreads, 3)
ssim_bwd_kernel(const float* __restrict__ xin, const float* __restrict__ yin, int W, int H,
                float lam, const Window win, const float2* __restrict__ abc_ab,
                const float* __restrict__ abc_c, float* __restrict__ grad) {
  pdl_prologue();
  extern __shared__ __align__(16) float sm[];
  float2* sAB = reinterpret_cast<float2*>(sm);             // [QR][QC]
  float* sC = reinterpret_cast<float*>(sAB + QR * QC);     // [QR][QC]
  float2* gAB = reinterpret_cast<float2*>(sC + QR * QC);   // [QH][QPM] windows of (A, B)
  float* gC = reinterpret_cast<float*>(gAB + QH * QPM);    // [QH][QPM] windows of C
  const int ox = blockIdx.x * QW, oy = blockIdx.y * QH, ch = blockIdx.z;
  const float inv = 1.f / (3.f * (float)W * (float)H);
  // x and y of the pixels this thread finishes in the last pass (one column of the tile, every
  // other row), loaded first so that their latency hides behind the window passes
  const int fc = threadIdx.x % QC, fr = threadIdx.x / QC;
  const int fx = ox + fc;
  const bool f_col = fc < QW && fx < W;
  float xq[QH / 2], yq[QH / 2];
#pragma unroll
  for (int j = 0; j < QH / 2; ++j) {
    const int gy = oy + fr + 2 * j;
    xq[j] = 0.f;
    yq[j] = 0.f;
    if (f_col && gy < H) {
      const int q = gy * W + fx;
      xq[j] = __ldg(xin + 4 * q + ch);
      yq[j] = __ldg(yin + 3 * q + ch);
    }
  }
  // ---- A, B, C on the tile + 5, zero outside the image (no pixel there contributes); a thread
  // stages one column, every other row
  {
    constexpr int kRows = QR / 2;
    const int c = threadIdx.x % QC, rb = threadIdx.x / QC;
    const int gx = ox - 5 + c;
    const bool col_in = gx >= 0 && gx < W;
    float2 ab[kRows];
    float cv[kRows];
#pragma unroll
    for (int j = 0; j < kRows; ++j) {
      const int gy = oy - 5 + rb + 2 * j;
      ab[j] = make_float2(0.f, 0.f);
      cv[j] = 0.f;
      if (col_in && gy >= 0 && gy < H) {
        const int q = (ch * H + gy) * W + gx;
        ab[j] = __ldcg(abc_ab + q);
        cv[j] = __ldcg(abc_c + q);
      }
    }
#pragma unroll
    for (int j = 0; j < kRows; ++j) {
      const int r = rb + 2 * j;
      sAB[r * QC + c] = ab[j];
      sC[r * QC + c] = cv[j];
    }
  }
  __syncthreads();
  // ---- vertical windows of (A, B) and C
  {
    const int c = threadIdx.x % QC, r0 = (threadIdx.x / QC) * QRUN;
    {
      float2 v[QRUN + 10], o2[QRUN];
#pragma unroll
      for (int t = 0; t < QRUN + 10; ++t) v[t] = sAB[(r0 + t) * QC + c];
      window_pairs<QRUN>(v, win, o2);
#pragma unroll
      for (int o = 0; o < QRUN; ++o) gAB[(r0 + o) * QPM + c] = o2[o];
    }
    {
      float v[QRUN + 10], o1[QRUN];
#pragma unroll
      for (int t = 0; t < QRUN + 10; ++t) v[t] = sC[(r0 + t) * QC + c];
      window_scalars<QRUN>(v, win, o1);
#pragma unroll
      for (int o = 0; o < QRUN; ++o) gC[(r0 + o) * QPM + c] = o1[o];
    }
  }
  __syncthreads();
  // ---- horizontal windows on the output tile, staged in the input region (free once the
  // vertical pass is done), then the gradient in a coalesced pass
  float2* oAB = sAB;                // [QH][QPO]
  float* oC = sC;                   // [QH][QPO]
  if (threadIdx.x < QH * QHSEG) {
    const int r = threadIdx.x % QH, k0 = (threadIdx.x / QH) * QRUN;
    const int c0 = min(k0, QW - QRUN), o0 = k0 - c0;
    {
      float2 v[QRUN + 10], wab[QRUN];
#pragma unroll
      for (int t = 0; t < QRUN + 10; ++t) v[t] = gAB[r * QPM + c0 + t];
      window_pairs<QRUN>(v, win, wab);
#pragma unroll
      for (int o = 0; o < QRUN; ++o) if (o >= o0) oAB[r * QPO + c0 + o] = wab[o];
    }
    {
      float v[QRUN + 10], wc[QRUN];
#pragma unroll
      for (int t = 0; t < QRUN + 10; ++t) v[t] = gC[r * QPM + c0 + t];
      window_scalars<QRUN>(v, win, wc);
#pragma unroll
      for (int o = 0; o < QRUN; ++o) if (o >= o0) oC[r * QPO + c0 + o] = wc[o];
    }
  }
  __syncthreads();
  if (!f_col) return;
#pragma unroll
  for (int j = 0; j < QH / 2; ++j) {
    const int r = fr + 2 * j, gy = oy + r;
    if (gy >= H) break;
    const int q = gy * W + fx;
    const float xv = xq[j], yv = yq[j];
    const float d = xv - yv;
    const float sgn = (d > 0.f) ? 1.f : ((d < 0.f) ? -1.f : 0.f);
    const float2 wab = oAB[r * QPO + fc];
    const float dS = wab.x + 2.f * xv * wab.y + yv * oC[r * QPO + fc];
    grad[3 * q + ch] = ((1.f - lam) * sgn - lam * dS) * inv;
  }
}

// The SSIM window, computed in double and rounded once per tap.
Window ssim_window() {
  Window win;
  double w[11], s = 0.0;
  for (int t = 0; t < 11; ++t) { const double d = t - 5.0; w[t] = std::exp(-d * d / 4.5); s += w[t]; }
  for (int t = 0; t < 11; ++t) win.w[t] = (float)(w[t] / s);
  return win;
}

dim3 loss_grid(int width, int height) {
  return dim3((width + TW - 1) / TW, (height + TH - 1) / TH, 3);
}

}  // namespace

abcd_status loss_launch(abcd_ctx* ctx, const float* out_rgba, const float* gt_rgb, int width,
                        int height, float lambda_ssim, float* loss_out, float* dL_dout) {
  if (!has_workspace(ctx)) return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_loss: no workspace");
  if (!out_rgba || !gt_rgb || width <= 0 || height <= 0 || !(lambda_ssim >= 0.f && lambda_ssim <= 1.f))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_loss: bad arguments");
  if ((long long)width * height > ctx->max_pixels)
    return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_loss: %d x %d pixels, the workspace holds %lld",
                width, height, ctx->max_pixels);
  const dim3 grid((width + QW - 1) / QW, (height + QH - 1) / QH, 3);
  if ((long long)grid.x * grid.y * grid.z > kMaxLossBlocks)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_loss: image too large (%d x %d)", width, height);
  const size_t smem_f = sizeof(float) * kQFwdFloats, smem_b = sizeof(float) * kQBwdFloats;
  cudaError_t e = ensure_smem(ctx, (const void*)ssim_fwd_kernel, smem_f);
  if (e == cudaSuccess && dL_dout) e = ensure_smem(ctx, (const void*)ssim_bwd_kernel, smem_b);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "loss smem attribute: %s", cudaGetErrorString(e));
  const Window win = ssim_window();
  float2* abc_ab = dL_dout ? ctx->ws.ssim_ab : nullptr;
  abcd_status s = check_launch(ctx, "ssim_fwd_kernel",
                               launch_pdl(ssim_fwd_kernel, grid, dim3(kQThreads), smem_f, ctx->stream,
                                          out_rgba, gt_rgb, width, height, lambda_ssim, win, abc_ab,
                                          ctx->ws.ssim_c, ctx->ws.loss_partials, ctx->ws.status + 1,
                                          loss_out));
  if (s != ABCD_OK || !dL_dout) return s;
  return check_launch(ctx, "ssim_bwd_kernel",
                      launch_pdl(ssim_bwd_kernel, grid, dim3(kQThreads), smem_b, ctx->stream, out_rgba,
                                 gt_rgb, width, height, lambda_ssim, win,
                                 (const float2*)ctx->ws.ssim_ab, (const float*)ctx->ws.ssim_c, dL_dout));
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

constexpr int kStaticLossMaxBlocks = 65536;            // CTAs (64x28 pixels, one channel): 8192 x 4096
constexpr long long kStaticLossMaxPixels = 8192LL * 4096;   // the image size the header states
constexpr int kStaticLossWords = 2 * kStaticLossMaxBlocks + 64;   // partial sums, then the ticket

// Device scratch shared by every abcd_loss_static call on a device (held until exit).
static __device__ __align__(256) unsigned g_loss_static_scratch[kStaticLossWords];

// Device address of the static scratch on the current device.  The first lookup on a device
// loads this library's device code there; every call looks the address up again (a host-side
// table read once the code is loaded), so an address never outlives a device reset that moved
// the array.
cudaError_t static_scratch(unsigned** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_loss_static_scratch);
  if (e != cudaSuccess) return e;
  *out = static_cast<unsigned*>(p);
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
  const dim3 grid = loss_grid(width, height);
  // the stated limit is on the image (whatever the tile shape), and the scratch must hold a
  // partial sum per CTA
  if ((long long)width * height > kStaticLossMaxPixels ||
      (long long)grid.x * grid.y * grid.z > kStaticLossMaxBlocks)
    return ABCD_ERR_WORKSPACE;
  unsigned* scratch = nullptr;
  if (static_scratch(&scratch) != cudaSuccess) return ABCD_ERR_CUDA;
  float* partials = reinterpret_cast<float*>(scratch);
  unsigned* ticket = scratch + 2 * kStaticLossMaxBlocks;
  cudaStream_t stream = (cudaStream_t)cuda_stream;
  // the ticket must start at zero whatever an earlier (possibly failed) call left there
  if (cudaMemsetAsync(ticket, 0, sizeof(unsigned), stream) != cudaSuccess) return ABCD_ERR_CUDA;
  const size_t smem = sizeof(float) * kSmemFloats;
  if (cudaFuncSetAttribute(loss_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
      cudaSuccess)
    return ABCD_ERR_CUDA;
  const cudaError_t e = launch_pdl(loss_kernel, grid, dim3(kThreads), smem, stream, out_rgba,
                                   gt_rgb, width, height, lambda_ssim, ssim_window(), dL_dout,
                                   partials, ticket, loss_out);
  return e == cudaSuccess ? ABCD_OK : ABCD_ERR_CUDA;   // the launch's own status, not a sticky one
}
