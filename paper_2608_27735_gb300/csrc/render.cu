// K5 (blend + composite forward, also the cache refresh K10) and K7 (its backward).
//
// Per pixel, front to back over its tile's list (3DGS blending): sigma = 1/2 d^T Q d with
// d = pixel centre - uv, alpha = min(alpha_max, o exp(-sigma)), skip alpha < alpha_min (and
// sigma < 0), stop before T (1 - alpha) < t_min; A = (sum T_i alpha_i c_i, 1 - T).  Then the
// frozen partitions enter through out = F over (A over B) (Section 2), over meaning
// X + (1 - X.a) Y on premultiplied RGBA, and out.rgb += (1 - out.a) bg.
//
// One warp per 8x8 block of pixels (four per 16x16 binning tile), two pixels per lane --
// (x, y) and (x + 4, y), which share the shared-memory loads and the dy terms of sigma -- so
// the few heavily covered tiles of a small active block spread over four times as many CTAs,
// each lane runs two independent blend chains, and each CTA stops as soon as its own 64
// pixels have terminated.  List entries are staged in shared memory; an entry whose opacity
// cannot reach alpha_min anywhere on the CTA's pixel-centre box (analytic minimum of the
// quadratic form over the box, with a margin far above fp32 rounding) is dropped while
// staging -- every pixel would skip it, so results are unchanged -- and staging keeps loading
// groups of 64 entries, all in flight at once, until a batch of survivors is full, so the
// blocks that walk a long list whose entries mostly miss them are bound by bandwidth rather
// than by one load round trip per 32 entries.  Every quantity that decides a branch per pixel
// (sigma, alpha, T) is computed with explicit round-to-nearest intrinsics in one shared
// function, so the backward kernel retraces exactly the forward's contributors.
//
// Work is very uneven across blocks (lists of a few entries next to lists of 15,000), so both
// kernels take their tiles in the order bin_sort left in the workspace (decreasing list
// length) when it was made for the ranges they are given: the longest blocks start in the
// first wave instead of trailing the launch.  The order changes no result (CTAs are
// independent; the backward's gradient sums are atomic either way).
#include "abcd_internal.cuh"

namespace abcd {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kHalfLog2e = 0.7213475204444817f;
constexpr float kLn2 = 0.6931471805599453f;

constexpr int kSub = 8;                          // CTA pixel block edge
constexpr int kSubThreads = 32;                  // one warp, two pixels per lane
constexpr int kSubPerTile = (kTile / kSub) * (kTile / kSub);
static_assert(kSubPerTile == kRenderSubPerTile, "tile order expands to kRenderSubPerTile CTAs per tile");
constexpr int kRounds = 2;                       // list entries per lane per staging group
constexpr int kGroup = kSubThreads * kRounds;    // 64 entries loaded together
constexpr int kBatch = kGroup;                   // staged survivors per batch (at most)
constexpr int kCkChunk = 128;                    // list positions per backward chunk
constexpr int kItemCtasPerSm = 16;               // backward CTAs that replay listed chunks
static_assert(kCkChunk % kGroup == 0, "checkpoints fall on staging group boundaries");

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Conic scaled for base-2 exponentials: (a/2, b, c/2) * log2(e), opacity kept.
__device__ __forceinline__ float4 scaled_conic(float4 c) {
  return make_float4(__fmul_rn(kHalfLog2e, c.x), __fmul_rn(kLog2e, c.y), __fmul_rn(kHalfLog2e, c.z), c.w);
}

// sigma * log2(e) = dx (a/2 dx + b dy) + c/2 dy^2 at the lane's two pixels (fx0, fy) and
// (fx1, fy); the dy terms are shared.  Both kernels take every branch decision from these bits.
// The two pixels go through the packed two-lane fp32 instructions, whose every component is
// rounded exactly as the scalar instruction would round it.
__device__ __forceinline__ void sigma_pair(float4 s, float2 m, float fx0, float fx1, float fy,
                                           float& dx0, float& dx1, float& dy, float& s0, float& s1) {
  dy = __fsub_rn(fy, m.y);
  const float2 dx = __fadd2_rn(make_float2(fx0, fx1), make_float2(-m.x, -m.x));
  dx0 = dx.x;
  dx1 = dx.y;
  const float bdy = __fmul_rn(s.y, dy);
  const float cdy2 = __fmul_rn(__fmul_rn(s.z, dy), dy);
  const float2 in = __ffma2_rn(make_float2(s.x, s.x), dx, make_float2(bdy, bdy));
  const float2 sg = __ffma2_rn(dx, in, make_float2(cdy2, cdy2));
  s0 = sg.x;
  s1 = sg.y;
}

// Lower bound of sigma * log2(e) over the box [X0, X1] x [Y0, Y1] of offsets d = pixel - uv:
// 0 if the box contains d = 0, else the least value on its four edges (convex quadratic; on
// each edge the minimiser of the other coordinate is clamped into the box).
__device__ __forceinline__ float box_min_sigma2(float4 s, float X0, float X1, float Y0, float Y1) {
  if (X0 <= 0.f && X1 >= 0.f && Y0 <= 0.f && Y1 >= 0.f) return 0.f;
  const float ry = __fdividef(-s.y, 2.f * s.z), rx = __fdividef(-s.y, 2.f * s.x);
  float best = 3.0e38f;
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const float X = e ? X1 : X0;
    const float dy = fminf(fmaxf(ry * X, Y0), Y1);
    best = fminf(best, X * (s.x * X + s.y * dy) + s.z * dy * dy);
    const float Y = e ? Y1 : Y0;
    const float dx = fminf(fmaxf(rx * Y, X0), X1);
    best = fminf(best, dx * (s.x * dx + s.y * Y) + s.z * Y * Y);
  }
  return best;
}

// True when no pixel centre of the CTA's box can give alpha >= alpha_min: alpha = o 2^-sigma'
// < alpha_min needs sigma' > log2(o / alpha_min); the margin (0.02 + 0.2% in log2 units) is
// orders of magnitude above the fp32 error of either evaluation.
__device__ __forceinline__ bool cull(float4 s, float2 m, float bx0, float by0, float alpha_min) {
  if (!(s.w >= alpha_min)) return true;
  const float thr = __log2f(__fdividef(s.w, alpha_min));
  const float lo = box_min_sigma2(s, bx0 - m.x, bx0 + (kSub - 1) - m.x, by0 - m.y, by0 + (kSub - 1) - m.y);
  return lo * 0.998f > thr + 0.02f;
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

// Stages list entries from position `next` on, in groups of kGroup whose loads are all issued
// before any is used, until more than kBatch - kGroup survivors of the CTA-box cull are staged
// or position n is reached; survivors are compacted in list order, each with its list
// position in s_rgb[.].w (bits) and, for the backward, its Gaussian id.  Returns the number
// staged.  next and the count are warp-uniform.
template <bool WITH_ID>
__device__ __forceinline__ int stage_fill(const unsigned* ids, unsigned start, int n, int& next,
                                          const float2* uv, const float4* co, const float* rgb,
                                          float bx0, float by0, float alpha_min, float2* s_uv,
                                          float4* s_co, float4* s_rgb, unsigned* s_id) {
  const int lane = threadIdx.x & 31;
  const unsigned lt = (1u << lane) - 1u;
  int total = 0;
  while (next < n && total <= kBatch - kGroup) {
    unsigned g[kRounds];
    float2 m[kRounds];
    float4 c[kRounds];
    float col[kRounds][3];
#pragma unroll
    for (int r = 0; r < kRounds; ++r) {
      const int pos = next + lane + r * kSubThreads;
      g[r] = pos < n ? __ldg(ids + start + pos) : 0xffffffffu;
    }
#pragma unroll
    for (int r = 0; r < kRounds; ++r) {
      if (g[r] != 0xffffffffu) {
        m[r] = __ldg(uv + g[r]);
        c[r] = __ldg(co + g[r]);
        col[r][0] = __ldg(rgb + 3 * g[r]);
        col[r][1] = __ldg(rgb + 3 * g[r] + 1);
        col[r][2] = __ldg(rgb + 3 * g[r] + 2);
      }
    }
#pragma unroll
    for (int r = 0; r < kRounds; ++r) {
      bool keep = false;
      float4 sc = make_float4(0.f, 0.f, 0.f, 0.f);
      if (g[r] != 0xffffffffu) {
        sc = scaled_conic(c[r]);
        keep = !cull(sc, m[r], bx0, by0, alpha_min);
      }
      const unsigned b = __ballot_sync(0xffffffffu, keep);
      if (keep) {
        const int slot = total + __popc(b & lt);
        s_uv[slot] = m[r];
        s_co[slot] = sc;
        s_rgb[slot] = make_float4(col[r][0], col[r][1], col[r][2],
                                  __uint_as_float((unsigned)(next + lane + r * kSubThreads)));
        if (WITH_ID) s_id[slot] = g[r];
      }
      total += __popc(b);
    }
    next += kGroup;
  }
  // the blend loops read up to one (forward) or two (backward) slots past the last survivor
  // as masked-out entries: they must hold finite zeros, not another kernel's leftovers (a
  // zero weight times a non-finite value is not zero)
  constexpr int kPad = WITH_ID ? 2 : 1;
  constexpr int kSlots = WITH_ID ? kBatch + 2 : kBatch;
  if (lane < kPad && total + lane < kSlots) {
    s_uv[total + lane] = make_float2(0.f, 0.f);
    s_co[total + lane] = make_float4(0.f, 0.f, 0.f, 0.f);
    s_rgb[total + lane] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (WITH_ID) s_id[total + lane] = 0u;
  }
  __syncwarp();
  return total;
}

// Render CTA b handles the 8x8 block tile_order[b / 4] * 4 + b % 4 (tile_order: a permutation
// of the tiles, longest list first), or block b.
__device__ __forceinline__ int block_index(const unsigned* tile_order, int b) {
  if (tile_order) return (int)tile_order[b / kSubPerTile] * kSubPerTile + b % kSubPerTile;
  return b;
}

// Index, within its 8x8 block, of the lane's first pixel (the second is 4 further).
__device__ __forceinline__ int block_pixel(int lane) { return (lane >> 2) * kSub + (lane & 3); }

// The CTA's 8x8 pixel block and the lane's two pixels (qx0, py), (qx1 = qx0 + 4, py).
struct Block {
  int tile, px0, py0, qx0, qx1, py;
  bool in0, in1;
};

__device__ __forceinline__ Block block_of(const Cam& cam, int blk) {
  Block b;
  b.tile = blk / kSubPerTile;
  const int sub = blk % kSubPerTile;
  const int tx = b.tile % cam.tiles_x, ty = b.tile / cam.tiles_x;
  b.px0 = tx * kTile + (sub % (kTile / kSub)) * kSub;
  b.py0 = ty * kTile + (sub / (kTile / kSub)) * kSub;
  const int lane = threadIdx.x & 31;
  b.qx0 = b.px0 + (lane & 3);
  b.qx1 = b.qx0 + 4;
  b.py = b.py0 + (lane >> 2);
  b.in0 = b.qx0 < cam.width && b.py < cam.height;
  b.in1 = b.qx1 < cam.width && b.py < cam.height;
  return b;
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
  uint2* refresh_packed;        // fp16 x4 per pixel of the tiles tile_map lists (packed layer)
  const int* tile_map;
  const unsigned* tile_order;   // tiles, longest list first (nullptr: launch order)
  float4* ckpt;                 // render checkpoints (nullptr: none), see the workspace
  uint4* ck_items;
  unsigned* ck_count;
  unsigned* ck_first;
  int ck_cap;
  const unsigned* status;       // the context's status word: after a timed-out wait the lists
                                // may hold stale ids, so every list reads as empty
};

// Blend state of one pixel.
struct PixF {
  float T, c0, c1, c2;
  unsigned last;       // one past the list position of the last contributor
  bool done;
};

// Blend state of the lane's two pixels, the first in .x, the second in .y.
struct PixF2 {
  float2 T, c0, c1, c2;
  unsigned last0, last1;
  bool done0, done1;
};

// One staged list entry as the blend loops read it.
struct Entry {
  float4 s;            // scaled conic, opacity
  float2 m;            // uv
  float4 col;          // rgb, list position (bits)
};

__device__ __forceinline__ Entry load_entry(const float2* s_uv, const float4* s_co,
                                            const float4* s_rgb, int j) {
  Entry e;
  e.s = s_co[j];
  e.m = s_uv[j];
  e.col = s_rgb[j];
  return e;
}

// alpha at the lane's two pixels for one entry and whether each passes the skip tests
// (sigma >= 0, alpha >= alpha_min).  Independent of the blend state, so the loops evaluate
// it for several entries before the transmittance chain needs it.
__device__ __forceinline__ void alpha_pair(const Entry& e, float fx0, float fx1, float fy,
                                           const Opts& op, float& a0, float& a1, bool& ok0,
                                           bool& ok1) {
  float dx0, dx1, dy, sg0, sg1;
  sigma_pair(e.s, e.m, fx0, fx1, fy, dx0, dx1, dy, sg0, sg1);
  a0 = fminf(op.alpha_max, __fmul_rn(e.s.w, ex2_approx(-sg0)));
  a1 = fminf(op.alpha_max, __fmul_rn(e.s.w, ex2_approx(-sg1)));
  ok0 = sg0 >= 0.f && a0 >= op.alpha_min;
  ok1 = sg1 >= 0.f && a1 >= op.alpha_min;
}

// Front-to-back step of the lane's two pixels for one entry (selects, no branches): a passing
// entry either ends a pixel (T (1 - alpha) < t_min; it does not contribute) or is blended in.
// A pixel the entry does not reach gets a zero weight, and fma(0, c, C) leaves C as it was.
__device__ __forceinline__ void blend2(PixF2& p, float a0, float a1, bool ok0, bool ok1,
                                       float4 col, const Opts& op) {
  ok0 = ok0 && !p.done0;
  ok1 = ok1 && !p.done1;
  const float2 al = make_float2(a0, a1);
  const float2 test = __fmul2_rn(p.T, __fadd2_rn(make_float2(1.f, 1.f), make_float2(-a0, -a1)));
  const bool term0 = ok0 && test.x < op.t_min, term1 = ok1 && test.y < op.t_min;
  const bool use0 = ok0 && !term0, use1 = ok1 && !term1;
  const float2 w = __fmul2_rn(al, p.T);
  const float2 wu = make_float2(use0 ? w.x : 0.f, use1 ? w.y : 0.f);
  p.done0 = p.done0 || term0;
  p.done1 = p.done1 || term1;
  p.c0 = __ffma2_rn(wu, make_float2(col.x, col.x), p.c0);
  p.c1 = __ffma2_rn(wu, make_float2(col.y, col.y), p.c1);
  p.c2 = __ffma2_rn(wu, make_float2(col.z, col.z), p.c2);
  p.T = make_float2(use0 ? test.x : p.T.x, use1 ? test.y : p.T.y);
  const unsigned nxt = __float_as_uint(col.w) + 1u;
  p.last0 = use0 ? nxt : p.last0;
  p.last1 = use1 ? nxt : p.last1;
}

__device__ __forceinline__ void store_pixel(const FwdArgs& a, long long p, const PixF& s, int qx,
                                            int qy, int tile) {
  const float Aa = 1.f - s.T;
  if (a.refresh || a.refresh_packed) {
    const __half2 lo = __floats2half2_rn(s.c0, s.c1), hi = __floats2half2_rn(s.c2, Aa);
    uint2 r;
    r.x = *reinterpret_cast<const unsigned*>(&lo);
    r.y = *reinterpret_cast<const unsigned*>(&hi);
    if (a.refresh) a.refresh[p] = r;
    if (a.refresh_packed) {
      const int m = a.tile_map[tile];
      if (m >= 0) a.refresh_packed[(size_t)m * kTileThreads + (qy % kTile) * kTile + qx % kTile] = r;
    }
  }
  if (a.state_at) {
    a.state_at[p] = make_float4(s.c0, s.c1, s.c2, s.T);
    a.n_last[p] = s.last;
  }
  if (a.out) {
    const float4 Bv = a.B ? load_px(a.B, a.fb_dtype, p) : make_float4(0.f, 0.f, 0.f, 0.f);
    const float4 Fv = a.F ? load_px(a.F, a.fb_dtype, p) : make_float4(0.f, 0.f, 0.f, 0.f);
    const float kb = 1.f - Aa;      // A over B
    const float m0 = s.c0 + kb * Bv.x, m1 = s.c1 + kb * Bv.y, m2 = s.c2 + kb * Bv.z, ma = Aa + kb * Bv.w;
    const float kf = 1.f - Fv.w;    // F over (A over B)
    float4 o = make_float4(Fv.x + kf * m0, Fv.y + kf * m1, Fv.z + kf * m2, Fv.w + kf * ma);
    const float kg = 1.f - o.w;
    o.x += kg * a.bg[0];
    o.y += kg * a.bg[1];
    o.z += kg * a.bg[2];
    a.out[p] = o;
  }
}

__global__ void __launch_bounds__(kSubThreads) render_fwd_kernel(FwdArgs a) {
  pdl_prologue();
  __shared__ float2 s_uv[kBatch];
  __shared__ float4 s_co[kBatch];
  __shared__ float4 s_rgb[kBatch];
  const int blk = block_index(a.tile_order, (int)blockIdx.x);
  const Block bk = block_of(a.cam, blk);
  const int lane = threadIdx.x & 31;
  const uint2 rg = a.ranges[bk.tile];
  const int n = (rg.y > rg.x && !(*a.status & kStatusTimeout)) ? (int)(rg.y - rg.x) : 0;
  const float fx0 = (float)bk.qx0 + 0.5f, fx1 = (float)bk.qx1 + 0.5f, fy = (float)bk.py + 0.5f;
  const float bx0 = (float)bk.px0 + 0.5f, by0 = (float)bk.py0 + 0.5f;
  PixF2 pp;
  pp.T = make_float2(1.f, 1.f);
  pp.c0 = pp.c1 = pp.c2 = make_float2(0.f, 0.f);
  pp.last0 = pp.last1 = 0u;
  pp.done0 = !bk.in0;
  pp.done1 = !bk.in1;
  int next = 0;
  bool ck_on = a.ckpt != nullptr;          // warp-uniform
  int n_items = 0;
  unsigned my_slot = 0u;                   // lane k: the slot of this block's item k
  while (next < n) {
    if (__all_sync(0xffffffffu, pp.done0 && pp.done1)) break;
    __syncwarp();
    // with checkpoints, a batch ends at the next multiple of kCkChunk
    const int lim = ck_on ? min(n, (next / kCkChunk + 1) * kCkChunk) : n;
    const int cnt = stage_fill<false>(a.ids, rg.x, lim, next, a.uv, a.co, a.rgb, bx0, by0,
                                      a.op.alpha_min, s_uv, s_co, s_rgb, nullptr);
    // two entries per iteration (slot j + 1 <= kBatch - 1 exists; unused when j + 1 == cnt)
    for (int j = 0; j < cnt; j += 2) {
      const Entry e0 = load_entry(s_uv, s_co, s_rgb, j);
      const Entry e1 = load_entry(s_uv, s_co, s_rgb, j + 1);
      float a00, a01, a10, a11;
      bool k00, k01, k10, k11;
      alpha_pair(e0, fx0, fx1, fy, a.op, a00, a01, k00, k01);
      alpha_pair(e1, fx0, fx1, fy, a.op, a10, a11, k10, k11);
      const bool v1 = j + 1 < cnt;
      blend2(pp, a00, a01, k00, k01, e0.col, a.op);
      blend2(pp, a10, a11, k10 && v1, k11 && v1, e1.col, a.op);
      if ((j & 30) == 30 && __all_sync(0xffffffffu, pp.done0 && pp.done1)) break;
    }
    if (ck_on && next == lim && lim < n && !__all_sync(0xffffffffu, pp.done0 && pp.done1)) {
      // the state after every position below lim, for the backward's chunk starting there
      unsigned slot = 0u;
      if (lane == 0) slot = atomicAdd(a.ck_count, 1u);
      slot = __shfl_sync(0xffffffffu, slot, 0);
      if (slot < (unsigned)a.ck_cap) {
        float4* ck = a.ckpt + (size_t)slot * (kSub * kSub);
        const int k0 = block_pixel(lane);
        ck[k0] = make_float4(pp.c0.x, pp.c1.x, pp.c2.x, pp.T.x);
        ck[k0 + 4] = make_float4(pp.c0.y, pp.c1.y, pp.c2.y, pp.T.y);
        if (lane == n_items) my_slot = slot;
        ++n_items;
      }
      // past 32 items or a full buffer the last item listed runs to the end of the walk
      ck_on = slot < (unsigned)a.ck_cap && n_items < 32;
    }
  }
  const PixF p0 = {pp.T.x, pp.c0.x, pp.c1.x, pp.c2.x, pp.last0, pp.done0};
  const PixF p1 = {pp.T.y, pp.c0.y, pp.c1.y, pp.c2.y, pp.last1, pp.done1};
  if (a.ckpt) {
    if (lane == 0) a.ck_first[blk] = n_items > 0 ? (unsigned)kCkChunk : 0xffffffffu;
    if (lane < n_items) {
      const unsigned start = (unsigned)((lane + 1) * kCkChunk);
      a.ck_items[my_slot] = make_uint4((unsigned)blk, start, lane == n_items - 1 ? 0xffffffffu : start + kCkChunk, 0u);
    }
  }
  if (bk.in0) store_pixel(a, (long long)bk.py * a.cam.width + bk.qx0, p0, bk.qx0, bk.py, bk.tile);
  if (bk.in1) store_pixel(a, (long long)bk.py * a.cam.width + bk.qx1, p1, bk.qx1, bk.py, bk.tile);
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
  const unsigned* tile_order;   // tiles, longest list first (nullptr: launch order)
  const float4* ckpt;           // the forward's checkpoints (nullptr: every block walks whole)
  const uint4* ck_items;
  const unsigned* ck_count;
  const unsigned* ck_first;
  int ck_cap;
  int n_item_ctas;              // the first CTAs of the launch replay the listed chunks
  const unsigned* status;       // as in FwdArgs
};

// Backward state of one pixel.  With G = dL/dA.rgb and G_a = dL/dA.a, the derivative of the
// loss w.r.t. an entry's alpha is
//   sum_ch G_ch (T col_ch - (A_ch - C_ch) / (1 - alpha)) + G_a T_final / (1 - alpha)
//   = T (G . col) - (K - G . C) / (1 - alpha),   K = G . A - G_a T_final,
// C the colour accumulated up to and including the entry: only the scalar G . C is replayed.
struct PixB {
  float T, Gc;                  // transmittance and G . C replayed up to the current entry
  float Gr, Gg, Gb, K;          // dL/dA.rgb; G . A - G_a T_final
  unsigned last;                // replay only list positions below this
};

__device__ __forceinline__ void load_pixel_grad(const BwdArgs& a, long long p, int n, PixB& q) {
  q.last = min(a.n_last[p], (unsigned)n);
  const float4 at = a.state_at[p];
  const float g0 = a.dl_dout[3 * p], g1 = a.dl_dout[3 * p + 1], g2 = a.dl_dout[3 * p + 2];
  const float4 Fv = a.F ? load_px(a.F, a.fb_dtype, p) : make_float4(0.f, 0.f, 0.f, 0.f);
  const float4 Bv = a.B ? load_px(a.B, a.fb_dtype, p) : make_float4(0.f, 0.f, 0.f, 0.f);
  const float kf = 1.f - Fv.w;
  q.Gr = kf * g0; q.Gg = kf * g1; q.Gb = kf * g2;
  // d final / d A.a = -(1 - F.a) (B.rgb + (1 - B.a) bg)
  const float Ga = -kf * (g0 * (Bv.x + (1.f - Bv.w) * a.bg[0]) + g1 * (Bv.y + (1.f - Bv.w) * a.bg[1]) +
                          g2 * (Bv.z + (1.f - Bv.w) * a.bg[2]));
  q.K = q.Gr * at.x + q.Gg * at.y + q.Gb * at.z - Ga * at.w;
}

// Backward of the lane's two pixels for one list entry (selects, no branches): when the entry
// contributed to a pixel (live: a position below the pixel's last contributor; sigma >= 0;
// alpha >= alpha_min) adds to v the opacity and colour gradients (v[5..8]) and the moments of
// d = pixel - uv weighted by dL/dsigma, (sum w dx, w dy, w dx^2, w dx dy, w dy^2) in v[0..4]
// (the conic and mean gradients follow from them once per entry), and advances the replayed
// transmittance exactly as the forward did.  With G = dL/dA.rgb and G_a = dL/dA.a, the
// derivative of the loss w.r.t. an entry's alpha is
//   T (G . col) - (K - G . C) / (1 - alpha),   K = G . A - G_a T_final,
// C the colour accumulated up to and including the entry.  The two pixels' arithmetic is paired through the packed two-lane fp32 instructions and the shared row
// offset dy factored out of the moment sums (sum t dy = (t0 + t1) dy).  The decisions (alpha,
// the skip tests, the replayed transmittance) are rounded exactly as the forward rounds them;
// the gradient terms only round in a different order.  who0 / who1: whether the entry
// contributed to each pixel.
struct PixB2 {
  float2 T, Gc, Gr, Gg, Gb, K;
};

__device__ __forceinline__ void pixel_backward2(PixB2& p, float4 s, float4 col, float sg0,
                                                float sg1, float dx0, float dx1, float dy,
                                                bool live0, bool live1, const Opts& op, float* v,
                                                bool& who0, bool& who1) {
  const float2 G = make_float2(ex2_approx(-sg0), ex2_approx(-sg1));
  const float2 raw = __fmul2_rn(make_float2(s.w, s.w), G);
  const float a0 = fminf(op.alpha_max, raw.x), a1 = fminf(op.alpha_max, raw.y);
  const bool ok0 = live0 && sg0 >= 0.f && a0 >= op.alpha_min;
  const bool ok1 = live1 && sg1 >= 0.f && a1 >= op.alpha_min;
  const float2 w = __fmul2_rn(make_float2(a0, a1), p.T);
  const float2 gcol = __ffma2_rn(p.Gb, make_float2(col.z, col.z),
                                 __ffma2_rn(p.Gg, make_float2(col.y, col.y),
                                            __fmul2_rn(p.Gr, make_float2(col.x, col.x))));
  const float2 gc = __ffma2_rn(w, gcol, p.Gc);                     // G . C including the entry
  const float2 oma = __fadd2_rn(make_float2(1.f, 1.f), make_float2(-a0, -a1));
  const float2 ioma = make_float2(__fdividef(1.f, oma.x), __fdividef(1.f, oma.y));
  const float2 km = __fadd2_rn(p.K, make_float2(-gc.x, -gc.y));
  const float2 dalpha = __ffma2_rn(make_float2(-km.x, -km.y), ioma, __fmul2_rn(p.T, gcol));
  const bool ga0 = ok0 && raw.x <= op.alpha_max, ga1 = ok1 && raw.y <= op.alpha_max;
  const float2 dg = __fmul2_rn(dalpha, G);                          // d alpha / d opacity = G
  const float2 dr = __fmul2_rn(dalpha, raw);                        // d alpha / d sigma = -alpha
  const float wk0 = ok0 ? w.x : 0.f, wk1 = ok1 ? w.y : 0.f;
  const float ds0 = ga0 ? -dr.x : 0.f, ds1 = ga1 ? -dr.y : 0.f;
  v[5] += (ga0 ? dg.x : 0.f) + (ga1 ? dg.y : 0.f);
  v[6] = fmaf(p.Gr.x, wk0, fmaf(p.Gr.y, wk1, v[6]));
  v[7] = fmaf(p.Gg.x, wk0, fmaf(p.Gg.y, wk1, v[7]));
  v[8] = fmaf(p.Gb.x, wk0, fmaf(p.Gb.y, wk1, v[8]));
  const float2 t = __fmul2_rn(make_float2(ds0, ds1), make_float2(dx0, dx1));
  const float ts = t.x + t.y, us = (ds0 + ds1) * dy;
  v[0] += ts;
  v[1] += us;
  v[2] = fmaf(t.x, dx0, fmaf(t.y, dx1, v[2]));
  v[3] = fmaf(ts, dy, v[3]);
  v[4] = fmaf(us, dy, v[4]);
  p.Gc = make_float2(ok0 ? gc.x : p.Gc.x, ok1 ? gc.y : p.Gc.y);
  const float2 Tn = __fmul2_rn(p.T, oma);
  p.T = make_float2(ok0 ? Tn.x : p.T.x, ok1 ? Tn.y : p.T.y);
  who0 = ok0;
  who1 = ok1;
}

// Warp sum of 27 per-lane values through shared memory: each lane writes its row, lane l < 27
// reads column l (32 values, 8 float4 loads; pitch 36 keeps stores and loads conflict-free)
// and returns its sum.
constexpr int kRedPitch = 36;

__device__ __forceinline__ float warp_sum27(const float (&x)[27], float* red, int lane) {
#pragma unroll
  for (int k = 0; k < 27; ++k) red[k * kRedPitch + lane] = x[k];
  __syncwarp();
  float r = 0.f;
  if (lane < 27) {
    const float4* col = reinterpret_cast<const float4*>(red + lane * kRedPitch);
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const float4 a = col[q];
      r += (a.x + a.y) + (a.z + a.w);
    }
  }
  __syncwarp();
  return r;
}

// Backward of list positions [start, end) of block blk (clipped to the block's walk), from the
// forward's checkpoint `ck` when start > 0.
__device__ __forceinline__ void bwd_chunk(const BwdArgs& a, int blk, int start, unsigned end,
                                          const float4* ck, float2* s_uv, float4* s_co,
                                          float4* s_rgb, unsigned* s_id, float* s_red) {
  const Block bk = block_of(a.cam, blk);
  const int lane = threadIdx.x & 31;
  const uint2 rg = a.ranges[bk.tile];
  const int n = (rg.y > rg.x && !(*a.status & kStatusTimeout)) ? (int)(rg.y - rg.x) : 0;
  const float fx0 = (float)bk.qx0 + 0.5f, fx1 = (float)bk.qx1 + 0.5f, fy = (float)bk.py + 0.5f;
  const float bx0 = (float)bk.px0 + 0.5f, by0 = (float)bk.py0 + 0.5f;
  PixB p0 = {}, p1 = {};
  p0.T = p1.T = 1.f;
  if (bk.in0) load_pixel_grad(a, (long long)bk.py * a.cam.width + bk.qx0, n, p0);
  if (bk.in1) load_pixel_grad(a, (long long)bk.py * a.cam.width + bk.qx1, n, p1);
  if (ck) {
    const int k0 = block_pixel(lane);
    const float4 c0 = ck[k0], c1 = ck[k0 + 4];
    p0.T = c0.w; p0.Gc = p0.Gr * c0.x + p0.Gg * c0.y + p0.Gb * c0.z;
    p1.T = c1.w; p1.Gc = p1.Gr * c1.x + p1.Gg * c1.y + p1.Gb * c1.z;
  }
  const int span = (int)min((unsigned)__reduce_max_sync(0xffffffffu, max(p0.last, p1.last)), end);
  PixB2 pp;
  pp.T = make_float2(p0.T, p1.T);
  pp.Gc = make_float2(p0.Gc, p1.Gc);
  pp.Gr = make_float2(p0.Gr, p1.Gr);
  pp.Gg = make_float2(p0.Gg, p1.Gg);
  pp.Gb = make_float2(p0.Gb, p1.Gb);
  pp.K = make_float2(p0.K, p1.K);
  const unsigned last0 = p0.last, last1 = p1.last;
  int next = start;
  while (next < span) {
    __syncwarp();
    const int cnt = stage_fill<true>(a.ids, rg.x, span, next, a.uv, a.co, a.rgb, bx0, by0,
                                     a.op.alpha_min, s_uv, s_co, s_rgb, s_id);
    // three entries per iteration, their 27 components summed over the warp at once (slots up
    // to j + 2 <= kBatch + 1 exist; unused past cnt)
    for (int j = 0; j < cnt; j += 3) {
      float x[27];
#pragma unroll
      for (int k = 0; k < 27; ++k) x[k] = 0.f;
      unsigned who[3];
#pragma unroll
      for (int i = 0; i < 3; ++i) {
        const Entry e = load_entry(s_uv, s_co, s_rgb, j + i);
        const unsigned pos = __float_as_uint(e.col.w);
        const bool valid = j + i < cnt;
        float dx0, dx1, dy, sg0, sg1;
        sigma_pair(e.s, e.m, fx0, fx1, fy, dx0, dx1, dy, sg0, sg1);
        bool c0, c1;
        pixel_backward2(pp, e.s, e.col, sg0, sg1, dx0, dx1, dy, valid && pos < last0,
                        valid && pos < last1, a.op, x + 9 * i, c0, c1);
        who[i] = __ballot_sync(0xffffffffu, c0 || c1);
      }
      if ((who[0] | who[1] | who[2]) == 0) continue;
      const float r = warp_sum27(x, s_red, lane);
      const int ei = min(lane / 9, 2), comp = lane - 9 * ei;
      // mean and conic gradients from the weighted moments of entry ei:
      // d/du = -(ca Sx + cb Sy), d/dv = -(cb Sx + cc Sy), d/da = Sxx / 2, d/db = Sxy,
      // d/dc = Syy / 2, with (ca, cb, cc) = ln 2 (2 a', b', 2 c') of the scaled conic
      const float sx = __shfl_sync(0xffffffffu, r, 9 * ei);
      const float sy = __shfl_sync(0xffffffffu, r, 9 * ei + 1);
      const unsigned wi = ei == 0 ? who[0] : (ei == 1 ? who[1] : who[2]);
      if (lane < 27 && wi != 0) {
        float g = r;
        if (comp <= 1) {
          const float4 sc = s_co[j + ei];
          const float ca = 2.f * kLn2 * sc.x, cb = kLn2 * sc.y, cc = 2.f * kLn2 * sc.z;
          g = comp == 0 ? -(ca * sx + cb * sy) : -(cb * sx + cc * sy);
        } else if (comp == 2 || comp == 4) {
          g = 0.5f * r;
        }
        atomicAdd(a.grad2d + 9 * (size_t)s_id[j + ei] + comp, g);
      }
    }
  }
}

__global__ void __launch_bounds__(kSubThreads, 24) render_bwd_kernel(BwdArgs a) {
  pdl_prologue();
  __shared__ float2 s_uv[kBatch + 2];
  __shared__ float4 s_co[kBatch + 2];
  __shared__ float4 s_rgb[kBatch + 2];
  __shared__ unsigned s_id[kBatch + 2];
  __shared__ __align__(16) float s_red[27 * kRedPitch];
  // the first n_item_ctas CTAs replay the listed chunks after the first of the long walks, the
  // others each a block's walk up to its first checkpoint
  const int b = (int)blockIdx.x;
  const bool item_cta = b < a.n_item_ctas;
  const unsigned items = item_cta ? min(*a.ck_count, (unsigned)a.ck_cap) : 0u;
  for (unsigned i = b; !item_cta || i < items; i += a.n_item_ctas) {
    int blk, start = 0;
    unsigned end = 0xffffffffu;
    const float4* ck = nullptr;
    if (item_cta) {
      const uint4 it = a.ck_items[i];
      blk = (int)it.x; start = (int)it.y; end = it.z;
      ck = a.ckpt + (size_t)i * (kSub * kSub);
    } else {
      blk = block_index(a.tile_order, b - a.n_item_ctas);
      if (a.ckpt) end = a.ck_first[blk];
    }
    __syncwarp();
    bwd_chunk(a, blk, start, end, ck, s_uv, s_co, s_rgb, s_id, s_red);
    if (!item_cta) break;
  }
}

// The tile order bin_sort left in the workspace, if it was made for these ranges.
const unsigned* tile_order_for(const abcd_ctx* ctx, const abcd_tiles* tiles, long long n_tiles) {
  return (has_workspace(ctx) && ctx->order_ranges == tiles->ranges && ctx->order_tiles == n_tiles)
             ? ctx->ws.tile_order : nullptr;
}

// Checkpoints need the workspace and room for a first-chunk end per block.
bool ckpt_ok(const abcd_ctx* ctx, long long n_blocks) {
  return has_workspace(ctx) && ctx->ws.ckpt && n_blocks <= kSubPerTile * ctx->ws.max_tiles;
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
  a.status = ctx->ws.status;
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
  a.refresh_packed = nullptr;
  a.tile_map = nullptr;
  const int n_tiles = a.cam.tiles_x * a.cam.tiles_y, n_blocks = n_tiles * kSubPerTile;
  a.tile_order = tile_order_for(ctx, tiles, n_tiles);
  a.ckpt = nullptr; a.ck_items = nullptr; a.ck_count = nullptr; a.ck_first = nullptr;
  a.ck_cap = 0;
  if (state && ckpt_ok(ctx, n_blocks)) {
    const abcd_status z = zero_async(ctx, ctx->ws.ck_count, sizeof(unsigned), "checkpoint count clear");
    if (z != ABCD_OK) return z;
    a.ckpt = ctx->ws.ckpt; a.ck_items = ctx->ws.ck_items; a.ck_count = ctx->ws.ck_count;
    a.ck_first = ctx->ws.ck_first; a.ck_cap = ctx->ws.ck_cap;
    ctx->ck_state = state->A_T;
    ctx->ck_blocks = n_blocks;
    ctx->ck_ranges = tiles->ranges;
  } else if (state && ctx->ck_state == state->A_T) {
    ctx->ck_state = nullptr;               // this state's checkpoints are gone
  }
  return check_launch(ctx, "render_fwd_kernel",
                      launch_pdl(render_fwd_kernel, dim3(n_blocks), dim3(kSubThreads), 0, ctx->stream, a));
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
  {
    const abcd_status z = zero_async(ctx, grad2d, sizeof(float) * 9 * (size_t)n, "grad2d clear");
    if (z != ABCD_OK) return z;
  }
  BwdArgs a;
  a.status = ctx->ws.status;
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
  const int n_tiles = a.cam.tiles_x * a.cam.tiles_y, n_blocks = n_tiles * kSubPerTile;
  a.tile_order = tile_order_for(ctx, tiles, n_tiles);
  a.ckpt = nullptr; a.ck_items = nullptr; a.ck_count = nullptr; a.ck_first = nullptr;
  a.ck_cap = 0; a.n_item_ctas = 0;
  if (ckpt_ok(ctx, n_blocks) && ctx->ck_state == state->A_T && ctx->ck_blocks == n_blocks &&
      ctx->ck_ranges == tiles->ranges) {
    a.ckpt = ctx->ws.ckpt; a.ck_items = ctx->ws.ck_items; a.ck_count = ctx->ws.ck_count;
    a.ck_first = ctx->ws.ck_first; a.ck_cap = ctx->ws.ck_cap;
    a.n_item_ctas = std::min(ctx->ws.ck_cap, kItemCtasPerSm * ctx->num_sms);
  }
  return check_launch(ctx, "render_bwd_kernel",
                      launch_pdl(render_bwd_kernel, dim3(a.n_item_ctas + n_blocks), dim3(kSubThreads),
                                 0, ctx->stream, a));
}

// ---- packed layers (the cache's tile-sparse format): tile t of a layer is stored iff its
// list is non-empty (a tile with no entry renders (0, 0, 0, 0) exactly), as the block
// tile_map[t] of 16 x 16 fp16 RGBA pixels in row-major order; blocks are numbered in tile order.
namespace abcd {
namespace {

__global__ void __launch_bounds__(1024)
tile_map_kernel(const uint2* ranges, int n_tiles, int* tile_map, int* count) {
  pdl_prologue();
  const int per = (n_tiles + (int)blockDim.x - 1) / (int)blockDim.x;
  const int lo = min(n_tiles, (int)threadIdx.x * per), hi = min(n_tiles, lo + per);
  unsigned long long s = 0;
  for (int t = lo; t < hi; ++t) s += ranges[t].y > ranges[t].x ? 1u : 0u;
  unsigned long long total = 0;
  __shared__ unsigned long long warp_sums[32];
  // exclusive block scan of s
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  unsigned long long x = s;
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[wid] = x;
  __syncthreads();
  if (wid == 0) {
    const int nw = blockDim.x >> 5;
    unsigned long long v = lane < nw ? warp_sums[lane] : 0ull;
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long y = __shfl_up_sync(0xffffffffu, v, o);
      if (lane >= o) v += y;
    }
    if (lane < nw) warp_sums[lane] = v;
  }
  __syncthreads();
  unsigned long long run = (wid > 0 ? warp_sums[wid - 1] : 0ull) + x - s;
  total = warp_sums[(blockDim.x >> 5) - 1];
  for (int t = lo; t < hi; ++t) {
    const bool used = ranges[t].y > ranges[t].x;
    tile_map[t] = used ? (int)run : -1;
    run += used ? 1u : 0u;
  }
  if (threadIdx.x == 0) *count = (int)total;
}

}  // namespace
}  // namespace abcd

extern "C" abcd_status abcd_render_refresh_packed(abcd_ctx* ctx, const abcd_camera* cam,
                                                  const abcd_render_opts* opts,
                                                  const abcd_projected* proj,
                                                  const abcd_tiles* tiles, int* tile_map,
                                                  void* packed, int* count) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!cam || cam->width <= 0 || cam->height <= 0 || !tiles || !tiles->ids || !tiles->ranges)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_refresh_packed: bad camera or tiles");
  if (!proj_ok(proj)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_refresh_packed: bad projected buffers");
  if (!tile_map || !packed || !count || ((uintptr_t)packed & 15) || ((uintptr_t)tile_map & 3))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_render_refresh_packed: bad or misaligned output");
  FwdArgs a;
  a.status = ctx->ws.status;
  a.cam = make_cam(cam, opts);
  a.op = make_opts(opts);
  a.uv = (const float2*)proj->uv;
  a.co = (const float4*)proj->conic_opacity;
  a.rgb = proj->rgb;
  a.ids = tiles->ids;
  a.ranges = (const uint2*)tiles->ranges;
  a.F = nullptr; a.B = nullptr; a.fb_dtype = ABCD_F16;
  for (int c = 0; c < 3; ++c) a.bg[c] = 0.f;
  a.out = nullptr;
  a.state_at = nullptr;
  a.n_last = nullptr;
  a.refresh = nullptr;
  a.refresh_packed = (uint2*)packed;
  a.tile_map = tile_map;
  const int n_tiles = a.cam.tiles_x * a.cam.tiles_y, n_blocks = n_tiles * kSubPerTile;
  a.tile_order = tile_order_for(ctx, tiles, n_tiles);
  a.ckpt = nullptr; a.ck_items = nullptr; a.ck_count = nullptr; a.ck_first = nullptr;
  a.ck_cap = 0;
  abcd_status s = check_launch(ctx, "tile_map_kernel",
                               launch_pdl(tile_map_kernel, dim3(1), dim3(1024), 0, ctx->stream,
                                          (const uint2*)tiles->ranges, n_tiles, tile_map, count));
  if (s) return s;
  return check_launch(ctx, "render_fwd_kernel",
                      launch_pdl(render_fwd_kernel, dim3(n_blocks), dim3(kSubThreads), 0, ctx->stream, a));
}
