// K3 (tile binning) and K4 (sort + tile ranges) of the ABCD active-block step.
//
// What is computed (3DGS binning, Section 1 of the paper by citation): every visible Gaussian
// is listed in each 16x16 tile met by its square [u-r, u+r] x [v-r, v+r] on which it can
// reach alpha >= alpha_min (the least sigma over the tile's pixel-centre box is at most
// ln(o / alpha_min), tested with a small margin, so the lists may hold a few more entries
// than the exact rule; every pixel skips those); each tile's list is ordered front to back by
// (fp32 depth, Gaussian id).  Dropping the tiles every pixel would skip leaves the image
// unchanged and halves the pairs to sort and to walk.
//
// How (GB300 design, different from sorting 64-bit (tile | depth) keys):
//   1. per Gaussian: its tile rectangle (kept in the workspace) and a sort key (fp32 depth
//      bits, all ones when culled); then, one thread per Gaussian: the contiguous run of kept
//      tiles in each of its tile rows (the kept set is convex), its pair (or run) count, and
//      +-1 at the run's ends in a per-row difference array over the tile grid (block-local
//      first);
//   2. stable LSD radix sort of the n Gaussians by the 32 depth bits, on the context's side
//      stream, while the main stream makes the row runs and then, in one block, the tile
//      ranges (row prefix sums of the difference array, an exclusive scan, K) and the tiles
//      ordered by decreasing pair count (the order the render kernels launch them in);
//   3. exclusive scan of the pair (run) counts in depth order: every Gaussian's output offset;
//   4. for tile grids up to 256 x 1024 tiles: emission of one item per non-empty (Gaussian,
//      tile row) run in depth order (row, x0, x1, id; the runs are recomputed with the same
//      round-to-nearest arithmetic, so they match step 1 bit for bit), a stable LSD radix sort
//      of the runs on the row bits, and the placement of every run's id in the ranges of the
//      tiles it covers (per row, chunks of runs count their runs per tile column, add the
//      counts of the row's earlier chunks by decoupled look-back and write one column per
//      lane, in run order): no pass over the K pairs but the final write;
//   5. for larger grids: emission of (tile << id_bits | id) items in depth order, 32-bit when
//      tile and id bits fit (else 64-bit), each warp writing its Gaussians' contiguous output
//      in order, then a stable LSD radix sort of the K items on the tile bits only, in passes
//      of equal width, which keeps depth order inside each tile; the last pass writes ids.
// Radix sorts are one-sweep: one kernel counts the digits of all passes, then each pass is a
// single kernel whose CTAs take tiles of items in order and find the offsets of their digits
// by decoupled look-back over the tiles before theirs (bounded waits on CTAs that are already
// running).  Lanes of equal digit are ranked with ballots on the low, scattered digits and
// with __match_any_sync on the high, grouped ones.
// Counts that live on the device (K) are read by the kernels themselves; grids are fixed, so
// the step has no host sync.
#include <algorithm>

#include "abcd_internal.cuh"

namespace abcd {
namespace {

typedef unsigned long long u64;

__device__ __forceinline__ long long dev_count(long long n_static, const long long* n_dev,
                                               long long cap) {
  if (!n_dev) return n_static;
  const long long k = *n_dev;
  return (k < 0 || k > cap) ? 0 : k;       // overflow: nothing valid to process
}

__device__ __forceinline__ void block_range(long long n, int G, long long* lo, long long* hi) {
  const long long chunk = (n + G - 1) / G;
  *lo = min(n, (long long)blockIdx.x * chunk);
  *hi = min(n, *lo + chunk);
}

__device__ __forceinline__ int4 tile_rect(float2 m, int r, int tiles_x, int tiles_y) {
  const float fr = (float)r;
  int4 q;
  q.x = (int)fminf(fmaxf(floorf((m.x - fr) * (1.f / kTile)), 0.f), (float)tiles_x);
  q.y = (int)fminf(fmaxf(floorf((m.y - fr) * (1.f / kTile)), 0.f), (float)tiles_y);
  q.z = (int)fminf(fmaxf(floorf((m.x + fr) * (1.f / kTile)) + 1.f, 0.f), (float)tiles_x);
  q.w = (int)fminf(fmaxf(floorf((m.y + fr) * (1.f / kTile)) + 1.f, 0.f), (float)tiles_y);
  return q;
}

// ---- per Gaussian: depth key (bits(depth) << 32 | id, all ones when culled) and the tile
// rectangle of its square
__global__ void keys_rects_kernel(const float* depth, const int* radius, const float2* uv, int n,
                                  int tiles_x, int tiles_y, u64* items, int4* rects,
                                  unsigned* gh_zero, int gh_words, unsigned* rows_zero,
                                  int rows_words, int* diff_zero, int diff_cells, unsigned* krange,
                                  unsigned* krange_next) {
  pdl_prologue();
  if (blockIdx.x == 0) {                  // the radix sorts' digit counts start from zero
    for (int k = threadIdx.x; k < gh_words; k += blockDim.x) gh_zero[k] = 0u;
    for (int k = threadIdx.x; k < rows_words; k += blockDim.x) rows_zero[k] = 0u;
    // the key range words of the next call (two pairs used in turn, so no memset is needed)
    if (threadIdx.x < 2) krange_next[threadIdx.x] = 0u;
  }
  // and so does the tile rows' difference array (here rather than by a memset, which would
  // end the programmatic overlap of the launches before and after it)
  for (int k = blockIdx.x * blockDim.x + threadIdx.x; k < diff_cells; k += gridDim.x * blockDim.x)
    diff_zero[k] = 0;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  int4 q = make_int4(0, 0, 0, 0);
  bool vis = false;
  unsigned key = 0xFFFFFFFFu;
  if (i < n) {
    const int r = radius[i];
    if (r > 0) q = tile_rect(uv[i], r, tiles_x, tiles_y);
    vis = r > 0 && q.x < q.z && q.y < q.w;
    if (!vis) q = make_int4(0, 0, 0, 0);
    rects[i] = q;
    if (vis) key = __float_as_uint(depth[i]);
    items[i] = ((u64)key << 32) | (unsigned)i;
  }
  // the range of the visible keys, for the depth sort's digits: the warps' extremes, then one
  // pair of atomics per block
  __shared__ unsigned s_kr[2][32];
  const unsigned kmax = __reduce_max_sync(0xffffffffu, vis ? key : 0u);
  const unsigned kcmin = __reduce_max_sync(0xffffffffu, vis ? ~key : 0u);
  if ((threadIdx.x & 31) == 0) { s_kr[0][threadIdx.x >> 5] = kcmin; s_kr[1][threadIdx.x >> 5] = kmax; }
  __syncthreads();
  if (threadIdx.x < 32) {
    const int nw = blockDim.x >> 5;
    const unsigned a = __reduce_max_sync(0xffffffffu, (int)threadIdx.x < nw ? s_kr[0][threadIdx.x] : 0u);
    const unsigned b = __reduce_max_sync(0xffffffffu, (int)threadIdx.x < nw ? s_kr[1][threadIdx.x] : 0u);
    if (threadIdx.x == 0 && b != 0u) {
      atomicMax(krange, a);
      atomicMax(krange + 1, b);
    }
  }
}

// The tiles of row ty kept for a Gaussian are those whose pixel-centre box meets the ellipse
// E = {d : sigma'(d) <= lim}, sigma'(d) = ha dx^2 + hb dx dy + hc dy^2 (log2-scaled conic).
// Over the row's band of centre offsets dy in [Y0, Y1], the x-extent of E is [xl, xr]: the
// leftmost point of E is (-m, hb m / (2 hc)) with m = sqrt(lim / (ha - hb^2 / (4 hc))), and
// the left boundary x(dy) = (-hb dy - sqrt(D(dy))) / (2 ha), D = hb^2 dy^2 - 4 ha (hc dy^2 -
// lim), is convex, so its least value over the band is at the leftmost point's dy clamped into
// the band (the rightmost side is symmetric).  lim = (1.001 log2(o / alpha_min) + 0.01) 1.001
// keeps every tile the exact rule keeps.  Round-to-nearest intrinsics only: count and emit
// kernels get the same bits.
struct Splat {
  float u, v, hb, lim;
  float ym;        // |dy| <= ym on E
  float dyl;       // dy of the leftmost point of E (the rightmost is at -dyl)
  float fal;       // 4 ha lim
  float det4;      // 4 ha hc - hb^2 > 0
  float inv2a;     // 1 / (2 ha)
};

__device__ __forceinline__ float diff_of_products(float a, float b, float c, float d) {
  // a b - c d with one rounding error at most (Kahan)
  const float w = __fmul_rn(c, d);
  const float e = __fmaf_rn(-c, d, w);
  const float f = __fmaf_rn(a, b, -w);
  return __fadd_rn(f, e);
}

__device__ __forceinline__ Splat load_splat(const float2* uv, const float4* co, unsigned g,
                                            float alpha_min) {
  const float2 m = uv[g];
  const float4 c = co[g];
  Splat s;
  s.u = m.x; s.v = m.y;
  const float ha = __fmul_rn(0.7213475204444817f, c.x);   // log2(e)/2
  s.hb = __fmul_rn(1.4426950408889634f, c.y);             // log2(e)
  const float hc = __fmul_rn(0.7213475204444817f, c.z);
  s.det4 = diff_of_products(__fmul_rn(4.f, ha), hc, s.hb, s.hb);
  // alpha = o 2^-sigma' >= alpha_min  <=>  sigma' <= log2(o / alpha_min); margin 0.01 + 0.1%
  const float thr = c.w >= alpha_min ? log2f(__fdiv_rn(c.w, alpha_min)) : -1.f;
  s.lim = (thr >= 0.f && s.det4 > 0.f && ha > 0.f && hc > 0.f)
              ? __fmul_rn(__fadd_rn(__fmul_rn(thr, 1.001f), 0.01f), 1.001f) : -1.f;
  s.fal = __fmul_rn(__fmul_rn(4.f, ha), s.lim);
  s.ym = 0.f; s.dyl = 0.f; s.inv2a = 0.f;
  if (s.lim >= 0.f) {
    // |dy| <= ym on E: D(dy) = 4 ha lim - det4 dy^2 >= 0
    s.ym = __fsqrt_rn(__fdiv_rn(s.fal, s.det4));
    // leftmost point of E: dx = -mx, dy = hb mx / (2 hc); mx = sqrt(4 hc lim / det4)
    const float mx = __fsqrt_rn(__fdiv_rn(__fmul_rn(__fmul_rn(4.f, hc), s.lim), s.det4));
    s.dyl = __fdiv_rn(__fmul_rn(s.hb, mx), __fmul_rn(2.f, hc));
    s.inv2a = __frcp_rn(__fmul_rn(2.f, ha));
  }
  return s;
}

// Run [xa, xb) of kept tiles in tile row ty of rectangle q (empty: xa == xb).
__device__ __forceinline__ int2 row_run(const Splat& s, int4 q, int ty) {
  if (!(s.lim >= 0.f)) return make_int2(0, 0);
  const float Y0 = __fsub_rn((float)(ty * kTile) + 0.5f, s.v);
  const float Y1 = __fadd_rn(Y0, (float)(kTile - 1));
  const float ylo = fmaxf(Y0, -s.ym), yhi = fminf(Y1, s.ym);
  if (!(ylo <= yhi)) return make_int2(0, 0);
  // boundary x at dy: (-hb dy -+ sqrt(D)) / (2 ha), D = 4 ha lim - det4 dy^2; the least x over
  // the band is at the leftmost point's dy clamped into it, the largest at -dyl clamped
  const float yl = fminf(fmaxf(s.dyl, ylo), yhi);
  const float Dl = fmaxf(__fmaf_rn(-s.det4, __fmul_rn(yl, yl), s.fal), 0.f);
  const float xl = __fmul_rn(__fsub_rn(__fmul_rn(-s.hb, yl), __fsqrt_rn(Dl)), s.inv2a);
  const float yr = fminf(fmaxf(-s.dyl, ylo), yhi);
  const float Dr = fmaxf(__fmaf_rn(-s.det4, __fmul_rn(yr, yr), s.fal), 0.f);
  const float xr = __fmul_rn(__fadd_rn(__fmul_rn(-s.hb, yr), __fsqrt_rn(Dr)), s.inv2a);
  // tiles whose centre box [16 tx + 0.5, 16 tx + 15.5] meets [u + xl, u + xr]
  const float fa = ceilf(__fmul_rn(__fsub_rn(__fadd_rn(s.u, xl), 15.5f), 1.f / kTile));
  const float fb = floorf(__fmul_rn(__fsub_rn(__fadd_rn(s.u, xr), 0.5f), 1.f / kTile)) + 1.f;
  const int xa = (int)fminf(fmaxf(fa, (float)q.x), (float)q.z);
  const int xb = (int)fminf(fmaxf(fb, (float)xa), (float)q.z);
  return make_int2(xa, xb);
}

// ---- one thread per Gaussian, looping over its tile rows: +1 / -1 at the ends of every row's
// run in the per-row difference array, and the Gaussian's count: its pairs, or (RUNS) its
// non-empty row runs, with the runs of every tile row added up in row_runs.  The +-1 go to a
// block-local copy of the difference array in shared memory first (the same few thousand cells
// are hit by every block), then only its non-zero cells to the global array.
constexpr int kSmemDiffCells = 12288;      // 48 KB: tile grids up to ~1900x1500 pixels

template <bool RUNS>
__global__ void __launch_bounds__(256)
tile_rows_kernel(const float2* uv, const float4* co, const int4* rects, int n, int tiles_x,
                 int tiles_y, float alpha_min, unsigned* counts, int* diff, unsigned* row_runs) {
  pdl_prologue();
  extern __shared__ int sdiff[];
  const int W1 = tiles_x + 1;
  const int cells = W1 * (tiles_y + 1);
  const bool local = cells <= kSmemDiffCells;      // always, with RUNS
  unsigned* srows = reinterpret_cast<unsigned*>(sdiff + cells);   // RUNS: [tiles_y]
  if (local) {
    for (int k = threadIdx.x; k < cells; k += blockDim.x) sdiff[k] = 0;
    if (RUNS)
      for (int k = threadIdx.x; k < tiles_y; k += blockDim.x) srows[k] = 0u;
    __syncthreads();
  }
  int* dst = local ? sdiff : diff;
  const int g = blockIdx.x * blockDim.x + threadIdx.x;
  if (g < n) {
    const int4 q = rects[g];
    unsigned c = 0;
    if (q.x < q.z) {
      const Splat s = load_splat(uv, co, (unsigned)g, alpha_min);
      for (int ty = q.y; ty < q.w; ++ty) {
        const int2 r = row_run(s, q, ty);
        if (r.y > r.x) {
          c += RUNS ? 1u : (unsigned)(r.y - r.x);
          atomicAdd(&dst[ty * W1 + r.x], 1);
          atomicAdd(&dst[ty * W1 + r.y], -1);
          if (RUNS) atomicAdd(&srows[ty], 1u);
        }
      }
    }
    counts[g] = c;
  }
  if (local) {
    __syncthreads();
    for (int k = threadIdx.x; k < cells; k += blockDim.x) {
      const int v = sdiff[k];
      if (v != 0) atomicAdd(&diff[k], v);
    }
    if (RUNS)
      for (int k = threadIdx.x; k < tiles_y; k += blockDim.x) {
        const unsigned v = srows[k];
        if (v != 0u) atomicAdd(&row_runs[k], v);
      }
  }
}

// Items j = 0..U-1 of a warp's run: in[b0 + 32 j + lane] below wh (zero past it).
template <typename T, int U>
__device__ __forceinline__ void load_items(const T* in, long long b0, long long wh, int lane,
                                           T (&xs)[U]) {
#pragma unroll
  for (int j = 0; j < U; ++j) {
    const long long i = b0 + 32 * j + lane;
    xs[j] = i < wh ? in[i] : (T)0;
  }
}

// Digit of item j of a round (0x100 past the end of the slice).
template <typename T>
__device__ __forceinline__ unsigned digit_of(T x, long long i, long long wh, int shift,
                                             unsigned mask) {
  return i < wh ? ((unsigned)(x >> shift) & mask) : 0x100u;
}

// The depth sort ranks keys relative to the smallest visible one (the positive depths' float
// bits keep their order under the subtraction), with the culled items' all-ones keys mapped
// just above the largest: when the visible keys span fewer than 2^24 - 1 values, every item's
// top byte is then zero and the last 8-bit pass has a single digit, so it runs as a copy.  The
// order is the one of the keys themselves.  krange: [0] the largest complement of a visible
// key, [1] the largest visible key (both zero when none is visible).  Its first pass writes the
// items with their keys mapped; only the id bits are read after the sort.
struct KeyMap {
  unsigned lo, sat;
  bool on;
};

__device__ __forceinline__ KeyMap key_map(const unsigned* kr) {
  KeyMap m{0u, 0xFFFFFFFFu, kr != nullptr};
  if (kr) {
    const unsigned lo = ~kr[0], hi = kr[1];
    m.lo = lo;
    m.sat = (hi >= lo && hi - lo < 0xFFFFFFu) ? 0xFFFFFFu : 0xFFFFFFFFu;
  }
  return m;
}

template <typename T>
__device__ __forceinline__ T map_item(T x, const KeyMap& m) {
  if constexpr (sizeof(T) == 8) {
    const unsigned k = (unsigned)(x >> 32);
    const unsigned kk = k == 0xFFFFFFFFu ? m.sat : k - m.lo;
    return ((T)kk << 32) | (x & 0xFFFFFFFFull);
  } else {
    return x;
  }
}

// Lanes holding the same BITS-bit digit as this lane, among the lanes of valid_mask: one
// ballot per bit (a cost independent of how many distinct digits the warp holds).
template <int BITS>
__device__ __forceinline__ unsigned match_digit(unsigned d, unsigned valid_mask) {
  unsigned peers = valid_mask;
#pragma unroll
  for (int b = 0; b < BITS; ++b) {
    const unsigned bit = (d >> b) & 1u;
    const unsigned m = __ballot_sync(0xffffffffu, bit);
    peers &= bit ? m : ~m;
  }
  return peers;
}

// Exclusive scan of a block of per-thread sums (any multiple of 32 threads up to 1024).
__device__ __forceinline__ unsigned long long block_exclusive_scan(unsigned long long v,
                                                                   unsigned long long* total) {
  __shared__ unsigned long long warp_sums[32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  unsigned long long x = v;
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[wid] = x;
  __syncthreads();
  if (wid == 0) {
    const int nw = blockDim.x >> 5;
    unsigned long long s = lane < nw ? warp_sums[lane] : 0ull;
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    if (lane < nw) warp_sums[lane] = s;
  }
  __syncthreads();
  const unsigned long long before = (wid > 0 ? warp_sums[wid - 1] : 0ull) + x - v;
  if (total) *total = warp_sums[(blockDim.x >> 5) - 1];
  __syncthreads();
  return before;
}

// Lanes of the warp holding the same digit: one ballot per bit (a cost independent of how many
// distinct digits the warp holds: the right choice for the low, scattered digits) or
// __match_any_sync (fast when a warp holds few distinct digits: the high digits of depth keys and
// of tile indices, whose items arrive nearly grouped).
template <int BITS, bool MATCH>
__device__ __forceinline__ unsigned rank_peers(unsigned d, bool valid) {
  if (MATCH) return __match_any_sync(0xffffffffu, d);
  return match_digit<BITS>(d, __ballot_sync(0xffffffffu, valid));
}

// ---- one-sweep radix sort (decoupled look-back)
// A sort of n items on bits [bit_lo, bit_hi) runs in passes of equal width.  One kernel counts
// the digits of every pass at once; then each pass is a single kernel: CTAs claim tiles of
// kOsWarps x 32 x U consecutive items in order (a global counter), rank each item among the
// tile's items of equal digit (stable), publish the tile's per-digit counts, and add up the
// counts of the tiles before theirs by looking back until a tile whose inclusive prefix is
// published.  Item position = digit base + prefix of earlier tiles + rank in the tile.
// A tile only waits for tiles claimed before it, whose CTAs are running, so the waits end;
// each is bounded all the same (on expiry the status word gets ABCD_ERR_TIMEOUT and the pass
// goes on with a wrong prefix instead of hanging).
struct SortPasses {
  int n;                 // passes (at most kMaxSortPasses)
  int shift[4];          // low bit of each pass's digit
  int bits[4];           // digit width of each pass (4..8)
};
// Passes of equal width (at least 4 bits) covering bits [bit_lo, bit_hi).
__host__ __device__ inline SortPasses make_passes(int bit_lo, int bit_hi) {
  SortPasses sp{};
  const int nbits = bit_hi - bit_lo;
  sp.n = (nbits + kRadixBits - 1) / kRadixBits;
  const int width = (nbits + sp.n - 1) / sp.n > 4 ? (nbits + sp.n - 1) / sp.n : 4;
  for (int p = 0; p < sp.n && p < 4; ++p) {
    sp.shift[p] = bit_lo + p * width;
    const int left = bit_hi - sp.shift[p];
    sp.bits[p] = left < width ? (left < 4 ? 4 : left) : width;
  }
  return sp;
}

// Adds the digit counts of one tile's c items ((tile << bit_lo | id) items of a sort whose
// passes `tp` are relative to the tile bits) to h.
__device__ __forceinline__ void tile_digit_counts(unsigned t, unsigned c, const SortPasses& tp,
                                                  unsigned (*h)[kRadixBins]) {
  if (c == 0) return;
  for (int p = 0; p < tp.n; ++p)
    atomicAdd(&h[p][(t >> tp.shift[p]) & ((1u << tp.bits[p]) - 1u)], c);
}

constexpr int kOsWarps = 8;
constexpr int kOsThreads = 32 * kOsWarps;

// Look-back state word: epoch (30 bits) | flag (2 bits: 1 aggregate, 2 inclusive) | count.
// The epoch changes with every pass launch, so words left by earlier passes read as "not
// published" and the array needs no clearing.
__device__ __forceinline__ u64 os_word(unsigned epoch, unsigned flag, unsigned count) {
  return ((u64)epoch << 34) | ((u64)flag << 32) | count;
}

__device__ __forceinline__ void os_publish(u64* p, u64 v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ u64 os_peek(const u64* p) {
  u64 v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

// Digit counts of every pass: gh[p * kRadixBins + d] += count (gh zeroed by keys_rects).
template <typename T>
__global__ void __launch_bounds__(256)
sort_digits_kernel(const T* in, long long n_static, const long long* n_dev, long long cap,
                   SortPasses sp, int match_from, unsigned* gh, const unsigned* krange) {
  pdl_prologue();
  __shared__ unsigned h[4][kRadixBins];
  for (int k = threadIdx.x; k < 4 * kRadixBins; k += blockDim.x) (&h[0][0])[k] = 0;
  __syncthreads();
  const long long n = dev_count(n_static, n_dev, cap);
  const int lane = threadIdx.x & 31;
  const unsigned lt = (1u << lane) - 1u;
  const long long stride = (long long)gridDim.x * blockDim.x;
  const KeyMap km = key_map(krange);
  // the loop runs while any lane of the warp has an item (the ranking is warp-collective)
  for (long long b = (long long)blockIdx.x * blockDim.x + (threadIdx.x & ~31); b < n; b += stride) {
    const long long i = b + lane;
    const bool valid = i < n;
    const T x = valid ? (km.on ? map_item(in[i], km) : in[i]) : (T)0;
    for (int p = 0; p < sp.n; ++p) {
      const unsigned d = valid ? (unsigned)(x >> sp.shift[p]) & ((1u << sp.bits[p]) - 1u) : 0x100u;
      const unsigned peers = p >= match_from ? __match_any_sync(0xffffffffu, d) : match_byte(d);
      if (valid && (peers & lt) == 0) atomicAdd(&h[p][d], __popc(peers));
    }
  }
  __syncthreads();
  for (int k = threadIdx.x; k < sp.n * kRadixBins; k += blockDim.x) {
    const unsigned c = (&h[0][0])[k];
    if (c) atomicAdd(gh + k, c);
  }
}

// One pass: stable scatter of the items of [0, n) by the BITS-bit digit at `shift`.  gh holds
// this pass's digit counts; ctr[0] hands out tiles and ctr[1] counts finished CTAs (the last
// one clears both); state holds kRadixBins words per tile.  On the last pass out_ids (when not
// null) receives the bits id_mask of each item instead of the item.  A look-back wait gives up
// after spin_limit polls.  Tile `withhold` (a test hook; -1 in normal use) publishes nothing,
// so the waits of the tiles after it run out.
template <typename T, int BITS, bool MATCH>
__global__ void __launch_bounds__(kOsThreads, 2)
onesweep_kernel(const T* in, T* out, unsigned* out_ids, unsigned id_mask, long long n_static,
                const long long* n_dev, long long cap, int shift, const unsigned* gh, u64* state,
                unsigned* ctr, unsigned epoch, unsigned* status, unsigned spin_limit,
                long long withhold, const unsigned* krange) {
  pdl_prologue();
  constexpr unsigned BINS = 1u << BITS, MASK = BINS - 1;
  constexpr int U = 64 / (int)sizeof(T);          // items per lane: 64 bytes in flight
  constexpr int TILE = kOsThreads * U;
  __shared__ unsigned cnt[kOsWarps][BINS];
  __shared__ unsigned s_base[BINS];
  __shared__ unsigned s_off[BINS];
  __shared__ unsigned s_run[BINS];
  __shared__ unsigned s_loc[BINS];                // start of each digit inside the tile
  __shared__ T s_items[TILE];                     // the tile's items in digit order
  __shared__ unsigned s_tile;
  __shared__ int s_copy;
  const long long n = dev_count(n_static, n_dev, cap);
  if (threadIdx.x == 0) s_copy = 0;
  __syncthreads();
  {
    const unsigned v = threadIdx.x < BINS ? gh[threadIdx.x] : 0u;
    // every item holds the same digit: the stable scatter is the identity, a copy
    if (n > 0 && (long long)v == n) s_copy = 1;
    const unsigned long long ex = block_exclusive_scan(v, nullptr);
    if (threadIdx.x < BINS) s_base[threadIdx.x] = (unsigned)ex;
  }
  const long long n_tiles = (n + TILE - 1) / TILE;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const unsigned lt = (1u << lane) - 1u;
  const KeyMap km = key_map(krange);
  while (s_copy) {                                   // block-uniform (set before the scan's barriers)
    if (threadIdx.x == 0) s_tile = atomicAdd(ctr, 1u);
    __syncthreads();
    const long long t = s_tile;
    __syncthreads();                                 // s_tile is read before the next claim
    if (t >= n_tiles) break;
    T xs[U];
#pragma unroll
    for (int j = 0; j < U; ++j) {                    // all loads in flight together
      const long long i = t * TILE + j * kOsThreads + threadIdx.x;
      xs[j] = i < n ? in[i] : (T)0;
    }
#pragma unroll
    for (int j = 0; j < U; ++j) {
      const long long i = t * TILE + j * kOsThreads + threadIdx.x;
      if (i >= n) continue;
      const T x = km.on ? map_item(xs[j], km) : xs[j];
      if (out_ids) out_ids[i] = (unsigned)x & id_mask;
      else out[i] = x;
    }
  }
  for (; !s_copy;) {
    if (threadIdx.x == 0) s_tile = atomicAdd(ctr, 1u);
    for (int k = threadIdx.x; k < kOsWarps * (int)BINS; k += kOsThreads) (&cnt[0][0])[k] = 0;
    __syncthreads();
    const long long t = s_tile;
    if (t >= n_tiles) break;                         // block-uniform
    const long long b0 = t * TILE + (long long)w * 32 * U;
    T xs[U];
    unsigned rk[U];
    load_items(in, b0, n, lane, xs);
    if (km.on) {
#pragma unroll
      for (int j = 0; j < U; ++j) xs[j] = map_item(xs[j], km);
    }
#pragma unroll
    for (int j = 0; j < U; ++j) {
      const unsigned d = digit_of(xs[j], b0 + 32 * j + lane, n, shift, MASK);
      const bool valid = d < 0x100u;
      const unsigned peers = rank_peers<BITS, MATCH>(d, valid);
      rk[j] = valid ? cnt[w][d] + __popc(peers & lt) : 0u;
      __syncwarp();
      if (valid && (peers & lt) == 0) cnt[w][d] += __popc(peers);
      __syncwarp();
    }
    __syncthreads();
    if (threadIdx.x < BINS) {
      // warp bases per digit (exclusive over warps) and the tile's count: published at once
      const unsigned d = threadIdx.x;
      unsigned run = 0;
#pragma unroll
      for (int k = 0; k < kOsWarps; ++k) { const unsigned c = cnt[k][d]; cnt[k][d] = run; run += c; }
      s_run[d] = run;
      if (t != withhold)
        os_publish(state + (size_t)t * kRadixBins + d, os_word(epoch, t == 0 ? 2u : 1u, run));
    }
    __syncthreads();
    {
      // look-back: R threads per digit read LB tiles each, nearest first, per round.  At least
      // 16 tiles per digit and round: when every CTA of a short pass starts at once, the
      // inclusive prefixes move back along the tiles by that many tiles per round trip.
      constexpr int R = kOsThreads / (int)BINS;
      constexpr int LB = 16 / R > 4 ? 16 / R : 4;
      const unsigned d = threadIdx.x / R;
      const int q = threadIdx.x % R;
      const unsigned gmask = R == 32 ? 0xffffffffu : (((1u << R) - 1u) << (lane & ~(R - 1)));
      const int g0 = lane & ~(R - 1);
      unsigned prefix = 0;
      long long k0 = t - 1;                          // nearest tile not summed yet
      unsigned spins = 0;
      while (t > 0) {
        u64 v[LB];
#pragma unroll
        for (int j = 0; j < LB; ++j) {
          const long long k = k0 - (long long)LB * q - j;
          v[j] = k >= 0 ? os_peek(state + (size_t)k * kRadixBins + d) : os_word(epoch, 2u, 0u);
        }
        unsigned sum = 0, used = LB;
        int kind = 0;                                // 0: all aggregates, 1: inclusive, 2: blocked
#pragma unroll
        for (int j = 0; j < LB; ++j) {
          if (kind != 0) continue;
          const unsigned flag = (unsigned)(v[j] >> 32) & 3u;
          if ((unsigned)(v[j] >> 34) != epoch || flag == 0u) { kind = 2; used = j; continue; }
          sum += (unsigned)v[j];
          if (flag == 2u) { kind = 1; used = j + 1; }
        }
        // combine the R windows in order (every thread of the group decides alike)
        unsigned add = 0;
        long long consumed = 0;
        int res = 0;
        for (int qq = 0; qq < R; ++qq) {
          const unsigned sq = __shfl_sync(gmask, sum, g0 + qq);
          const int kq = __shfl_sync(gmask, kind, g0 + qq);
          const unsigned uq = __shfl_sync(gmask, used, g0 + qq);
          if (res == 0) { add += sq; consumed += uq; res = kq; }
        }
        prefix += add;
        k0 -= consumed;
        if (res == 1) break;
        if (res == 2) {
          if (++spins > spin_limit) { if (q == 0) atomicOr(status, kStatusTimeout); break; }
          __nanosleep(32);
        }
      }
      if (q == 0) {
        if (t > 0 && t != withhold)
          os_publish(state + (size_t)t * kRadixBins + d, os_word(epoch, 2u, prefix + s_run[d]));
        s_off[d] = s_base[d] + prefix;
      }
    }
    {
      // the tile's items in digit order in shared memory, then written out in that order:
      // consecutive threads store consecutive addresses of a digit's run
      const unsigned v = threadIdx.x < BINS ? s_run[threadIdx.x] : 0u;
      const unsigned long long ex = block_exclusive_scan(v, nullptr);
      if (threadIdx.x < BINS) s_loc[threadIdx.x] = (unsigned)ex;
      __syncthreads();
    }
#pragma unroll
    for (int j = 0; j < U; ++j) {
      const unsigned d = digit_of(xs[j], b0 + 32 * j + lane, n, shift, MASK);
      if (d < 0x100u) s_items[s_loc[d] + cnt[w][d] + rk[j]] = xs[j];
    }
    __syncthreads();
    const int in_tile = (int)min((long long)TILE, n - t * TILE);
    for (int i = threadIdx.x; i < in_tile; i += kOsThreads) {
      const T x = s_items[i];
      const unsigned d = (unsigned)(x >> shift) & MASK;
      const unsigned long long pos = (unsigned long long)s_off[d] + (unsigned)(i - (int)s_loc[d]);
      if (pos < (unsigned long long)n) {             // always, unless a wait expired
        if (out_ids) out_ids[pos] = (unsigned)x & id_mask;
        else out[pos] = x;
      }
    }
    __syncthreads();                                 // before the next tile reuses cnt, s_off
  }
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(ctr + 1, 1u) == gridDim.x - 1) { ctr[0] = 0u; ctr[1] = 0u; }
  }
}

// ---- binning: per-block sums of pair counts in depth order
__global__ void __launch_bounds__(256)
count_kernel(const u64* sorted, int n, const unsigned* counts, unsigned long long* block_sums,
             int G) {
  pdl_prologue();
  long long lo, hi;
  block_range(n, G, &lo, &hi);
  unsigned long long s = 0;
  for (long long i = lo + threadIdx.x; i < hi; i += blockDim.x) {
    const unsigned id = (unsigned)sorted[i];
    if (id < (unsigned)n) s += counts[id];           // (a timed-out sort may leave stale items)
  }
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  __shared__ unsigned long long ws[8];
  if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long t = 0;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) t += ws[k];
    block_sums[blockIdx.x] = t;
  }
}

__global__ void __launch_bounds__(1024)
scan_blocks_kernel(unsigned long long* block_sums, int G, long long* count, long long cap,
                   unsigned* status) {
  pdl_prologue();
  const unsigned long long v = (int)threadIdx.x < G ? block_sums[threadIdx.x] : 0ull;
  unsigned long long total = 0;
  const unsigned long long ex = block_exclusive_scan(v, &total);
  if ((int)threadIdx.x < G) block_sums[threadIdx.x] = ex;
  if (threadIdx.x == 0) {
    *count = (long long)total;
    if ((long long)total > cap) atomicOr(status, kStatusCapacity);
  }
}

// ---- tile ranges from the per-row difference array: prefix sums along each row -> per-tile
// counts -> exclusive scan (one block).  Empty ranges when K overflowed the capacity.
__global__ void __launch_bounds__(1024)
ranges_from_diff_kernel(int* diff, int tiles_x, int tiles_y, long long cap, unsigned* ranges,
                        SortPasses tp, unsigned* gh) {
  pdl_prologue();
  __shared__ unsigned dh[4][kRadixBins];
  for (int k = threadIdx.x; k < 4 * kRadixBins; k += blockDim.x) (&dh[0][0])[k] = 0u;
  const int W1 = tiles_x + 1;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
  for (int y = wid; y < tiles_y; y += nw) {                        // prefix along each row
    int carry = 0;
    for (int x0 = 0; x0 < tiles_x; x0 += 32) {
      const int x = x0 + lane;
      int v = x < tiles_x ? diff[y * W1 + x] : 0;
      for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += u;
      }
      if (x < tiles_x) diff[y * W1 + x] = v + carry;
      carry += __shfl_sync(0xffffffffu, v, 31);
    }
  }
  __syncthreads();
  const int nt = tiles_x * tiles_y;
  const int per = (nt + blockDim.x - 1) / blockDim.x;
  const int lo = min(nt, (int)threadIdx.x * per), hi = min(nt, lo + per);
  unsigned long long s = 0;
  for (int t = lo; t < hi; ++t) s += (unsigned)diff[(t / tiles_x) * W1 + (t % tiles_x)];
  unsigned long long total = 0;
  unsigned long long run = block_exclusive_scan(s, &total);
  const bool ok = (long long)total <= cap;          // K: the same total the count scan finds
  for (int t = lo; t < hi; ++t) {
    const unsigned c = (unsigned)diff[(t / tiles_x) * W1 + (t % tiles_x)];
    ranges[2 * t] = ok ? (unsigned)run : 0u;
    ranges[2 * t + 1] = ok ? (unsigned)(run + c) : 0u;
    tile_digit_counts((unsigned)t, c, tp, dh);
    run += c;
  }
  __syncthreads();
  for (int k = threadIdx.x; k < tp.n * kRadixBins; k += blockDim.x) gh[k] = (&dh[0][0])[k];
}

// ---- the same, with the difference array staged in shared memory (one load round trip
// instead of a chain of dependent ones), followed by the render order: tiles sorted by
// decreasing pair count (16 buckets per octave; a counting sort, in no particular order inside
// a bucket) into tile_order, so that the render kernels start the longest lists first.  The
// order changes no result.
constexpr int kOrderBuckets = 256;

__device__ __forceinline__ unsigned count_bucket(unsigned c) {
  if (c == 0) return kOrderBuckets - 1;
  const int b = (int)(__log2f((float)c) * 16.f) + 1;
  return (unsigned)(kOrderBuckets - 1 - min(b, kOrderBuckets - 1));
}

// With row_runs (binning through tile-row runs) the digit counts are those of the runs' row
// sort, and K goes to k_out (an overflow is flagged in status).
__global__ void __launch_bounds__(1024)
ranges_order_kernel(const int* diff, int tiles_x, int tiles_y, long long cap, unsigned* ranges,
                    unsigned* tile_order, SortPasses tp, unsigned* gh, const unsigned* row_runs,
                    long long* k_out, unsigned* status) {
  pdl_prologue();
  extern __shared__ int sd[];              // [(tiles_x + 1) (tiles_y + 1)] cells, then [nt] keys
  __shared__ unsigned hist[kOrderBuckets];
  __shared__ unsigned dh[4][kRadixBins];   // digit counts of the tile sort's passes
  for (int k = threadIdx.x; k < 4 * kRadixBins; k += blockDim.x) (&dh[0][0])[k] = 0u;
  const int W1 = tiles_x + 1, cells = W1 * (tiles_y + 1), nt = tiles_x * tiles_y;
  unsigned char* skey = reinterpret_cast<unsigned char*>(sd + cells);
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const unsigned lt = (1u << lane) - 1u;
  constexpr int kLoads = 8;
  for (int i0 = threadIdx.x; i0 < cells; i0 += blockDim.x * kLoads) {
    int v[kLoads];
#pragma unroll
    for (int k = 0; k < kLoads; ++k) {
      const int i = i0 + k * (int)blockDim.x;
      v[k] = i < cells ? diff[i] : 0;
    }
#pragma unroll
    for (int k = 0; k < kLoads; ++k) {
      const int i = i0 + k * (int)blockDim.x;
      if (i < cells) sd[i] = v[k];
    }
  }
  for (int i = threadIdx.x; i < kOrderBuckets; i += blockDim.x) hist[i] = 0;
  __syncthreads();
  for (int y = wid; y < tiles_y; y += nw) {                        // prefix along each row
    int carry = 0;
    for (int x0 = 0; x0 < tiles_x; x0 += 32) {
      const int x = x0 + lane;
      int v = x < tiles_x ? sd[y * W1 + x] : 0;
      for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += u;
      }
      if (x < tiles_x) sd[y * W1 + x] = v + carry;
      carry += __shfl_sync(0xffffffffu, v, 31);
    }
  }
  __syncthreads();
  const int per = (nt + blockDim.x - 1) / blockDim.x;
  const int lo = min(nt, (int)threadIdx.x * per), hi = min(nt, lo + per);
  unsigned long long s = 0;
  for (int t = lo; t < hi; ++t) s += (unsigned)sd[(t / tiles_x) * W1 + (t % tiles_x)];
  unsigned long long total = 0;
  unsigned long long run = block_exclusive_scan(s, &total);
  const bool ok = (long long)total <= cap;          // K: the same total the count scan finds
  for (int t = lo; t < hi; ++t) {
    const unsigned c = (unsigned)sd[(t / tiles_x) * W1 + (t % tiles_x)];
    ranges[2 * t] = ok ? (unsigned)run : 0u;
    ranges[2 * t + 1] = ok ? (unsigned)(run + c) : 0u;
    skey[t] = (unsigned char)count_bucket(ok ? c : 0u);
    if (!row_runs) tile_digit_counts((unsigned)t, c, tp, dh);
    run += c;
  }
  if (row_runs) {
    for (int y = threadIdx.x; y < tiles_y; y += blockDim.x)
      tile_digit_counts((unsigned)y, row_runs[y], tp, dh);
    if (threadIdx.x == 0) {
      *k_out = (long long)total;
      if (!ok) atomicOr(status, kStatusCapacity);
    }
  }
  __syncthreads();
  for (int k = threadIdx.x; k < tp.n * kRadixBins; k += blockDim.x) gh[k] = (&dh[0][0])[k];
  for (int i0 = 0; i0 < nt; i0 += blockDim.x) {
    const int i = i0 + threadIdx.x;
    const unsigned key = i < nt ? skey[i] : (unsigned)kOrderBuckets;
    const unsigned peers = __match_any_sync(0xffffffffu, key);
    if (key < kOrderBuckets && (peers & lt) == 0) atomicAdd(&hist[key], (unsigned)__popc(peers));
  }
  __syncthreads();
  if (threadIdx.x < 32) {                  // exclusive scan of the 256 counts, 8 per lane
    constexpr int kPer = kOrderBuckets / 32;
    unsigned v[kPer], sum = 0;
#pragma unroll
    for (int k = 0; k < kPer; ++k) { v[k] = hist[lane * kPer + k]; sum += v[k]; }
    unsigned incl = sum;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const unsigned o = __shfl_up_sync(0xffffffffu, incl, d);
      if (lane >= d) incl += o;
    }
    unsigned r = incl - sum;
#pragma unroll
    for (int k = 0; k < kPer; ++k) { hist[lane * kPer + k] = r; r += v[k]; }
  }
  __syncthreads();
  for (int i0 = 0; i0 < nt; i0 += blockDim.x) {
    const int i = i0 + threadIdx.x;
    const unsigned key = i < nt ? skey[i] : (unsigned)kOrderBuckets;
    const unsigned peers = __match_any_sync(0xffffffffu, key);
    const int leader = __ffs(peers) - 1;
    unsigned base = 0;
    if (key < kOrderBuckets && lane == leader) base = atomicAdd(&hist[key], (unsigned)__popc(peers));
    base = __shfl_sync(0xffffffffu, base, leader);
    if (key < kOrderBuckets) tile_order[base + __popc(peers & lt)] = (unsigned)i;
  }
}

// ---- emission of (tile << id_bits | id) in depth order.  A warp takes 32 consecutive
// Gaussians of the depth order, whose pairs fill one contiguous range of the output, and
// writes that range in order with coalesced stores, all lanes busy whatever the Gaussians'
// sizes: the warp's (Gaussian, tile row) pairs are taken 32 at a time (lane l: pair l of the
// round, its Gaussian found by a search over the scan of row counts), each lane computes its
// row's run of tiles, a warp scan places the runs, and consecutive lanes take consecutive
// output pairs (the run of pair k found by a search over that scan).
constexpr int kEmitThreads = 256;

// Lanes 0..31 hold an inclusive scan `incl`; returns the number of lanes whose value is <= k
// (clamped to 31): the lane whose range holds k.  Every lane must call it.
__device__ __forceinline__ int scan_search(unsigned incl, unsigned k) {
  int rl = 0;
#pragma unroll
  for (int step = 16; step > 0; step >>= 1) {
    const unsigned v = __shfl_sync(0xffffffffu, incl, rl + step - 1);
    if (v <= k) rl += step;
  }
  return min(rl, 31);
}

__device__ __forceinline__ unsigned warp_inclusive_scan(unsigned v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned y = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += y;
  }
  return v;
}

template <typename T>
__global__ void __launch_bounds__(kEmitThreads)
emit_kernel(const u64* sorted, int n, const float2* uv, const float4* co, const int4* rects,
            const unsigned* counts, const unsigned long long* block_off, const long long* count,
            long long cap, int tiles_x, float alpha_min, int id_bits, T* pairs, int G) {
  pdl_prologue();
  __shared__ Splat s_sp[kEmitThreads];
  __shared__ int4 s_q[kEmitThreads];
  __shared__ unsigned s_id[kEmitThreads];
  if (*count > cap) return;
  long long lo, hi;
  block_range(n, G, &lo, &hi);
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  unsigned long long run = block_off[blockIdx.x];
  for (long long base = lo; base < hi; base += blockDim.x) {
    const long long i = base + threadIdx.x;
    unsigned id = 0, t = 0;
    int4 qm = make_int4(0, 0, 0, 0);
    Splat sm_ = {};
    if (i < hi) {
      id = (unsigned)sorted[i];
      t = id < (unsigned)n ? counts[id] : 0u;
      if (t > 0) { qm = rects[id]; sm_ = load_splat(uv, co, id, alpha_min); }
    }
    unsigned long long tot = 0;
    const unsigned long long off = run + block_exclusive_scan(t, &tot);
    run += tot;
    s_sp[threadIdx.x] = sm_;
    s_q[threadIdx.x] = qm;
    s_id[threadIdx.x] = id;
    const unsigned long long off0 = __shfl_sync(0xffffffffu, off, 0);
    const unsigned R = (unsigned)(__shfl_sync(0xffffffffu, off + t, 31) - off0);   // warp's pairs
    const unsigned rows = t > 0 ? (unsigned)(qm.w - qm.y) : 0u;
    const unsigned rincl = warp_inclusive_scan(rows, lane);
    const unsigned P = __shfl_sync(0xffffffffu, rincl, 31);
    __syncwarp();
    unsigned done = 0;                               // pairs written by this warp so far
    for (unsigned p0 = 0; p0 < P; p0 += 32) {
      const unsigned pr = p0 + lane;                 // this lane's (Gaussian, row) pair
      const int j = scan_search(rincl, pr);
      const unsigned jfirst = __shfl_sync(0xffffffffu, rincl - rows, j);
      int2 r = make_int2(0, 0);
      int ty = 0;
      unsigned idj = 0;
      if (pr < P) {
        const int slot = w * 32 + j;
        const int4 q = s_q[slot];
        ty = q.y + (int)(pr - jfirst);
        r = row_run(s_sp[slot], q, ty);
        idj = s_id[slot];
      }
      const unsigned c = (unsigned)(r.y - r.x);
      const unsigned cincl = warp_inclusive_scan(c, lane);
      const unsigned total = __shfl_sync(0xffffffffu, cincl, 31);
      for (unsigned k0 = 0; k0 < total; k0 += 32) {  // uniform trip count: every lane
        const unsigned k = k0 + lane;                // takes part in the shuffles
        const int rl = scan_search(cincl, k);
        const unsigned before = __shfl_sync(0xffffffffu, cincl - c, rl);
        const int xa = __shfl_sync(0xffffffffu, r.x, rl);
        const int tyl = __shfl_sync(0xffffffffu, ty, rl);
        const unsigned idl = __shfl_sync(0xffffffffu, idj, rl);
        const unsigned at = done + k;
        if (k < total && at < R)
          pairs[off0 + at] = ((T)(unsigned)(tyl * tiles_x + xa + (int)(k - before)) << id_bits) | (T)idl;
      }
      done += total;
    }
    __syncthreads();                                 // s_sp, s_q, s_id are refilled next round
  }
}

// ---- binning through tile-row runs (tile grids up to kMaxRunCols x kMaxRunRows).  Each
// Gaussian's kept tiles in a tile row form one run [x0, x1) (the kept set is convex), so instead
// of emitting every (tile, Gaussian) pair and sorting the pairs by tile, the runs (about a
// seventh as many) are emitted in depth order, sorted stably by row, and each run's Gaussian
// is written straight into the tiles' ranges: within a row, the pairs of tile column x come
// from the row's runs that cover x, in order, so the position of a run's entry in column x is
// the column's range start + the runs before it in the row that cover x.  The row's runs are
// cut into chunks of kPlaceRuns; a chunk counts its runs per column (a difference array),
// adds the counts of the row's earlier chunks by decoupled look-back over the columns, and
// writes its entries one column per lane.

// Run item: row (16 bits) | x0 (8) | x1 - 1 (8) | Gaussian id (32).
constexpr int kRunRowShift = 48;

__device__ __forceinline__ u64 run_item(int ty, int2 r, unsigned id) {
  return ((u64)ty << kRunRowShift) | ((u64)r.x << 40) | ((u64)(r.y - 1) << 32) | id;
}

// The same traversal as emit_kernel, one item per non-empty (Gaussian, tile row) run, in depth
// order then row order; run offsets from the scan of the per-Gaussian run counts.
__global__ void __launch_bounds__(kEmitThreads)
emit_runs_kernel(const u64* sorted, int n, const float2* uv, const float4* co, const int4* rects,
                 const unsigned* counts, const unsigned long long* block_off, const long long* K,
                 long long cap, float alpha_min, u64* runs, int G) {
  pdl_prologue();
  __shared__ Splat s_sp[kEmitThreads];
  __shared__ int4 s_q[kEmitThreads];
  __shared__ unsigned s_id[kEmitThreads];
  if (*K > cap) return;
  long long lo, hi;
  block_range(n, G, &lo, &hi);
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const unsigned lt = (1u << lane) - 1u;
  unsigned long long run = block_off[blockIdx.x];
  for (long long base = lo; base < hi; base += blockDim.x) {
    const long long i = base + threadIdx.x;
    unsigned id = 0, t = 0;
    int4 qm = make_int4(0, 0, 0, 0);
    Splat sm_ = {};
    if (i < hi) {
      id = (unsigned)sorted[i];
      t = id < (unsigned)n ? counts[id] : 0u;
      if (t > 0) { qm = rects[id]; sm_ = load_splat(uv, co, id, alpha_min); }
    }
    unsigned long long tot = 0;
    const unsigned long long off = run + block_exclusive_scan(t, &tot);
    run += tot;
    s_sp[threadIdx.x] = sm_;
    s_q[threadIdx.x] = qm;
    s_id[threadIdx.x] = id;
    const unsigned long long off0 = __shfl_sync(0xffffffffu, off, 0);   // the warp's first run
    const unsigned rows = t > 0 ? (unsigned)(qm.w - qm.y) : 0u;
    const unsigned rincl = warp_inclusive_scan(rows, lane);
    const unsigned P = __shfl_sync(0xffffffffu, rincl, 31);
    __syncwarp();
    unsigned long long at = off0;
    for (unsigned p0 = 0; p0 < P; p0 += 32) {
      const unsigned pr = p0 + lane;                 // this lane's (Gaussian, row) pair
      const int j = scan_search(rincl, pr);
      const unsigned jfirst = __shfl_sync(0xffffffffu, rincl - rows, j);
      int2 r = make_int2(0, 0);
      int ty = 0;
      unsigned idj = 0;
      if (pr < P) {
        const int slot = w * 32 + j;
        const int4 q = s_q[slot];
        ty = q.y + (int)(pr - jfirst);
        r = row_run(s_sp[slot], q, ty);
        idj = s_id[slot];
      }
      const bool ne = r.y > r.x;
      const unsigned b = __ballot_sync(0xffffffffu, ne);
      const unsigned long long dst = at + __popc(b & lt);
      if (ne && dst < (unsigned long long)cap) runs[dst] = run_item(ty, r, idj);
      at += __popc(b);
    }
    __syncthreads();                                 // s_sp, s_q, s_id are refilled next round
  }
}

constexpr int kPlaceThreads = 128;
constexpr int kPlaceRuns = 512;                      // runs per chunk: 4 per thread
constexpr int kPlaceWords = kPlaceRuns / 32;         // words of a column's run mask
constexpr int kPlacePitch = kPlaceWords + 1;         // odd pitch: a column per thread, no conflicts
constexpr int kPlaceLB = 8;                          // look-back words read per column and round
static_assert(kMaxRunRows % kPlaceThreads == 0 && kPlaceRuns % kPlaceThreads == 0, "tiling");

// Runs sorted by row (depth order inside a row) -> ids in the tile ranges.  row_runs: runs per
// row; chunks are claimed in order through ctr (the last CTA clears it); state: tiles_x look-back
// words per chunk.  Inside a chunk, column x keeps a bit mask of the runs that cover it and the
// number of covering runs before each mask word, so the rank of run j in column x is a
// popcount.  A wait gives up after spin_limit polls (status gets ABCD_ERR_TIMEOUT).
// Dynamic shared memory of place_kernel, sized for the grid (so that, with at most 64
// registers, eight CTAs fit on an SM): the rows' run and chunk starts, then per tile column the
// run mask, the chunk's count and base, and the popcounts before each mask word.
inline size_t place_smem_bytes(int rows, int tiles_x) {
  return sizeof(unsigned) * (2 * (size_t)(rows + 1) + (size_t)tiles_x * (kPlacePitch + 2)) +
         sizeof(unsigned short) * (size_t)tiles_x * kPlacePitch;
}

__global__ void __launch_bounds__(kPlaceThreads, 8)
place_kernel(const u64* runs, const long long* n_runs, long long cap, const unsigned* row_runs,
             int rows, int tiles_x, const unsigned* ranges, const long long* K, unsigned* ids,
             u64* state, unsigned* ctr, unsigned epoch, unsigned* status, unsigned spin_limit) {
  pdl_prologue();
  extern __shared__ __align__(16) unsigned place_sm[];
  unsigned* s_rs = place_sm;                                  // [rows + 1] first run of a row
  unsigned* s_cs = s_rs + (rows + 1);                         // [rows + 1] first chunk of a row
  unsigned* s_mask = s_cs + (rows + 1);                       // [column][word]
  unsigned* s_cnt = s_mask + tiles_x * kPlacePitch;           // the chunk's runs per column
  unsigned* s_base = s_cnt + tiles_x;                         // where a column's entries start
  unsigned short* s_pc = reinterpret_cast<unsigned short*>(s_base + tiles_x);   // before a word
  __shared__ unsigned s_c, s_row;
  if (*K > cap) return;                              // the ranges are empty: nothing to place
  const long long nr = dev_count(0, n_runs, cap);
  {
    constexpr int PER = kMaxRunRows / kPlaceThreads;
    unsigned a[PER], b[PER], sa = 0, sb = 0;
#pragma unroll
    for (int k = 0; k < PER; ++k) {
      const int y = threadIdx.x * PER + k;
      a[k] = y < rows ? row_runs[y] : 0u;
      b[k] = (a[k] + kPlaceRuns - 1) / kPlaceRuns;
      sa += a[k];
      sb += b[k];
    }
    unsigned long long ta = 0, tb = 0;
    unsigned long long ea = block_exclusive_scan(sa, &ta);
    unsigned long long eb = block_exclusive_scan(sb, &tb);
#pragma unroll
    for (int k = 0; k < PER; ++k) {
      const int y = threadIdx.x * PER + k;
      if (y < rows) { s_rs[y] = (unsigned)ea; s_cs[y] = (unsigned)eb; }
      ea += a[k];
      eb += b[k];
    }
    if (threadIdx.x == 0) { s_rs[rows] = (unsigned)ta; s_cs[rows] = (unsigned)tb; }
  }
  __syncthreads();
  const unsigned n_chunks = s_cs[rows];
  for (;;) {
    if (threadIdx.x == 0) {
      const unsigned c = atomicAdd(ctr, 1u);
      unsigned y = 0;
      if (c < n_chunks) {                            // the row with s_cs[y] <= c < s_cs[y + 1]
        int lo = 0, hi = rows;
        while (hi - lo > 1) {
          const int mid = (lo + hi) >> 1;
          if (s_cs[mid] <= c) lo = mid; else hi = mid;
        }
        y = (unsigned)lo;
      }
      s_c = c;
      s_row = y;
    }
    for (int k = threadIdx.x; k < tiles_x * kPlacePitch; k += kPlaceThreads) s_mask[k] = 0u;
    __syncthreads();
    const unsigned c = s_c;
    if (c >= n_chunks) break;                        // block-uniform
    const int ty = (int)s_row;
    const unsigned c0 = s_cs[ty], k = c - c0;
    const unsigned r0 = s_rs[ty] + k * kPlaceRuns;
    const unsigned r1 = min(s_rs[ty + 1], r0 + (unsigned)kPlaceRuns);
    // this thread's runs j = threadIdx.x + 128 q, kept in registers for the placement
    unsigned rx0[kPlaceRuns / kPlaceThreads], rxm[kPlaceRuns / kPlaceThreads];
    unsigned rid[kPlaceRuns / kPlaceThreads];
#pragma unroll
    for (int q = 0; q < kPlaceRuns / kPlaceThreads; ++q) {
      const int j = threadIdx.x + q * kPlaceThreads;
      rx0[q] = 1u;
      rxm[q] = 0u;                                   // empty
      rid[q] = 0u;
      if (r0 + j < r1 && (long long)(r0 + j) < nr) {
        const u64 v = runs[r0 + j];
        rx0[q] = (unsigned)(v >> 40) & 255u;
        rxm[q] = min((unsigned)(v >> 32) & 255u, (unsigned)tiles_x - 1u);
        rid[q] = (unsigned)v;
      }
    }
#pragma unroll
    for (int q = 0; q < kPlaceRuns / kPlaceThreads; ++q) {
      const int j = threadIdx.x + q * kPlaceThreads;
      const unsigned bit = 1u << (j & 31);
      for (unsigned x = rx0[q]; x <= rxm[q]; ++x) atomicOr(&s_mask[x * kPlacePitch + (j >> 5)], bit);
    }
    __syncthreads();
    // per column: covering runs before each word, and in all
    for (int x = threadIdx.x; x < tiles_x; x += kPlaceThreads) {
      unsigned run = 0;
#pragma unroll
      for (int w = 0; w < kPlaceWords; ++w) {
        s_pc[x * kPlacePitch + w] = (unsigned short)run;
        run += __popc(s_mask[x * kPlacePitch + w]);
      }
      s_cnt[x] = run;
    }
    // publish the chunk's counts (the row's first chunk: as inclusive prefixes) ...
    for (int x = threadIdx.x; x < tiles_x; x += kPlaceThreads)
      os_publish(state + (size_t)c * tiles_x + x, os_word(epoch, k == 0 ? 2u : 1u, s_cnt[x]));
    // ... then add up the row's earlier chunks per column, nearest first
    for (int x = threadIdx.x; x < tiles_x; x += kPlaceThreads) {
      unsigned prefix = 0;
      if (k > 0) {
        long long j0 = (long long)c - 1;             // nearest chunk not summed yet
        unsigned spins = 0;
        for (;;) {
          u64 v[kPlaceLB];
#pragma unroll
          for (int q = 0; q < kPlaceLB; ++q) {
            const long long idx = j0 - q;
            v[q] = idx >= (long long)c0 ? os_peek(state + (size_t)idx * tiles_x + x)
                                        : os_word(epoch, 2u, 0u);
          }
          unsigned sum = 0;
          int used = kPlaceLB, kind = 0;             // 0: all aggregates, 1: inclusive, 2: blocked
#pragma unroll
          for (int q = 0; q < kPlaceLB; ++q) {
            if (kind != 0) continue;
            const unsigned flag = (unsigned)(v[q] >> 32) & 3u;
            if ((unsigned)(v[q] >> 34) != epoch || flag == 0u) { kind = 2; used = q; continue; }
            sum += (unsigned)v[q];
            if (flag == 2u) { kind = 1; used = q + 1; }
          }
          prefix += sum;
          j0 -= used;
          if (kind == 1) break;
          if (kind == 2) {
            if (++spins > spin_limit) { atomicOr(status, kStatusTimeout); break; }
            __nanosleep(32);
          }
        }
        os_publish(state + (size_t)c * tiles_x + x, os_word(epoch, 2u, prefix + s_cnt[x]));
      }
      s_base[x] = ranges[2 * (ty * tiles_x + x)] + prefix;
    }
    __syncthreads();
    // entries: run j in column x goes to base(x) + the runs before j that cover x
#pragma unroll
    for (int q = 0; q < kPlaceRuns / kPlaceThreads; ++q) {
      const int j = threadIdx.x + q * kPlaceThreads;
      const unsigned below = (1u << (j & 31)) - 1u;
      for (unsigned x = rx0[q]; x <= rxm[q]; ++x) {
        const int at = (int)x * kPlacePitch + (j >> 5);
        const unsigned pos = s_base[x] + s_pc[at] + __popc(s_mask[at] & below);
        if ((long long)pos < cap) ids[pos] = rid[q];
      }
    }
    __syncthreads();                                 // before the next chunk reuses the arrays
  }
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(ctr + 1, 1u) == gridDim.x - 1) { ctr[0] = 0u; ctr[1] = 0u; }
  }
}

// Launches one pass for a digit of `bits` bits (4..8).
template <typename T>
abcd_status launch_onesweep(abcd_ctx* ctx, cudaStream_t st, int bits, bool match, int G,
                            const T* src, T* dst, unsigned* ids, unsigned id_mask,
                            long long n_static, const long long* n_dev, long long cap, int shift,
                            const unsigned* gh, unsigned* ctr, long long withhold,
                            const unsigned* krange) {
  const unsigned epoch = ++ctx->os_epoch;
  const unsigned spin = ctx->wait_limit;
#define ABCD_PASS(B)                                                                              \
  case B:                                                                                         \
    e = match ? launch_pdl(onesweep_kernel<T, B, true>, dim3(G), dim3(kOsThreads), 0, st, src, dst, \
                           ids, id_mask, n_static, n_dev, cap, shift, gh, ctx->ws.os_state, ctr,   \
                           epoch, ctx->ws.status, spin, withhold, krange)                          \
              : launch_pdl(onesweep_kernel<T, B, false>, dim3(G), dim3(kOsThreads), 0, st, src,    \
                           dst, ids, id_mask, n_static, n_dev, cap, shift, gh, ctx->ws.os_state,   \
                           ctr, epoch, ctx->ws.status, spin, withhold, krange);                    \
    break;
  cudaError_t e = cudaSuccess;
  switch (bits) {
    ABCD_PASS(4) ABCD_PASS(5) ABCD_PASS(6) ABCD_PASS(7) ABCD_PASS(8)
    default: return fail(ctx, ABCD_ERR_INVALID_ARG, "radix digit of %d bits", bits);
  }
#undef ABCD_PASS
  return check_launch(ctx, "onesweep_kernel", e);
}

// First pass ranked with __match_any_sync (earlier passes use ballots): the depth keys' two
// high bytes and the tile index's high bits come nearly grouped.
constexpr int kDepthMatchFrom = 2;
constexpr int kTileMatchFrom = 1;

// Stable LSD radix sort of 32- or 64-bit items on bits [bit_lo, bit_hi), in the fewest
// one-sweep passes of at most 8 bits, of equal width (fewer bits per pass: fewer ballots per
// ranked item); returns the buffer holding the result, or writes the bits id_mask of the
// sorted items to ids_out on the last pass.  `slot` (0: depth sort, 1: tile sort) selects the
// digit counts and tile counters.  n_max bounds the item count (it sizes the grid).
template <typename T>
abcd_status radix_sort(abcd_ctx* ctx, cudaStream_t st, T* a, T* b, long long n_static,
                       const long long* n_dev, long long cap, long long n_max, int bit_lo,
                       int bit_hi, int slot, bool counted, T** result, unsigned* ids_out,
                       unsigned id_mask, int match_from, const unsigned* krange = nullptr) {
  const SortPasses sp = make_passes(bit_lo, bit_hi);
  if (sp.n < 1 || sp.n > 4) return fail(ctx, ABCD_ERR_INVALID_ARG, "radix sort of %d bits", bit_hi - bit_lo);
  unsigned* gh = ctx->ws.os_gh + (size_t)slot * 4 * kRadixBins;
  unsigned* ctr = ctx->ws.os_ctr + 2 * slot;
  const long long tile = (long long)kOsThreads * (64 / (int)sizeof(T));
  const long long tiles = (n_max + tile - 1) / tile;
  if (tiles > ctx->ws.os_tiles) return fail(ctx, ABCD_ERR_WORKSPACE, "radix sort: %lld tiles exceed the workspace", tiles);
  const int G = (int)std::max<long long>(1, std::min<long long>(tiles, 4LL * ctx->num_sms));
  const int Gd = (int)std::max<long long>(1, std::min<long long>((n_max + 255) / 256, 2LL * ctx->num_sms));
  abcd_status s = ABCD_OK;
  if (!counted &&                              // the tile sort's counts come with the ranges
      (s = check_launch(ctx, "sort_digits_kernel",
                        launch_pdl(sort_digits_kernel<T>, dim3(Gd), dim3(256), 0, st, (const T*)a,
                                   n_static, n_dev, cap, sp, match_from, gh, krange))))
    return s;
  T* src = a;
  T* dst = b;
  for (int p = 0; p < sp.n; ++p) {
    const bool last = p == sp.n - 1;
    // the test hook withholds a tile of the depth sort's first pass only
    const long long withhold = (slot == 0 && p == 0) ? ctx->withhold_tile : -1;
    if ((s = launch_onesweep<T>(ctx, st, sp.bits[p], p >= match_from, G, src, dst,
                                last ? ids_out : nullptr, id_mask, n_static, n_dev, cap,
                                sp.shift[p], gh + p * kRadixBins, ctr, withhold,
                                p == 0 ? krange : nullptr)))
      return s;
    if (slot == 0 && p == 0) ctx->withhold_tile = -1;
    T* t = src; src = dst; dst = t;
  }
  if (result) *result = src;
  return ABCD_OK;
}

}  // namespace
}  // namespace abcd

using namespace abcd;

extern "C" abcd_status abcd_bin_sort(abcd_ctx* ctx, const abcd_projected* proj, int n,
                                     const abcd_camera* cam, const abcd_render_opts* opts,
                                     abcd_tiles* out) {
  if (!ctx) return ABCD_ERR_INVALID_ARG;
  if (!has_workspace(ctx)) return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_bin_sort: no workspace");
  if (!proj || !cam || !out || n < 0 || cam->width <= 0 || cam->height <= 0)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_bin_sort: bad arguments");
  if (n > ctx->max_g) return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_bin_sort: n=%d exceeds workspace max_gaussians=%d", n, ctx->max_g);
  if (!out->ids || !out->ranges || !out->count || out->capacity < 0)
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_bin_sort: null tiles output");
  const long long cap = std::min(out->capacity, ctx->max_pairs);
  const int tiles_x = (cam->width + kTile - 1) / kTile, tiles_y = (cam->height + kTile - 1) / kTile;
  const long long n_tiles = (long long)tiles_x * tiles_y;
  if (n_tiles >= (1LL << 24)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_bin_sort: too many tiles");
  if (cap >= (1LL << 32)) return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_bin_sort: capacity must be < 2^32");
  if (n > 0 && (!proj->depth || !proj->radius || !proj->uv || !proj->conic_opacity ||
                ((uintptr_t)proj->uv & 7) || ((uintptr_t)proj->conic_opacity & 15)))
    return fail(ctx, ABCD_ERR_INVALID_ARG, "abcd_bin_sort: null projected field");
  cudaError_t e = cudaSuccess;
  if (n == 0) {
    e = cudaMemsetAsync(out->ranges, 0, sizeof(unsigned) * 2 * n_tiles, ctx->stream);
    if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "ranges memset: %s", cudaGetErrorString(e));
    e = cudaMemsetAsync(out->count, 0, sizeof(long long), ctx->stream);
    return e == cudaSuccess ? ABCD_OK : fail(ctx, ABCD_ERR_CUDA, "count memset: %s", cudaGetErrorString(e));
  }
  if (ctx->os_epoch > (1u << 30) - 64) {     // look-back epochs wrap: clear the old words
    e = cudaMemsetAsync(ctx->ws.os_state, 0, 8ull * kRadixBins * (size_t)ctx->ws.os_tiles, ctx->stream);
    if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "sort state memset: %s", cudaGetErrorString(e));
    ctx->os_epoch = 0;
  }
  const size_t diff_bytes = sizeof(int) * (size_t)(tiles_x + 1) * (tiles_y + 1);
  if (diff_bytes > ctx->ws.diff_bytes)
    return fail(ctx, ABCD_ERR_WORKSPACE, "abcd_bin_sort: tile grid exceeds the workspace");
  abcd_status s;
  // the visible depth keys' range: two pairs of words used in turn, each call's keys_rects
  // clearing the other pair for the next call (zero initially: the workspace set-up clears them)
  unsigned* krange = ctx->ws.os_ctr + 8 + 2 * (int)(ctx->krange_parity & 1u);
  unsigned* krange_next = ctx->ws.os_ctr + 8 + 2 * (int)((ctx->krange_parity + 1u) & 1u);
  const float alpha_min = make_opts(opts).alpha_min;
  int tile_bits = 1;
  while ((1LL << tile_bits) < n_tiles) ++tile_bits;
  int row_bits = 1;
  while ((1 << row_bits) < tiles_y) ++row_bits;
  const int cells = (tiles_x + 1) * (tiles_y + 1);
  // tile grids up to kMaxRunCols x kMaxRunRows bin through tile-row runs (the run placement's
  // look-back words must fit the workspace); larger ones sort (tile, Gaussian) pairs
  const long long max_chunks = cap / kPlaceRuns + tiles_y + 1;
  const bool by_runs = tiles_x <= kMaxRunCols && tiles_y <= kMaxRunRows &&
                       cells <= kSmemDiffCells && n_tiles <= ctx->ws.max_tiles &&
                       max_chunks * tiles_x <= ctx->ws.os_tiles * kRadixBins;
  // digit counts of the tile sort's passes (or of the runs' row sort), made with the ranges;
  // the passes count from the tile (row) bits' lowest, the sorts' own from the items' field
  const SortPasses tile_passes = make_passes(0, by_runs ? row_bits : tile_bits);
  unsigned* tile_gh = ctx->ws.os_gh + 4 * kRadixBins;
  if ((s = check_launch(ctx, "keys_rects_kernel",
                        launch_pdl(keys_rects_kernel,
                                   dim3((unsigned)std::max<size_t>((n + 255) / 256, (cells + 4095) / 4096)),
                                   dim3(256), 0, ctx->stream,
                                   (const float*)proj->depth, (const int*)proj->radius,
                                   (const float2*)proj->uv, n, tiles_x, tiles_y, ctx->ws.dsort[0],
                                   ctx->ws.rects, ctx->ws.os_gh, 2 * 4 * kRadixBins,
                                   ctx->ws.row_runs, by_runs ? tiles_y : 0, ctx->ws.diff, cells,
                                   krange, krange_next))))
    return s;
  ++ctx->krange_parity;                              // the next call's pair is being cleared
  // the tile rows and ranges only need the rectangles: they run on the side stream while the
  // depth sort, the longer branch, runs here (its launches chained to keys_rects_kernel's
  // without the fork's event wait)
  e = cudaEventRecord(ctx->ev_fork, ctx->stream);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(ctx->side, ctx->ev_fork, 0);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "tile rows fork: %s", cudaGetErrorString(e));
  {
    const size_t smem = cells <= kSmemDiffCells
                            ? sizeof(int) * cells + (by_runs ? sizeof(unsigned) * tiles_y : 0)
                            : 0;
    auto kern = by_runs ? tile_rows_kernel<true> : tile_rows_kernel<false>;
    {
      const cudaError_t e2 = ensure_smem(ctx, (const void*)kern, smem);
      if (e2 != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "tile_rows smem: %s", cudaGetErrorString(e2));
    }
    if ((s = check_launch(ctx, "tile_rows_kernel",
                          launch_pdl(kern, dim3((n + 255) / 256), dim3(256), smem,
                                     ctx->side, (const float2*)proj->uv,
                                     (const float4*)proj->conic_opacity, (const int4*)ctx->ws.rects,
                                     n, tiles_x, tiles_y, alpha_min, ctx->ws.counts, ctx->ws.diff,
                                     ctx->ws.row_runs))))
      return s;
  }
  {
    ctx->order_ranges = nullptr;
    if (cells <= kSmemDiffCells && n_tiles <= ctx->ws.max_tiles) {
      const size_t smem = sizeof(int) * cells + (size_t)n_tiles;
      {
        const cudaError_t e2 = ensure_smem(ctx, (const void*)ranges_order_kernel, smem);
        if (e2 != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "ranges smem: %s", cudaGetErrorString(e2));
      }
      if ((s = check_launch(ctx, "ranges_order_kernel",
                            launch_pdl(ranges_order_kernel, dim3(1), dim3(1024), smem, ctx->side,
                                       (const int*)ctx->ws.diff, tiles_x, tiles_y, cap, out->ranges,
                                       ctx->ws.tile_order, tile_passes, tile_gh,
                                       by_runs ? (const unsigned*)ctx->ws.row_runs : nullptr,
                                       by_runs ? (long long*)out->count : nullptr, ctx->ws.status))))
        return s;
      ctx->order_ranges = out->ranges;           // the order belongs to these ranges
      ctx->order_tiles = n_tiles;
    } else {
      if ((s = check_launch(ctx, "ranges_from_diff_kernel",
                            launch_pdl(ranges_from_diff_kernel, dim3(1), dim3(1024), 0, ctx->side,
                                       ctx->ws.diff, tiles_x, tiles_y, cap, out->ranges,
                                       tile_passes, tile_gh))))
        return s;
    }
  }
  e = cudaEventRecord(ctx->ev_join, ctx->side);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "tile rows join: %s", cudaGetErrorString(e));
  u64* by_depth = nullptr;
  if ((s = radix_sort<u64>(ctx, ctx->stream, ctx->ws.dsort[0], ctx->ws.dsort[1], n, nullptr, n, n,
                           32, 64, 0, false, &by_depth, nullptr, 0xffffffffu, kDepthMatchFrom,
                           krange)))
    return s;
  e = cudaStreamWaitEvent(ctx->stream, ctx->ev_join, 0);
  if (e != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "tile rows join: %s", cudaGetErrorString(e));
  const int Ge = std::min(kMaxRadixBlocks, 6 * ctx->num_sms);   // blocks of count / emit
  if ((s = check_launch(ctx, "count_kernel",
                        launch_pdl(count_kernel, dim3(Ge), dim3(256), 0, ctx->stream,
                                   (const u64*)by_depth, n, (const unsigned*)ctx->ws.counts,
                                   ctx->ws.block_sums, Ge))))
    return s;
  if ((s = check_launch(ctx, "scan_blocks_kernel",
                        launch_pdl(scan_blocks_kernel, dim3(1), dim3(1024), 0, ctx->stream,
                                   ctx->ws.block_sums, Ge,
                                   by_runs ? ctx->ws.n_runs : (long long*)out->count, cap,
                                   ctx->ws.status))))
    return s;
  if (by_runs) {
    u64* runs = ctx->ws.pairs[0];
    if ((s = check_launch(ctx, "emit_runs_kernel",
                          launch_pdl(emit_runs_kernel, dim3(Ge), dim3(kEmitThreads), 0, ctx->stream,
                                     (const u64*)by_depth, n, (const float2*)proj->uv,
                                     (const float4*)proj->conic_opacity, (const int4*)ctx->ws.rects,
                                     (const unsigned*)ctx->ws.counts,
                                     (const unsigned long long*)ctx->ws.block_sums,
                                     (const long long*)out->count, cap, alpha_min, runs, Ge))))
      return s;
    u64* by_row = nullptr;
    if ((s = radix_sort<u64>(ctx, ctx->stream, runs, ctx->ws.pairs[1], 0, ctx->ws.n_runs, cap, cap,
                             kRunRowShift, kRunRowShift + row_bits, 1, true, &by_row, nullptr,
                             0xffffffffu, 1)))
      return s;
    const unsigned epoch = ++ctx->os_epoch;
    const int Gp = (int)std::max<long long>(1, std::min<long long>(max_chunks, 8LL * ctx->num_sms));
    const size_t psm = place_smem_bytes(tiles_y, tiles_x);
    {
      const cudaError_t e2 = ensure_smem(ctx, (const void*)place_kernel, psm);
      if (e2 != cudaSuccess) return fail(ctx, ABCD_ERR_CUDA, "place smem: %s", cudaGetErrorString(e2));
    }
    return check_launch(ctx, "place_kernel",
                        launch_pdl(place_kernel, dim3(Gp), dim3(kPlaceThreads), psm, ctx->stream,
                                   (const u64*)by_row, (const long long*)ctx->ws.n_runs, cap,
                                   (const unsigned*)ctx->ws.row_runs, tiles_y, tiles_x,
                                   (const unsigned*)out->ranges, (const long long*)out->count,
                                   (unsigned*)out->ids, ctx->ws.os_state, ctx->ws.os_ctr + 4, epoch,
                                   ctx->ws.status, ctx->wait_limit));
  }
  int id_bits = 1;
  while ((1LL << id_bits) < n) ++id_bits;
  // K lives on the device: the tile passes take the largest grid; blocks past K exit at once.
  // (tile, id) pairs pack into 32 bits when they fit (half the bytes per pass), else 64.
  if (tile_bits + id_bits <= 32) {
    unsigned* pairs = reinterpret_cast<unsigned*>(ctx->ws.pairs[0]);
    unsigned* pairs_b = reinterpret_cast<unsigned*>(ctx->ws.pairs[1]);
    if ((s = check_launch(ctx, "emit_kernel",
                          launch_pdl(emit_kernel<unsigned>, dim3(Ge), dim3(kEmitThreads), 0,
                                     ctx->stream, (const u64*)by_depth, n, (const float2*)proj->uv,
                                     (const float4*)proj->conic_opacity, (const int4*)ctx->ws.rects,
                                     (const unsigned*)ctx->ws.counts,
                                     (const unsigned long long*)ctx->ws.block_sums,
                                     (const long long*)out->count, cap, tiles_x, alpha_min, id_bits,
                                     pairs, Ge))))
      return s;
    return radix_sort<unsigned>(ctx, ctx->stream, pairs, pairs_b, 0, out->count, cap, cap, id_bits,
                                id_bits + tile_bits, 1, true, nullptr, out->ids,
                                (1u << id_bits) - 1u, kTileMatchFrom);
  }
  if ((s = check_launch(ctx, "emit_kernel",
                        launch_pdl(emit_kernel<u64>, dim3(Ge), dim3(kEmitThreads), 0,
                                   ctx->stream, (const u64*)by_depth, n, (const float2*)proj->uv,
                                   (const float4*)proj->conic_opacity, (const int4*)ctx->ws.rects,
                                   (const unsigned*)ctx->ws.counts,
                                   (const unsigned long long*)ctx->ws.block_sums,
                                   (const long long*)out->count, cap, tiles_x, alpha_min, 32,
                                   ctx->ws.pairs[0], Ge))))
    return s;
  return radix_sort<u64>(ctx, ctx->stream, ctx->ws.pairs[0], ctx->ws.pairs[1], 0, out->count, cap,
                         cap, 32, 32 + tile_bits, 1, true, nullptr, out->ids, 0xffffffffu,
                         kTileMatchFrom);
}
