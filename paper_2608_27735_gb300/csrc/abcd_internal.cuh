// Internal declarations shared by the libabcd translation units (not part of the ABI).
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "../../include/abcd.h"

namespace abcd {

constexpr int kTile = 16;                 // tile edge (pixels)
constexpr int kTileThreads = kTile * kTile;
constexpr int kRadixBits = 8;
constexpr int kRadixBins = 1 << kRadixBits;
constexpr int kMaxRadixBlocks = 1024;     // upper bound used to size the histogram scratch
constexpr int kMaxLossBlocks = 1 << 16;
constexpr int kMaxLayers = 256;
constexpr long long kMaxDiffCells = 1LL << 20;   // (tiles_x + 1) * (tiles_y + 1)
constexpr int kMaxRunRows = 1024;     // tile grids that bin through tile-row runs: rows ...
constexpr int kMaxRunCols = 256;      // ... and columns at most
constexpr int kVisSumCopies = 8;          // copies of the layer visibility sums

// Device status bits (OR-ed into the status word; abcd_sync reports the lowest set code).
constexpr unsigned kStatusCapacity = 1u << ABCD_ERR_CAPACITY;
constexpr unsigned kStatusTimeout = 1u << ABCD_ERR_TIMEOUT;

struct Cam {               // camera as the kernels read it (by value)
  float R[9], t[3];
  float fx, fy, cx, cy;
  float campos[3];         // -R^T t (host fp64, rounded)
  float limx, limy;        // guard * tan(fov/2)
  int width, height, tiles_x, tiles_y;
};

struct Opts {
  float near_z, dilation, alpha_max, alpha_min, t_min, guard;
};

struct SHConst { float k[16]; };    // normalisation factors of the real SH basis

struct Workspace {
  unsigned* status;                 // [0] status word, [1] loss ticket
  unsigned long long* dsort[2];     // depth sort items [max_g]
  unsigned long long* pairs[2];     // (tile << 32 | id) items [max_pairs]
  unsigned* os_gh;                  // [2 sorts][4 passes][kRadixBins] digit counts
  unsigned* os_ctr;                 // [2 sorts][2] tile and finished-CTA counters of a pass
  unsigned long long* os_state;     // [os_tiles][kRadixBins] look-back words
  long long os_tiles;
  int4* rects;                      // [max_g] tile rectangle per Gaussian
  unsigned* counts;                 // [max_g] listed tiles (or tile-row runs) per Gaussian
  unsigned* row_runs;               // [kMaxRunRows] tile-row runs per tile row
  long long* n_runs;                // tile-row runs of the last binning
  int* diff;                        // 2-D difference array over the tile grid
  size_t diff_bytes;
  unsigned long long* block_sums;   // [kMaxRadixBlocks + 1]
  float* grad2d;                    // [max_g][9]
  float* dl_dout;                   // [max_pixels][3]
  float* loss_partials;             // [kMaxLossBlocks][2]
  float2* ssim_ab;                  // [3][max_pixels] SSIM partials (A, B) per channel and pixel
  float* ssim_c;                    // [3][max_pixels] SSIM partial C
  unsigned* tile_order;             // [max_tiles] tiles by decreasing list length (bin_sort)
  long long max_tiles;
  // render checkpoints: the forward saves each pixel's (colour, T) where a block's walk crosses
  // a multiple of kCkChunk list positions, and lists the chunks after the first as work items
  // (block, start, end) that the backward replays in parallel CTAs
  float4* ckpt;                     // [ck_cap][64]
  uint4* ck_items;                  // [ck_cap]
  unsigned* ck_count;               // items allocated by the last forward with a state
  unsigned* ck_first;               // [4 max_tiles] end of each block's first chunk, or ~0
  int ck_cap;
  unsigned long long* vis_sums;     // [kVisSumCopies][2][kMaxLayers] layer visibility sums (zero between calls)
  unsigned* vis_ticket;             // CTAs of the visibility call that finished
};

constexpr int kRenderSubPerTile = 4;      // render CTAs (8x8 pixel blocks) per 16x16 tile

// Programmatic dependent launch.  Every kernel of the library starts with pdl_prologue(): it
// waits until the grid before it in the stream has completed and its writes are visible
// (griddepcontrol.wait; immediate when the kernel was launched without the attribute), then
// lets the next grid be launched (griddepcontrol.launch_dependents), whose CTAs wait the same
// way before touching memory.  Launching and rasterising a kernel thus overlaps the tail of the
// one before it instead of following it.  The next grid only starts once every CTA of this one
// is resident, so it takes resources this grid no longer needs.
__device__ __forceinline__ void pdl_prologue() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launches kernel on stream with programmatic stream serialisation allowed.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Mask of the lanes whose value equals this lane's, for values 0..256 (256 marks an unused
// lane; it matches only other unused lanes).  Nine ballots: the cost does not depend on how
// many distinct values the warp holds, unlike __match_any_sync's.
__device__ __forceinline__ unsigned match_byte(unsigned d) {
  unsigned peers = 0xffffffffu;
#pragma unroll
  for (int b = 0; b < 9; ++b) {
    const unsigned bit = (d >> b) & 1u;
    const unsigned m = __ballot_sync(0xffffffffu, bit);
    peers &= bit ? m : ~m;
  }
  return peers;
}

// Tiles the workspace orders for images of up to max_pixels pixels with sides up to 16384.
inline long long max_order_tiles(long long max_pixels) { return max_pixels / 256 + 2048; }

}  // namespace abcd

struct abcd_ctx {
  int device = 0;
  cudaStream_t stream = nullptr;
  cudaStream_t side = nullptr;          // forked work inside one call, joined before it returns
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  // host tier of the layer cache (cache.cu): copy streams and per-slot events, made on first use
  cudaStream_t h2d = nullptr, d2h = nullptr;
  cudaEvent_t ev_store = nullptr;
  cudaEvent_t* cache_ready = nullptr;           // [ABCD_MAX_CACHE_SLOTS]
  cudaEvent_t* cache_released = nullptr;        // [ABCD_MAX_CACHE_SLOTS]
  cudaEvent_t* cache_stored = nullptr;          // [ABCD_MAX_CACHE_SLOTS]
  unsigned char* cache_has_release = nullptr;   // [ABCD_MAX_CACHE_SLOTS]
  int num_sms = 0;
  int radix_blocks = 0;
  char* ws_base = nullptr;
  size_t ws_bytes = 0;
  int max_g = 0;
  long long max_pairs = 0;
  long long max_pixels = 0;
  abcd::Workspace ws{};
  const void* order_ranges = nullptr;   // tile ranges the order in ws.tile_order belongs to
  const void* ck_state = nullptr;       // forward state the render checkpoints belong to
  const void* ck_ranges = nullptr;      // and the tile ranges and block count they were made for
  long long ck_blocks = 0;
  long long order_tiles = 0;
  abcd::SHConst sh{};
  long long launches = 0;
  unsigned os_epoch = 0;                // last look-back epoch handed to a sort pass
  unsigned krange_parity = 0;           // which pair of depth-key range words bin_sort uses next
  unsigned wait_limit = 1u << 20;       // polls before a device-side wait gives up
  long long withhold_tile = -1;         // test hook: a look-back tile that publishes nothing
  // dynamic shared memory limits already raised on this context's device, per kernel (the
  // attribute call costs host time on every step otherwise)
  const void* smem_fn[16] = {nullptr};
  int smem_set[16] = {0};
  char err[512] = {0};
};

namespace abcd {

abcd_status fail(abcd_ctx* ctx, abcd_status code, const char* fmt, ...);
void cache_destroy(abcd_ctx* ctx);            // copy streams and slot events (cache.cu)
abcd_status check_launch(abcd_ctx* ctx, const char* what);
abcd_status check_launch(abcd_ctx* ctx, const char* what, cudaError_t launched);
// Raises kernel fn's dynamic shared-memory limit to at least `bytes` (once per context and size).
cudaError_t ensure_smem(abcd_ctx* ctx, const void* fn, size_t bytes);
// Zeroes bytes at p on the context's stream with a programmatically serialised kernel (a memset
// when p or bytes is not a multiple of 4).
abcd_status zero_async(abcd_ctx* ctx, void* p, size_t bytes, const char* what);
bool has_workspace(const abcd_ctx* ctx);
Cam make_cam(const abcd_camera* c, const abcd_render_opts* o);
Opts make_opts(const abcd_render_opts* o);
void sh_constants(SHConst* out);

// translation-unit entry points used by the composite calls
abcd_status loss_launch(abcd_ctx* ctx, const float* out_rgba, const float* gt_rgb, int width,
                        int height, float lambda_ssim, float* loss_out, float* dL_dout);

}  // namespace abcd
