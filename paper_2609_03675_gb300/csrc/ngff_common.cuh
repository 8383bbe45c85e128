// Internal declarations shared by the NGFF kernels and the C ABI layer.
//
// Data layout in device memory (per handle):
//   frames   uint8  [rows][H][W][3]   caller-owned (or a staging buffer)
//   hist     uint32 [rows][B]         integer histograms of the push (kept zero
//                                     between pushes: the scan clears its rows)
//   l1       uint32 [rows][L_max]     L1[t][k-1] = sum_b |c_t[b] - c_{t-k}[b]|
//   mask     uint32 [rows][W_m]       bit g-1 of row t: keep decision of frame t
//                                     if its gap t - r(t) were g (W_m = ceil(L_max/32))
//   ring     uint32 [streams][L_max][B]  histogram of frame t at slot t mod L_max
//                                     (L_max = 0: [streams][2][B], the previous
//                                     frame's and the reference frame's rows)
//   state    StreamState [streams]    frames seen and current gap
//   record   uint32 [streams][R]      retention record: bit t of stream s is set
//                                     when frame t was retained (any nonzero keep
//                                     code), for t < 32 R (cofie_ngff_candidates)
#pragma once

#include <atomic>
#include <cstdint>
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

namespace cofie {

constexpr int kMaxSegs = 64;
constexpr int kMaxBins = 256;
constexpr int kMaxLmax = 256;

// One stream's frames inside a push: rows [row0, row0 + n) of the tables.
struct Segment {
  const uint8_t* frames;  // device pointer of the first frame
  float* scores;          // device, n entries, or nullptr
  uint8_t* keep;          // device, n entries, or nullptr
  uint32_t n;
  uint32_t row0;
  uint32_t stream;
  uint32_t halo;          // histogram rows before row0 that hold the frames just before it
};

struct SegTable {
  Segment s[kMaxSegs];
  uint32_t count;
  uint32_t rows;
};

// Grayscale weights packed for the two-way 16x8-bit dot product (dp2a):
// dp2a.lo(a, b, c) = a.h0 * b.byte0 + a.h1 * b.byte1 + c, .hi uses bytes 2, 3.
struct LumaConsts {
  uint32_t w_rg;     // (wG << 16) | wR
  uint32_t w_b0;     // wB
  uint32_t w_0r;     // wR << 16
  uint32_t w_gb;     // (wB << 16) | wG
  uint32_t half;     // floor(den / 2), the rounding term
  uint32_t magic;    // bin = umulhi(v, magic) when the fast bin path holds
  uint32_t magic_y;  // Y = umulhi(v, magic_y) on the two-step path
  uint32_t bins;
  uint32_t w[3];     // plain weights and divisor for the generic kernel
  uint32_t den;
};

// kCells: the fast kernel's consumers sum grayscale per cell of a grid
// (the spatial signals) instead of counting bins.
enum BinPath : int { kBinFast = 0, kBinTwoStep = 1, kCells = 2 };

struct StreamState {
  unsigned long long t;    // frames seen
  uint32_t g;              // t - r(t) of the next frame (valid when t > 0)
  uint32_t pad;
  unsigned long long acc;  // scene-change signal: L1 numerator summed over the open gradual run (0: none)
};

// Programmatic dependent launch: the first-stage kernel lets the selection
// kernels that follow it be scheduled early (pdl_trigger), and those wait
// for it (pdl_wait) before their first read of its output, so their launch
// and set-up overlap its tail. The small-push selection kernel does the same
// for the next push's first-stage kernel, whose producer waits before it
// reads a frame (a caller's kernel writing those frames may be the kernel
// before it instead: the wait then covers that kernel). Both instructions are
// no-ops for a kernel launched without the attribute.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// A launch that is a programmatic dependent of the kernel before it when pdl.
template <typename... Params, typename... Args>
inline cudaError_t launch_dependent(bool pdl, void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem,
                                    cudaStream_t st, Args... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// Index checks of the checked build (-DCOFIE_DEBUG_CHECKS=1), which stands in
// for a memory checker: COFIE_BOUND(c) is true in normal builds (and
// compiles away); in checked builds a false c sets this translation unit's
// bounds error word and the guarded access is skipped. cofie_ngff_status
// collects the words (COFIE_EDEVICE). Each check relates an index to the
// kernel's own launch arguments (rows, L_max, bins, tile sizes).
#ifndef COFIE_DEBUG_CHECKS
#define COFIE_DEBUG_CHECKS 0
#endif
namespace {
#if COFIE_DEBUG_CHECKS
__device__ uint32_t g_bounds_err;
__device__ __forceinline__ bool bound_ok(bool c) {
  if (!c) atomicOr(&g_bounds_err, 1u);
  return c;
}
#define COFIE_BOUND(c) (::cofie::bound_ok(static_cast<bool>(c)))
// this translation unit's word, read and cleared (host; synchronous)
inline uint32_t take_local_bounds_errors() {
  uint32_t v = 0, z = 0;
  if (cudaMemcpyFromSymbol(&v, g_bounds_err, sizeof v) != cudaSuccess) return 0;
  cudaMemcpyToSymbol(g_bounds_err, &z, sizeof z);
  return v;
}
#else
#define COFIE_BOUND(c) true
inline uint32_t take_local_bounds_errors() { return 0; }
#endif
}  // namespace
// one reader per translation unit with checked kernels
uint32_t take_bounds_errors_hist();
uint32_t take_bounds_errors_features();
uint32_t take_bounds_errors_select();
uint32_t take_bounds_errors_lazy();
uint32_t take_bounds_errors_finalize();
bool checked_build();

// Bits of the device error word.
constexpr uint32_t kErrConsumerTimeout = 1u;
constexpr uint32_t kErrProducerTimeout = 2u;
constexpr uint32_t kErrDrainTimeout = 4u;
constexpr uint32_t kErrBadIndex = 8u;  // a gather index outside the frame buffer
constexpr uint32_t kErrBounds = 16u;   // checked build: an index check failed
constexpr uint32_t kErrRecord = 32u;   // candidates of a stream that has run past its retention record

struct HistArgs {
  uint64_t frame_bytes;      // 3 W H
  uint32_t npix;             // W H
  uint32_t groups_per_frame; // frame_bytes / 48 (fast kernel)
  uint32_t chunks_per_frame; // ceil(groups_per_frame / chunk groups)
  uint64_t timeout_ns;
  // kCells only (width a multiple of 16): the grid (output row stride grid_h * grid_w),
  // groups per image row, and multiply-high constants for / gpr and / height
  uint32_t width, height, grid_h, grid_w;
  uint32_t gpr, m_gpr, m_h;
  uint32_t wide;  // every cell column is at least 16 pixels wide
  uint32_t m_gw;  // multiply-high constant for / grid_w (wide path)
  uint32_t slice_groups;  // generic kernel only: 16-pixel groups per CTA
};

struct SelectArgs {
  uint32_t bins;
  uint32_t l_max;
  uint32_t mask_words;
  float tau;
  float two_n;        // fp32 of the distance's denominator: 2 W H (histogram), 255 W H (low-res), 64 (dHash)
  uint32_t zero_hist;  // the scan zeroes the push's histogram rows after use
  uint32_t dist_kind;  // 0: sum of |differences| (histogram, low-res); 1: Hamming (dHash)
  uint32_t scd;        // twin-comparison scene changes are added to the rule
  float scd_cut, scd_grad;
  // the same three decisions as integer thresholds on the L1 numerator: the
  // smallest x with fp32(x) / two_n >= tau, T_b, T_s (2^64 - 1: never)
  unsigned long long x_tau, x_cut, x_grad;
  // the streams' retention records ([streams][rec_words]; nullptr: none)
  uint32_t* record;
  uint32_t rec_words;
};

// Sets the record bits of retained frames: bit i of `bits` stands for frame
// t_first + i of the stream whose record is `rec` (rec_words words). Frames
// at or past the record's end are not recorded. One thread per call.
__device__ __forceinline__ void record_bits(uint32_t* rec, uint32_t rec_words, unsigned long long t_first,
                                            uint32_t bits) {
  const unsigned long long cap = 32ull * rec_words;
  if (!rec || !bits || t_first >= cap) return;
  if (cap - t_first < 32) bits &= (1u << (cap - t_first)) - 1u;
  const unsigned long long w = t_first >> 5;
  const uint32_t sh = static_cast<uint32_t>(t_first & 31);
  if (bits << sh) atomicOr(rec + w, bits << sh);
  if (sh && (bits >> (32 - sh))) atomicOr(rec + w + 1, bits >> (32 - sh));
}

// The spatial signals: per-frame grayscale sums on a grid of cells.
struct FeatArgs {
  uint64_t frame_bytes;
  uint32_t width, height, npix;
  uint32_t grid_h, grid_w;    // cell rows, cell columns
  uint32_t kind;              // 1: low-res (writes the cell sums), 2: dHash (writes 64 bits)
  uint32_t use_magic;         // Y = umulhi(v, magic_y) (host-verified), else v / den
  uint32_t row_h[16], col_w[16];  // pixels per cell row / cell column
};

// An NVTX range over one C-ABI call (a no-op unless a profiler is attached).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// Host-side fault injection for tests: when >= 0, that many further device
// allocations of the library succeed and the next one fails (then the hook
// switches itself off). Set through cofie_ngff_debug_fail_alloc.
extern std::atomic<int> g_fail_alloc;
inline bool injected_alloc_failure() {
  int left = g_fail_alloc.load();
  while (left >= 0 && !g_fail_alloc.compare_exchange_weak(left, left - 1)) {
  }
  return left == 0;
}

// Launchers (stream-ordered; return the launch error).
int hist_blocks_per_sm(int bin_path, uint32_t bins);
uint32_t hist_chunk_groups();
size_t hist_smem_bytes(uint32_t bins);
cudaError_t launch_hist_fast(const SegTable& segs, const HistArgs& a, const LumaConsts& lc, int bin_path,
                             uint32_t* hist, uint32_t* err, int grid, cudaStream_t st, bool pdl = false);
// The generic kernel over CTAs of slice_groups 16-pixel groups (0: the
// default 2048); with pdl a programmatic dependent of the kernel before it.
cudaError_t launch_hist_generic(const SegTable& segs, const HistArgs& a, const LumaConsts& lc, int bin_path,
                                uint32_t* hist, cudaStream_t st, uint32_t slice_groups = 0, bool pdl = false);
// the generic kernel's CTAs per frame (slices of slice_groups groups, 0: the
// default), and its resident CTAs per SM (-1 on error)
uint32_t hist_generic_slices(uint32_t npix, uint32_t slice_groups = 0);
int hist_generic_blocks_per_sm(int bin_path, uint32_t bins);
cudaError_t launch_window(const SegTable& segs, const SelectArgs& a, const uint32_t* hist, const uint32_t* ring,
                          const StreamState* state, uint32_t* l1, uint32_t* mask, cudaStream_t st, bool pdl = false);
cudaError_t launch_scan(const SegTable& segs, const SelectArgs& a, const uint32_t* l1, const uint32_t* mask,
                        uint32_t* hist, uint32_t* ring, StreamState* state, cudaStream_t st, bool pdl = false);
uint32_t select_small_max();
cudaError_t launch_select_small(const SegTable& segs, const SelectArgs& a, uint32_t* hist, uint32_t* ring,
                                StreamState* state, uint32_t* l1, uint32_t* mask, cudaStream_t st, bool pdl = false);
// pushes of at most select_walk_max_frames() frames per stream with L_max <= select_walk_max_lmax()
uint32_t select_walk_max_frames();
uint32_t select_walk_max_lmax();
cudaError_t launch_select_walk(const SegTable& segs, const SelectArgs& a, uint32_t* hist, uint32_t* ring,
                               StreamState* state, cudaStream_t st, bool pdl = false);
cudaError_t launch_features(const SegTable& segs, const FeatArgs& fa, const LumaConsts& lc, uint32_t* feat, uint32_t fw,
                            cudaStream_t st);
int cells_blocks_per_sm();
cudaError_t launch_cells_fast(const SegTable& segs, const HistArgs& a, const LumaConsts& lc, uint32_t* cells,
                              uint32_t* err, int grid, cudaStream_t st, bool pdl = false);
cudaError_t launch_dhash_finish(uint32_t* cells, uint32_t rows, const FeatArgs& fa, uint32_t* bits, cudaStream_t st,
                                bool pdl = false);
cudaError_t launch_wait_probe(uint64_t timeout_ns, uint32_t* err, cudaStream_t st);
cudaError_t launch_lazy_select(const SegTable& segs, const SelectArgs& a, const uint32_t* feat, uint32_t* ring,
                               StreamState* state, cudaStream_t st, bool pdl = false);
cudaError_t launch_debug_bins(const uint8_t* px, uint64_t n_groups, const LumaConsts& lc, int bin_path,
                              uint8_t* bins_out, cudaStream_t st);
cudaError_t scan_prepare(uint32_t mask_words, uint32_t l_max);
cudaError_t launch_gap_map(const Segment& seg, const SelectArgs& a, unsigned long long t0, const uint32_t* mask,
                           uint16_t* map_out, cudaStream_t st);
cudaError_t launch_ring_store(const uint32_t* hist, uint32_t rows, unsigned long long t_first, uint32_t stream,
                              const SelectArgs& a, uint32_t* ring, cudaStream_t st);
cudaError_t launch_candidates(const uint8_t* keep, uint32_t T, uint32_t m_min, uint32_t* idx, uint32_t* m_out,
                              cudaStream_t st);
cudaError_t launch_stream_candidates(const uint32_t* rec, uint32_t rec_words, const StreamState* state,
                                     uint32_t m_min, uint32_t* idx, uint32_t cap, uint32_t* m_out, uint32_t* err,
                                     cudaStream_t st);
cudaError_t launch_stream_reset(StreamState* state, uint32_t* rec, uint32_t rec_words, cudaStream_t st);
cudaError_t launch_gather(const uint8_t* frames, uint32_t n_frames, uint64_t frame_bytes, const uint32_t* idx, uint32_t m,
                          uint8_t* out, uint32_t* err, bool host_src, cudaStream_t st);

}  // namespace cofie
