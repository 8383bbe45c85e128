// C ABI of the NGFF library (declared in include/cofie_ngff.h).
//
// A push of n frames of one stream runs, in stream order:
//   memset(hist) -> K1 histograms -> K2 windowed distances + gap masks ->
//   K3 scan (scores, keep codes, stream state)
// in pieces of at most max_frames_per_push frames. Frames in host memory are
// copied into one of two device staging buffers on an internal copy stream,
// overlapping the copy of piece i+1 with the kernels of piece i. Outputs in
// host memory are written to device scratch and copied back on the caller's
// stream.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstddef>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "cofie_ngff.h"
#include "ngff_common.cuh"

using namespace cofie;

namespace cofie {
bool checked_build() { return COFIE_DEBUG_CHECKS != 0; }
std::atomic<int> g_fail_alloc{-1};
}

namespace {

thread_local std::string g_global_error;

enum MemKind { kNull = 0, kDevice = 1, kHostPinned = 2, kHostPageable = 3 };

constexpr uint64_t kDefaultStageBytes = 256ull << 20;
constexpr uint32_t kSmallSliceGroups = 256;  // the generic kernel's slice for small launches (12 KiB of frame)
constexpr uint32_t kDefaultRecordFrames = 1u << 20;  // frames per stream the retention record covers
constexpr uint64_t kTimeoutNs = 2000000000ull;  // bounded device waits: 2 s
constexpr size_t kMaxTimedEvents = 1u << 16;

struct DeviceGuard {
  int prev = -1;
  bool ok = true;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

}  // namespace

struct cofie_ngff {
  cofie_ngff_params p{};
  int device = 0;
  int num_sms = 0;
  uint64_t frame_bytes = 0;
  uint32_t npix = 0;
  uint32_t mask_words = 0;
  uint32_t fw = 0;       // uint32 feature words per frame: bins, 256 (low-res) or 2 (dHash)
  FeatArgs fa{};         // the spatial signals' grid
  LumaConsts lc{};
  int bin_path = -1;  // kBinFast, kBinTwoStep, or -1 (generic kernel only)
  bool size_fast = false;
  int hist_grid = 0;
  uint64_t generic_wave = 0;  // CTAs of the generic kernel resident at once (0: never chosen over K1)
  int cells_grid = 0;    // the TMA kernel's grid for the spatial signals (0: not usable)
  unsigned long long x_tau = 0, x_cut = 0, x_grad = 0;  // integer forms of the fp32 decisions
  uint32_t m_gpr = 0, m_h = 0, m_gw = 0;  // its multiply-high divisors (16-pixel groups per row, height, grid columns)
  uint32_t* d_cells = nullptr;  // dHash only: [F][72] cell sums, kept zero between pushes
  float two_n = 0.f;
  uint32_t* d_hist = nullptr;
  uint32_t* d_l1 = nullptr;
  uint32_t* d_mask = nullptr;
  uint32_t* d_ring = nullptr;
  StreamState* d_state = nullptr;
  uint32_t* d_record = nullptr;  // [S][rec_words] retention record (bit t: frame t retained)
  uint32_t rec_words = 0;
  float* d_scores = nullptr;
  uint8_t* d_keep = nullptr;
  uint32_t* d_err = nullptr;
  uint32_t* d_count = nullptr;  // candidate count when the caller's m_out is host memory
  uint32_t* d_idx = nullptr;    // candidate indices when the caller's idx_out is host memory (allocated on first use)
  uint64_t dirty_rows = 0;      // histogram rows [0, dirty_rows) may be nonzero
  uint16_t* d_map = nullptr;    // a shard's gap map
  struct {                      // the shard prepared and not yet committed
    bool ready = false;
    uint32_t stream = 0, n_halo = 0, n = 0;
    uint64_t t0 = 0;
  } shard;
  uint8_t* d_stage[2] = {nullptr, nullptr};
  uint64_t stage_bytes = 0;
  uint32_t stage_frames = 0;
  uint32_t stage_next = 0;
  cudaStream_t copy_stream = nullptr;
  cudaEvent_t ev_copied[2] = {nullptr, nullptr};
  cudaEvent_t ev_free[2] = {nullptr, nullptr};
  std::vector<uint64_t> seen;
  std::string err;
  // launch counters and optional event timing of the histogram kernel
  uint64_t n_hist = 0, n_select = 0, n_other = 0, hist_bytes = 0;
  bool time_kernels = false;
  std::vector<cudaEvent_t> ev_pool;  // pairs: [2i] start, [2i+1] end
  size_t ev_used = 0;
  std::vector<cudaEvent_t> ev_sel;  // the same for distance + scan pairs
  size_t ev_sel_used = 0;

  int fail(int code, const std::string& msg) {
    err = msg;
    return code;
  }
  int cuda_fail(cudaError_t e, const char* what) {
    err = std::string(what) + ": " + cudaGetErrorString(e);
    return COFIE_ECUDA;
  }
};

namespace {

MemKind classify(const void* ptr, int* dev_out = nullptr) {
  if (!ptr) return kNull;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, ptr) != cudaSuccess) {
    cudaGetLastError();
    return kHostPageable;
  }
  if (dev_out) *dev_out = a.device;
  switch (a.type) {
    case cudaMemoryTypeDevice:
    case cudaMemoryTypeManaged:
      return kDevice;
    case cudaMemoryTypeHost:
      return kHostPinned;
    default:
      return kHostPageable;
  }
}

// The allocation a pointer was last found in, with its kind: a batched call
// names three pointers per stream but usually few allocations (one frames
// tensor per stream, one scores and one keep tensor for all of them), so
// each descriptor field keeps the range of the last pointer it classified
// and a pointer inside it needs no query.
struct KindRange {
  uintptr_t lo = 0, hi = 0;
  MemKind kind = kNull;
  int dev = -1;
};

PFN_cuPointerGetAttributes_v7000 pointer_attributes_fn() {
  static PFN_cuPointerGetAttributes_v7000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    return cudaGetDriverEntryPointByVersion("cuPointerGetAttributes", &p, 7000, cudaEnableDefault, &q) ==
                       cudaSuccess &&
                   q == cudaDriverEntryPointSuccess
               ? reinterpret_cast<PFN_cuPointerGetAttributes_v7000>(p)
               : nullptr;
  }();
  return fn;
}

// classify() with the range cache: one driver query gives the kind, the
// device and the allocation's address range (a pointer the driver does not
// know, such as pageable host memory, gets null attributes and is not cached).
MemKind classify_in(const void* ptr, int* dev_out, KindRange* last) {
  if (!ptr) return kNull;
  const uintptr_t a = reinterpret_cast<uintptr_t>(ptr);
  if (a >= last->lo && a < last->hi) {
    if (dev_out) *dev_out = last->dev;
    return last->kind;
  }
  const PFN_cuPointerGetAttributes_v7000 fn = pointer_attributes_fn();
  if (!fn) return classify(ptr, dev_out);
  unsigned int type = 0, managed = 0;
  int ordinal = -1;
  CUdeviceptr start = 0;
  size_t size = 0;
  CUpointer_attribute attrs[5] = {CU_POINTER_ATTRIBUTE_MEMORY_TYPE, CU_POINTER_ATTRIBUTE_IS_MANAGED,
                                  CU_POINTER_ATTRIBUTE_DEVICE_ORDINAL, CU_POINTER_ATTRIBUTE_RANGE_START_ADDR,
                                  CU_POINTER_ATTRIBUTE_RANGE_SIZE};
  void* data[5] = {&type, &managed, &ordinal, &start, &size};
  if (fn(5, attrs, data, static_cast<CUdeviceptr>(a)) != CUDA_SUCCESS) return classify(ptr, dev_out);
  const MemKind k = (managed || type == CU_MEMORYTYPE_DEVICE) ? kDevice
                    : type == CU_MEMORYTYPE_HOST              ? kHostPinned
                                                              : kHostPageable;
  if (dev_out) *dev_out = ordinal;
  if (k != kHostPageable && size > 0 && a >= start && a - start < size) {
    last->lo = static_cast<uintptr_t>(start);
    last->hi = static_cast<uintptr_t>(start) + size;
    last->kind = k;
    last->dev = ordinal;
  }
  return k;
}

// m = ceil(2^32 / d) with e = m d - 2^32 gives umulhi(n, m) = floor(n / d)
// for every n with n e < 2^32: n m / 2^32 = n / d + n e / (d 2^32), and the
// fraction of n / d is at most (d - 1) / d. Returns 0 when d < 2 or n_max is
// out of that range.
uint32_t magic_for(uint32_t d, uint64_t n_max) {
  if (d < 2) return 0;
  const uint64_t m = ((1ull << 32) + d - 1) / d;
  const uint64_t e = m * d - (1ull << 32);
  if (m > 0xffffffffull || (e && n_max >= (1ull << 32) / e)) return 0;
  return static_cast<uint32_t>(m);
}

bool verify_magic(uint32_t magic, uint32_t vmax, uint32_t den, uint32_t bins, bool divide_only) {
  for (uint32_t v = 0; v <= vmax; ++v) {
    const uint32_t y = v / den;
    const uint32_t want = divide_only ? y : (y * bins) / 256u;
    const uint32_t got = static_cast<uint32_t>((static_cast<uint64_t>(v) * magic) >> 32);
    if (got != want) return false;
  }
  return true;
}

int validate_params(const cofie_ngff_params* p, std::string& why) {
  if (!p) return why = "params is NULL", COFIE_EINVAL;
  if (p->width == 0 || p->height == 0) return why = "width and height must be >= 1", COFIE_EINVAL;
  const uint64_t npix = static_cast<uint64_t>(p->width) * p->height;
  if (npix > 0x7fffffffull) return why = "width * height must be < 2^31", COFIE_EINVAL;
  if (p->bins < 1 || p->bins > COFIE_NGFF_MAX_BINS) return why = "bins must be in [1, 256]", COFIE_EINVAL;
  if (p->l_max > COFIE_NGFF_MAX_LMAX) return why = "l_max must be in [0, 256]", COFIE_EINVAL;
  if (p->tau != p->tau) return why = "tau is NaN", COFIE_EINVAL;
  if (p->luma_den == 0 || p->luma_den > 65535) return why = "luma_den must be in [1, 65535]", COFIE_EINVAL;
  if (static_cast<uint64_t>(p->luma_w[0]) + p->luma_w[1] + p->luma_w[2] != p->luma_den)
    return why = "luma weights must sum to luma_den", COFIE_EINVAL;
  if (p->max_streams < 1) return why = "max_streams must be >= 1", COFIE_EINVAL;
  if (p->max_frames_per_push < 1) return why = "max_frames_per_push must be >= 1", COFIE_EINVAL;
  if (p->signal > COFIE_SIGNAL_SCD) return why = "signal must be one of COFIE_SIGNAL_*", COFIE_EINVAL;
  if (p->signal == COFIE_SIGNAL_SCD && (p->scd_cut != p->scd_cut || p->scd_gradual != p->scd_gradual))
    return why = "scd_cut or scd_gradual is NaN", COFIE_EINVAL;
  if (p->signal == COFIE_SIGNAL_LOWRES && (p->width < 16 || p->height < 16 || npix > (1ull << 24)))
    return why = "the low-res signal needs width, height >= 16 and width * height <= 2^24", COFIE_EINVAL;
  if (p->signal == COFIE_SIGNAL_DHASH && (p->width < 9 || p->height < 8))
    return why = "the dHash signal needs width >= 9 and height >= 8", COFIE_EINVAL;
  if (p->signal == COFIE_SIGNAL_DHASH &&
      255ull * ((p->height + 7) / 8) * ((p->width + 8) / 9) > 0xffffffffull)  // a cell's grayscale sum in 32 bits
    return why = "the dHash signal's cells are too large for 32-bit sums", COFIE_EINVAL;
  return COFIE_OK;
}

template <typename T>
cudaError_t dalloc(T** p, size_t count) {
  if (injected_alloc_failure()) return cudaErrorMemoryAllocation;
  return cudaMalloc(reinterpret_cast<void**>(p), count * sizeof(T) + 16);
}

// Takes the next event pair from a pool (growing it up to kMaxTimedEvents).
bool take_pair(std::vector<cudaEvent_t>& pool, size_t& used, cudaEvent_t* a, cudaEvent_t* b) {
  if (used + 2 > kMaxTimedEvents) return false;
  while (pool.size() < used + 2) {
    cudaEvent_t ev;
    if (cudaEventCreate(&ev) != cudaSuccess) return false;
    pool.push_back(ev);
  }
  *a = pool[used];
  *b = pool[used + 1];
  used += 2;
  return true;
}

double sum_pairs(const std::vector<cudaEvent_t>& pool, size_t used, cudaError_t* err) {
  double ms = 0.0;
  *err = cudaSuccess;
  for (size_t i = 0; i + 1 < used; i += 2) {
    cudaError_t e = cudaEventSynchronize(pool[i + 1]);
    float t = 0.f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&t, pool[i], pool[i + 1]);
    if (e != cudaSuccess) {
      *err = e;
      return 0.0;
    }
    ms += t;
  }
  return ms;
}

// Whether the first stage over segs runs on the bulk-copy kernel (K1 or its
// cells mode): frames of a multiple of 16 pixels, 16-byte aligned, and a bin
// or grid path the host has verified.
bool first_stage_fast(const cofie_ngff* h, const SegTable& segs) {
  const bool cells = h->p.signal == COFIE_SIGNAL_LOWRES || h->p.signal == COFIE_SIGNAL_DHASH;
  bool fast = cells ? h->cells_grid > 0 : h->size_fast && h->bin_path >= 0;
  for (uint32_t i = 0; i < segs.count && fast; ++i)
    if (reinterpret_cast<uintptr_t>(segs.s[i].frames) % 16 != 0) fast = false;
  return fast;
}

// The first stage over the rows of segs: grayscale histograms (K1), or the
// spatial signal's per-frame features. With pdl the bulk-copy kernels are
// programmatic dependents of the kernel before them (they wait for it before
// reading a frame).
cudaError_t launch_first_stage(cofie_ngff* h, const SegTable& segs, cudaStream_t st, bool pdl = false) {
  const bool cells = h->p.signal == COFIE_SIGNAL_LOWRES || h->p.signal == COFIE_SIGNAL_DHASH;
  const bool fast = first_stage_fast(h, segs);
  HistArgs ha{};
  ha.frame_bytes = h->frame_bytes;
  ha.npix = h->npix;
  ha.groups_per_frame = static_cast<uint32_t>(h->frame_bytes / 48);
  ha.chunks_per_frame = (ha.groups_per_frame + hist_chunk_groups() - 1) / hist_chunk_groups();
  ha.timeout_ns = kTimeoutNs;
  if (cells) {
    if (!fast) return launch_features(segs, h->fa, h->lc, h->d_hist, h->fw, st);
    ha.width = h->p.width;
    ha.height = h->p.height;
    ha.grid_h = h->fa.grid_h;
    ha.grid_w = h->fa.grid_w;
    ha.gpr = h->p.width / 16;
    ha.m_gpr = h->m_gpr;
    ha.m_h = h->m_h;
    ha.m_gw = h->m_gw;
    ha.wide = (h->p.width / h->fa.grid_w >= 16 && h->m_gw) ? 1u : 0u;
    const uint64_t chunks = static_cast<uint64_t>(segs.rows) * ha.chunks_per_frame;
    const int grid = static_cast<int>(chunks < static_cast<uint64_t>(h->cells_grid) ? chunks : h->cells_grid);
    const bool dhash = h->p.signal == COFIE_SIGNAL_DHASH;
    cudaError_t e = launch_cells_fast(segs, ha, h->lc, dhash ? h->d_cells : h->d_hist, h->d_err, grid, st, pdl);
    if (e == cudaSuccess && dhash) e = launch_dhash_finish(h->d_cells, segs.rows, h->fa, h->d_hist, st, true);
    return e;
  }
  // A launch whose generic grid fills the GPU in one wave of resident CTAs
  // (at least two per SM, and at most an eighth of a second wave) runs the
  // generic kernel: its CTAs start as SMs free and need no ring to fill,
  // which K1's persistent CTAs, each with a fixed share of the chunks, pay on
  // launches of that size (a batched call of 32 streams of 640x360: 23.2
  // against 20.8 us). Launches too small for that window with the default
  // slices take slices of kSmallSliceGroups groups if those land in it, as a
  // programmatic dependent of the kernel before them (8-frame 448x448 pushes:
  // 7.27 against 6.56 us per push); a grid near one wave stays an ordinary
  // launch, because CTAs made resident ahead of time keep SMs the previous
  // kernel still holds (the serving call went from 21 to 27 us). Smaller
  // launches keep K1, whose CTAs are scheduled while the kernel before it
  // runs; larger ones too, where the generic grid would end in a larger
  // partial wave (a quarter of a wave already loses 6 %).
  if (fast) {
    const uint64_t lo = 2ull * h->num_sms, hi = h->generic_wave + h->generic_wave / 8;
    const uint64_t gen_ctas = static_cast<uint64_t>(hist_generic_slices(h->npix)) * segs.rows;
    if (gen_ctas >= lo && gen_ctas <= hi) return launch_hist_generic(segs, ha, h->lc, h->bin_path, h->d_hist, st);
    const uint64_t small_ctas = static_cast<uint64_t>(hist_generic_slices(h->npix, kSmallSliceGroups)) * segs.rows;
    if (gen_ctas < lo && small_ctas >= lo && small_ctas <= hi)
      return launch_hist_generic(segs, ha, h->lc, h->bin_path, h->d_hist, st, kSmallSliceGroups, pdl);
  }
  if (fast) {
    const uint64_t chunks = static_cast<uint64_t>(segs.rows) * ha.chunks_per_frame;
    const int grid = static_cast<int>(chunks < static_cast<uint64_t>(h->hist_grid) ? chunks : h->hist_grid);
    return launch_hist_fast(segs, ha, h->lc, h->bin_path, h->d_hist, h->d_err, grid, st, pdl);
  }
  return launch_hist_generic(segs, ha, h->lc, h->bin_path, h->d_hist, st);
}

// The smallest numerator x with fp32(x) / den >= thr, or 2^64 - 1 if none.
// fp32(x) and the correctly rounded division never decrease as x grows, so
// "x >= result" is exactly the fp32 decision; found by bisection with the
// host's IEEE arithmetic (the device's __ull2float_rn and __fdiv_rn round
// the same way).
unsigned long long numerator_threshold(float thr, float den) {
  const auto reaches = [&](unsigned long long x) { return static_cast<float>(x) / den >= thr; };
  if (reaches(0)) return 0;
  unsigned long long lo = 0, hi = ~0ull;  // reaches(lo) false; reaches(hi) decides "never"
  if (!reaches(hi)) return ~0ull;
  while (hi - lo > 1) {
    const unsigned long long mid = lo + (hi - lo) / 2;
    (reaches(mid) ? hi : lo) = mid;
  }
  return hi;
}

// Ring rows per stream: the last L_max feature rows, or for L_max = 0 the
// previous frame's row and the reference frame's row.
uint32_t ring_rows(const cofie_ngff* h) { return h->p.l_max ? h->p.l_max : 2u; }

SelectArgs select_args(const cofie_ngff* h) {
  SelectArgs sa{};
  sa.bins = h->fw;
  sa.l_max = h->p.l_max;
  sa.mask_words = h->mask_words;
  sa.tau = h->p.tau;
  sa.two_n = h->two_n;
  sa.dist_kind = h->p.signal == COFIE_SIGNAL_DHASH ? 1u : 0u;
  sa.scd = h->p.signal == COFIE_SIGNAL_SCD ? 1u : 0u;
  sa.scd_cut = h->p.scd_cut;
  sa.scd_grad = h->p.scd_gradual;
  sa.x_tau = h->x_tau;
  sa.x_cut = h->x_cut;
  sa.x_grad = h->x_grad;
  sa.record = h->d_record;
  sa.rec_words = h->rec_words;
  return sa;
}

// Zeroes histogram rows [0, rows) (dHash rows are written whole and need it not).
cudaError_t clear_rows(cofie_ngff* h, uint64_t rows, cudaStream_t st) {
  if (rows == 0 || h->p.signal == COFIE_SIGNAL_DHASH) return cudaSuccess;
  return cudaMemsetAsync(h->d_hist, 0, static_cast<size_t>(rows) * h->fw * 4, st);
}

// Runs K1-K3 over the rows described by segs (device frames). Histogram rows
// are zero between calls, so that a push enqueues the same work whatever came
// before it (which is what lets a push be captured into a CUDA graph and
// replayed): the fused small-push kernel clears its rows after use, and
// otherwise one memset after the selection does, or, with keep_hist, the
// caller after copying them out. Rows that an earlier call left nonzero (a
// prepared shard, a push that failed part way) are cleared first.
// While `capturing`, nothing here runs until the graph is launched, so the
// host's record of dirty rows is left as it was and no timing events are taken.
int run_segments(cofie_ngff* h, const SegTable& segs, cudaStream_t st, bool keep_hist, bool capturing) {
  if (segs.rows == 0) return COFIE_OK;
  cudaError_t e = clear_rows(h, h->dirty_rows, st);
  if (e != cudaSuccess) return h->cuda_fail(e, "memset histograms");
  if (!capturing) h->dirty_rows = h->p.max_frames_per_push;  // until the clean-up is enqueued
  cudaEvent_t ev0 = nullptr, ev1 = nullptr;
  const bool timed = h->time_kernels && !capturing;
  if (timed && take_pair(h->ev_pool, h->ev_used, &ev0, &ev1)) cudaEventRecord(ev0, st);
  e = launch_first_stage(h, segs, st, !ev0);
  if (e != cudaSuccess) return h->cuda_fail(e, "histogram kernel launch");
  if (ev1) cudaEventRecord(ev1, st);
  h->n_hist += 1;
  h->hist_bytes += static_cast<uint64_t>(segs.rows) * (h->frame_bytes + 4ull * h->fw);
  SelectArgs sa = select_args(h);
  uint32_t longest = 0;
  for (uint32_t i = 0; i < segs.count; ++i) longest = segs.s[i].n > longest ? segs.s[i].n : longest;
  // small pushes clear their rows inside the selection kernel (saving a
  // launch); large ones with one device-wide memset after the selection
  const bool walk = h->p.l_max > 0 && h->p.l_max <= select_walk_max_lmax() && longest <= select_walk_max_frames();
  const bool fused = longest <= select_small_max();
  sa.zero_hist = ((walk || fused) && !keep_hist && h->p.l_max > 0) ? 1u : 0u;
  cudaEvent_t es0 = nullptr, es1 = nullptr;
  if (timed && take_pair(h->ev_sel, h->ev_sel_used, &es0, &es1)) cudaEventRecord(es0, st);
  if (h->p.l_max == 0) {  // no forced retention: the rule walked in frame order
    e = launch_lazy_select(segs, sa, h->d_hist, h->d_ring, h->d_state, st, !ev0);
    if (e != cudaSuccess) return h->cuda_fail(e, "lazy selection kernel launch");
    h->n_select += 1;
  } else if (walk) {  // distances and the rule walked in frame order, in one small launch per stream
    e = launch_select_walk(segs, sa, h->d_hist, h->d_ring, h->d_state, st, !ev0);
    if (e != cudaSuccess) return h->cuda_fail(e, "selection kernel launch");
    h->n_select += 1;
  } else if (fused) {  // distances and scan in one launch
    e = launch_select_small(segs, sa, h->d_hist, h->d_ring, h->d_state, h->d_l1, h->d_mask, st, !ev0);
    if (e != cudaSuccess) return h->cuda_fail(e, "selection kernel launch");
    h->n_select += 1;
  } else {
    e = launch_window(segs, sa, h->d_hist, h->d_ring, h->d_state, h->d_l1, h->d_mask, st, !ev0);
    if (e != cudaSuccess) return h->cuda_fail(e, "window kernel launch");
    e = launch_scan(segs, sa, h->d_l1, h->d_mask, h->d_hist, h->d_ring, h->d_state, st, !es0);
    if (e != cudaSuccess) return h->cuda_fail(e, "scan kernel launch");
    h->n_select += 2;
  }
  if (es1) cudaEventRecord(es1, st);
  if (keep_hist) {  // the caller clears the rows once it has copied them
    if (!capturing) h->dirty_rows = segs.rows;
    return COFIE_OK;
  }
  if (!sa.zero_hist) {
    e = clear_rows(h, segs.rows, st);
    if (e != cudaSuccess) return h->cuda_fail(e, "memset histograms");
  }
  if (!capturing) h->dirty_rows = 0;
  return COFIE_OK;
}

// One piece of a single-stream push: n <= max_frames_per_push device frames.
int run_piece(cofie_ngff* h, uint32_t stream, const uint8_t* dframes, uint32_t n, float* scores, MemKind ks,
              uint8_t* keep, MemKind kk, uint32_t* hist_out, MemKind kh, cudaStream_t st, bool capturing) {
  SegTable segs;
  memset(&segs, 0, sizeof segs);
  segs.count = 1;
  segs.rows = n;
  Segment& s = segs.s[0];
  s.frames = dframes;
  s.n = n;
  s.row0 = 0;
  s.stream = stream;
  s.scores = ks == kDevice ? scores : (ks == kNull ? nullptr : h->d_scores);
  s.keep = kk == kDevice ? keep : (kk == kNull ? nullptr : h->d_keep);
  int rc = run_segments(h, segs, st, kh != kNull, capturing);
  if (rc != COFIE_OK) return rc;
  cudaError_t e = cudaSuccess;
  if (ks == kHostPinned || ks == kHostPageable)
    e = cudaMemcpyAsync(scores, h->d_scores, n * sizeof(float), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess && (kk == kHostPinned || kk == kHostPageable))
    e = cudaMemcpyAsync(keep, h->d_keep, n, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess && kh != kNull)
    e = cudaMemcpyAsync(hist_out, h->d_hist, static_cast<size_t>(n) * h->fw * 4, cudaMemcpyDefault, st);
  if (e == cudaSuccess && kh != kNull) e = clear_rows(h, n, st);
  if (e != cudaSuccess) return h->cuda_fail(e, "output copy");
  if (kh != kNull && !capturing) h->dirty_rows = 0;
  return COFIE_OK;
}

// 1 while st is capturing into a CUDA graph, 0 when it is not, -1 when the
// state cannot be read or the capture has been invalidated.
int capture_state(cudaStream_t st) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) {
    cudaGetLastError();
    return -1;
  }
  return cs == cudaStreamCaptureStatusActive ? 1 : (cs == cudaStreamCaptureStatusNone ? 0 : -1);
}

int ensure_staging(cofie_ngff* h) {
  if (h->d_stage[0]) return COFIE_OK;
  for (int i = 0; i < 2; ++i) {
    cudaError_t e = injected_alloc_failure() ? cudaErrorMemoryAllocation
                                             : cudaMalloc(reinterpret_cast<void**>(&h->d_stage[i]), h->stage_bytes);
    if (e != cudaSuccess) {
      cudaGetLastError();
      for (int j = 0; j < 2; ++j) {
        if (h->d_stage[j]) cudaFree(h->d_stage[j]);
        h->d_stage[j] = nullptr;
      }
      return h->fail(COFIE_ENOMEM, "staging buffer allocation failed");
    }
  }
  return COFIE_OK;
}

int push_impl(cofie_ngff* h, uint32_t stream, const uint8_t* frames, uint32_t n, float* scores, uint8_t* keep,
              uint32_t* hist_out, void* cuda_stream) {
  NvtxRange nvtx("ngff.push");
  if (!h) return COFIE_EINVAL;
  if (stream >= h->p.max_streams) return h->fail(COFIE_EINVAL, "stream index out of range");
  if (n == 0) return COFIE_OK;
  if (!frames) return h->fail(COFIE_EINVAL, "frames is NULL");
  DeviceGuard guard(h->device);
  if (!guard.ok) return h->fail(COFIE_ECUDA, "cannot select the handle's device");
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  int fdev = -1;
  const MemKind kf = classify(frames, &fdev);
  const MemKind ks = classify(scores), kk = classify(keep), kh = classify(hist_out);
  if (kf == kDevice && fdev != h->device) return h->fail(COFIE_EINVAL, "frames live on another device");
  const int cap = capture_state(st);
  if (cap < 0) return h->fail(COFIE_ECUDA, "cannot read the CUDA stream's capture state");
  const auto dev_or_null = [](MemKind k) { return k == kDevice || k == kNull; };
  if (cap && !(kf == kDevice && dev_or_null(ks) && dev_or_null(kk) && dev_or_null(kh)))
    return h->fail(COFIE_EINVAL, "a push captured into a CUDA graph takes device frames and outputs only");
  h->shard.ready = false;  // a push between shard_prepare and shard_commit reuses the shard's rows
  const uint32_t B = h->fw;
  if (kf == kDevice) {
    const uint32_t step = h->p.max_frames_per_push;
    for (uint32_t off = 0; off < n; off += step) {
      const uint32_t m = n - off < step ? n - off : step;
      int rc = run_piece(h, stream, frames + off * h->frame_bytes, m, scores ? scores + off : nullptr, ks,
                         keep ? keep + off : nullptr, kk, hist_out ? hist_out + static_cast<size_t>(off) * B : nullptr,
                         kh, st, cap == 1);
      if (rc != COFIE_OK) return rc;
    }
  } else {
    int rc = ensure_staging(h);
    if (rc != COFIE_OK) return rc;
    const uint32_t step = h->stage_frames < h->p.max_frames_per_push ? h->stage_frames : h->p.max_frames_per_push;
    for (uint32_t off = 0; off < n; off += step) {
      const uint32_t m = n - off < step ? n - off : step;
      const uint32_t slot = h->stage_next;
      h->stage_next ^= 1u;
      cudaError_t e = cudaStreamWaitEvent(h->copy_stream, h->ev_free[slot], 0);
      if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->d_stage[slot], frames + off * h->frame_bytes, m * h->frame_bytes,
                            cudaMemcpyHostToDevice, h->copy_stream);
      if (e == cudaSuccess) e = cudaEventRecord(h->ev_copied[slot], h->copy_stream);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(st, h->ev_copied[slot], 0);
      if (e != cudaSuccess) return h->cuda_fail(e, "host frame staging");
      rc = run_piece(h, stream, h->d_stage[slot], m, scores ? scores + off : nullptr, ks, keep ? keep + off : nullptr,
                     kk, hist_out ? hist_out + static_cast<size_t>(off) * B : nullptr, kh, st, false);
      // the slot is free again only behind whatever of this piece was enqueued, failed or not
      e = cudaEventRecord(h->ev_free[slot], st);
      if (rc != COFIE_OK) return rc;
      if (e != cudaSuccess) return h->cuda_fail(e, "staging event");
    }
  }
  if (!cap) h->seen[stream] += n;
  h->err.clear();
  return COFIE_OK;
}

void free_handle(cofie_ngff* h) {
  if (!h) return;
  DeviceGuard guard(h->device);
  cudaDeviceSynchronize();
  void* bufs[] = {h->d_hist,     h->d_l1,       h->d_mask,  h->d_ring, h->d_state, h->d_scores, h->d_keep,
                  h->d_err,      h->d_stage[0], h->d_stage[1], h->d_count, h->d_map, h->d_cells, h->d_record, h->d_idx};
  for (void* b : bufs)
    if (b) cudaFree(b);
  for (cudaEvent_t ev : h->ev_pool) cudaEventDestroy(ev);
  for (cudaEvent_t ev : h->ev_sel) cudaEventDestroy(ev);
  for (int i = 0; i < 2; ++i) {
    if (h->ev_copied[i]) cudaEventDestroy(h->ev_copied[i]);
    if (h->ev_free[i]) cudaEventDestroy(h->ev_free[i]);
  }
  if (h->copy_stream) cudaStreamDestroy(h->copy_stream);
  delete h;
}

}  // namespace

extern "C" {

uint32_t cofie_ngff_feature_words(const cofie_ngff_t* h) { return h ? h->fw : 0; }

void cofie_ngff_default_params(cofie_ngff_params* p, uint32_t width, uint32_t height) {
  if (!p) return;
  memset(p, 0, sizeof *p);
  p->width = width;
  p->height = height;
  p->bins = 32;     // App. A
  p->l_max = 30;    // App. B.2
  p->m_min = 4;     // App. B.2
  p->tau = 0.30f;   // App. B.2
  p->luma_w[0] = 299;
  p->luma_w[1] = 587;
  p->luma_w[2] = 114;
  p->luma_den = 1000;
  p->max_streams = 1;
  p->max_frames_per_push = 4096;
  p->device = -1;
  p->host_stage_bytes = 0;
  p->signal = COFIE_SIGNAL_HISTOGRAM;
  p->scd_cut = 0.30f;     // twin-comparison thresholds of the scene-change signal
  p->scd_gradual = 0.10f;
  p->max_stream_frames = kDefaultRecordFrames;
}

int cofie_ngff_create(const cofie_ngff_params* p, cofie_ngff_t** out) {
  std::string why;
  if (!out) {
    g_global_error = "out is NULL";
    return COFIE_EINVAL;
  }
  int rc = validate_params(p, why);
  if (rc != COFIE_OK) {
    g_global_error = why;
    return rc;
  }
  int dev = p->device;
  if (dev < 0 && cudaGetDevice(&dev) != cudaSuccess) {
    g_global_error = "no CUDA device";
    return COFIE_ECUDA;
  }
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || dev >= ndev) {
    cudaGetLastError();
    g_global_error = "device ordinal out of range";
    return COFIE_EINVAL;
  }
  DeviceGuard guard(dev);
  if (!guard.ok) {
    g_global_error = "cannot select the device";
    return COFIE_ECUDA;
  }
  cofie_ngff* h = new (std::nothrow) cofie_ngff();
  if (!h) {
    g_global_error = "host allocation failed";
    return COFIE_ENOMEM;
  }
  h->p = *p;
  h->device = dev;
  h->p.device = dev;
  cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, dev);
  h->npix = p->width * p->height;
  h->frame_bytes = 3ull * h->npix;
  h->mask_words = (p->l_max + 31) / 32;
  if (p->signal == COFIE_SIGNAL_LOWRES) {
    h->fw = 256;
    h->two_n = static_cast<float>(255ull * h->npix);
  } else if (p->signal == COFIE_SIGNAL_DHASH) {
    h->fw = 2;
    h->two_n = 64.0f;
  } else {
    h->fw = p->bins;
    h->two_n = static_cast<float>(2ull * h->npix);
  }
  h->x_tau = numerator_threshold(p->tau, h->two_n);
  h->x_cut = numerator_threshold(p->scd_cut, h->two_n);
  h->x_grad = numerator_threshold(p->scd_gradual, h->two_n);
  if (p->signal == COFIE_SIGNAL_LOWRES || p->signal == COFIE_SIGNAL_DHASH) {
    FeatArgs& fa = h->fa;
    fa.frame_bytes = 3ull * h->npix;
    fa.width = p->width;
    fa.height = p->height;
    fa.npix = h->npix;
    fa.grid_h = p->signal == COFIE_SIGNAL_LOWRES ? 16 : 8;
    fa.grid_w = p->signal == COFIE_SIGNAL_LOWRES ? 16 : 9;
    fa.kind = p->signal;
    for (uint32_t y = 0; y < p->height; ++y) fa.row_h[y * fa.grid_h / p->height] += 1;
    for (uint32_t x = 0; x < p->width; ++x) fa.col_w[x * fa.grid_w / p->width] += 1;
  }
  h->size_fast = (h->npix % 16) == 0;
  h->seen.assign(p->max_streams, 0);
  const uint32_t rec_frames = p->max_stream_frames ? p->max_stream_frames : kDefaultRecordFrames;
  h->rec_words = static_cast<uint32_t>((static_cast<uint64_t>(rec_frames) + 31) / 32);
  // the record holds whole words: it covers rec_frames rounded up to a multiple of 32
  h->p.max_stream_frames = static_cast<uint32_t>(std::min<uint64_t>(32ull * h->rec_words, 0xffffffffull));

  LumaConsts& lc = h->lc;
  const uint32_t wr = p->luma_w[0], wg = p->luma_w[1], wb = p->luma_w[2], den = p->luma_den;
  lc.w_rg = (wg << 16) | wr;
  lc.w_b0 = wb;
  lc.w_0r = wr << 16;
  lc.w_gb = (wb << 16) | wg;
  lc.half = den / 2;
  lc.bins = p->bins;
  lc.w[0] = wr;
  lc.w[1] = wg;
  lc.w[2] = wb;
  lc.den = den;
  const uint32_t vmax = 255u * den + den / 2;
  h->bin_path = -1;
  if (256 % p->bins == 0) {
    const uint64_t D = static_cast<uint64_t>(den) * (256 / p->bins);
    const uint64_t M = ((1ull << 32) + D - 1) / D;
    if (D >= 2 && M <= 0xffffffffull && verify_magic(static_cast<uint32_t>(M), vmax, den, p->bins, false)) {
      lc.magic = static_cast<uint32_t>(M);
      h->bin_path = kBinFast;
    }
  }
  bool magic_y_ok = false;
  if (den >= 2) {
    const uint64_t M = ((1ull << 32) + den - 1) / den;
    if (M <= 0xffffffffull && verify_magic(static_cast<uint32_t>(M), vmax, den, p->bins, true)) {
      lc.magic_y = static_cast<uint32_t>(M);
      magic_y_ok = true;
    }
  }
  if (h->bin_path < 0 && magic_y_ok) h->bin_path = kBinTwoStep;
  h->fa.use_magic = magic_y_ok ? 1u : 0u;

  const uint64_t F = p->max_frames_per_push, S = p->max_streams;
  cudaError_t e = cudaSuccess;
  if (e == cudaSuccess) e = dalloc(&h->d_hist, F * h->fw);
  if (e == cudaSuccess) e = dalloc(&h->d_l1, F * p->l_max);
  if (e == cudaSuccess) e = dalloc(&h->d_mask, F * h->mask_words);
  if (e == cudaSuccess) e = dalloc(&h->d_ring, S * ring_rows(h) * h->fw);
  if (e == cudaSuccess) e = dalloc(&h->d_state, S);
  if (e == cudaSuccess) e = dalloc(&h->d_scores, F);
  if (e == cudaSuccess) e = dalloc(&h->d_keep, F);
  if (e == cudaSuccess) e = dalloc(&h->d_err, 1);
  if (e == cudaSuccess) e = dalloc(&h->d_count, 1);
  if (e == cudaSuccess) e = dalloc(&h->d_map, COFIE_NGFF_MAX_LMAX);
  if (e == cudaSuccess) e = dalloc(&h->d_record, S * h->rec_words);
  if (e == cudaSuccess && p->signal == COFIE_SIGNAL_DHASH) {
    e = dalloc(&h->d_cells, F * 72);
    if (e == cudaSuccess) e = cudaMemset(h->d_cells, 0, F * 72 * sizeof(uint32_t));
  }
  if (e != cudaSuccess) {
    cudaGetLastError();
    free_handle(h);
    g_global_error = "device allocation failed";
    return COFIE_ENOMEM;
  }
  if (e == cudaSuccess) e = cudaMemset(h->d_state, 0, S * sizeof(StreamState));
  if (e == cudaSuccess) e = cudaMemset(h->d_record, 0, S * h->rec_words * sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMemset(h->d_hist, 0, F * h->fw * sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMemset(h->d_err, 0, sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&h->copy_stream, cudaStreamNonBlocking);
  for (int i = 0; i < 2 && e == cudaSuccess; ++i) {
    e = cudaEventCreateWithFlags(&h->ev_copied[i], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&h->ev_free[i], cudaEventDisableTiming);
  }
  if (e == cudaSuccess && p->l_max > 0) e = scan_prepare(h->mask_words, p->l_max);
  if (e == cudaSuccess && h->bin_path >= 0) {
    const int per_sm = hist_blocks_per_sm(h->bin_path, p->bins);
    if (per_sm <= 0) e = cudaGetLastError() != cudaSuccess ? cudaErrorInvalidConfiguration : cudaErrorInvalidValue;
    h->hist_grid = h->num_sms * (per_sm > 0 ? per_sm : 1);
    const int gen_per_sm = hist_generic_blocks_per_sm(h->bin_path, p->bins);
    if (gen_per_sm < 0) cudaGetLastError();
    h->generic_wave = gen_per_sm > 0 ? static_cast<uint64_t>(h->num_sms) * gen_per_sm : 0;
  }
  if (p->signal == COFIE_SIGNAL_LOWRES || p->signal == COFIE_SIGNAL_DHASH) {
    const uint32_t gpr = p->width / 16, gw = h->fa.grid_w, gh = h->fa.grid_h;
    const uint64_t groups = h->npix / 16;
    const uint64_t n_gpr = std::max<uint64_t>(groups, static_cast<uint64_t>(gpr) * gw);
    h->m_gpr = magic_for(gpr, n_gpr);
    h->m_h = magic_for(p->height, static_cast<uint64_t>(p->height) * gh);
    h->m_gw = magic_for(gw, static_cast<uint64_t>(p->width) * gw + gw);
  }
  if (e == cudaSuccess && (p->signal == COFIE_SIGNAL_LOWRES || p->signal == COFIE_SIGNAL_DHASH) &&
      p->width % 16 == 0 && h->fa.use_magic &&
      h->m_gpr && h->m_h && static_cast<uint64_t>(p->width) * h->fa.grid_w < (1ull << 32)) {
    const int per_sm = cells_blocks_per_sm();
    if (per_sm <= 0) e = cudaGetLastError() != cudaSuccess ? cudaErrorInvalidConfiguration : cudaErrorInvalidValue;
    h->cells_grid = h->num_sms * (per_sm > 0 ? per_sm : 1);
  }
  if (e != cudaSuccess) {
    g_global_error = std::string("CUDA setup failed: ") + cudaGetErrorString(e);
    cudaGetLastError();
    free_handle(h);
    return COFIE_ECUDA;
  }
  uint64_t sb = p->host_stage_bytes ? p->host_stage_bytes : kDefaultStageBytes;
  if (sb < h->frame_bytes) sb = h->frame_bytes;
  h->stage_frames = static_cast<uint32_t>(sb / h->frame_bytes);
  h->stage_bytes = static_cast<uint64_t>(h->stage_frames) * h->frame_bytes;
  *out = h;
  return COFIE_OK;
}

void cofie_ngff_destroy(cofie_ngff_t* h) { free_handle(h); }

int cofie_ngff_push(cofie_ngff_t* h, uint32_t stream, const uint8_t* frames, uint32_t n, float* scores_out,
                    uint8_t* keep_out, void* cuda_stream) {
  return push_impl(h, stream, frames, n, scores_out, keep_out, nullptr, cuda_stream);
}

int cofie_ngff_push_ex(cofie_ngff_t* h, uint32_t stream, const uint8_t* frames, uint32_t n, float* scores_out,
                       uint8_t* keep_out, uint32_t* hist_out, void* cuda_stream) {
  return push_impl(h, stream, frames, n, scores_out, keep_out, hist_out, cuda_stream);
}

int cofie_ngff_push_batch(cofie_ngff_t* h, const cofie_ngff_push_desc* desc, uint32_t nd, void* cuda_stream) {
  NvtxRange nvtx("ngff.push_batch");
  if (!h) return COFIE_EINVAL;
  if (nd == 0) return COFIE_OK;
  if (!desc) return h->fail(COFIE_EINVAL, "desc is NULL");
  if (nd > COFIE_NGFF_MAX_BATCH) return h->fail(COFIE_EINVAL, "more than COFIE_NGFF_MAX_BATCH descriptors");
  DeviceGuard guard(h->device);
  if (!guard.ok) return h->fail(COFIE_ECUDA, "cannot select the handle's device");
  SegTable segs;
  memset(&segs, 0, sizeof segs);
  uint64_t rows = 0, staged_bytes = 0;
  bool host_frames = false, host_out = false;
  MemKind kf[COFIE_NGFF_MAX_BATCH], ks[COFIE_NGFF_MAX_BATCH], kk[COFIE_NGFF_MAX_BATCH];
  KindRange rf, rs, rk;  // the allocations the last frames, scores and keep pointers were found in
  uint64_t stage_off[COFIE_NGFF_MAX_BATCH];
  for (uint32_t i = 0; i < nd; ++i) {
    const cofie_ngff_push_desc& d = desc[i];
    if (d.stream >= h->p.max_streams) return h->fail(COFIE_EINVAL, "stream index out of range");
    for (uint32_t j = 0; j < i; ++j)  // at most 64 descriptors: no table the size of max_streams
      if (desc[j].stream == d.stream) return h->fail(COFIE_EINVAL, "a stream appears twice in one batch");
    kf[i] = ks[i] = kk[i] = kNull;
    stage_off[i] = 0;
    if (d.n > 0) {
      int fdev = -1;
      kf[i] = d.frames ? classify_in(d.frames, &fdev, &rf) : kNull;
      if (kf[i] == kNull || (kf[i] == kDevice && fdev != h->device))
        return h->fail(COFIE_EINVAL, "batched frames must be device memory on the handle's device, or host memory");
      int sdev = -1, kdev = -1;
      ks[i] = classify_in(d.scores_out, &sdev, &rs);
      kk[i] = classify_in(d.keep_out, &kdev, &rk);
      if ((ks[i] == kDevice && sdev != h->device) || (kk[i] == kDevice && kdev != h->device))
        return h->fail(COFIE_EINVAL, "batched outputs live on another device");
      if (kf[i] != kDevice) {  // staged back to back, each descriptor's frames from a 16-byte boundary
        host_frames = true;
        stage_off[i] = staged_bytes;
        staged_bytes += (static_cast<uint64_t>(d.n) * h->frame_bytes + 15) & ~uint64_t(15);
      }
      host_out = host_out || (ks[i] != kDevice && ks[i] != kNull) || (kk[i] != kDevice && kk[i] != kNull);
    }
    rows += d.n;
  }
  if (rows > h->p.max_frames_per_push) return h->fail(COFIE_EINVAL, "batch exceeds max_frames_per_push frames");
  const cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const int cap = capture_state(st);
  if (cap < 0) return h->fail(COFIE_ECUDA, "cannot read the CUDA stream's capture state");
  if (cap && (host_frames || host_out))
    return h->fail(COFIE_EINVAL, "a batch captured into a CUDA graph takes device frames and outputs only");
  uint32_t slot = 0;
  if (host_frames) {
    int rc = ensure_staging(h);
    if (rc != COFIE_OK) return rc;
    if (staged_bytes > h->stage_bytes)
      return h->fail(COFIE_EINVAL, "the batch's host frames exceed one staging buffer (host_stage_bytes)");
    // one copy per host descriptor on the copy stream, into the staging slot
    // the kernels of the call before the last have finished reading
    slot = h->stage_next;
    h->stage_next ^= 1u;
    cudaError_t e = cudaStreamWaitEvent(h->copy_stream, h->ev_free[slot], 0);
    for (uint32_t i = 0; i < nd && e == cudaSuccess; ++i)
      if (desc[i].n > 0 && kf[i] != kDevice)
        e = cudaMemcpyAsync(h->d_stage[slot] + stage_off[i], desc[i].frames,
                            static_cast<uint64_t>(desc[i].n) * h->frame_bytes, cudaMemcpyHostToDevice, h->copy_stream);
    if (e == cudaSuccess) e = cudaEventRecord(h->ev_copied[slot], h->copy_stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(st, h->ev_copied[slot], 0);
    if (e != cudaSuccess) return h->cuda_fail(e, "host frame staging");
  }
  rows = 0;
  for (uint32_t i = 0; i < nd; ++i) {
    const cofie_ngff_push_desc& d = desc[i];
    Segment& s = segs.s[segs.count++];
    s.frames = (d.n > 0 && kf[i] != kDevice) ? h->d_stage[slot] + stage_off[i] : d.frames;
    s.n = d.n;
    s.row0 = static_cast<uint32_t>(rows);
    s.stream = d.stream;
    // host outputs are written to the row's place in the device scratch and copied back below
    s.scores = ks[i] == kDevice ? d.scores_out : (ks[i] == kNull ? nullptr : h->d_scores + rows);
    s.keep = kk[i] == kDevice ? d.keep_out : (kk[i] == kNull ? nullptr : h->d_keep + rows);
    rows += d.n;
  }
  segs.rows = static_cast<uint32_t>(rows);
  h->shard.ready = false;
  int rc = run_segments(h, segs, st, false, cap == 1);
  if (rc != COFIE_OK) {
    if (host_frames) cudaEventRecord(h->ev_free[slot], st);  // behind whatever of the call was enqueued
    return rc;
  }
  cudaError_t e = cudaSuccess;
  for (uint32_t i = 0; i < nd && e == cudaSuccess; ++i) {
    const Segment& s = segs.s[i];
    if (desc[i].n == 0) continue;
    if (ks[i] == kHostPinned || ks[i] == kHostPageable)
      e = cudaMemcpyAsync(desc[i].scores_out, s.scores, desc[i].n * sizeof(float), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess && (kk[i] == kHostPinned || kk[i] == kHostPageable))
      e = cudaMemcpyAsync(desc[i].keep_out, s.keep, desc[i].n, cudaMemcpyDeviceToHost, st);
  }
  if (e == cudaSuccess && host_frames) e = cudaEventRecord(h->ev_free[slot], st);
  if (e != cudaSuccess) return h->cuda_fail(e, "batched output copy");
  if (!cap)
    for (uint32_t i = 0; i < nd; ++i) h->seen[desc[i].stream] += desc[i].n;
  h->err.clear();
  return COFIE_OK;
}

namespace {

constexpr uint32_t kStateMagic = 0x5346474Eu;  // "NGFS" little-endian
constexpr uint32_t kStateVersion = 3;
constexpr size_t kStateHeader = 64;

struct StateHeader {  // the first 64 bytes of a saved state
  uint32_t magic, version, width, height, bins, l_max;
  uint32_t pad0, pad1;
  StreamState st;  // frames seen, current gap, open scene-change run (24 bytes)
  uint32_t rec_words;  // words of the retention record that follows the ring
  uint32_t reserved;
};
static_assert(sizeof(StateHeader) == kStateHeader, "state header layout");

}  // namespace

size_t cofie_ngff_state_bytes(const cofie_ngff_t* h) {
  return h ? kStateHeader + (static_cast<size_t>(ring_rows(h)) * h->fw + h->rec_words) * sizeof(uint32_t) : 0;
}

int cofie_ngff_state_save(cofie_ngff_t* h, uint32_t stream, void* buf, void* cuda_stream) {
  NvtxRange nvtx("ngff.state_save");
  if (!h) return COFIE_EINVAL;
  if (stream >= h->p.max_streams) return h->fail(COFIE_EINVAL, "stream index out of range");
  if (!buf) return h->fail(COFIE_EINVAL, "buf is NULL");
  DeviceGuard guard(h->device);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const MemKind kb = classify(buf);
  StateHeader hdr{};
  hdr.magic = kStateMagic;
  hdr.version = kStateVersion;
  hdr.width = h->p.width;
  hdr.height = h->p.height;
  hdr.bins = h->p.bins;
  hdr.l_max = h->p.l_max;
  hdr.pad0 = h->p.signal;
  hdr.rec_words = h->rec_words;
  uint8_t* b = static_cast<uint8_t*>(buf);
  const size_t ring_bytes = static_cast<size_t>(ring_rows(h)) * h->fw * sizeof(uint32_t);
  const uint32_t* ring = h->d_ring + static_cast<size_t>(stream) * ring_rows(h) * h->fw;
  cudaError_t e;
  if (kb == kDevice) {
    // the header's fixed part travels through the handle's pinned-free path: a
    // synchronous copy of 32 host bytes, then the device-resident parts
    e = cudaMemcpyAsync(b, &hdr, offsetof(StateHeader, st), cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(b + offsetof(StateHeader, rec_words), &hdr.rec_words, 8, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  } else {
    memcpy(b, &hdr, kStateHeader);
    e = cudaSuccess;
  }
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(b + offsetof(StateHeader, st), h->d_state + stream, sizeof(StreamState), cudaMemcpyDefault, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(b + kStateHeader, ring, ring_bytes, cudaMemcpyDefault, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(b + kStateHeader + ring_bytes, h->d_record + static_cast<size_t>(stream) * h->rec_words,
                        h->rec_words * sizeof(uint32_t), cudaMemcpyDefault, st);
  if (e == cudaSuccess && kb != kDevice) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return h->cuda_fail(e, "state save");
  return COFIE_OK;
}

int cofie_ngff_state_load(cofie_ngff_t* h, uint32_t stream, const void* buf, void* cuda_stream) {
  NvtxRange nvtx("ngff.state_load");
  if (!h) return COFIE_EINVAL;
  if (stream >= h->p.max_streams) return h->fail(COFIE_EINVAL, "stream index out of range");
  if (!buf) return h->fail(COFIE_EINVAL, "buf is NULL");
  DeviceGuard guard(h->device);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  StateHeader hdr{};
  cudaError_t e = cudaMemcpyAsync(&hdr, buf, kStateHeader, cudaMemcpyDefault, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return h->cuda_fail(e, "state load");
  if (hdr.magic != kStateMagic || hdr.version != kStateVersion)
    return h->fail(COFIE_EINVAL, "not a saved stream state (format tag or version)");
  if (hdr.width != h->p.width || hdr.height != h->p.height || hdr.bins != h->p.bins || hdr.l_max != h->p.l_max ||
      hdr.pad0 != h->p.signal)
    return h->fail(COFIE_EINVAL, "saved state has another width, height, bins, l_max or signal");
  if (hdr.rec_words != h->rec_words)
    return h->fail(COFIE_EINVAL, "saved state has another retention record size (max_stream_frames)");
  if (hdr.st.t > 0 && h->p.l_max > 0 && (hdr.st.g < 1 || hdr.st.g > h->p.l_max))
    return h->fail(COFIE_EINVAL, "saved state has a gap outside [1, l_max]");
  const uint8_t* b = static_cast<const uint8_t*>(buf);
  const size_t ring_bytes = static_cast<size_t>(ring_rows(h)) * h->fw * sizeof(uint32_t);
  uint32_t* ring = h->d_ring + static_cast<size_t>(stream) * ring_rows(h) * h->fw;
  e = cudaMemcpyAsync(ring, b + kStateHeader, ring_bytes, cudaMemcpyDefault, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(h->d_record + static_cast<size_t>(stream) * h->rec_words, b + kStateHeader + ring_bytes,
                        h->rec_words * sizeof(uint32_t), cudaMemcpyDefault, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(h->d_state + stream, b + offsetof(StateHeader, st), sizeof(StreamState), cudaMemcpyDefault, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);  // buf may be released when this returns
  if (e != cudaSuccess) return h->cuda_fail(e, "state load");
  h->seen[stream] = hdr.st.t;
  return COFIE_OK;
}

int cofie_ngff_shard_prepare(cofie_ngff_t* h, uint32_t stream, const uint8_t* frames, uint32_t n_halo, uint32_t n,
                             uint64_t t0, uint16_t* map_out, void* cuda_stream) {
  NvtxRange nvtx("ngff.shard_prepare");
  if (!h) return COFIE_EINVAL;
  if (stream >= h->p.max_streams) return h->fail(COFIE_EINVAL, "stream index out of range");
  if (!frames || !map_out || n == 0) return h->fail(COFIE_EINVAL, "frames and map_out are required, n >= 1");
  if (h->p.signal == COFIE_SIGNAL_SCD)  // a scene-change run can reach back past any halo
    return h->fail(COFIE_EINVAL, "streams of the scene-change signal cannot be sharded");
  if (h->p.l_max == 0)  // without forced retention the reference frame can lie any distance back
    return h->fail(COFIE_EINVAL, "streams with l_max = 0 cannot be sharded");
  const uint64_t want_halo = t0 < h->p.l_max ? t0 : h->p.l_max;
  if (n_halo != want_halo) return h->fail(COFIE_EINVAL, "n_halo must be min(t0, l_max)");
  if (static_cast<uint64_t>(n_halo) + n > h->p.max_frames_per_push)
    return h->fail(COFIE_EINVAL, "n_halo + n exceeds max_frames_per_push");
  int fdev = -1;
  if (classify(frames, &fdev) != kDevice || fdev != h->device)
    return h->fail(COFIE_EINVAL, "shard frames must be device memory on the handle's device");
  DeviceGuard guard(h->device);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  h->shard.ready = false;
  // K1 over halo + shard frames; the stream's clock starts at t0 for K2
  SegTable all;
  memset(&all, 0, sizeof all);
  all.count = 1;
  all.rows = n_halo + n;
  all.s[0].frames = frames;
  all.s[0].n = n_halo + n;
  all.s[0].stream = stream;
  StreamState ss{t0, 1u, 0u, 0ull};
  cudaError_t e = cudaMemcpyAsync(h->d_state + stream, &ss, sizeof ss, cudaMemcpyHostToDevice, st);
  // the record of a sharded stream holds the committed shard's frames only
  if (e == cudaSuccess)
    e = cudaMemsetAsync(h->d_record + static_cast<size_t>(stream) * h->rec_words, 0, h->rec_words * sizeof(uint32_t),
                        st);
  if (e != cudaSuccess) return h->cuda_fail(e, "shard state");
  // the first stage only (histograms or features): the selection runs later
  e = clear_rows(h, h->dirty_rows, st);
  if (e != cudaSuccess) return h->cuda_fail(e, "memset histograms");
  h->dirty_rows = h->p.max_frames_per_push;
  e = launch_first_stage(h, all, st);
  if (e != cudaSuccess) return h->cuda_fail(e, "histogram kernel launch");
  h->n_hist += 1;
  h->hist_bytes += static_cast<uint64_t>(all.rows) * (h->frame_bytes + 4ull * h->fw);
  // K2 over the shard's rows, reading the halo rows before them
  SegTable sh;
  memset(&sh, 0, sizeof sh);
  sh.count = 1;
  sh.rows = n_halo + n;
  sh.s[0].frames = frames + static_cast<uint64_t>(n_halo) * h->frame_bytes;
  sh.s[0].n = n;
  sh.s[0].row0 = n_halo;
  sh.s[0].stream = stream;
  sh.s[0].halo = n_halo;
  SelectArgs sa = select_args(h);
  e = launch_window(sh, sa, h->d_hist, h->d_ring, h->d_state, h->d_l1, h->d_mask, st);
  if (e == cudaSuccess) e = launch_gap_map(sh.s[0], sa, t0, h->d_mask, h->d_map, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(map_out, h->d_map, h->p.l_max * sizeof(uint16_t), cudaMemcpyDefault, st);
  if (e == cudaSuccess && classify(map_out) != kDevice) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return h->cuda_fail(e, "shard preparation");
  h->n_select += 2;
  h->dirty_rows = n_halo + n;
  h->shard.ready = true;
  h->shard.stream = stream;
  h->shard.n_halo = n_halo;
  h->shard.n = n;
  h->shard.t0 = t0;
  return COFIE_OK;
}

int cofie_ngff_shard_commit(cofie_ngff_t* h, uint32_t stream, uint32_t entry_gap, float* scores_out, uint8_t* keep_out,
                            void* cuda_stream) {
  NvtxRange nvtx("ngff.shard_commit");
  if (!h) return COFIE_EINVAL;
  if (!h->shard.ready || h->shard.stream != stream)
    return h->fail(COFIE_EINVAL, "no shard of this stream is prepared on this handle");
  if (h->shard.t0 > 0 && (entry_gap < 1 || entry_gap > h->p.l_max))
    return h->fail(COFIE_EINVAL, "entry_gap must be in [1, l_max]");
  DeviceGuard guard(h->device);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const uint32_t n_halo = h->shard.n_halo, n = h->shard.n;
  SelectArgs sa = select_args(h);
  // the stream's ring holds the halo frames (the last frames before t0) ...
  cudaError_t e = launch_ring_store(h->d_hist, n_halo, h->shard.t0 - n_halo, stream, sa, h->d_ring, st);
  // ... and its gap is the resolved entry gap
  StreamState ss{h->shard.t0, h->shard.t0 > 0 ? entry_gap : 1u, 0u, 0ull};
  if (e == cudaSuccess) e = cudaMemcpyAsync(h->d_state + stream, &ss, sizeof ss, cudaMemcpyHostToDevice, st);
  if (e != cudaSuccess) return h->cuda_fail(e, "shard commit");
  const MemKind ks = classify(scores_out), kk = classify(keep_out);
  SegTable sh;
  memset(&sh, 0, sizeof sh);
  sh.count = 1;
  sh.rows = n_halo + n;
  sh.s[0].n = n;
  sh.s[0].row0 = n_halo;
  sh.s[0].stream = stream;
  sh.s[0].halo = n_halo;
  sh.s[0].scores = ks == kDevice ? scores_out : (ks == kNull ? nullptr : h->d_scores);
  sh.s[0].keep = kk == kDevice ? keep_out : (kk == kNull ? nullptr : h->d_keep);
  e = launch_scan(sh, sa, h->d_l1, h->d_mask, h->d_hist, h->d_ring, h->d_state, st);
  if (e == cudaSuccess && (ks == kHostPinned || ks == kHostPageable))
    e = cudaMemcpyAsync(scores_out, h->d_scores, n * sizeof(float), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess && (kk == kHostPinned || kk == kHostPageable))
    e = cudaMemcpyAsync(keep_out, h->d_keep, n, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = clear_rows(h, static_cast<uint64_t>(n_halo) + n, st);  // rows are zero between calls
  if (e != cudaSuccess) return h->cuda_fail(e, "shard commit");
  h->dirty_rows = 0;
  h->n_select += 1;
  h->shard.ready = false;
  h->seen[stream] = h->shard.t0 + n;
  return COFIE_OK;
}

int cofie_ngff_reset(cofie_ngff_t* h, uint32_t stream, void* cuda_stream) {
  if (!h) return COFIE_EINVAL;
  if (stream >= h->p.max_streams) return h->fail(COFIE_EINVAL, "stream index out of range");
  DeviceGuard guard(h->device);
  const cudaError_t e = launch_stream_reset(h->d_state + stream, h->d_record + static_cast<size_t>(stream) * h->rec_words,
                                            h->rec_words, static_cast<cudaStream_t>(cuda_stream));
  if (e != cudaSuccess) return h->cuda_fail(e, "reset");
  h->n_other += 1;
  h->seen[stream] = 0;
  return COFIE_OK;
}

int cofie_ngff_status(cofie_ngff_t* h, void* cuda_stream) {
  if (!h) return COFIE_EINVAL;
  DeviceGuard guard(h->device);
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(cuda_stream));
  if (e != cudaSuccess) return h->cuda_fail(e, "stream synchronise");
  uint32_t word = 0;
  e = cudaMemcpy(&word, h->d_err, sizeof word, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return h->cuda_fail(e, "error word read");
  if (checked_build()) {  // the index checks of every kernel file (checked builds only)
    const uint32_t b = take_bounds_errors_hist() | take_bounds_errors_features() | take_bounds_errors_select() |
                       take_bounds_errors_lazy() | take_bounds_errors_finalize();
    if (b) word |= kErrBounds;
  }
  if (word) {
    cudaMemset(h->d_err, 0, sizeof word);
    char buf[128];
    snprintf(buf, sizeof buf,
             "device-side failure (error bits 0x%x: 1/2/4 a wait ran out, 8 a bad gather index, 16 an index check "
             "of the checked build, 32 candidates of a stream past its retention record)",
             word);
    return h->fail((word & (kErrConsumerTimeout | kErrProducerTimeout | kErrDrainTimeout)) ? COFIE_ETIMEOUT
                                                                                          : COFIE_EDEVICE,
                   buf);
  }
  return COFIE_OK;
}

int cofie_ngff_frames_seen(const cofie_ngff_t* h, uint32_t stream, uint64_t* t_out) {
  if (!h || !t_out || stream >= h->p.max_streams) return COFIE_EINVAL;
  *t_out = h->seen[stream];
  return COFIE_OK;
}

int cofie_ngff_checked_build(void) { return checked_build() ? 1 : 0; }

void cofie_ngff_debug_fail_alloc(int32_t after) { g_fail_alloc.store(after < 0 ? -1 : after); }

int cofie_ngff_debug_wait(cofie_ngff_t* h, uint64_t timeout_ns, void* cuda_stream) {
  if (!h) return COFIE_EINVAL;
  if (timeout_ns > 1000000000ull) return h->fail(COFIE_EINVAL, "timeout_ns must be at most 1 s");
  DeviceGuard guard(h->device);
  const cudaError_t e = launch_wait_probe(timeout_ns, h->d_err, static_cast<cudaStream_t>(cuda_stream));
  return e == cudaSuccess ? COFIE_OK : h->cuda_fail(e, "wait probe launch");
}

int cofie_ngff_debug_bins(cofie_ngff_t* h, const uint8_t* pixels, uint64_t n_pixels, uint8_t* bins_out,
                          void* cuda_stream) {
  if (!h) return COFIE_EINVAL;
  if (n_pixels == 0) return COFIE_OK;
  if (!pixels || !bins_out || n_pixels % 4 != 0) return h->fail(COFIE_EINVAL, "pixels/bins_out NULL or n_pixels % 4");
  if (h->bin_path < 0) return h->fail(COFIE_EINVAL, "these parameters use the generic histogram kernel only");
  if (classify(pixels) != kDevice || classify(bins_out) != kDevice)
    return h->fail(COFIE_EINVAL, "debug buffers must be device memory");
  DeviceGuard guard(h->device);
  cudaError_t e = launch_debug_bins(pixels, n_pixels / 4, h->lc, h->bin_path, bins_out,
                                    static_cast<cudaStream_t>(cuda_stream));
  if (e != cudaSuccess) return h->cuda_fail(e, "debug kernel launch");
  return COFIE_OK;
}

int cofie_ngff_candidates(cofie_ngff_t* h, uint32_t stream, uint32_t* idx_out, uint32_t cap, uint32_t* m_out,
                          void* cuda_stream) {
  NvtxRange nvtx("ngff.candidates");
  if (!h) return COFIE_EINVAL;
  if (stream >= h->p.max_streams) return h->fail(COFIE_EINVAL, "stream index out of range");
  if (!m_out) return h->fail(COFIE_EINVAL, "m_out is NULL");
  DeviceGuard guard(h->device);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  int di = -1;
  const MemKind ki = cap > 0 ? classify(idx_out, &di) : kNull;
  if (cap > 0 && (ki == kNull || (ki == kDevice && di != h->device)))
    return h->fail(COFIE_EINVAL, "idx_out must be device memory on the handle's device, or host memory");
  const MemKind km = classify(m_out);
  const int capturing = capture_state(st);
  if (capturing < 0) return h->fail(COFIE_ECUDA, "cannot read the CUDA stream's capture state");
  if (capturing && (km != kDevice || (ki != kDevice && ki != kNull)))
    return h->fail(COFIE_EINVAL, "a captured call takes device idx_out and m_out");
  if (ki != kDevice && ki != kNull && km == kDevice)
    return h->fail(COFIE_EINVAL, "a host idx_out needs a host m_out");
  if (!capturing && h->seen[stream] > h->p.max_stream_frames)
    return h->fail(COFIE_EINVAL, "the stream has run past its retention record (max_stream_frames)");
  uint32_t* idx = idx_out;
  if (ki != kDevice && ki != kNull) {  // host indices: through a device buffer of the record's size
    if (!h->d_idx) {
      if (dalloc(&h->d_idx, static_cast<size_t>(h->rec_words) * 32) != cudaSuccess) {
        cudaGetLastError();
        h->d_idx = nullptr;
        return h->fail(COFIE_ENOMEM, "index buffer allocation failed");
      }
    }
    idx = h->d_idx;
    if (cap > h->p.max_stream_frames) cap = h->p.max_stream_frames;  // |S_c| <= T <= the record's frames
  }
  uint32_t* count = km == kDevice ? m_out : h->d_count;
  cudaError_t e = launch_stream_candidates(h->d_record + static_cast<size_t>(stream) * h->rec_words, h->rec_words,
                                           h->d_state + stream, h->p.m_min, idx, cap, count, h->d_err, st);
  if (e != cudaSuccess) return h->cuda_fail(e, "candidates kernel launch");
  h->n_other += 1;
  if (km != kDevice) {
    e = cudaMemcpyAsync(m_out, count, sizeof(uint32_t), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e == cudaSuccess && idx != idx_out && *m_out > 0)
      e = cudaMemcpy(idx_out, idx, static_cast<size_t>(std::min(*m_out, cap)) * sizeof(uint32_t),
                     cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return h->cuda_fail(e, "candidates count");
  }
  return COFIE_OK;
}

int cofie_ngff_candidates_from_keep(cofie_ngff_t* h, const uint8_t* keep, uint32_t T, uint32_t* idx_out,
                                    uint32_t* m_out, void* cuda_stream) {
  NvtxRange nvtx("ngff.candidates_from_keep");
  if (!h) return COFIE_EINVAL;
  if (!m_out) return h->fail(COFIE_EINVAL, "m_out is NULL");
  DeviceGuard guard(h->device);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const MemKind km = classify(m_out);
  if (T == 0) {
    if (km == kDevice) {
      cudaError_t e = cudaMemsetAsync(m_out, 0, sizeof(uint32_t), st);
      return e == cudaSuccess ? COFIE_OK : h->cuda_fail(e, "candidates count");
    }
    *m_out = 0;
    return COFIE_OK;
  }
  int dk = -1, di = -1;
  if (!keep || !idx_out || classify(keep, &dk) != kDevice || classify(idx_out, &di) != kDevice || dk != h->device ||
      di != h->device)
    return h->fail(COFIE_EINVAL, "keep and idx_out must be device memory on the handle's device");
  uint32_t* count = km == kDevice ? m_out : h->d_count;
  cudaError_t e = launch_candidates(keep, T, h->p.m_min, idx_out, count, st);
  if (e != cudaSuccess) return h->cuda_fail(e, "candidates kernel launch");
  h->n_other += 1;
  if (km != kDevice) {
    e = cudaMemcpyAsync(m_out, count, sizeof(uint32_t), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return h->cuda_fail(e, "candidates count");
  }
  return COFIE_OK;
}

int cofie_ngff_gather(cofie_ngff_t* h, const uint8_t* frames, uint32_t n_frames, const uint32_t* idx, uint32_t m,
                      uint8_t* out, void* cuda_stream) {
  NvtxRange nvtx("ngff.gather");
  if (!h) return COFIE_EINVAL;
  if (m == 0) return COFIE_OK;
  DeviceGuard guard(h->device);
  if (!guard.ok) return h->fail(COFIE_ECUDA, "cannot select the handle's device");
  int d0 = -1, d1 = -1, d2 = -1;
  const MemKind kf = frames ? classify(frames, &d0) : kNull;
  if (!idx || !out || classify(idx, &d1) != kDevice || classify(out, &d2) != kDevice || d1 != h->device ||
      d2 != h->device)
    return h->fail(COFIE_EINVAL, "idx and out must be device memory on the handle's device");
  // frames: device memory, or pinned host memory that the kernel reads through the device's mapping of it
  const uint8_t* src = nullptr;
  if (kf == kDevice && d0 == h->device) {
    src = frames;
  } else if (kf == kHostPinned) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, frames) == cudaSuccess) src = static_cast<const uint8_t*>(a.devicePointer);
    cudaGetLastError();
  }
  if (!src)
    return h->fail(COFIE_EINVAL, "frames must be device memory on the handle's device, or pinned host memory");
  cudaError_t e = launch_gather(src, n_frames, h->frame_bytes, idx, m, out, h->d_err, kf == kHostPinned,
                                static_cast<cudaStream_t>(cuda_stream));
  if (e != cudaSuccess) return h->cuda_fail(e, "gather kernel launch");
  h->n_other += 1;
  return COFIE_OK;
}

int cofie_ngff_profile_reset(cofie_ngff_t* h, int time_kernels) {
  if (!h) return COFIE_EINVAL;
  h->n_hist = h->n_select = h->n_other = h->hist_bytes = 0;
  h->ev_used = h->ev_sel_used = 0;
  h->time_kernels = time_kernels != 0;
  return COFIE_OK;
}

int cofie_ngff_profile_read(cofie_ngff_t* h, cofie_ngff_profile* out) {
  if (!h || !out) return COFIE_EINVAL;
  DeviceGuard guard(h->device);
  cudaError_t e;
  const double hist_ms = sum_pairs(h->ev_pool, h->ev_used, &e);
  if (e != cudaSuccess) return h->cuda_fail(e, "kernel timing events");
  const double sel_ms = sum_pairs(h->ev_sel, h->ev_sel_used, &e);
  if (e != cudaSuccess) return h->cuda_fail(e, "kernel timing events");
  out->hist_launches = h->n_hist;
  out->select_launches = h->n_select;
  out->hist_bytes = h->hist_bytes;
  out->hist_timed = h->ev_used / 2;
  out->hist_ms = hist_ms;
  out->select_timed = h->ev_sel_used / 2;
  out->select_ms = sel_ms;
  out->other_launches = h->n_other;
  return COFIE_OK;
}

const char* cofie_ngff_last_error(const cofie_ngff_t* h) { return h ? h->err.c_str() : ""; }

const char* cofie_ngff_global_error(void) { return g_global_error.c_str(); }

}  // extern "C"
