// internal.h — host-side declarations shared by the efsparse translation
// units: the per-stream workspace and the kernel launchers.
#pragma once

#include <cstddef>
#include <cstdint>
#include <vector>
#include <cuda_runtime.h>

#include "common.cuh"

namespace efs {

// Layout of the workspace header (bytes from the workspace base).
constexpr size_t kOffBarGen = 0;        // uint32: grid-barrier generation (never reset)
constexpr size_t kOffError = 8;         // uint32: latched device error bits
constexpr size_t kOffBarArrive = 16;    // uint32: grid-barrier arrivals (zero after each barrier)
constexpr size_t kOffTileClaim = 24;    // uint32[3]: work dispenser: handed out, CTAs finished,
                                        // groups resolved (zero between calls)
constexpr size_t kOffTkListCount = 72;  // uint32: candidates emitted by the streaming pass
constexpr size_t kOffErrArrive = 80;    // uint32: arrivals of the e' norm pass (zero after it)
constexpr size_t kOffStreamErr = 88;    // double: the streaming pass's share of ||e'||^2
// Per-call Top-k state that must start at zero, in two blocks used by
// alternate calls on a workspace: a call's candidate stream zeroes the
// other block (the previous call's, complete by then) for the next call.
constexpr size_t kOffTkState = 256;
constexpr size_t kStStreamArrive = 0;   // uint32: arrivals at the candidate stream's barrier
constexpr size_t kStListFlags = 4;      // uint32: that pass's latched bits (overflow, timeout)
constexpr size_t kStErrArrive = 8;      // uint32: select CTAs that published their ||e'||^2 share
constexpr size_t kStSelect = 16;        // uint32[4]: short-list threshold published by CTA 0
constexpr size_t kStCandCount = 32;     // uint32[6]: refine-level candidate counts
constexpr size_t kStLowerBound = 64;    // uint64: sampled lower bound of the candidates' keys
constexpr size_t kStMode = 72;          // uint32: 0 candidates, 1 full array
constexpr size_t kStHist = 256;         // uint32[6][2048]: refine-level histograms
constexpr int kHistLevels = 6;
constexpr int kHistBins = 2048;
constexpr int kSampleBits = 13;         // the sample histogram: top 13 bits of |a|
constexpr int kSampleBins = 1 << kSampleBits;
constexpr size_t kStSampleHist = kStHist + sizeof(uint32_t) * kHistLevels * kHistBins;
constexpr size_t kTkStateBytes = kStSampleHist + sizeof(uint32_t) * kSampleBins;
static_assert(kTkStateBytes % 256 == 0, "state block alignment");
constexpr size_t kHeaderBytes = kOffTkState + 2 * kTkStateBytes;
constexpr uint32_t kMaxChunks = 1024;   // per-CTA chunk sums of the streaming compaction
constexpr uint32_t kCountsPerTile = 16; // per-segment counts of the streaming compaction

// ---- layer-wise Top-k: one Top-k selection per segment of the vector.
// Segment kinds: nothing sent (k = 0); a short segment selected from e in
// one CTA's shared memory; a sampled candidate bound, then a selection over
// the candidates; every coordinate sent (k = d_s).
constexpr uint32_t kLwNone = 0, kLwWhole = 1, kLwSampled = 2, kLwAll = 3;
constexpr uint32_t kLwSmemElems = 48u * 1024u;  // values one select CTA holds in shared memory
constexpr uint32_t kLwWholeMax = 4096;          // segments at most this long: selected from e
constexpr uint32_t kLwSampleGroups = 4096;      // groups of 4 coordinates sampled per CTA
constexpr uint32_t kLwMaxParts = 32;            // sampling CTAs of one long segment, at most
constexpr int kLwSampleBits = 15;               // the sample histogram: top 15 bits of |a|
constexpr uint32_t kLwSampleBins = 1u << kLwSampleBits;  // (1/128 of a binade each)
constexpr uint32_t kLwPartHistWords = kLwSampleBins + 32;  // merged histogram + arrival word
// Candidate bounds that admit nothing: the residual of the segment's
// coordinates is then a, final in the streaming pass (kLwNoBound: segments
// that send nothing), or decided by the select (kLwDeferred: short segments,
// segments that send everything, sampled segments whose sample found no bound).
constexpr uint32_t kLwNoBound = 0xffffffffu;
constexpr uint32_t kLwDeferred = 0xfffffffeu;
constexpr uint32_t kLwTileUniform = 0x80000000u;  // tile_info: the tile lies in one segment

struct LwSeg {      // one segment (device and host layout, 32 bytes)
  uint64_t step;    // sampled: spacing of the groups, in aligned groups, 32.32 fixed point
  uint32_t lo, hi;  // coordinates [lo, hi)
  uint32_t k;       // pairs it sends
  uint32_t out;     // output position of its first pair
  uint32_t groups;  // sampled: its sampled groups of 4 consecutive coordinates
  uint16_t kind;    // kLw*
  uint16_t exact;   // sampled: the groups are every aligned group of the segment
};
// A select CTA: either the segments work_seg[a, b) one after another
// (team == kLwNoTeam), or member `rank` of a team of b CTAs that selects
// segment a together (team = the team's index).
constexpr uint32_t kLwNoTeam = 0xffffffffu;
constexpr uint32_t kLwMaxTeam = 32;
struct LwCta {
  uint32_t team, a, b, rank;
};
// Per-team state of the select kernel: histograms of the three magnitude
// digit levels and a barrier (zero at a call's start; the team's rank 0
// clears the histograms at the end), and per-rank counts.
struct LwTeamState {
  uint32_t hist[3][2048];
  uint32_t arrive, gen, last, pad0;
  uint32_t cnt[kLwMaxTeam];
  uint32_t tie_cnt[kLwMaxTeam];
  uint32_t pad[60];
};
static_assert(sizeof(LwTeamState) % 256 == 0, "team state alignment");

// The device tables of a segment table, rebuilt when the table changes.
struct LwPlan {
  std::vector<uint64_t> seg_end, seg_k;  // the host table this plan was built from
  uint64_t d = 0;
  bool valid = false;
  uint32_t n_seg = 0, n_sampled = 0, n_select_ctas = 0, n_teams = 0, tiles = 0;
  uint32_t n_part_hist = 0;  // merged sample histograms (segments sampled in parts), per copy
  uint64_t total_k = 0;
  std::vector<char> image;  // host image of the uploaded part
  char* dev = nullptr;
  size_t dev_bytes = 0;
  // byte offsets in dev: uploaded tables, then zero-initialised counters
  // and histograms (each user resets its own), then per-call outputs
  size_t off_segs = 0, off_seg_end = 0, off_mbound = 0, off_tile_info = 0, off_samples = 0,
         off_ctas = 0, off_work_seg = 0, off_teams = 0, off_part_hist = 0, off_tile_base = 0,
         total = 0;
};

struct Workspace {
  int device = -1;
  cudaStream_t stream = nullptr;
  char* base = nullptr;
  size_t bytes = 0;
  uint32_t status_tiles = 0;   // capacity of the per-tile arrays (status, counts)
  uint32_t cand_cap = 0;       // capacity of each Top-k candidate buffer
  size_t offsets_cap = 0;      // capacity of the aggregation offsets (uint32)
  size_t stage_cap = 0;        // capacity of the pair staging buffers (pairs)
  uint32_t epoch = 0;          // last epoch handed to a compaction launch
  uint32_t topk_calls = 0;     // Top-k calls so far: their parity picks the state block
  // Balanced chunks of the streaming hard-threshold kernel: each call computes
  // the next call's chunk boundaries from the previous call's chunk totals.
  uint32_t ht_seq = 0;          // streaming hard-threshold calls so far
  uint32_t ht_last_tiles = 0;   // the previous such call's tiles, grid and epoch
  uint32_t ht_last_grid = 0;
  uint32_t ht_last_epoch = 0;
  bool ht_part_ready = false;   // the previous call wrote the boundaries for this one
  bool ht_prev_balanced = false;  // the previous call used written boundaries
  // Host-mapped word the claimed-group hard-threshold kernel writes (the
  // call's pairs * 65536 / d): read without synchronising, it may be a few
  // calls old, and only picks the next calls' ring depth (never a result).
  uint32_t* density_host = nullptr;
  uint32_t* density_dev = nullptr;
  bool dirty = false;          // header must be re-cleared (failed launch or device timeout)
  LwPlan* lw = nullptr;        // layer-wise Top-k tables (created on first use)

  // Regions after the header, each 256-byte aligned.
  static size_t align(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }
  size_t off_status() const { return kHeaderBytes; }
  size_t off_cand() const { return align(off_status() + sizeof(uint64_t) * status_tiles); }
  // three candidate buffers: the streamed (index, value) list and two key buffers
  size_t off_offsets() const { return align(off_cand() + 3 * sizeof(uint64_t) * cand_cap); }
  size_t off_counts() const { return align(off_offsets() + sizeof(uint32_t) * offsets_cap); }
  size_t off_chunks() const {
    return align(off_counts() + sizeof(uint32_t) * kCountsPerTile * status_tiles);
  }
  size_t off_errparts() const { return align(off_chunks() + sizeof(uint64_t) * kMaxChunks); }
  size_t off_cntparts() const { return align(off_errparts() + sizeof(FF) * kMaxChunks); }
  size_t off_stage() const { return align(off_cntparts() + sizeof(uint32_t) * kMaxChunks); }
  // hard-threshold balancing: chunk totals of the last two calls (by call
  // parity), then three boundary arrays (by call number mod 3)
  size_t off_ht() const { return align(off_stage() + 8 * stage_cap); }
  size_t total_bytes() const {
    return align(off_ht() + 2 * sizeof(uint64_t) * kMaxChunks + 3 * sizeof(uint32_t) * (kMaxChunks + 1));
  }
  uint64_t* ht_chunks(uint32_t parity) const {
    return reinterpret_cast<uint64_t*>(base + off_ht()) + (parity & 1u) * kMaxChunks;
  }
  uint32_t* ht_part(uint32_t which) const {
    return reinterpret_cast<uint32_t*>(base + off_ht() + 2 * sizeof(uint64_t) * kMaxChunks) +
           (which % 3u) * (kMaxChunks + 1);
  }

  uint64_t* status() const { return reinterpret_cast<uint64_t*>(base + off_status()); }
  uint64_t* cand(int i) const {
    return reinterpret_cast<uint64_t*>(base + off_cand()) + static_cast<size_t>(i) * cand_cap;
  }
  uint32_t* offsets() const { return reinterpret_cast<uint32_t*>(base + off_offsets()); }
  uint32_t* counts() const { return reinterpret_cast<uint32_t*>(base + off_counts()); }
  uint64_t* chunks() const { return reinterpret_cast<uint64_t*>(base + off_chunks()); }
  FF* errparts() const { return reinterpret_cast<FF*>(base + off_errparts()); }
  uint32_t* cntparts() const { return reinterpret_cast<uint32_t*>(base + off_cntparts()); }
  double* stream_err() const { return reinterpret_cast<double*>(base + kOffStreamErr); }
  uint32_t* stage_idx() const { return reinterpret_cast<uint32_t*>(base + off_stage()); }
  float* stage_val() const {
    return reinterpret_cast<float*>(base + off_stage() + sizeof(uint32_t) * stage_cap);
  }
  uint32_t* u32(size_t off) const { return reinterpret_cast<uint32_t*>(base + off); }
  uint32_t* topk_state(uint32_t parity) const {
    return u32(kOffTkState + (parity & 1u) * kTkStateBytes);
  }
  uint64_t* u64(size_t off) const { return reinterpret_cast<uint64_t*>(base + off); }
};

// Per-device facts queried once.
struct DeviceInfo {
  int sm_count = 0;
  int refine_blocks = 0;          // co-resident CTAs for the cooperative Top-k select
  int finalize_blocks = 0;        // co-resident CTAs for the Top-k finalize
  int ht_stream_per_sm_f32 = 0;   // streaming hard-threshold CTAs per SM (0: unavailable)
  int ht_stream_per_sm_bf16 = 0;
  int ht_group_per_sm_f32 = 0;    // hard-threshold claimed-group CTAs per SM (0: unavailable)
  int ht_group_per_sm_bf16 = 0;
  int ht_dense_per_sm_f32 = 0;    // the same with the shallow ring
  int ht_dense_per_sm_bf16 = 0;
  int tk_stream_per_sm_f32 = 0;   // streaming Top-k candidate pass CTAs per SM
  int tk_stream_per_sm_bf16 = 0;
  int tk_group_per_sm_f32 = 0;    // Top-k candidate pass, claimed-group kernel CTAs per SM
  int tk_group_per_sm_bf16 = 0;
  int lw_stream_per_sm_f32 = 0;   // streaming layer-wise candidate pass CTAs per SM
  int lw_stream_per_sm_bf16 = 0;
  int lw_group_per_sm_f32 = 0;    // layer-wise candidate pass, claimed-group kernel CTAs per SM
  int lw_group_per_sm_bf16 = 0;
  int lw_select_per_sm = 0;       // co-resident layer-wise select CTAs per SM
};

// Per-device set-up of the Top-k kernels (shared-memory opt-in, occupancy).
void topk_init_device(DeviceInfo& info);

// Per-device set-up of the layer-wise Top-k kernels.
void topk_layerwise_init_device(DeviceInfo& info);

// Per-device set-up of the aggregation kernels (prefer the largest shared
// memory carve-out, so that 8 of their CTAs are resident per SM).
void aggregate_init_device();

// Per-device set-up of the streaming hard-threshold kernels (opts them into
// their shared-memory ring on the current device and records occupancy).
void ht_init_device(DeviceInfo& info);

// Scaled integer rounding under error feedback, and the exact exchange of
// its integer messages (round.cu).
cudaError_t launch_scaled_round(const void* g, bool g_bf16, float* e, float gamma, int m,
                                uint32_t d, int32_t* q, uint32_t* unsent, double* err_out,
                                Workspace& ws, const DeviceInfo& dev);
cudaError_t launch_int_aggregate(uint32_t n, const int32_t* const* q, uint32_t d, int m,
                                 float* dense_out, Workspace& ws, const DeviceInfo& dev);

// ||e'||^2 of e[0, d) after a step, by one plain pass (the paths that do
// not stream through stream_compact.cuh); written to *err_out.
cudaError_t launch_error_norm(const float* e, uint32_t d, double* err_out, Workspace& ws,
                              const DeviceInfo& dev);

// Launch bookkeeping.
// A launch that may begin while the previous kernel on the stream finishes
// (programmatic dependent launch: the kernel waits for its predecessor with
// griddepcontrol.wait before reading what it wrote), optionally cooperative.
cudaError_t launch_pdl(const void* fn, dim3 grid, uint32_t block, uint32_t smem,
                       cudaStream_t stream, void** params, bool cooperative);
void count_launch();
uint64_t wait_limit_ns();
int64_t withheld_tile();
// ef_test_set_stream_kernel: 0 by size (and density), 1 static chunks, 2 claimed
// groups, 3 claimed groups with the shallow ring (hard-threshold; the other
// streaming passes treat it as 2)
int stream_kernel_mode();

// The streaming passes (hard-threshold, Top-k and layer-wise candidates) use
// the claimed-group look-back kernel from this many tiles on (16.8 M
// coordinates), the static-chunk kernel below, whose call has less fixed cost
// (no look-back chain to drain at the end of a short call); the test hook
// ef_test_set_stream_kernel can force either.
constexpr uint32_t kGroupKernelMinTiles = 4096;
inline bool use_group_kernel(uint32_t tiles) {
  const int mode = stream_kernel_mode();
  return mode >= 2 || (mode == 0 && tiles >= kGroupKernelMinTiles);
}
// Dense calls (the claimed-group hard-threshold kernel's last call on this
// workspace sent at least this share of its coordinates, in 1/65536) run the
// kernel with one ring stage fewer and the freed shared memory added to the
// warps' pair buffers: fewer segments go through their global slots.
constexpr uint32_t kDenseRingHint = 65536u / 12u;  // 8.3 %
ScanCtx next_scan_ctx(Workspace& ws, uint32_t num_tiles);

// ---- launchers (return the launch's cudaError_t) ----
// err_out (optional, device): ||e'||^2 of the step.
// tiles_out (optional, device, uint32[tiles_for(d) + 1]): the message's tile
// index, tiles_out[t] = pairs with index < t * kTileElems, the last = count.
cudaError_t launch_hard_threshold(const void* g, bool g_bf16, float* e, float gamma,
                                  float lambda, uint32_t d, uint32_t* idx_out, float* val_out,
                                  uint32_t* count_out, double* err_out, uint32_t* tiles_out,
                                  Workspace& ws, const DeviceInfo& dev);
// The tile index of one ascending list (binary searches), for the paths whose
// kernel does not produce it.
cudaError_t launch_list_tiles(const uint32_t* idx, const uint32_t* count, uint32_t d,
                              uint32_t* tiles_out, Workspace& ws);
cudaError_t launch_hard_threshold_lookback(const float* g, float* e, float gamma, float lambda,
                                           uint32_t d, uint32_t* idx_out, float* val_out,
                                           uint32_t* count_out, const ScanCtx& ctx,
                                           cudaStream_t stream);
cudaError_t launch_topk(const void* g, bool g_bf16, float* e, float gamma, uint32_t k,
                        uint32_t d, uint32_t* idx_out, float* val_out, uint32_t* count_out,
                        double* err_out, Workspace& ws, const DeviceInfo& dev);
// Layer-wise Top-k: lw_prepare builds and uploads the plan of a segment
// table (a no-op when the workspace already holds that table's plan).
cudaError_t lw_prepare(Workspace& ws, const uint64_t* seg_end, const uint64_t* seg_k,
                       uint32_t n_seg, uint64_t d, const DeviceInfo& dev);
cudaError_t launch_topk_layerwise(const void* g, bool g_bf16, float* e, float gamma, uint32_t d,
                                  uint32_t* idx_out, float* val_out, uint32_t* count_out,
                                  double* err_out, Workspace& ws, const DeviceInfo& dev);
// tiles (optional): HOST array of n DEVICE pointers to the lists' tile
// indexes; without it the kernel before the reduction finds them.
cudaError_t launch_aggregate(uint32_t n, const uint32_t* const* idx, const float* const* val,
                             const uint32_t* const* tiles, const uint32_t* counts, uint32_t d,
                             float* dense_out, Workspace& ws);
cudaError_t launch_aggregate_apply(uint32_t n, const uint32_t* const* idx,
                                   const float* const* val, const uint32_t* const* tiles,
                                   const uint32_t* counts, uint32_t d, float alpha, float* x,
                                   float* m, float mu, float lr, Workspace& ws);


// Workspace sizing helpers.
inline uint32_t tiles_for(uint64_t d) {
  return static_cast<uint32_t>((d + kTileElems - 1) / kTileElems);
}
constexpr int kAggTile = 4096;             // dense elements per aggregation CTA
constexpr int kAggStage = 1024;            // pairs an aggregation CTA stages per round trip
static_assert(kAggTile == kTileElems, "a message's tile index serves the aggregation");
constexpr uint32_t kMaxWorkers = 256;
inline uint32_t agg_tiles_for(uint64_t d) {
  return static_cast<uint32_t>((d + kAggTile - 1) / kAggTile);
}
uint32_t topk_candidate_capacity(uint64_t d);

}  // namespace efs
