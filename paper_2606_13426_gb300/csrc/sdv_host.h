// sdv_host.h - internal launch parameters and workspace layout of libspecdiff.
#pragma once

#include <cstddef>
#include <cstdint>

#include "../../include/specdiff.h"

namespace sdv {

// Fused verify kernel: threads per CTA and 16-byte vectors per thread per tensor per sweep.
constexpr int kK1Threads = 256;
constexpr int kK1Vpt = 4;
// Resident CTAs per SM the fused kernel is built for (its register budget): the
// chain-finishing code needs more than the streaming loop.
constexpr int kK1MinBlocks = 4;
// Many-chain path (B >= kManyChainMin): resident CTAs per SM of the streaming
// kernel k_tiles (its register budget: 3 x vpt 16-byte buffers per thread), and
// the finishing kernel k_finish: threads per chain and groups of four elements per
// thread per residual sweep.
constexpr int kManyChainMin = 512;
// Plain calls with fewer chains than this run the fused kernel (one launch; its
// staggered per-chain finishing wins for small batches); from this many on, k_tiles +
// k_finish (measured per call, pixel rows: B = 16 18.5 against 22.5 us, B = 64 24.9
// against 24.3, B = 256 38.2 against 34.8 in block mode).
constexpr int kFusedMaxChains = 64;
// Three vectors per thread fit 48 registers, so that four k_tiles CTAs still leave
// room for two 64-thread k_finish CTAs of the previous pipelined call on the same SM
// (pipelined pixel rows 16.4 -> 16.3 us per call in block mode, 16.2 -> 15.7 in sample).
constexpr int tile_min_blocks(int vpt) { return vpt <= 1 ? 8 : (vpt == 2 ? 6 : (vpt == 3 ? 5 : 4)); }
constexpr int kFinishThreads = 64;
constexpr int kFinishWideThreads = 256;
constexpr int kFinishResidUnroll = 4;
// Stand-alone acceptance scan: one warp per chain.
constexpr int kK2Threads = 128;
// Long-row residual kernels: threads per CTA, and the elements of the rejected row
// per CTA, chosen per call between kK4MinChunk and kK4MaxChunk so that the grid is
// about kK4TargetCtas CTAs (short kernels want many CTAs; long rows want fewer,
// longer ones).
constexpr int kK4Threads = 256;
constexpr int64_t kK4MinChunk = 1024;
constexpr int64_t kK4MaxChunk = 4096;
constexpr int64_t kK4TargetCtas = 1024;
// Pipelined calls: at most this many CTAs per long-row residual kernel (they sit
// resident, waiting for the chain states, while the next call streams).
constexpr int64_t kK4PipeCtas = 128;
// Rows of up to kFusedMaxGroups groups of 4 elements are written by the CTA that
// finishes the chain inside the fused kernel, kFinishMaxGroups by k_finish on the
// many-chain path, and kPipeMaxGroups by k_finish on the pipelined path (in each case
// the residual's noise cached in dynamic shared memory: 16 KB, or up to 64 KB);
// longer rows by k_resid_dot/_write.  The fused kernel's residual sweeps take
// kFusedResidUnroll groups per thread, their loads issued together.
constexpr int64_t kFusedMaxGroups = 1024;
constexpr int64_t kFinishMaxGroups = 1024;
constexpr int64_t kPipeMaxGroups = 4096;
constexpr int kFusedResidUnroll = 3;

enum : int32_t {
  kKindInactive = 0,
  kKindResid = 1,      // decomposition residual
  kKindReflect = 2,    // reflection residual
  kKindZeroDelta = 3,  // |Delta_tau| = 0: m^q + sigma G
  kKindCopy = 4,       // full accept, last draft row
  kKindBonus = 5,      // full accept, bonus step
};

// Per-chain result of the scan, consumed by the residual writer (48 bytes).
struct ChainState {
  int32_t tau;      // 1-based
  int32_t row;      // row of the window the residual writer reads (tau-1, or the last draft)
  float U;          // residual 1-D draw
  float la_res;     // log alpha_{tau-1}
  float sigma;      // sigma_tau
  float dnorm;      // |Delta_tau|
  float inv_norm;   // 1/|delta_tau|, delta = m^p - m^q
  float refl;       // 1 + 2 S1/S2 (reflection: y = x - delta * refl)
  uint32_t status;
  int32_t kind;
  int32_t pad[2];
};

struct ScanArgs {
  const float2* part;     // fused kernel: [B, L, C] (S1, S2) per tile
  const uint64_t* tpart;  // k_tiles: [B, L, C] pairs of words (S1 | tag << 32, S2 | tag << 32)
  uint32_t* consumed;     // [B, L, C] beside tpart: the tag of the partial last read from each slot
  uint32_t tag;           // this call's tag of its k_tiles partials (never 0)
  bool fresh_set;         // the set held another layout before: k_tiles waits before its stores
  int C;
  const float* sigma;
  int64_t sstride;
  const float* ell_in;
  const float* dn_in;
  int B, L;
  const int32_t* L_eff;
  uint64_t seed;
  const uint64_t* seed_dev;  // nullable: the seed is read from device memory instead
  int mode;
  float inv_omega2;
  int residual_kind;
  bool has_bonus;
  bool ratios_only;
  float* ell_out;
  float* dn_out;
  int32_t* accepted_len;
  int32_t* tau_out;
  float* la_res_out;
  uint32_t* status_out;
  float* aux_out;
  bool draw_u;  // draw the residual U (the whole verify step) or stop at tau
};

struct WsLayout {
  int vpt1;        // K1 16-byte vectors per thread per tensor
  int64_t chunk1;  // elements of a row per K1 tile
  int C1;          // K1 tiles per row
  int64_t chunk4;  // K4 elements per tile
  int C4;          // K4 tiles per chain
  // tickets [B] u32 (fused kernel); two sets of tile partials [B, L, C1], 16 bytes
  // each (the fused kernel's float2, in set 0, or k_tiles' tagged pair of words), each
  // followed by its consumed tags [B, L, C1] u32; chain states; long-row partials
  size_t ticket_off, part_off, part_set_bytes, cons_off, state_off, part4_off, total;
};

WsLayout ws_layout(int B, int L, int64_t d, int dtype);

// sdv_verify_ex with the seed taken from device memory when seed_dev is not null (it
// is read by the kernels, so a captured call follows the value at replay), event
// timing skipped when timed is false, and, with overlap, the permission to start
// before the previous kernel on the stream has finished (sdv_verify_pipelined).  Same
// validation and return codes.
int verify_ex_impl(const void* x_draft, const void* mu_target, const void* mu_draft,
                   const float* sigma, int64_t sigma_stride_b, int B, int L, int64_t d, int dtype,
                   uint64_t seed, const uint64_t* seed_dev, int mode, const int32_t* L_eff,
                   const void* mu_target_bonus, const float* sigma_bonus, int residual_kind,
                   float omega, int32_t* accepted_len, void* y_out, float* log_ratio_out,
                   float* delta_norm_out, uint32_t* status_out, float* chain_aux_out,
                   void* workspace, size_t workspace_bytes, bool timed, void* stream,
                   bool overlap = false);

// Records a cudaError_t for sdv_last_cuda_error() (this host thread).
void set_last_cuda_error(int err);

// Largest number of mixture components of the analytic target.
constexpr int kSdvMaxComponents = SDV_MAX_COMPONENTS;

}  // namespace sdv
