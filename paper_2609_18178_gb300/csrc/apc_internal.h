// Launch plans shared by the host side of the C ABI and the kernels.
//
// A plan is a kernel parameter block (__grid_constant__, at most 32,764
// bytes): the chunk table is copied by the driver at launch, so nothing is
// staged in device memory and no allocation is needed.  Tables larger than
// one block are split over several launches that add into the same digests.
#pragma once

#include <stdint.h>

namespace apc {

constexpr int kThreads = 256;              // threads per CTA
constexpr int kVec = 8;                    // elements per thread-vector (16-byte bf16, 2 x 16-byte fp32)
constexpr int kCommitUnroll = 2;           // thread-vectors per thread per tile (commit)
constexpr int kDigestUnroll = 4;           // thread-vectors per thread per tile (digest)
constexpr uint64_t kCommitTile = (uint64_t)kThreads * kVec * kCommitUnroll;  // 4096 elements
constexpr uint64_t kDigestTile = (uint64_t)kThreads * kVec * kDigestUnroll;  // 8192 elements
constexpr uint32_t kScalarMode = 0xFFFFFFFFu;  // `head` value of an entry run without vectors

// One chunk-table entry of the commit kernel (64 bytes).
//   head: elements [0, head) are scalar, then 16-byte vectors of 8 elements
//         up to vec_end = head + 8 * floor((n - head) / 8), then a scalar tail;
//         kScalarMode when the five buffers are not mutually 16-byte aligned.
//   tile_begin: index of the entry's first tile in the launch's tile space.
//   key_base: global_offset mod 2^32 (the digest key of element 0).
struct CommitEntry {
  float *p, *m, *v;
  const uint16_t *g;
  uint16_t *w;
  uint64_t n;
  uint64_t tile_begin;
  uint32_t key_base;
  uint32_t head;
};

template <int MAXE>
struct CommitPlan {
  float h[8];            // b1, 1-b1, b2, 1-b2, eps, 1-lr*wd, lr/bc1, 1/sqrt(bc2)
  uint64_t total_tiles;
  uint32_t count;
  uint32_t pad_;
  CommitEntry e[MAXE];
};

constexpr int kCommitSmall = 16;
constexpr int kCommitLarge = 480;
static_assert(sizeof(CommitEntry) == 64, "entry layout");
static_assert(sizeof(CommitPlan<kCommitLarge>) <= 32764, "kernel parameter limit");

// One buffer of the digest kernel (32 bytes).
struct DigestEntry {
  const void *data;
  uint64_t n;
  uint64_t tile_begin;
  uint32_t key_base;
  uint8_t head;         // scalar elements before the first 16-byte vector (<= 7)
  uint8_t dtype;        // 0 fp32, 1 bf16
  uint8_t slot;
  uint8_t pad_;         // a single buffer always reaches 16-byte alignment within 7 elements
};

template <int MAXE>
struct DigestPlan {
  uint64_t total_tiles;
  uint32_t count;
  uint32_t pad_;
  DigestEntry e[MAXE];
};

constexpr int kDigestSmall = 16;
constexpr int kDigestLarge = 1000;
static_assert(sizeof(DigestEntry) == 32, "entry layout");
static_assert(sizeof(DigestPlan<kDigestLarge>) <= 32764, "kernel parameter limit");

// Launch wrappers (apc_commit.cu, apc_digest.cu).  They return a cudaError_t
// value and launch on `stream` with `grid` CTAs of kThreads threads.
int launch_commit_small(const CommitPlan<kCommitSmall> &plan, unsigned grid, void *stream,
                        unsigned long long *out);
int launch_commit_large(const CommitPlan<kCommitLarge> &plan, unsigned grid, void *stream,
                        unsigned long long *out);
int launch_digest_small(const DigestPlan<kDigestSmall> &plan, unsigned grid, void *stream,
                        unsigned long long *out);
int launch_digest_large(const DigestPlan<kDigestLarge> &plan, unsigned grid, void *stream,
                        unsigned long long *out);

// Resident CTAs per SM of each kernel (cudaOccupancyMaxActiveBlocksPerMultiprocessor).
int commit_blocks_per_sm(bool large, int *out);
int digest_blocks_per_sm(bool large, int *out);

}  // namespace apc
