// The fused committed-step kernel: AdamW over a chunk table of ragged
// tensors and the state digests, in one pass over HBM.  Two state layouts
// share the pipeline:
//  * F32State  -- fp32 master p and moments m, v, bf16 gradient g, and a bf16
//    working copy w of p'; four digests (p', m', v', w); 28 bytes per element
//    (p, m, v read and written, g read, w written).
//  * BF16State -- p, m, v kept in bf16 (the paper's setting, arxiv 2609.18178
//    Section IV-A "Workloads"): loaded exactly into binary32, updated in the
//    same fixed order, rounded once to bf16 (nearest even) at the store;
//    three digests (p', m', v'); 14 bytes per element.
// With ZERO (APC_COMMIT_ZERO_GRAD) each gradient tile is also overwritten
// with +0 once its copy has landed: 2 more bytes per element.
//
// Warp-specialized pipeline (one persistent CTA per SM by default):
//  * The producer warp walks the CTA's run of the launch's tiles (one
//    contiguous run per CTA; a tile is L::kTile elements of one entry's
//    16-byte aligned body: 4,864 for fp32 state, 10,368 for bf16 state)
//    and, for each, waits until a ring stage is free and issues four
//    bulk asynchronous copies -- p, m, v and g -- that complete on the
//    stage's "full" mbarrier.  Loads never occupy consumer registers, and up
//    to L::kStages tiles per CTA are in flight.
//  * With each stage the producer also writes a 48-byte descriptor (the
//    tile's first-element addresses in p, m, v, w, g, its element count and
//    first digest index) into shared memory before arming the stage, so the
//    consumers never search the chunk table themselves.
//  * The consumer warps (19 for fp32 state, 27 for bf16 state) wait for a
//    stage, read its descriptor and their elements from shared memory
//    (thread t of C takes the groups 4kC+4t..4kC+4t+3 for k < L::kGroups, 2
//    for fp32 state and 3 for bf16 state, so both the shared-memory reads and
//    the global stores are contiguous across the warp), release the
//    stage to the producer, then apply AdamW, store the results with
//    streaming stores, and fold the digest terms into 64-bit registers.
//  * Elements outside the aligned bodies (entry heads and tails under 8
//    elements, and entries whose buffers are not mutually 16-byte aligned)
//    are "scalar items", done afterwards by the consumers with a grid-stride
//    loop straight from global memory.
//  * At exit the CTA sums each digest (warp shuffles, shared memory) and adds
//    it into the caller's output with one 64-bit atomic; addition mod 2^64 is
//    order-free, so digests do not depend on grid size or table split.
//
// Every mbarrier wait is bounded (apc_tma.cuh).  A wait that gives up sets
// the translation unit's device status word, makes the CTA stop issuing and
// consuming, drains the copies already issued (bounded again) and returns.
#include <cuda_runtime.h>

#include <atomic>

#include "../../include/apc.h"
#include "apc_device.cuh"
#include "apc_internal.h"
#include "apc_tma.cuh"

namespace apc {
namespace {

__device__ unsigned int g_commit_status;

struct Acc {
  uint64_t p, m, v, w;
};

__device__ __forceinline__ uint64_t umin64(uint64_t a, uint64_t b) { return a < b ? a : b; }

__device__ __forceinline__ void fail_wait(int *abort_flag) {
  atomicOr(&g_commit_status, (unsigned)APC_ETIMEOUT);
  *(volatile int *)abort_flag = 1;
}

__device__ __forceinline__ uint32_t bf16_rne_bits(float x) {
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(x));
}

__device__ __forceinline__ float bf16_value(uint32_t h) { return __uint_as_float(h << 16); }

// Two binary32 values rounded to bf16 (nearest even) by one paired
// conversion, `lo` in the low half: each half equals bf16_rne_bits of its
// input for every non-NaN value.
// The bf16 layout rounds its three outputs this way, in pairs of elements
// (2.5% faster there); for the fp32 layout's single w per element pairing
// measured 0.2% slower, so it keeps one conversion per element.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t *>(&h);
}

// A consumer thread's output addresses in the current tile: element
// start + 4t of the entry (t the consumer index).  Group k of the thread then
// sits at a compile-time element offset k * 4 * L::kConsumers, which the
// stores carry as an immediate.
struct Dst {
  void *p, *m, *v;
  uint16_t *w, *g;
};

// What the consumers need of a stage's tile, written into shared memory by
// the producer before it arms the stage's "full" barrier (whose completion
// makes it visible to them): the addresses of the tile's first element in
// p, m, v, w and g, its element count and its first digest index.  The
// consumers then spend no instructions locating the tile in the chunk table.
struct __align__(16) StageDesc {
  uint8_t *p, *m, *v;
  uint16_t *w, *g;
  uint32_t cnt, G;
};
static_assert(sizeof(StageDesc) == 48, "three 16-byte shared-memory loads");

// A commit digest term.  With SHARED the caller has established that the
// whole group's terms share the top two bits of their incremented key high
// word (top_bits_shared) and passes them as `top`.
template <uint32_t K, bool SHARED>
__device__ __forceinline__ uint64_t cterm(uint32_t G, uint32_t bits, uint32_t one, uint32_t top) {
  if constexpr (SHARED) return digest_term<K>(G, bits, one, top);
  else return digest_term<K>(G, bits, one);
}

// The term of a 16-bit word (w, and the bf16 layout's p', m', v'): with the
// shared top bits, the 16-bit form digest_term_u16.
template <uint32_t K, bool SHARED>
__device__ __forceinline__ uint64_t hterm(uint32_t G, uint32_t bits, uint32_t one, uint32_t top) {
  if constexpr (SHARED) return digest_term_u16<K>(G, bits, one, top);
  else return digest_term<K>(G, bits, one);
}

// ------------------------------------------------------------ fp32 state

struct F32State {
  static constexpr uint32_t kES = 4;        // bytes per state element
  static constexpr int kDigests = 4;
  static constexpr int kConsumerWarps = kCommitConsumerWarps;
  static constexpr int kStages = kCommitStages;
  static constexpr int kConsumers = 32 * kConsumerWarps;
  static constexpr int kThreads = kConsumers + 32;  // + the producer warp
  static constexpr int kBoundThreads = kThreads > APC_COMMIT_BOUND_THREADS ? kThreads : APC_COMMIT_BOUND_THREADS;
  static constexpr int kGroups = kCommitGroups;
  static constexpr uint64_t kTile = kCommitTile;
  struct Regs {
    float4 p, m, v;
    uint2 g;
  };

  __device__ static void load(const uint8_t *st, uint32_t e, Regs &r) {
    r.p = *reinterpret_cast<const float4 *>(st + 4 * e);
    r.m = *reinterpret_cast<const float4 *>(st + 4 * (kTile + e));
    r.v = *reinterpret_cast<const float4 *>(st + 4 * (2 * kTile + e));
    r.g = *reinterpret_cast<const uint2 *>(st + 12 * kTile + 2 * e);
  }

  // Four consecutive elements at the compile-time element offset OFF from
  // the thread's output addresses, whose first element has digest index G.
  template <uint32_t OFF, bool PAIRED>
  __device__ static void compute_store(const Dst &d, uint32_t G, const Regs &r, const Scalars &s, Acc &a) {
    constexpr uint32_t off = OFF;
    float p[4] = {r.p.x, r.p.y, r.p.z, r.p.w};
    float m[4] = {r.m.x, r.m.y, r.m.z, r.m.w};
    float v[4] = {r.v.x, r.v.y, r.v.z, r.v.w};
    const uint32_t gw[4] = {r.g.x & 0xFFFFu, r.g.x >> 16, r.g.y & 0xFFFFu, r.g.y >> 16};
    uint32_t w[4];
    if constexpr (PAIRED) {
      adamw_pair(p[0], p[1], m[0], m[1], v[0], v[1], gw[0], gw[1], s, w[0], w[1]);
      adamw_pair(p[2], p[3], m[2], m[3], v[2], v[3], gw[2], gw[3], s, w[2], w[3]);
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) w[j] = adamw_element(p[j], m[j], v[j], gw[j], s);
    }
    __stcs(reinterpret_cast<float4 *>(static_cast<float *>(d.p) + off), make_float4(p[0], p[1], p[2], p[3]));
    __stcs(reinterpret_cast<float4 *>(static_cast<float *>(d.m) + off), make_float4(m[0], m[1], m[2], m[3]));
    __stcs(reinterpret_cast<float4 *>(static_cast<float *>(d.v) + off), make_float4(v[0], v[1], v[2], v[3]));
    __stcs(reinterpret_cast<uint2 *>(d.w + off), make_uint2(w[0] | (w[1] << 16), w[2] | (w[3] << 16)));
    // the group's keys are G + OFF .. G + OFF + 3
    const uint32_t B = G + (0x9E3779B9u + OFF);
    const uint32_t pb[4] = {__float_as_uint(p[0]), __float_as_uint(p[1]), __float_as_uint(p[2]), __float_as_uint(p[3])};
    const uint32_t mb[4] = {__float_as_uint(m[0]), __float_as_uint(m[1]), __float_as_uint(m[2]), __float_as_uint(m[3])};
    const uint32_t vb[4] = {__float_as_uint(v[0]), __float_as_uint(v[1]), __float_as_uint(v[2]), __float_as_uint(v[3])};
    if (top_bits_shared(B, 4)) {
      fold<OFF, true>(G, pb, mb, vb, w, s.one, B >> 30, a);
    } else {
      fold<OFF, false>(G, pb, mb, vb, w, s.one, 0, a);
    }
  }

  template <uint32_t OFF, bool SHARED>
  __device__ static void fold(uint32_t G, const uint32_t (&p)[4], const uint32_t (&m)[4], const uint32_t (&v)[4],
                              const uint32_t (&w)[4], uint32_t one, uint32_t top, Acc &a) {
    a.p += cterm<OFF, SHARED>(G, p[0], one, top) + cterm<OFF + 1, SHARED>(G, p[1], one, top);
    a.p += cterm<OFF + 2, SHARED>(G, p[2], one, top) + cterm<OFF + 3, SHARED>(G, p[3], one, top);
    a.m += cterm<OFF, SHARED>(G, m[0], one, top) + cterm<OFF + 1, SHARED>(G, m[1], one, top);
    a.m += cterm<OFF + 2, SHARED>(G, m[2], one, top) + cterm<OFF + 3, SHARED>(G, m[3], one, top);
    a.v += cterm<OFF, SHARED>(G, v[0], one, top) + cterm<OFF + 1, SHARED>(G, v[1], one, top);
    a.v += cterm<OFF + 2, SHARED>(G, v[2], one, top) + cterm<OFF + 3, SHARED>(G, v[3], one, top);
    a.w += hterm<OFF, SHARED>(G, w[0], one, top) + hterm<OFF + 1, SHARED>(G, w[1], one, top);
    a.w += hterm<OFF + 2, SHARED>(G, w[2], one, top) + hterm<OFF + 3, SHARED>(G, w[3], one, top);
  }

  __device__ static void one(const CommitEntry &E, uint64_t i, const Scalars &s, Acc &a) {
    float *P = static_cast<float *>(E.p), *M = static_cast<float *>(E.m), *V = static_cast<float *>(E.v);
    float p = P[i], m = M[i], v = V[i];
    const uint32_t w = adamw_element(p, m, v, (uint32_t)E.g[i], s);
    P[i] = p;
    M[i] = m;
    V[i] = v;
    E.w[i] = (uint16_t)w;
    const uint32_t G = E.key_base + (uint32_t)i;
    acc_add(a.p, digest_term(G, __float_as_uint(p), s.one), s.one);
    acc_add(a.m, digest_term(G, __float_as_uint(m), s.one), s.one);
    acc_add(a.v, digest_term(G, __float_as_uint(v), s.one), s.one);
    acc_add(a.w, digest_term(G, w, s.one), s.one);
  }
};

// ------------------------------------------------------------ bf16 state

struct BF16State {
  static constexpr uint32_t kES = 2;
  static constexpr int kDigests = 3;
  static constexpr int kConsumerWarps = kCommitConsumerWarpsBF16;
  static constexpr int kStages = kCommitStagesBF16;
  static constexpr int kConsumers = 32 * kConsumerWarps;
  static constexpr int kThreads = kConsumers + 32;
  static constexpr int kBoundThreads = kThreads;
  static constexpr int kGroups = kCommitGroupsBF16;
  static constexpr uint64_t kTile = kCommitTileBF16;
  struct Regs {
    uint2 p, m, v, g;
  };

  __device__ static void load(const uint8_t *st, uint32_t e, Regs &r) {
    r.p = *reinterpret_cast<const uint2 *>(st + 2 * e);
    r.m = *reinterpret_cast<const uint2 *>(st + 2 * (kTile + e));
    r.v = *reinterpret_cast<const uint2 *>(st + 2 * (2 * kTile + e));
    r.g = *reinterpret_cast<const uint2 *>(st + 6 * kTile + 2 * e);
  }

  template <uint32_t OFF, bool PAIRED>
  __device__ static void compute_store(const Dst &d, uint32_t G, const Regs &r, const Scalars &s, Acc &a) {
    constexpr uint32_t off = OFF;
    const uint32_t pw[4] = {r.p.x & 0xFFFFu, r.p.x >> 16, r.p.y & 0xFFFFu, r.p.y >> 16};
    const uint32_t mw[4] = {r.m.x & 0xFFFFu, r.m.x >> 16, r.m.y & 0xFFFFu, r.m.y >> 16};
    const uint32_t vw[4] = {r.v.x & 0xFFFFu, r.v.x >> 16, r.v.y & 0xFFFFu, r.v.y >> 16};
    const uint32_t gw[4] = {r.g.x & 0xFFFFu, r.g.x >> 16, r.g.y & 0xFFFFu, r.g.y >> 16};
    float pf[4], mf[4], vf[4];
    if constexpr (PAIRED) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        pf[j] = bf16_value(pw[j]);
        mf[j] = bf16_value(mw[j]);
        vf[j] = bf16_value(vw[j]);
      }
      uint32_t unused[4];
      adamw_pair(pf[0], pf[1], mf[0], mf[1], vf[0], vf[1], gw[0], gw[1], s, unused[0], unused[1]);
      adamw_pair(pf[2], pf[3], mf[2], mf[3], vf[2], vf[3], gw[2], gw[3], s, unused[2], unused[3]);
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        pf[j] = bf16_value(pw[j]);
        mf[j] = bf16_value(mw[j]);
        vf[j] = bf16_value(vw[j]);
        (void)adamw_element(pf[j], mf[j], vf[j], gw[j], s);
      }
    }
    const uint32_t p01 = pack_bf16x2(pf[0], pf[1]), p23 = pack_bf16x2(pf[2], pf[3]);
    const uint32_t m01 = pack_bf16x2(mf[0], mf[1]), m23 = pack_bf16x2(mf[2], mf[3]);
    const uint32_t v01 = pack_bf16x2(vf[0], vf[1]), v23 = pack_bf16x2(vf[2], vf[3]);
    __stcs(reinterpret_cast<uint2 *>(static_cast<uint16_t *>(d.p) + off), make_uint2(p01, p23));
    __stcs(reinterpret_cast<uint2 *>(static_cast<uint16_t *>(d.m) + off), make_uint2(m01, m23));
    __stcs(reinterpret_cast<uint2 *>(static_cast<uint16_t *>(d.v) + off), make_uint2(v01, v23));
    const uint32_t po[4] = {p01 & 0xFFFFu, p01 >> 16, p23 & 0xFFFFu, p23 >> 16};
    const uint32_t mo[4] = {m01 & 0xFFFFu, m01 >> 16, m23 & 0xFFFFu, m23 >> 16};
    const uint32_t vo[4] = {v01 & 0xFFFFu, v01 >> 16, v23 & 0xFFFFu, v23 >> 16};
    const uint32_t B = G + (0x9E3779B9u + OFF);  // the group's keys are G + OFF .. G + OFF + 3
    if (top_bits_shared(B, 4)) {
      fold<OFF, true>(G, po, mo, vo, s.one, B >> 30, a);
    } else {
      fold<OFF, false>(G, po, mo, vo, s.one, 0, a);
    }
  }

  template <uint32_t OFF, bool SHARED>
  __device__ static void fold(uint32_t G, const uint32_t (&p)[4], const uint32_t (&m)[4], const uint32_t (&v)[4],
                              uint32_t one, uint32_t top, Acc &a) {
    a.p += hterm<OFF, SHARED>(G, p[0], one, top) + hterm<OFF + 1, SHARED>(G, p[1], one, top);
    a.p += hterm<OFF + 2, SHARED>(G, p[2], one, top) + hterm<OFF + 3, SHARED>(G, p[3], one, top);
    a.m += hterm<OFF, SHARED>(G, m[0], one, top) + hterm<OFF + 1, SHARED>(G, m[1], one, top);
    a.m += hterm<OFF + 2, SHARED>(G, m[2], one, top) + hterm<OFF + 3, SHARED>(G, m[3], one, top);
    a.v += hterm<OFF, SHARED>(G, v[0], one, top) + hterm<OFF + 1, SHARED>(G, v[1], one, top);
    a.v += hterm<OFF + 2, SHARED>(G, v[2], one, top) + hterm<OFF + 3, SHARED>(G, v[3], one, top);
  }

  __device__ static void one(const CommitEntry &E, uint64_t i, const Scalars &s, Acc &a) {
    uint16_t *P = static_cast<uint16_t *>(E.p), *M = static_cast<uint16_t *>(E.m), *V = static_cast<uint16_t *>(E.v);
    float p = bf16_value(P[i]), m = bf16_value(M[i]), v = bf16_value(V[i]);
    const uint32_t po = adamw_element(p, m, v, (uint32_t)E.g[i], s);
    const uint32_t mo = bf16_rne_bits(m), vo = bf16_rne_bits(v);
    P[i] = (uint16_t)po;
    M[i] = (uint16_t)mo;
    V[i] = (uint16_t)vo;
    const uint32_t G = E.key_base + (uint32_t)i;
    acc_add(a.p, digest_term(G, po, s.one), s.one);
    acc_add(a.m, digest_term(G, mo, s.one), s.one);
    acc_add(a.v, digest_term(G, vo, s.one), s.one);
  }
};

// Group K of a consumer thread's tile: its elements sit at the compile-time
// offset K * 4 * L::kConsumers from the thread's output addresses, which
// the stores carry as immediates and the digest terms fold into their
// increment.
template <class L, bool ZERO, int K>
__device__ __forceinline__ void store_groups(const Dst &d, uint32_t G1, const typename L::Regs *r, const bool *ok,
                                             const Scalars &s, Acc &a) {
  constexpr uint32_t off = (uint32_t)(K * L::kConsumers) * 4;
  if (ok[K]) {
    if (ZERO) __stcs(reinterpret_cast<uint2 *>(d.g + off), make_uint2(0u, 0u));
    // the gradient-zeroing pass is bound by its 30 bytes per element, and the
    // packed multiplies measured slower there (33.9 against 33.5 ms on the
    // full model): it keeps one element at a time
    L::template compute_store<off, APC_PAIRED_ADAMW != 0 && !ZERO>(d, G1, r[K], s, a);
  }
  if constexpr (K + 1 < L::kGroups) store_groups<L, ZERO, K + 1>(d, G1, r, ok, s, a);
}

template <class L>
__host__ __device__ constexpr uint32_t stage_bytes() {
  return (uint32_t)L::kTile * (3 * L::kES + 2);
}

template <class L>
__host__ __device__ constexpr uint32_t smem_bytes() {
  return (uint32_t)L::kStages * stage_bytes<L>();
}

static_assert(smem_bytes<F32State>() <= 227 * 1024 && smem_bytes<BF16State>() <= 227 * 1024, "shared memory per CTA");

template <int MAXE>
__device__ __forceinline__ uint32_t find_tile(const CommitPlan<MAXE> &plan, uint32_t cur, uint64_t tile) {
  while (cur + 1 < plan.count && tile >= plan.e[cur + 1].tile_begin) ++cur;
  return cur;
}

// This CTA's tiles: tile = t0, t0 + ts, ... while tile < t1 (the same walk
// for the producer and the consumers).
struct TileWalk {
  uint64_t t0, t1, ts;
};
__device__ __forceinline__ TileWalk tile_walk(uint64_t total) {
  const uint64_t b = blockIdx.x;
  if (APC_COMMIT_CONTIGUOUS) {
    const uint64_t per = total / gridDim.x, rem = total % gridDim.x;
    const uint64_t t0 = b * per + (b < rem ? b : rem);
    return {t0, t0 + per + (b < rem ? 1 : 0), 1};
  }
  return {b, total, gridDim.x};
}

template <class L, int MAXE, bool ZERO>
__global__ void __launch_bounds__(L::kBoundThreads, kCommitBlocksPerSm)
    commit_kernel(const __grid_constant__ CommitPlan<MAXE> plan, unsigned long long *out) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ __align__(8) uint64_t full[L::kStages];
  __shared__ __align__(8) uint64_t empty[L::kStages];
  __shared__ StageDesc desc[L::kStages];
  __shared__ uint64_t red[L::kThreads / 32];
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < L::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], L::kConsumerWarps);
    }
    abort_flag = 0;
    mbar_init_fence();
  }
  __syncthreads();

  Acc a{0, 0, 0, 0};
  if (warp == L::kConsumerWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t policy = l2_evict_first();
      uint32_t cur = 0, phase = 0;
      int stage = 0;
      uint64_t issued = 0;
      const TileWalk w = tile_walk(plan.total_tiles);
      for (uint64_t tile = w.t0; tile < w.t1; tile += w.ts) {
        if (*(volatile int *)&abort_flag) break;
        cur = find_tile(plan, cur, tile);
        const CommitEntry &E = plan.e[cur];
        const uint64_t start = E.head + (tile - E.tile_begin) * L::kTile;
        const uint64_t vec_end = E.head + ((E.n - E.head) & ~(uint64_t)7);
        const uint32_t cnt = (uint32_t)umin64(L::kTile, vec_end - start);
        if (!mbar_wait(&empty[stage], phase ^ 1)) {
          fail_wait(&abort_flag);
          break;
        }
        uint8_t *st = smem + (size_t)stage * stage_bytes<L>();
        desc[stage] = StageDesc{static_cast<uint8_t *>(E.p) + start * L::kES,
                                static_cast<uint8_t *>(E.m) + start * L::kES,
                                static_cast<uint8_t *>(E.v) + start * L::kES,
                                L::kDigests == 4 ? E.w + start : nullptr,
                                const_cast<uint16_t *>(E.g) + start,
                                cnt,
                                E.key_base + (uint32_t)start};
        mbar_arrive_expect_tx(&full[stage], cnt * (3 * L::kES + 2));
        bulk_g2s(st, static_cast<const uint8_t *>(E.p) + start * L::kES, cnt * L::kES, &full[stage], policy);
        bulk_g2s(st + L::kES * L::kTile, static_cast<const uint8_t *>(E.m) + start * L::kES, cnt * L::kES,
                 &full[stage], policy);
        bulk_g2s(st + 2 * L::kES * L::kTile, static_cast<const uint8_t *>(E.v) + start * L::kES,
                 cnt * L::kES, &full[stage], policy);
        bulk_g2s(st + 3 * L::kES * L::kTile, E.g + start, cnt * 2, &full[stage], policy);
        ++issued;
        if (++stage == L::kStages) {
          stage = 0;
          phase ^= 1;
        }
      }
      // Drain: the last min(issued, stages) copies must have landed before
      // the CTA may exit (normally the consumers already waited for them).
      const int n_drain = (int)umin64(issued, (uint64_t)L::kStages);
      for (int k = 0; k < n_drain; ++k) {
        if (--stage < 0) {
          stage = L::kStages - 1;
          phase ^= 1;
        }
        if (!mbar_wait(&full[stage], phase)) atomicOr(&g_commit_status, (unsigned)APC_ETIMEOUT);
      }
    }
    __syncwarp();
  } else {
    // ----------------------------------------------------------- consumers
    const Scalars s{plan.h, plan.one};
    const int ct = threadIdx.x;  // 0 .. L::kConsumers-1
    uint32_t phase = 0;
    int stage = 0;
    const TileWalk w = tile_walk(plan.total_tiles);
    for (uint64_t tile = w.t0; tile < w.t1; tile += w.ts) {
      if (!mbar_wait(&full[stage], phase)) {
        fail_wait(&abort_flag);
        break;
      }
      if (*(volatile int *)&abort_flag) break;
      const StageDesc sd = desc[stage];
      const uint8_t *st = smem + (size_t)stage * stage_bytes<L>();
      typename L::Regs r[L::kGroups];
      bool ok[L::kGroups];
#pragma unroll
      for (int k = 0; k < L::kGroups; ++k) {
        const uint32_t e = (uint32_t)(k * L::kConsumers + ct) * 4;
        ok[k] = e < sd.cnt;
        if (ok[k]) L::load(st, e, r[k]);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[stage]);
      // this thread's first element in the tile is element 4 * ct
      const uint32_t ob = 4u * (uint32_t)ct;
      const Dst d{sd.p + ob * L::kES, sd.m + ob * L::kES, sd.v + ob * L::kES,
                  L::kDigests == 4 ? sd.w + ob : nullptr, sd.g + ob};
      store_groups<L, ZERO, 0>(d, sd.G + ob, r, ok, s, a);
      if (++stage == L::kStages) {
        stage = 0;
        phase ^= 1;
      }
    }
    // scalar items: entry heads and tails, and entries without vectors
    if (!*(volatile int *)&abort_flag) {
      uint32_t cur = 0;
      for (uint64_t it = (uint64_t)blockIdx.x * L::kConsumers + ct; it < plan.total_scalar;
           it += (uint64_t)gridDim.x * L::kConsumers) {
        while (cur + 1 < plan.count && it >= plan.e[cur + 1].scalar_begin) ++cur;
        const CommitEntry &E = plan.e[cur];
        const uint64_t k = it - E.scalar_begin;
        uint64_t i;
        if (E.head == kScalarMode) {
          i = k;
        } else {
          const uint64_t vec_end = E.head + ((E.n - E.head) & ~(uint64_t)7);
          i = k < E.head ? k : vec_end + (k - E.head);
        }
        L::one(E, i, s, a);
        if (ZERO) const_cast<uint16_t *>(E.g)[i] = 0;
      }
    }
  }

  const bool ok = !*(volatile int *)&abort_flag;
  uint64_t r;
  r = cta_sum<L::kThreads>(a.p, red);
  if (threadIdx.x == 0 && ok && r) atomicAdd(&out[0], (unsigned long long)r);
  r = cta_sum<L::kThreads>(a.m, red);
  if (threadIdx.x == 0 && ok && r) atomicAdd(&out[1], (unsigned long long)r);
  r = cta_sum<L::kThreads>(a.v, red);
  if (threadIdx.x == 0 && ok && r) atomicAdd(&out[2], (unsigned long long)r);
  if (L::kDigests == 4) {
    r = cta_sum<L::kThreads>(a.w, red);
    if (threadIdx.x == 0 && ok && r) atomicAdd(&out[3], (unsigned long long)r);
  }
}

// One thread waits on an mbarrier that nothing completes: the bounded wait
// must give up after `limit_ns` and record APC_ETIMEOUT.
__global__ void wait_timeout_kernel(uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  mbar_init(&bar, 1);
  mbar_init_fence();
  if (!mbar_wait(&bar, 0, limit_ns)) atomicOr(&g_commit_status, (unsigned)APC_ETIMEOUT);
}

// The dynamic shared-memory limit of one kernel instantiation, raised once
// per device (the first launch on a device sets it; later launches, for
// example inside a stream capture, only enqueue).
template <class L, int MAXE, bool ZERO>
int ensure_smem_attribute() {
  static std::atomic<uint64_t> done_mask{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return (int)e;
  const uint64_t bit = dev < 64 ? (1ull << dev) : 0;
  if (bit && (done_mask.load(std::memory_order_acquire) & bit)) return 0;
  e = cudaFuncSetAttribute(commit_kernel<L, MAXE, ZERO>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem_bytes<L>());
  if (e != cudaSuccess) return (int)e;
  if (APC_SMEM_CARVEOUT >= 0) {
    e = cudaFuncSetAttribute(commit_kernel<L, MAXE, ZERO>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             APC_SMEM_CARVEOUT);
    if (e != cudaSuccess) return (int)e;
  }
  if (bit) done_mask.fetch_or(bit, std::memory_order_acq_rel);
  return 0;
}

template <class L, int MAXE, bool ZERO>
int launch_t(const CommitPlan<MAXE> &plan, unsigned grid, void *stream, unsigned long long *out) {
  int e = ensure_smem_attribute<L, MAXE, ZERO>();
  if (e) return e;
  commit_kernel<L, MAXE, ZERO><<<grid, L::kThreads, smem_bytes<L>(), (cudaStream_t)stream>>>(plan, out);
  return (int)cudaGetLastError();
}

template <int MAXE>
int launch(const CommitPlan<MAXE> &plan, int layout, bool zero_grad, unsigned grid, void *stream,
           unsigned long long *out) {
  if (layout == kLayoutBF16)
    return zero_grad ? launch_t<BF16State, MAXE, true>(plan, grid, stream, out)
                     : launch_t<BF16State, MAXE, false>(plan, grid, stream, out);
  return zero_grad ? launch_t<F32State, MAXE, true>(plan, grid, stream, out)
                   : launch_t<F32State, MAXE, false>(plan, grid, stream, out);
}

template <class L, int MAXE>
int blocks_per_sm(int *out) {
  int e = ensure_smem_attribute<L, MAXE, false>();
  if (e) return e;
  return (int)cudaOccupancyMaxActiveBlocksPerMultiprocessor(out, commit_kernel<L, MAXE, false>, L::kThreads,
                                                            smem_bytes<L>());
}

}  // namespace

int launch_commit_small(const CommitPlan<kCommitSmall> &plan, int layout, bool zero_grad, unsigned grid,
                        void *stream, unsigned long long *out) {
  return launch(plan, layout, zero_grad, grid, stream, out);
}

int launch_commit_large(const CommitPlan<kCommitLarge> &plan, int layout, bool zero_grad, unsigned grid,
                        void *stream, unsigned long long *out) {
  return launch(plan, layout, zero_grad, grid, stream, out);
}

int commit_blocks_per_sm(bool large, int *out) {
  // one grid size serves both layouts: the smaller of their residencies
  int f = 0, b = 0;
  int e = large ? blocks_per_sm<F32State, kCommitLarge>(&f) : blocks_per_sm<F32State, kCommitSmall>(&f);
  if (e) return e;
  e = large ? blocks_per_sm<BF16State, kCommitLarge>(&b) : blocks_per_sm<BF16State, kCommitSmall>(&b);
  if (e) return e;
  *out = f < b ? f : b;
  return 0;
}

int launch_wait_timeout(uint64_t limit_ns, void *stream) {
  wait_timeout_kernel<<<1, 1, 0, (cudaStream_t)stream>>>(limit_ns);
  return (int)cudaGetLastError();
}

int read_commit_status(unsigned *out) {
  cudaError_t e = cudaMemcpyFromSymbol(out, g_commit_status, sizeof(unsigned));
  if (e != cudaSuccess) return (int)e;
  const unsigned zero = 0;
  return (int)cudaMemcpyToSymbol(g_commit_status, &zero, sizeof(unsigned));
}

}  // namespace apc
