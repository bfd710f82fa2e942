// Host side of the C ABI declared in include/apc.h: argument validation,
// resolution of the step's binary32 scalars (in double, rounded once),
// conversion of chunk tables, buffer lists and upload segments into launch
// plans, the persistent grid sizes (SM count x residency, less the SMs
// reserved with apc_set_reserved_sms), and the launches.
//
// The library allocates nothing.  Each plan travels in the kernel's
// parameter block; the digests are accumulated with atomics straight into
// the caller's output, which is zeroed on the stream first.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <memory>
#include <mutex>
#include <vector>

#include "../../include/apc.h"
#include "apc_internal.h"

#define APC_EXPORT extern "C" __attribute__((visibility("default")))

namespace {

thread_local char g_last_error[512] = "";

apc_status fail(apc_status s, const char *fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof g_last_error, fmt, ap);
  va_end(ap);
  return s;
}

apc_status cuda_fail(int err, const char *what) {
  return fail(APC_ECUDA, "%s: %s", what, cudaGetErrorString((cudaError_t)err));
}

// Scalars of step t (see apc_resolve_hparams).
apc_status resolve(const apc_adamw_hparams *hp, int64_t step, float out[8]) {
  if (!hp) return fail(APC_EINVAL, "hparams pointer is null");
  if (step < 1) return fail(APC_EINVAL, "step %lld < 1", (long long)step);
  const double lr = hp->lr, b1 = hp->beta1, b2 = hp->beta2, eps = hp->eps, wd = hp->weight_decay;
  if (!std::isfinite(lr) || !std::isfinite(b1) || !std::isfinite(b2) || !std::isfinite(eps) || !std::isfinite(wd))
    return fail(APC_EINVAL, "non-finite hyper-parameter");
  if (!(b1 >= 0.0 && b1 < 1.0) || !(b2 >= 0.0 && b2 < 1.0)) return fail(APC_EINVAL, "beta outside [0, 1)");
  if (!(eps > 0.0)) return fail(APC_EINVAL, "eps must be > 0");
  if (lr < 0.0 || wd < 0.0) return fail(APC_EINVAL, "lr and weight_decay must be >= 0");
  // bias corrections in double; each scalar rounded once to binary32
  const double bc1 = 1.0 - std::pow(b1, (double)step);
  const double bc2 = 1.0 - std::pow(b2, (double)step);
  out[0] = (float)b1;
  out[1] = (float)(1.0 - b1);
  out[2] = (float)b2;
  out[3] = (float)(1.0 - b2);
  out[4] = (float)eps;
  out[5] = (float)(1.0 - lr * wd);
  out[6] = (float)(lr / bc1);
  out[7] = (float)(1.0 / std::sqrt(bc2));
  return APC_OK;
}

struct Range {
  uintptr_t lo, hi;  // [lo, hi)
  bool written;
};

// Written ranges must be pairwise disjoint and disjoint from read ranges.
bool overlaps(std::vector<Range> &r) {
  std::sort(r.begin(), r.end(), [](const Range &a, const Range &b) { return a.lo < b.lo; });
  uintptr_t hi_any = 0, hi_written = 0;
  bool have_any = false, have_written = false;
  for (const Range &x : r) {
    if (have_written && x.lo < hi_written) return true;
    if (x.written && have_any && x.lo < hi_any) return true;
    if (!have_any || x.hi > hi_any) hi_any = x.hi;
    have_any = true;
    if (x.written) {
      if (!have_written || x.hi > hi_written) hi_written = x.hi;
      have_written = true;
    }
  }
  return false;
}

struct Device {
  int sms = 0;
  int commit_small = 0, commit_large = 0, digest_small = 0, digest_large = 0, count_small = 0, count_large = 0;
};

constexpr int kMaxDevices = 64;
Device g_devices[kMaxDevices];
std::atomic<bool> g_device_ready[kMaxDevices];
std::mutex g_device_mu;

// SM count and occupancy of the current device, queried once per device.
apc_status device_info(Device *out) {
  int dev = 0;
  int e = (int)cudaGetDevice(&dev);
  if (e) return cuda_fail(e, "cudaGetDevice");
  if (dev >= 0 && dev < kMaxDevices && g_device_ready[dev].load(std::memory_order_acquire)) {
    *out = g_devices[dev];
    return APC_OK;
  }
  Device dd, *d = &dd;
  e = (int)cudaDeviceGetAttribute(&d->sms, cudaDevAttrMultiProcessorCount, dev);
  if (e) return cuda_fail(e, "cudaDeviceGetAttribute");
  if ((e = apc::commit_blocks_per_sm(false, &d->commit_small))) return cuda_fail(e, "occupancy query");
  if ((e = apc::commit_blocks_per_sm(true, &d->commit_large))) return cuda_fail(e, "occupancy query");
  if ((e = apc::digest_blocks_per_sm(false, &d->digest_small))) return cuda_fail(e, "occupancy query");
  if ((e = apc::digest_blocks_per_sm(true, &d->digest_large))) return cuda_fail(e, "occupancy query");
  if ((e = apc::count_blocks_per_sm(false, &d->count_small))) return cuda_fail(e, "occupancy query");
  if ((e = apc::count_blocks_per_sm(true, &d->count_large))) return cuda_fail(e, "occupancy query");
  if (dev >= 0 && dev < kMaxDevices) {
    std::lock_guard<std::mutex> lock(g_device_mu);
    if (!g_device_ready[dev].load(std::memory_order_relaxed)) {
      g_devices[dev] = dd;
      g_device_ready[dev].store(true, std::memory_order_release);
    }
  }
  *out = dd;
  return APC_OK;
}

// SMs that the persistent kernels leave free (apc_set_reserved_sms).
std::atomic<int> g_reserved_sms{0};

// The persistent grid: one CTA per resident slot on the SMs not reserved
// (at least one SM's worth), capped by APC_GRID_LIMIT (read at every call)
// when that is a positive integer.
unsigned grid_for(uint64_t tiles, int sms, int per_sm) {
  const int avail = std::max(1, sms - g_reserved_sms.load(std::memory_order_relaxed));
  uint64_t cap = (uint64_t)avail * (uint64_t)std::max(per_sm, 1);
  if (const char *lim = std::getenv("APC_GRID_LIMIT")) {
    char *end = nullptr;
    const unsigned long long v = std::strtoull(lim, &end, 10);
    if (end != lim && *end == 0 && v > 0) cap = std::min<uint64_t>(cap, v);
  }
  return (unsigned)std::max<uint64_t>(1, std::min(tiles, cap));
}

// A pointer that a kernel will dereference, with what it is for the error
// message: `list` ("table", "bufs", "out"), entry index and field name.
struct Owned {
  const void *p;
  const char *list;
  int index;
  const char *field;
};

// Every buffer a kernel reads or writes must be memory of the calling
// thread's current device (or managed memory): a pointer into another GPU's
// memory, or host memory, would otherwise be dereferenced by this device's
// copies.  One attribute query per distinct address.  Returns APC_ECUDA if
// the runtime cannot answer (for example, no device) and APC_EINVAL naming the
// first foreign pointer (lowest address first).
apc_status check_device_pointers(std::vector<Owned> &ptrs) {
  if (ptrs.empty()) return APC_OK;
  int dev = 0;
  int e = (int)cudaGetDevice(&dev);
  if (e) return cuda_fail(e, "cudaGetDevice");
  std::sort(ptrs.begin(), ptrs.end(), [](const Owned &a, const Owned &b) { return a.p < b.p; });
  const void *last = nullptr;
  for (const Owned &o : ptrs) {
    if (o.p == last) continue;
    last = o.p;
    cudaPointerAttributes a;
    e = (int)cudaPointerGetAttributes(&a, o.p);
    if (e) {
      cudaGetLastError();  // clear the runtime's error state of the failed query
      return cuda_fail(e, "cudaPointerGetAttributes");
    }
    const bool own = (a.type == cudaMemoryTypeDevice && a.device == dev) || a.type == cudaMemoryTypeManaged;
    if (!own) {
      if (o.index >= 0)
        return fail(APC_EINVAL, "%s[%d].%s is not memory of the current device %d (memory type %d, device %d)",
                    o.list, o.index, o.field, dev, (int)a.type, a.device);
      return fail(APC_EINVAL, "%s is not memory of the current device %d (memory type %d, device %d)", o.list, dev,
                  (int)a.type, a.device);
    }
  }
  return APC_OK;
}

// Entries arrive with their tile count in tile_begin and their scalar-item
// count in scalar_begin; each batch turns both into prefix offsets.
template <int MAXE, typename Launch>
apc_status run_commit_batches(const std::vector<apc::CommitEntry> &entries, const float h[8], int layout,
                              bool zero_grad, unsigned grid_cap, void *stream, unsigned long long *out,
                              Launch launch) {
  auto plan = std::make_unique<apc::CommitPlan<MAXE>>();
  std::memcpy(plan->h, h, sizeof plan->h);
  plan->one = 1;
  size_t i = 0;
  while (i < entries.size()) {
    const size_t k = std::min(entries.size() - i, (size_t)MAXE);
    uint64_t tiles = 0, scalars = 0;
    for (size_t j = 0; j < k; ++j) {
      apc::CommitEntry e = entries[i + j];
      const uint64_t t = e.tile_begin, sc = e.scalar_begin;
      e.tile_begin = tiles;
      e.scalar_begin = scalars;
      tiles += t;
      scalars += sc;
      plan->e[j] = e;
    }
    plan->count = (uint32_t)k;
    plan->total_tiles = tiles;
    plan->total_scalar = scalars;
    const uint64_t consumers = (uint64_t)apc::commit_consumers(layout);
    const uint64_t want = std::max<uint64_t>(tiles, (scalars + consumers - 1) / consumers);
    const unsigned grid = (unsigned)std::max<uint64_t>(1, std::min<uint64_t>(want, grid_cap));
    int e = launch(*plan, layout, zero_grad, grid, stream, out);
    if (e) return cuda_fail(e, "commit kernel launch");
    i += k;
  }
  return APC_OK;
}

template <int MAXE, typename Launch>
apc_status run_digest_batches(const std::vector<apc::DigestEntry> &entries, unsigned grid_cap, void *stream,
                              unsigned long long *out, Launch launch, const char *what) {
  auto plan = std::make_unique<apc::DigestPlan<MAXE>>();
  plan->one = 1;
  size_t i = 0;
  while (i < entries.size()) {
    const size_t k = std::min(entries.size() - i, (size_t)MAXE);
    uint64_t tiles = 0;
    for (size_t j = 0; j < k; ++j) {
      apc::DigestEntry e = entries[i + j];
      const uint64_t t = e.tile_begin;  // holds the entry's tile count until placed
      e.tile_begin = tiles;
      tiles += t;
      plan->e[j] = e;
    }
    plan->count = (uint32_t)k;
    plan->total_tiles = tiles;
    const unsigned grid = (unsigned)std::max<uint64_t>(1, std::min<uint64_t>(tiles, grid_cap));
    int e = launch(*plan, grid, stream, out);
    if (e) return cuda_fail(e, what);
    i += k;
  }
  return APC_OK;
}

uint64_t ceil_div(uint64_t a, uint64_t b) { return a / b + (a % b != 0); }

}  // namespace

APC_EXPORT apc_status apc_resolve_hparams(const apc_adamw_hparams *hp, int64_t step, float out[8]) {
  g_last_error[0] = 0;
  if (!out) return fail(APC_EINVAL, "output pointer is null");
  return resolve(hp, step, out);
}

namespace {

// One table entry in layout-neutral form.
struct TableRow {
  void *p, *m, *v;
  const uint16_t *g;
  uint16_t *w;  // null for the bf16 layout
  uint64_t n, goff;
};

// Shared by both layouts: validation, scalar resolution, overlap check,
// planning and launches.  nslots digests are zeroed and accumulated.
apc_status commit_common(int layout, const std::vector<TableRow> &rows, const apc_adamw_hparams *hp, int64_t step,
                         uint32_t flags, apc_stream_t stream, uint64_t *out_digests, int nslots) {
  if (flags & ~(uint32_t)APC_COMMIT_ZERO_GRAD) return fail(APC_EINVAL, "unknown flag bits 0x%x", flags);
  const bool zero_grad = (flags & APC_COMMIT_ZERO_GRAD) != 0;
  if (!out_digests) return fail(APC_EINVAL, "out_digests pointer is null");
  if ((uintptr_t)out_digests % 8) return fail(APC_EALIGN, "out_digests not 8-byte aligned");
  float h[8];
  apc_status st = resolve(hp, step, h);
  if (st != APC_OK) return st;
  const uint64_t es = layout == apc::kLayoutF32 ? 4 : 2;  // bytes per state element

  std::vector<apc::CommitEntry> entries;
  std::vector<Range> ranges;
  std::vector<Owned> owned;
  entries.reserve(rows.size());
  ranges.reserve(rows.size() * 5 + 1);
  owned.reserve(rows.size() * 5 + 1);
  for (size_t k = 0; k < rows.size(); ++k) {
    const TableRow &t = rows[k];
    if (t.n == 0) continue;
    if (!t.p || !t.m || !t.v || !t.g || (layout == apc::kLayoutF32 && !t.w))
      return fail(APC_EINVAL, "table[%zu]: null buffer pointer", k);
    if (t.n > (UINT64_MAX - t.goff)) return fail(APC_ERANGE, "table[%zu]: global_offset + n overflows", k);
    if (t.n > ((uint64_t)1 << 61)) return fail(APC_ERANGE, "table[%zu]: n too large", k);
    const uintptr_t p = (uintptr_t)t.p, m = (uintptr_t)t.m, v = (uintptr_t)t.v, g = (uintptr_t)t.g,
                    w = (uintptr_t)t.w;
    if (p % es || m % es || v % es)
      return fail(APC_EALIGN, "table[%zu]: state buffer not %u-byte aligned", k, (unsigned)es);
    if (g % 2 || w % 2) return fail(APC_EALIGN, "table[%zu]: bf16 buffer not 2-byte aligned", k);
    ranges.push_back({p, p + es * t.n, true});
    ranges.push_back({m, m + es * t.n, true});
    ranges.push_back({v, v + es * t.n, true});
    if (t.w) ranges.push_back({w, w + 2 * t.n, true});
    ranges.push_back({g, g + 2 * t.n, zero_grad});
    const int ki = (int)k;
    owned.push_back({t.p, "table", ki, "p"});
    owned.push_back({t.m, "table", ki, "m"});
    owned.push_back({t.v, "table", ki, "v"});
    owned.push_back({t.g, "table", ki, "g"});
    if (t.w) owned.push_back({t.w, "table", ki, "w"});
    // first element at which all buffers sit on a 16-byte boundary
    const uint64_t h0 = ((16 - g % 16) % 16) / 2;
    const bool aligned = (p + es * h0) % 16 == 0 && (m + es * h0) % 16 == 0 && (v + es * h0) % 16 == 0 &&
                         (!t.w || (w + 2 * h0) % 16 == 0);
    apc::CommitEntry e;
    e.p = t.p;
    e.m = t.m;
    e.v = t.v;
    e.g = t.g;
    e.w = t.w;
    e.n = t.n;
    e.key_base = (uint32_t)t.goff;
    if (aligned) {
      const uint64_t head = std::min<uint64_t>(h0, t.n);
      const uint64_t body = (t.n - head) / apc::kVec * apc::kVec;
      e.head = (uint32_t)head;
      e.tile_begin = ceil_div(body, apc::commit_tile(layout));  // tile count until placed
      e.scalar_begin = t.n - body;                       // head + tail items
    } else {
      e.head = apc::kScalarMode;
      e.tile_begin = 0;
      e.scalar_begin = t.n;
    }
    entries.push_back(e);
  }
  const uintptr_t o = (uintptr_t)out_digests;
  ranges.push_back({o, o + (uintptr_t)nslots * sizeof(uint64_t), true});
  if (overlaps(ranges))
    return fail(APC_EINVAL, "table buffers or out_digests overlap (a written range meets another range)");
  owned.push_back({out_digests, "out_digests", -1, ""});
  if ((st = check_device_pointers(owned)) != APC_OK) return st;

  int e = (int)cudaMemsetAsync(out_digests, 0, (size_t)nslots * sizeof(uint64_t), (cudaStream_t)stream);
  if (e) return cuda_fail(e, "cudaMemsetAsync(out_digests)");
  if (entries.empty()) return APC_OK;
  Device d;
  if ((st = device_info(&d)) != APC_OK) return st;
  unsigned long long *out = reinterpret_cast<unsigned long long *>(out_digests);
  if (entries.size() <= (size_t)apc::kCommitSmall)
    return run_commit_batches<apc::kCommitSmall>(entries, h, layout, zero_grad,
                                                 grid_for(UINT64_MAX, d.sms, d.commit_small), stream, out,
                                                 apc::launch_commit_small);
  return run_commit_batches<apc::kCommitLarge>(entries, h, layout, zero_grad,
                                               grid_for(UINT64_MAX, d.sms, d.commit_large), stream, out,
                                               apc::launch_commit_large);
}

}  // namespace

APC_EXPORT apc_status apc_commit_step_ex(const apc_tensor *table, int32_t num_tensors,
                                         const apc_adamw_hparams *hp, int64_t step, uint32_t flags,
                                         apc_stream_t stream, uint64_t *out_digests) {
  g_last_error[0] = 0;
  if (num_tensors < 0) return fail(APC_EINVAL, "num_tensors %d < 0", num_tensors);
  if (num_tensors > 0 && !table) return fail(APC_EINVAL, "table pointer is null");
  std::vector<TableRow> rows((size_t)num_tensors);
  for (int32_t k = 0; k < num_tensors; ++k)
    rows[k] = TableRow{table[k].p, table[k].m, table[k].v, table[k].g, table[k].w, table[k].n,
                       table[k].global_offset};
  return commit_common(apc::kLayoutF32, rows, hp, step, flags, stream, out_digests, 4);
}

APC_EXPORT apc_status apc_commit_step(const apc_tensor *table, int32_t num_tensors, const apc_adamw_hparams *hp,
                                      int64_t step, apc_stream_t stream, uint64_t *out_digests) {
  return apc_commit_step_ex(table, num_tensors, hp, step, 0u, stream, out_digests);
}

APC_EXPORT apc_status apc_commit_step_bf16(const apc_tensor_bf16 *table, int32_t num_tensors,
                                           const apc_adamw_hparams *hp, int64_t step, uint32_t flags,
                                           apc_stream_t stream, uint64_t *out_digests) {
  g_last_error[0] = 0;
  if (num_tensors < 0) return fail(APC_EINVAL, "num_tensors %d < 0", num_tensors);
  if (num_tensors > 0 && !table) return fail(APC_EINVAL, "table pointer is null");
  std::vector<TableRow> rows((size_t)num_tensors);
  for (int32_t k = 0; k < num_tensors; ++k)
    rows[k] = TableRow{table[k].p, table[k].m, table[k].v, table[k].g, nullptr, table[k].n,
                       table[k].global_offset};
  return commit_common(apc::kLayoutBF16, rows, hp, step, flags, stream, out_digests, 3);
}

namespace {

// Validate a buffer list and turn it into digest/count plan entries for a
// kernel whose tiles hold `tile` elements.
apc_status buffer_entries(const apc_buffer *bufs, int32_t num_bufs, int32_t num_slots, uint64_t *out,
                          uint64_t tile, std::vector<apc::DigestEntry> *entries) {
  if (num_bufs < 0) return fail(APC_EINVAL, "num_bufs %d < 0", num_bufs);
  if (num_bufs > 0 && !bufs) return fail(APC_EINVAL, "bufs pointer is null");
  if (num_slots < 1 || num_slots > APC_MAX_SLOTS)
    return fail(APC_EINVAL, "num_slots %d outside 1..%d", num_slots, APC_MAX_SLOTS);
  if (!out) return fail(APC_EINVAL, "output pointer is null");
  if ((uintptr_t)out % 8) return fail(APC_EALIGN, "output not 8-byte aligned");
  entries->reserve((size_t)num_bufs);
  std::vector<Range> ranges;
  std::vector<Owned> owned;
  ranges.reserve((size_t)num_bufs + 1);
  owned.reserve((size_t)num_bufs + 1);
  for (int32_t k = 0; k < num_bufs; ++k) {
    const apc_buffer &b = bufs[k];
    if (b.dtype != APC_F32 && b.dtype != APC_BF16) return fail(APC_EINVAL, "bufs[%d]: unknown dtype %u", k, b.dtype);
    if (b.slot >= (uint32_t)num_slots) return fail(APC_EINVAL, "bufs[%d]: slot %u >= num_slots", k, b.slot);
    if (b.n == 0) continue;
    if (!b.data) return fail(APC_EINVAL, "bufs[%d]: null data pointer", k);
    if (b.n > (UINT64_MAX - b.global_offset)) return fail(APC_ERANGE, "bufs[%d]: global_offset + n overflows", k);
    if (b.n > ((uint64_t)1 << 61)) return fail(APC_ERANGE, "bufs[%d]: n too large", k);
    const uintptr_t a = (uintptr_t)b.data;
    const uint64_t es = b.dtype == APC_F32 ? 4 : 2;
    if (a % es) return fail(APC_EALIGN, "bufs[%d]: data not %u-byte aligned", k, (unsigned)es);
    ranges.push_back({a, a + es * b.n, false});
    owned.push_back({b.data, "bufs", (int)k, "data"});
    apc::DigestEntry e;
    e.data = b.data;
    e.n = b.n;
    e.key_base = (uint32_t)b.global_offset;
    e.head = (uint8_t)std::min<uint64_t>(((16 - a % 16) % 16) / es, b.n);
    e.dtype = (uint8_t)b.dtype;
    e.slot = (uint8_t)b.slot;
    e.pad_ = 0;
    const uint64_t body = (b.n - e.head) / apc::kVec * apc::kVec;
    e.tile_begin = std::max<uint64_t>(1, ceil_div(body, tile));  // tile count until placed
    entries->push_back(e);
  }
  const uintptr_t o = (uintptr_t)out;
  ranges.push_back({o, o + (uintptr_t)num_slots * sizeof(uint64_t), true});
  if (overlaps(ranges)) return fail(APC_EINVAL, "the output overlaps a buffer of the list");
  owned.push_back({out, "output", -1, ""});
  return check_device_pointers(owned);
}

}  // namespace

APC_EXPORT apc_status apc_digest(const apc_buffer *bufs, int32_t num_bufs, int32_t num_slots, apc_stream_t stream,
                                 uint64_t *out_digests) {
  g_last_error[0] = 0;
  std::vector<apc::DigestEntry> entries;
  apc_status st = buffer_entries(bufs, num_bufs, num_slots, out_digests, apc::kDigestTile, &entries);
  if (st != APC_OK) return st;
  int e = (int)cudaMemsetAsync(out_digests, 0, (size_t)num_slots * sizeof(uint64_t), (cudaStream_t)stream);
  if (e) return cuda_fail(e, "cudaMemsetAsync(out_digests)");
  if (entries.empty()) return APC_OK;
  Device d;
  if ((st = device_info(&d)) != APC_OK) return st;
  unsigned long long *out = reinterpret_cast<unsigned long long *>(out_digests);
  if (entries.size() <= (size_t)apc::kDigestSmall)
    return run_digest_batches<apc::kDigestSmall>(entries, grid_for(UINT64_MAX, d.sms, d.digest_small), stream, out,
                                                 apc::launch_digest_small, "digest kernel launch");
  return run_digest_batches<apc::kDigestLarge>(entries, grid_for(UINT64_MAX, d.sms, d.digest_large), stream, out,
                                               apc::launch_digest_large, "digest kernel launch");
}

APC_EXPORT apc_status apc_count_nonzero(const apc_buffer *bufs, int32_t num_bufs, int32_t num_slots,
                                        apc_stream_t stream, uint64_t *out_counts) {
  g_last_error[0] = 0;
  std::vector<apc::DigestEntry> entries;
  apc_status st = buffer_entries(bufs, num_bufs, num_slots, out_counts, apc::kCountTile, &entries);
  if (st != APC_OK) return st;
  int e = (int)cudaMemsetAsync(out_counts, 0, (size_t)num_slots * sizeof(uint64_t), (cudaStream_t)stream);
  if (e) return cuda_fail(e, "cudaMemsetAsync(out_counts)");
  if (entries.empty()) return APC_OK;
  Device d;
  if ((st = device_info(&d)) != APC_OK) return st;
  unsigned long long *out = reinterpret_cast<unsigned long long *>(out_counts);
  if (entries.size() <= (size_t)apc::kDigestSmall)
    return run_digest_batches<apc::kDigestSmall>(entries, grid_for(UINT64_MAX, d.sms, d.count_small), stream, out,
                                                 apc::launch_count_small, "count kernel launch");
  return run_digest_batches<apc::kDigestLarge>(entries, grid_for(UINT64_MAX, d.sms, d.count_large), stream, out,
                                               apc::launch_count_large, "count kernel launch");
}

namespace {

// The device-side address of a source the current device `dev` can read:
// its own device memory, managed memory, page-locked host memory mapped for
// the device, or pageable host memory where the device reads it through the
// host's page tables.  Null if the device cannot read it.
const void *device_readable(const void *p, int dev, bool pageable_ok) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();  // clear the error state of the failed query
    return pageable_ok ? p : nullptr;
  }
  switch (a.type) {
    case cudaMemoryTypeDevice:
      return a.device == dev ? p : nullptr;
    case cudaMemoryTypeManaged:
      return p;
    case cudaMemoryTypeHost:
      return a.devicePointer;
    default:
      return pageable_ok ? p : nullptr;
  }
}

// Device memory of `dev` (or managed memory) that a kernel may write.
bool device_writable(void *p, int dev) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return (a.type == cudaMemoryTypeDevice && a.device == dev) || a.type == cudaMemoryTypeManaged;
}

}  // namespace

APC_EXPORT apc_status apc_upload(const apc_segment *segs, int32_t num_segments, int32_t max_ctas,
                                 apc_stream_t stream) {
  g_last_error[0] = 0;
  if (num_segments < 0) return fail(APC_EINVAL, "num_segments %d < 0", num_segments);
  if (num_segments > 0 && !segs) return fail(APC_EINVAL, "segments pointer is null");
  if (max_ctas < 0 || max_ctas > 4096) return fail(APC_EINVAL, "max_ctas %d outside 0..4096", max_ctas);
  std::vector<apc::UploadEntry> entries;
  entries.reserve((size_t)num_segments);
  int dev = 0, pageable = 0;
  bool queried = false;
  for (int32_t k = 0; k < num_segments; ++k) {
    const apc_segment &g = segs[k];
    if (g.bytes == 0) continue;
    if (!g.dst || !g.src) return fail(APC_EINVAL, "segments[%d]: null pointer", k);
    if (g.bytes > UINTPTR_MAX - (uintptr_t)g.dst || g.bytes > UINTPTR_MAX - (uintptr_t)g.src)
      return fail(APC_ERANGE, "segments[%d]: address + bytes overflows", k);
    if (!queried) {
      int e = (int)cudaGetDevice(&dev);
      if (e) return cuda_fail(e, "cudaGetDevice");
      if ((e = (int)cudaDeviceGetAttribute(&pageable, cudaDevAttrPageableMemoryAccess, dev)))
        return cuda_fail(e, "cudaDeviceGetAttribute");
      queried = true;
    }
    const void *src = device_readable(g.src, dev, pageable != 0);
    if (!src) return fail(APC_EINVAL, "segments[%d]: the current device cannot read the source", k);
    if (!device_writable(g.dst, dev))
      return fail(APC_EINVAL, "segments[%d]: destination is not memory of the current device", k);
    apc::UploadEntry e{};
    e.dst = static_cast<uint8_t *>(g.dst);
    e.src = static_cast<const uint8_t *>(src);
    e.bytes = g.bytes;
    const uintptr_t d = (uintptr_t)e.dst, s = (uintptr_t)e.src;
    const uint64_t head = (16 - (d & 15)) & 15;
    e.body = ((d ^ s) & 15) == 0 && g.bytes > head ? (g.bytes - head) & ~(uint64_t)15 : 0;
    e.tile_begin = (e.body + apc::kUploadTile - 1) / apc::kUploadTile;  // tile count until placed
    e.scalar_begin = g.bytes - e.body;                                  // scalar count until placed
    entries.push_back(e);
  }
  // destinations must not overlap each other or any source (sorted sweep)
  std::vector<Range> rs;
  rs.reserve(2 * entries.size());
  for (const auto &e : entries) {
    rs.push_back(Range{(uintptr_t)e.dst, (uintptr_t)e.dst + e.bytes, true});
    rs.push_back(Range{(uintptr_t)e.src, (uintptr_t)e.src + e.bytes, false});
  }
  if (overlaps(rs)) return fail(APC_EINVAL, "a destination range overlaps another destination or a source");
  if (entries.empty()) return APC_OK;
  Device d;
  apc_status st = device_info(&d);
  if (st != APC_OK) return st;
  const unsigned cap = max_ctas > 0 ? (unsigned)max_ctas : (unsigned)d.sms;
  auto plan = std::make_unique<apc::UploadPlan<apc::kUploadMax>>();
  size_t i = 0;
  while (i < entries.size()) {
    const size_t k = std::min(entries.size() - i, (size_t)apc::kUploadMax);
    uint64_t tiles = 0, scalars = 0;
    for (size_t j = 0; j < k; ++j) {
      apc::UploadEntry e = entries[i + j];
      const uint64_t t = e.tile_begin, c = e.scalar_begin;
      e.tile_begin = tiles;
      e.scalar_begin = scalars;
      tiles += t;
      scalars += c;
      plan->e[j] = e;
    }
    plan->count = (uint32_t)k;
    plan->total_tiles = tiles;
    plan->total_scalar = scalars;
    const uint64_t want = std::max<uint64_t>(tiles, (scalars + apc::kUploadThreads - 1) / apc::kUploadThreads);
    const unsigned grid = (unsigned)std::max<uint64_t>(1, std::min<uint64_t>(want, cap));
    int e = apc::launch_upload(*plan, grid, stream);
    if (e) return cuda_fail(e, "upload kernel launch");
    i += k;
  }
  return APC_OK;
}

APC_EXPORT apc_status apc_set_reserved_sms(int32_t n) {
  g_last_error[0] = 0;
  if (n < 0 || n > 1024) return fail(APC_EINVAL, "reserved SMs %d outside 0..1024", n);
  g_reserved_sms.store(n, std::memory_order_relaxed);
  return APC_OK;
}

APC_EXPORT apc_status apc_device_status(void) {
  g_last_error[0] = 0;
  int e = (int)cudaDeviceSynchronize();
  if (e) return cuda_fail(e, "cudaDeviceSynchronize");
  unsigned word = 0;
  if ((e = apc::read_commit_status(&word))) return cuda_fail(e, "reading the device status word");
  if (word & APC_ETIMEOUT) return fail(APC_ETIMEOUT, "a bounded wait inside a kernel gave up");
  return APC_OK;
}

APC_EXPORT apc_status apc_selftest_wait_timeout(uint64_t limit_ns, apc_stream_t stream) {
  g_last_error[0] = 0;
  if (limit_ns < 1 || limit_ns > 10000000000ull) return fail(APC_EINVAL, "limit_ns outside 1..1e10");
  int e = apc::launch_wait_timeout(limit_ns, stream);
  if (e) return cuda_fail(e, "self-test kernel launch");
  return APC_OK;
}

APC_EXPORT const char *apc_status_string(apc_status s) {
  switch (s) {
    case APC_OK: return "APC_OK: success";
    case APC_EINVAL: return "APC_EINVAL: invalid argument";
    case APC_EALIGN: return "APC_EALIGN: misaligned pointer";
    case APC_ERANGE: return "APC_ERANGE: index range overflow";
    case APC_ECUDA: return "APC_ECUDA: CUDA runtime error";
    case APC_ETIMEOUT: return "APC_ETIMEOUT: a bounded wait inside a kernel gave up";
  }
  return "unknown apc_status";
}

APC_EXPORT const char *apc_last_error(void) { return g_last_error; }

APC_EXPORT int32_t apc_version(void) { return 3; }
