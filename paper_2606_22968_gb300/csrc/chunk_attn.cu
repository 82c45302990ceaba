// chunk_attn.cu -- host side of the chunked causal GQA prefill attention:
// tensor maps, the split-KV plan, launches of the attention kernel
// (attn_kernel.cuh) and of the split-KV combine (attn_combine.cuh), and the
// C entry points (mocap_chunk_attn, _varlen, _varlen_dev, _append,
// _varlen_append, _workspace_size, _noalloc).
//
// Sec. 2.2 / Eq. 1: chunk i's queries (global rows prefix .. prefix+len-1)
// attend to the KV of every earlier chunk plus a causal block over their own
// chunk; the attention work grows with the prefix, which is what LBCP
// balances.
#include <cmath>
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <functional>
#include <cstdlib>
#include <cstring>
#include <map>
#include <mutex>
#include <tuple>
#include <vector>

#include "internal.h"
#include "sm103_ptx.cuh"
#include "attn_kernel.cuh"
#include "attn_combine.cuh"
#include "attn_varlen_dev.cuh"

namespace mocap {
namespace {

// ------------------------------------------------------------------ host --

// [rows, heads, d] bf16 tensor, box = 64 columns x 1 head x box_rows rows,
// 128B swizzle.
bool make_map(CUtensorMap *map, const void *ptr, int64_t rows, int heads, int d,
              int box_rows = kBlockM) {
  auto fn = tensor_map_encoder();
  if (fn == nullptr) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(heads),
                        static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(d) * 2,
                           static_cast<cuuint64_t>(heads) * static_cast<cuuint64_t>(d) * 2};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(kBoxCols), 1u, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t elem[3] = {1u, 1u, 1u};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), dims, strides, box,
            elem, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct Shape {
  int n_q_heads, n_kv_heads, head_dim;
};

mocap_status check_shape(const Shape &sh, float scale) {
  if (sh.n_q_heads < 1 || sh.n_kv_heads < 1 || sh.n_q_heads % sh.n_kv_heads != 0)
    return MOCAP_EINVAL;
  if (!(scale > 0.0f) || !std::isfinite(scale)) return MOCAP_EINVAL;
  if (sh.head_dim != 64 && sh.head_dim != 128) return MOCAP_EUNSUPPORTED;
  return MOCAP_OK;
}

struct HostItem {
  int64_t q_row, kv_row, prefix, len;
};

// KV appends a launch carries (validated by the entry points): K/V sources
// of `rows` rows each, written to cache rows [dst_row, dst_row + rows).
struct HostAppend {
  const void *k_src, *v_src;
  int64_t dst_row, rows;
};

// Split-KV scratch (single item): o_part [splits, len, Hq, D] fp32 followed by
// lse_part [splits, Hq, len] fp32, the latter 256-byte aligned.
struct SplitPlan {
  int splits = 1;
  size_t o_bytes = 0, lse_off = 0, bytes = 0;
};

SplitPlan split_layout(int splits, int64_t len, int n_q_heads, int head_dim) {
  SplitPlan sp;
  sp.splits = splits;
  if (splits <= 1) return sp;
  sp.o_bytes = static_cast<size_t>(splits) * len * n_q_heads * head_dim * sizeof(float);
  sp.lse_off = (sp.o_bytes + 255) / 256 * 256;
  sp.bytes = sp.lse_off + static_cast<size_t>(splits) * n_q_heads * len * sizeof(float);
  return sp;
}

// Split count for one chunk: list-schedule the CTAs (heaviest first, one per
// SM at a time) for 1..4 key-range splits and keep the fastest estimate.
// Cost units: one 128-key tile of a head pair ~ 1.4 us; a CTA's fixed cost
// ~ 4 us; the combine reads splits x (4D + 4) and writes 2D + 4 bytes per
// (row, head) at ~5 TB/s, plus ~3 us for its launch.
int choose_splits_uncached(int64_t prefix, int64_t len, int n_q_heads, int n_kv_heads,
                           int head_dim, int sms) {
  const int group = n_q_heads / n_kv_heads;
  const int64_t pairs = (group + 1) / 2;
  const int64_t q_blocks = (len + kBlockM - 1) / kBlockM;
  const int64_t units = q_blocks * n_kv_heads * pairs;
  if (units <= 0 || units >= 8LL * sms) return 1;  // many waves: little to gain
  const int64_t min_tiles = (std::min<int64_t>(prefix + kBlockM, prefix + len) + kBlockN - 1) / kBlockN;
  const double tile_us = 1.4 * (head_dim / 128.0), cta_us = 4.0;
  double best_t = 0.0;
  int best = 1;
  for (int sp = 1; sp <= kMaxSplits && sp <= min_tiles; ++sp) {
    // SM loads as a min-heap: each CTA goes to a least-loaded SM (which of
    // several equally loaded SMs does not change the multiset of loads)
    std::vector<double> sm(static_cast<size_t>(sms), 0.0);
    for (int64_t qb = q_blocks - 1; qb >= 0; --qb) {
      const int64_t kv_end = std::min<int64_t>(prefix + qb * kBlockM + kBlockM, prefix + len);
      const int64_t tiles = (kv_end + kBlockN - 1) / kBlockN;
      for (int64_t u = 0; u < n_kv_heads * pairs; ++u)
        for (int k = 0; k < sp; ++k) {
          const int64_t nk = (k + 1) * tiles / sp - k * tiles / sp;
          std::pop_heap(sm.begin(), sm.end(), std::greater<double>());
          sm.back() += cta_us + tile_us * static_cast<double>(nk);
          std::push_heap(sm.begin(), sm.end(), std::greater<double>());
        }
    }
    double t = *std::max_element(sm.begin(), sm.end());
    if (sp > 1)
      t += 3.0 + static_cast<double>(len) * n_q_heads *
                     (sp * (4.0 * head_dim + 4.0) + 2.0 * head_dim + 4.0) / 5e6;
    if (sp == 1 || t < best_t) {
      best_t = t;
      best = sp;
    }
  }
  return best;
}

// The plan depends only on the shape and the SM count, and a prompt repeats
// its chunk shapes step after step, so plans are kept (up to 4096 shapes;
// the table is cleared when full).
int choose_splits(int64_t prefix, int64_t len, int n_q_heads, int n_kv_heads, int head_dim,
                  int sms) {
  using Key = std::tuple<int64_t, int64_t, int, int, int, int>;
  static std::map<Key, int> cache;
  static std::mutex mu;
  const Key key{prefix, len, n_q_heads, n_kv_heads, head_dim, sms};
  {
    std::lock_guard<std::mutex> lock(mu);
    const auto it = cache.find(key);
    if (it != cache.end()) return it->second;
  }
  const int splits = choose_splits_uncached(prefix, len, n_q_heads, n_kv_heads, head_dim, sms);
  std::lock_guard<std::mutex> lock(mu);
  if (cache.size() >= 4096) cache.clear();
  cache.emplace(key, splits);
  return splits;
}

// CTA pairs (cta_group::2) serve d = 128 with a multiple of four query heads
// per KV group.  MOCAP_ATTN_PAIR=0 selects the single-CTA kernel for every
// shape (tests compare the two).
bool pair_enabled() {
  const char *env = std::getenv("MOCAP_ATTN_PAIR");
  return env == nullptr || std::atoi(env) != 0;
}

// One attention launch of `kern` with `prm` on `ctas` CTAs, as CTA pairs
// (clusters of two) or single CTAs.  Once per kernel and context (`once`):
// the register-count check (the setmaxnreg split assumes kLaunchRegs) and
// the dynamic shared-memory limit.
template <typename Kern, typename P>
mocap_status start_attn(Kern kern, const P &prm, int64_t ctas, bool as_pair, int smem,
                        ContextOnce &once, cudaStream_t stream) {
  const uint64_t ctx = current_context();
  if (ctx == 0) return MOCAP_ECUDA;
  if (!once.done(ctx)) {
    cudaFuncAttributes fa{};
    if (cudaFuncGetAttributes(&fa, kern) != cudaSuccess) return MOCAP_ECUDA;
    if (fa.numRegs != kLaunchRegs) return MOCAP_EUNSUPPORTED;  // split would not balance
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
        cudaSuccess)
      return MOCAP_ECUDA;
    once.mark(ctx);
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(ctas));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = static_cast<size_t>(smem);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = as_pair ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, prm) == cudaSuccess ? MOCAP_OK : MOCAP_ECUDA;
}

template <int D, int MAXI>
mocap_status launch(const void *q, const void *k_cache, const void *v_cache,
                    const std::vector<HostItem> &items, int64_t lse_stride, const Shape &sh,
                    float scale, void *out, float *lse, cudaStream_t stream,
                    const SplitPlan &sp = SplitPlan(), void *workspace = nullptr,
                    const std::vector<HostAppend> &apps = {}) {
  using L = Layout<D>;
  static AttnParams<MAXI> prm;  // large: build in static storage, guarded below
  static std::mutex mu;
  std::lock_guard<std::mutex> lock(mu);
  std::memset(&prm, 0, sizeof(prm));
  uint32_t *status = device_status_ptr();
  if (status == nullptr) return MOCAP_ECUDA;
  const int group = sh.n_q_heads / sh.n_kv_heads;
  const int pairs = (group + 1) / 2;
  int64_t ctas = 0;
  int n = 0;
  // CTA pairs need an even number of head pairs per KV group
  const bool pair = D == 128 && group % 4 == 0 && pair_enabled();
  const size_t qrow_bytes = static_cast<size_t>(sh.n_q_heads) * D * 2;
  const size_t kvrow_bytes = static_cast<size_t>(sh.n_kv_heads) * D * 2;
  for (const HostItem &h : items) {
    const auto *qb = static_cast<const uint8_t *>(q) + h.q_row * qrow_bytes;
    const auto *kb = static_cast<const uint8_t *>(k_cache) + h.kv_row * kvrow_bytes;
    const auto *vb = static_cast<const uint8_t *>(v_cache) + h.kv_row * kvrow_bytes;
    if (!make_map(&prm.tq[n], qb, h.len, sh.n_q_heads, D) ||
        !make_map(&prm.tk[n], kb, h.prefix + h.len, sh.n_kv_heads, D,
                  pair ? kBlockN / 2 : kBlockN) ||
        !make_map(&prm.tv[n], vb, h.prefix + h.len, sh.n_kv_heads, D))
      return MOCAP_ECUDA;
    ItemDesc &d = prm.items[n];
    d.q_row = h.q_row;
    d.prefix = static_cast<int32_t>(h.prefix);
    d.len = static_cast<int32_t>(h.len);
    d.q_blocks = static_cast<int32_t>((h.len + kBlockM - 1) / kBlockM);
    d.cta_begin = static_cast<int32_t>(ctas);
    ctas += static_cast<int64_t>(d.q_blocks) * sh.n_kv_heads * pairs * sp.splits;
    ++n;
  }
  if (n == 0) return MOCAP_OK;
  if (ctas > 0x7fffffff) return MOCAP_EINVAL;
  prm.out = static_cast<__nv_bfloat16 *>(out);
  prm.lse = lse;
  prm.status = status;
  prm.lse_stride = lse_stride;
  prm.n_items = n;
  prm.n_q_heads = sh.n_q_heads;
  prm.n_kv_heads = sh.n_kv_heads;
  prm.heads_per_group = group;
  prm.pairs_per_group = pairs;
  prm.scale_log2 = static_cast<float>(static_cast<double>(scale) * 1.4426950408889634074);
  prm.splits = sp.splits;
  if (sp.splits > 1) {
    if (n != 1 || workspace == nullptr || sp.splits > kMaxSplits) return MOCAP_EINVAL;
    prm.o_part = static_cast<float *>(workspace);
    prm.lse_part = reinterpret_cast<float *>(static_cast<uint8_t *>(workspace) + sp.lse_off);
  }
  if (apps.size() > static_cast<size_t>(kMaxAppends)) return MOCAP_EINVAL;
  prm.k_cache_vec = static_cast<uint4 *>(const_cast<void *>(k_cache));
  prm.v_cache_vec = static_cast<uint4 *>(const_cast<void *>(v_cache));
  const int64_t row_vec = static_cast<int64_t>(sh.n_kv_heads) * D / 8;  // 16-byte vectors per row
  for (const HostAppend &a : apps) {
    if (a.rows <= 0) continue;
    AppendSeg &g = prm.app[prm.n_app++];
    g.k_src = static_cast<const uint4 *>(a.k_src);
    g.v_src = static_cast<const uint4 *>(a.v_src);
    g.dst_vec = a.dst_row * row_vec;
    g.n_vec = a.rows * row_vec;
    g.begin = prm.app_total;
    prm.app_total += 2 * g.n_vec;
  }

  // the CTA-pair or single-CTA form, each with or without the append copy
  auto launch_form = [&](auto kern, bool as_pair, int smem, ContextOnce &once) -> mocap_status {
    return start_attn(kern, prm, ctas, as_pair, smem, once, stream);
  };
  const bool append = prm.n_app > 0;
  mocap_status lst = MOCAP_OK;
  bool launched = false;
  if constexpr (D == 128) {
    if (pair) {
      if (ctas % 2 != 0) return MOCAP_EINVAL;  // whole pairs by construction
      constexpr int kSmem = Layout<D, true>::kBytes;
      if (append) {
        static ContextOnce once;
        lst = launch_form(chunk_attn_kernel<D, MAXI, true, true>, true, kSmem, once);
      } else {
        static ContextOnce once;
        lst = launch_form(chunk_attn_kernel<D, MAXI, true, false>, true, kSmem, once);
      }
      launched = true;
    }
  }
  if (!launched) {
    if (append) {
      static ContextOnce once;
      lst = launch_form(chunk_attn_kernel<D, MAXI, false, true>, false, L::kBytes, once);
    } else {
      static ContextOnce once;
      lst = launch_form(chunk_attn_kernel<D, MAXI, false, false>, false, L::kBytes, once);
    }
  }
  if (lst != MOCAP_OK) return lst;
  if (cudaGetLastError() != cudaSuccess) return MOCAP_ECUDA;
  if (sp.splits > 1) {
    // the item's rows start at q_row of the packed out / lse (0 for a
    // single-chunk call)
    const int64_t len = items[0].len, q_row = items[0].q_row;
    const dim3 grid(static_cast<unsigned>(len),
                    static_cast<unsigned>((sh.n_q_heads + kCombineHeadsPerBlock - 1) /
                                          kCombineHeadsPerBlock));
    static ContextOnce combine_once;  // shared-memory limit set, per context
    const uint64_t ctx = current_context();
    if (ctx == 0) return MOCAP_ECUDA;
    if (!combine_once.done(ctx)) {
      if (cudaFuncSetAttribute(attn_combine_kernel<D>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(combine_smem_bytes<D>(kMaxSplits))) !=
          cudaSuccess)
        return MOCAP_ECUDA;
      combine_once.mark(ctx);
    }
    attn_combine_kernel<D><<<grid, kCombineThreads, combine_smem_bytes<D>(sp.splits), stream>>>(
        prm.o_part, prm.lse_part, sp.splits, len, sh.n_q_heads,
        prm.out + q_row * sh.n_q_heads * D, lse + q_row, lse_stride, status);
    if (cudaGetLastError() != cudaSuccess) return MOCAP_ECUDA;
  }
  return MOCAP_OK;
}

template <int MAXI>
mocap_status dispatch(const void *q, const void *k_cache, const void *v_cache,
                      const std::vector<HostItem> &items, int64_t lse_stride, const Shape &sh,
                      float scale, void *out, float *lse, cudaStream_t stream,
                      const SplitPlan &sp = SplitPlan(), void *workspace = nullptr,
                      const std::vector<HostAppend> &apps = {}) {
  if (sh.head_dim == 128)
    return launch<128, MAXI>(q, k_cache, v_cache, items, lse_stride, sh, scale, out, lse, stream,
                             sp, workspace, apps);
  return launch<64, MAXI>(q, k_cache, v_cache, items, lse_stride, sh, scale, out, lse, stream, sp,
                          workspace, apps);
}

// Validates the KV appends an attention launch is to carry and converts
// them: each must fit the cache (kv_rows_total rows), have 16-byte aligned
// sources, and write only rows that no item of the launch reads (item r
// reads cache rows [kv_row, kv_row + prefix + len)).  Appends must not write
// overlapping rows either.
mocap_status check_appends(const mocap_kv_append_item *appends, int32_t n_appends,
                           int64_t kv_rows_total, const std::vector<HostItem> &items,
                           std::vector<HostAppend> *out) {
  if (n_appends < 0 || n_appends > kMaxAppends) return MOCAP_EINVAL;
  if (n_appends > 0 && appends == nullptr) return MOCAP_EINVAL;
  for (int i = 0; i < n_appends; ++i) {
    const mocap_kv_append_item &a = appends[i];
    if (a.rows < 0 || a.dst_row < 0 || a.dst_row > kv_rows_total - a.rows) return MOCAP_EINVAL;
    if (a.rows == 0) continue;
    if (!a.k_src || !a.v_src || !aligned16(a.k_src) || !aligned16(a.v_src)) return MOCAP_EINVAL;
    const int64_t lo = a.dst_row, hi = a.dst_row + a.rows;
    for (const HostItem &it : items)
      if (lo < it.kv_row + it.prefix + it.len && it.kv_row < hi) return MOCAP_EINVAL;
    for (const HostAppend &b : *out)
      if (lo < b.dst_row + b.rows && b.dst_row < hi) return MOCAP_EINVAL;
    out->push_back({a.k_src, a.v_src, a.dst_row, a.rows});
  }
  return MOCAP_OK;
}

bool pointers_ok(const void *q, const void *k, const void *v, const void *out, const float *lse) {
  if (!q || !k || !v || !out || !lse) return false;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out)) return false;
  return (reinterpret_cast<uintptr_t>(lse) & 3u) == 0;
}

constexpr int64_t kMaxRows = 0x7fffffffLL;

// ---- mocap_chunk_attn_varlen_dev -------------------------------------------
// Scratch of the device-descriptor form (offsets in bytes; the tensor maps,
// three per item, start at 0): ItemDescs, the CTA -> item table of the
// grid's upper bound, the CTA count.
struct DevLayout {
  int64_t max_ctas = 0;
  size_t descs = 0, cta_item = 0, total = 0, bytes = 0;
};

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

bool dev_layout(int32_t n_items, int64_t max_rows, const Shape &sh, DevLayout *out) {
  if (n_items < 1 || n_items > MOCAP_VARLEN_DEV_MAX_ITEMS || max_rows < 0 || max_rows > kMaxRows)
    return false;
  const int64_t group = sh.n_q_heads / sh.n_kv_heads;
  const int64_t per_block = static_cast<int64_t>(sh.n_kv_heads) * ((group + 1) / 2);
  // sum over items of ceil(len / 128) <= ceil(max_rows / 128) + n_items when
  // the items' lengths add up to at most max_rows
  const int64_t blocks = (max_rows + kBlockM - 1) / kBlockM + n_items;
  if (per_block > 0x7fffffffLL / blocks) return false;
  DevLayout l;
  l.max_ctas = blocks * per_block;
  l.descs = align256(static_cast<size_t>(n_items) * 3 * sizeof(CUtensorMap));
  l.cta_item = align256(l.descs + static_cast<size_t>(n_items) * sizeof(ItemDesc));
  l.total = align256(l.cta_item + static_cast<size_t>(l.max_ctas) * sizeof(int32_t));
  l.bytes = l.total + 256;
  *out = l;
  return true;
}

template <int D>
mocap_status launch_dev(const void *q, const void *k_cache, const void *v_cache,
                        const mocap_varlen_item *items, int32_t n_items, int64_t q_rows_total,
                        int64_t kv_rows_total, const Shape &sh, float scale, void *out, float *lse,
                        const DevLayout &dl, void *workspace, cudaStream_t stream) {
  static AttnParams<1> prm;  // large: built in static storage, guarded below
  static DevPrep prep;
  static std::mutex mu;
  std::lock_guard<std::mutex> lock(mu);
  std::memset(&prm, 0, sizeof(prm));
  std::memset(&prep, 0, sizeof(prep));
  uint32_t *status = device_status_ptr();
  if (status == nullptr) return MOCAP_ECUDA;
  const int group = sh.n_q_heads / sh.n_kv_heads;
  const int pairs = (group + 1) / 2;
  const bool pair = D == 128 && group % 4 == 0 && pair_enabled();
  // templates over the whole buffers; the prepare kernel sets each item's
  // first row and row count
  const int64_t q_rows = std::min<int64_t>(std::max<int64_t>(q_rows_total, 1), kMaxRows);
  const int64_t kv_rows = std::min<int64_t>(std::max<int64_t>(kv_rows_total, 1), kMaxRows);
  if (!make_map(&prep.tq, q, q_rows, sh.n_q_heads, D) ||
      !make_map(&prep.tk, k_cache, kv_rows, sh.n_kv_heads, D, pair ? kBlockN / 2 : kBlockN) ||
      !make_map(&prep.tv, v_cache, kv_rows, sh.n_kv_heads, D))
    return MOCAP_ECUDA;
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  int32_t *cta_item = reinterpret_cast<int32_t *>(ws + dl.cta_item);
  prep.items = items;
  prep.cta_item = cta_item;
  prep.descs = reinterpret_cast<ItemDesc *>(ws + dl.descs);
  prep.maps = reinterpret_cast<CUtensorMap *>(ws);
  prep.total = reinterpret_cast<int32_t *>(ws + dl.total);
  prep.status = status;
  prep.q = static_cast<const uint8_t *>(q);
  prep.k = static_cast<const uint8_t *>(k_cache);
  prep.v = static_cast<const uint8_t *>(v_cache);
  prep.q_rows_total = q_rows_total;
  prep.kv_rows_total = kv_rows_total;
  prep.qrow_bytes = static_cast<int64_t>(sh.n_q_heads) * D * 2;
  prep.kvrow_bytes = static_cast<int64_t>(sh.n_kv_heads) * D * 2;
  prep.max_ctas = dl.max_ctas;
  prep.n_items = n_items;
  prep.ctas_per_block = sh.n_kv_heads * pairs;
  varlen_dev_prepare<<<1, kPrepThreads, 0, stream>>>(prep);
  if (cudaGetLastError() != cudaSuccess) return MOCAP_ECUDA;

  prm.out = static_cast<__nv_bfloat16 *>(out);
  prm.lse = lse;
  prm.status = status;
  prm.lse_stride = q_rows_total;
  prm.n_items = 1;
  prm.n_q_heads = sh.n_q_heads;
  prm.n_kv_heads = sh.n_kv_heads;
  prm.heads_per_group = group;
  prm.pairs_per_group = pairs;
  prm.scale_log2 = static_cast<float>(static_cast<double>(scale) * 1.4426950408889634074);
  prm.splits = 1;
  prm.k_cache_vec = static_cast<uint4 *>(const_cast<void *>(k_cache));
  prm.v_cache_vec = static_cast<uint4 *>(const_cast<void *>(v_cache));
  prm.dev_items = prep.descs;
  prm.dev_cta_item = cta_item;
  prm.dev_maps = prep.maps;
  prm.dev_total = prep.total;
  mocap_status st = MOCAP_OK;
  bool launched = false;
  if constexpr (D == 128) {
    if (pair) {
      if (dl.max_ctas % 2 != 0) return MOCAP_EINVAL;  // whole pairs by construction
      static ContextOnce once;
      st = start_attn(chunk_attn_kernel<D, 1, true, false, true>, prm, dl.max_ctas, true,
                      Layout<D, true>::kBytes, once, stream);
      launched = true;
    }
  }
  if (!launched) {
    static ContextOnce once;
    st = start_attn(chunk_attn_kernel<D, 1, false, false, true>, prm, dl.max_ctas, false,
                    Layout<D>::kBytes, once, stream);
  }
  if (st != MOCAP_OK) return st;
  return cudaGetLastError() == cudaSuccess ? MOCAP_OK : MOCAP_ECUDA;
}

}  // namespace

}  // namespace mocap

using mocap::HostItem;

namespace {
// The split the library uses for this shape when given enough workspace.
mocap::SplitPlan plan_for(int64_t prefix, int64_t len, int32_t n_q_heads, int32_t n_kv_heads,
                          int32_t head_dim) {
  const mocap::Shape sh{n_q_heads, n_kv_heads, head_dim};
  if (mocap::check_shape(sh, 1.0f) != MOCAP_OK || prefix < 0 || len <= 0 ||
      prefix > mocap::kMaxRows - len)
    return mocap::SplitPlan();
  if (n_q_heads > mocap::kCombineHeadsPerBlock * 65535)  // the combine's grid has y <= 65535
    return mocap::SplitPlan();
  int splits =
      mocap::choose_splits(prefix, len, n_q_heads, n_kv_heads, head_dim, mocap::device_sm_count());
  // MOCAP_SPLIT_KV: 0 never splits; 1..4 forces that count (tests, tuning),
  // capped so the first row block still has a key tile per split.
  if (const char *env = std::getenv("MOCAP_SPLIT_KV")) {
    const int forced = std::atoi(env);
    if (forced >= 0 && forced <= mocap::kMaxSplits) {
      const int64_t min_tiles = (std::min<int64_t>(prefix + mocap::kBlockM, prefix + len) +
                                 mocap::kBlockN - 1) / mocap::kBlockN;
      splits = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(forced, min_tiles)));
    }
  }
  return mocap::split_layout(splits, len, n_q_heads, head_dim);
}
}  // namespace

extern "C" size_t mocap_chunk_attn_workspace_size(int64_t prefix, int64_t len, int32_t n_q_heads,
                                                  int32_t n_kv_heads, int32_t head_dim) {
  return plan_for(prefix, len, n_q_heads, n_kv_heads, head_dim).bytes;
}

namespace {
// mocap_chunk_attn, optionally carrying KV appends (checked by the caller).
mocap_status chunk_attn_impl(const void *q, const void *k_cache, const void *v_cache,
                             int64_t prefix, int64_t len, int32_t n_q_heads, int32_t n_kv_heads,
                             int32_t head_dim, float scale, void *out, float *lse,
                             void *workspace, size_t workspace_bytes, mocap_stream_t stream,
                             bool with_appends = false,
                             const mocap_kv_append_item *appends = nullptr,
                             int32_t n_appends = 0, int64_t cache_rows = 0) {
  const mocap::Shape sh{n_q_heads, n_kv_heads, head_dim};
  const mocap_status st = mocap::check_shape(sh, scale);
  if (st != MOCAP_OK) return st;
  if (prefix < 0 || len < 0 || prefix > mocap::kMaxRows - len) return MOCAP_EINVAL;
  if (!mocap::pointers_ok(q, k_cache, v_cache, out, lse)) return MOCAP_EINVAL;
  if (workspace != nullptr && !mocap::aligned16(workspace)) return MOCAP_EINVAL;
  std::vector<HostItem> items{{0, 0, prefix, len}};
  std::vector<mocap::HostAppend> apps;
  if (with_appends) {
    if (cache_rows < prefix + len) return MOCAP_EINVAL;
    const mocap_status sa = mocap::check_appends(appends, n_appends, cache_rows, items, &apps);
    if (sa != MOCAP_OK) return sa;
  }
  if (len == 0) {
    // no attention work: the appends run as plain append launches
    for (const mocap::HostAppend &a : apps) {
      const mocap_status sa = mocap_kv_append(a.k_src, a.v_src, const_cast<void *>(k_cache),
                                              const_cast<void *>(v_cache), cache_rows, a.dst_row,
                                              a.rows, n_kv_heads, head_dim, stream);
      if (sa != MOCAP_OK) return sa;
    }
    return MOCAP_OK;
  }
  // Split the key range only when the caller's scratch holds the partials.
  mocap::SplitPlan sp = plan_for(prefix, len, n_q_heads, n_kv_heads, head_dim);
  if (sp.splits > 1 && (workspace == nullptr || workspace_bytes < sp.bytes)) sp = mocap::SplitPlan();
  return mocap::dispatch<1>(q, k_cache, v_cache, items, len, sh, scale, out, lse,
                            reinterpret_cast<cudaStream_t>(stream), sp, workspace, apps);
}

// mocap_chunk_attn_varlen, optionally carrying KV appends.
mocap_status varlen_impl(const void *q, const void *k_cache, const void *v_cache,
                         const mocap_varlen_item *items, int32_t n_items, int64_t q_rows_total,
                         int64_t kv_rows_total, int32_t n_q_heads, int32_t n_kv_heads,
                         int32_t head_dim, float scale, void *out, float *lse, void *workspace,
                         size_t workspace_bytes, mocap_stream_t stream,
                         const mocap_kv_append_item *appends = nullptr, int32_t n_appends = 0) {
  const mocap::Shape sh{n_q_heads, n_kv_heads, head_dim};
  const mocap_status st = mocap::check_shape(sh, scale);
  if (st != MOCAP_OK) return st;
  if (n_items < 0 || n_items > MOCAP_VARLEN_MAX_ITEMS) return MOCAP_EINVAL;
  if (n_items > 0 && items == nullptr) return MOCAP_EINVAL;
  if (q_rows_total < 0 || kv_rows_total < 0) return MOCAP_EINVAL;
  if (!mocap::pointers_ok(q, k_cache, v_cache, out, lse)) return MOCAP_EINVAL;
  if (workspace != nullptr && !mocap::aligned16(workspace)) return MOCAP_EINVAL;
  std::vector<HostItem> list;
  for (int i = 0; i < n_items; ++i) {
    const mocap_varlen_item &x = items[i];
    if (x.q_row < 0 || x.kv_row < 0 || x.prefix < 0 || x.len < 0) return MOCAP_EINVAL;
    if (x.prefix > mocap::kMaxRows - x.len) return MOCAP_EINVAL;
    if (x.q_row > q_rows_total - x.len) return MOCAP_EINVAL;
    if (x.kv_row > kv_rows_total - (x.prefix + x.len)) return MOCAP_EINVAL;
    if (x.len > 0) list.push_back({x.q_row, x.kv_row, x.prefix, x.len});
  }
  std::vector<mocap::HostAppend> apps;
  const mocap_status sa = mocap::check_appends(appends, n_appends, kv_rows_total, list, &apps);
  if (sa != MOCAP_OK) return sa;
  if (list.empty()) {
    for (const mocap::HostAppend &a : apps) {
      const mocap_status sk = mocap_kv_append(a.k_src, a.v_src, const_cast<void *>(k_cache),
                                              const_cast<void *>(v_cache), kv_rows_total,
                                              a.dst_row, a.rows, n_kv_heads, head_dim, stream);
      if (sk != MOCAP_OK) return sk;
    }
    return MOCAP_OK;
  }
  if (list.size() == 1) {
    // One item: the single-chunk plan, key-range split included when the
    // caller's workspace holds its partials.
    const HostItem &x = list[0];
    mocap::SplitPlan sp = plan_for(x.prefix, x.len, n_q_heads, n_kv_heads, head_dim);
    if (sp.splits > 1 && (workspace == nullptr || workspace_bytes < sp.bytes))
      sp = mocap::SplitPlan();
    return mocap::dispatch<1>(q, k_cache, v_cache, list, q_rows_total, sh, scale, out, lse,
                              reinterpret_cast<cudaStream_t>(stream), sp, workspace, apps);
  }
  // Heaviest items first (their last row blocks see the most keys).
  std::stable_sort(list.begin(), list.end(), [](const HostItem &a, const HostItem &b) {
    return a.prefix + a.len > b.prefix + b.len;
  });
  return mocap::dispatch<MOCAP_VARLEN_MAX_ITEMS>(q, k_cache, v_cache, list, q_rows_total, sh,
                                                 scale, out, lse,
                                                 reinterpret_cast<cudaStream_t>(stream),
                                                 mocap::SplitPlan(), nullptr, apps);
}
}  // namespace

extern "C" mocap_status mocap_chunk_attn(const void *q, const void *k_cache, const void *v_cache,
                                         int64_t prefix, int64_t len, int32_t n_q_heads,
                                         int32_t n_kv_heads, int32_t head_dim, float scale,
                                         void *out, float *lse, void *workspace,
                                         size_t workspace_bytes, mocap_stream_t stream) {
  return chunk_attn_impl(q, k_cache, v_cache, prefix, len, n_q_heads, n_kv_heads, head_dim, scale,
                         out, lse, workspace, workspace_bytes, stream);
}

extern "C" mocap_status mocap_chunk_attn_append(
    const void *q, const void *k_cache, const void *v_cache, int64_t prefix, int64_t len,
    int32_t n_q_heads, int32_t n_kv_heads, int32_t head_dim, float scale, void *out, float *lse,
    void *workspace, size_t workspace_bytes, const mocap_kv_append_item *appends,
    int32_t n_appends, int64_t cache_capacity, mocap_stream_t stream) {
  return chunk_attn_impl(q, k_cache, v_cache, prefix, len, n_q_heads, n_kv_heads, head_dim, scale,
                         out, lse, workspace, workspace_bytes, stream, true, appends, n_appends,
                         cache_capacity);
}

extern "C" mocap_status mocap_chunk_attn_varlen(const void *q, const void *k_cache,
                                                const void *v_cache,
                                                const mocap_varlen_item *items, int32_t n_items,
                                                int64_t q_rows_total, int64_t kv_rows_total,
                                                int32_t n_q_heads, int32_t n_kv_heads,
                                                int32_t head_dim, float scale, void *out,
                                                float *lse, void *workspace,
                                                size_t workspace_bytes, mocap_stream_t stream) {
  return varlen_impl(q, k_cache, v_cache, items, n_items, q_rows_total, kv_rows_total, n_q_heads,
                     n_kv_heads, head_dim, scale, out, lse, workspace, workspace_bytes, stream);
}

extern "C" size_t mocap_chunk_attn_varlen_dev_workspace_size(int32_t n_items, int64_t max_rows,
                                                             int32_t n_q_heads,
                                                             int32_t n_kv_heads,
                                                             int32_t head_dim) {
  const mocap::Shape sh{n_q_heads, n_kv_heads, head_dim};
  if (mocap::check_shape(sh, 1.0f) != MOCAP_OK) return 0;
  mocap::DevLayout dl;
  return mocap::dev_layout(n_items, max_rows, sh, &dl) ? dl.bytes : 0;
}

extern "C" mocap_status mocap_chunk_attn_varlen_dev(
    const void *q, const void *k_cache, const void *v_cache, const mocap_varlen_item *items,
    int32_t n_items, int64_t q_rows_total, int64_t kv_rows_total, int64_t max_rows,
    int32_t n_q_heads, int32_t n_kv_heads, int32_t head_dim, float scale, void *out, float *lse,
    void *workspace, size_t workspace_bytes, mocap_stream_t stream) {
  const mocap::Shape sh{n_q_heads, n_kv_heads, head_dim};
  const mocap_status st = mocap::check_shape(sh, scale);
  if (st != MOCAP_OK) return st;
  if (n_items < 0 || n_items > MOCAP_VARLEN_DEV_MAX_ITEMS) return MOCAP_EINVAL;
  if (q_rows_total < 0 || kv_rows_total < 0 || q_rows_total > mocap::kMaxRows)
    return MOCAP_EINVAL;
  if (max_rows < 0 || max_rows > mocap::kMaxRows) return MOCAP_EINVAL;
  if (!mocap::pointers_ok(q, k_cache, v_cache, out, lse)) return MOCAP_EINVAL;
  if (n_items == 0) return MOCAP_OK;
  if (items == nullptr || (reinterpret_cast<uintptr_t>(items) & 7u) != 0) return MOCAP_EINVAL;
  mocap::DevLayout dl;
  if (!mocap::dev_layout(n_items, max_rows, sh, &dl)) return MOCAP_EINVAL;
  if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) & 127u) != 0 ||
      workspace_bytes < dl.bytes)
    return MOCAP_EINVAL;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (head_dim == 128)
    return mocap::launch_dev<128>(q, k_cache, v_cache, items, n_items, q_rows_total,
                                  kv_rows_total, sh, scale, out, lse, dl, workspace, s);
  return mocap::launch_dev<64>(q, k_cache, v_cache, items, n_items, q_rows_total, kv_rows_total,
                               sh, scale, out, lse, dl, workspace, s);
}

extern "C" mocap_status mocap_chunk_attn_varlen_append(
    const void *q, const void *k_cache, const void *v_cache, const mocap_varlen_item *items,
    int32_t n_items, int64_t q_rows_total, int64_t kv_rows_total, int32_t n_q_heads,
    int32_t n_kv_heads, int32_t head_dim, float scale, void *out, float *lse, void *workspace,
    size_t workspace_bytes, const mocap_kv_append_item *appends, int32_t n_appends,
    mocap_stream_t stream) {
  return varlen_impl(q, k_cache, v_cache, items, n_items, q_rows_total, kv_rows_total, n_q_heads,
                     n_kv_heads, head_dim, scale, out, lse, workspace, workspace_bytes, stream,
                     appends, n_appends);
}

// ---------------------------------------------------------------------------
// mocap_chunk_attn_noalloc: mocap_chunk_attn for callers that cannot allocate
// device memory.  The split-KV partials go to a fixed scratch array that is
// part of this library's device image; nothing is allocated per call.
//
// Every context that loads the library holds its own copy of the array, from
// load until the context ends, and all calls in a context share it.  Every
// byte a call reads from it was written earlier in the same call, so nothing
// needs clearing; two calls whose work overlaps on the GPU (for example on
// two streams) would overwrite each other's partials.
static __device__ __align__(256) uint8_t g_noalloc_scratch[MOCAP_NOALLOC_SCRATCH_BYTES];

namespace {
std::vector<std::pair<uint64_t, uint8_t *>> g_noalloc_ptr;  // per context ID
std::mutex g_noalloc_mu;

// Device address of g_noalloc_scratch in the current context.  The name is
// only a host-side handle in host code, so the address is looked up once per
// context and cached; nullptr if the lookup fails.  The status word is
// resolved first, which binds the runtime's context to the thread if none
// was current.
uint8_t *noalloc_scratch() {
  if (mocap::device_status_ptr() == nullptr) return nullptr;
  const uint64_t ctx = mocap::current_context();
  if (ctx == 0) return nullptr;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  for (const auto &e : g_noalloc_ptr)
    if (e.first == ctx) return e.second;
  void *ptr = nullptr;
  if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess) return nullptr;
  g_noalloc_ptr.emplace_back(ctx, static_cast<uint8_t *>(ptr));
  return static_cast<uint8_t *>(ptr);
}
}  // namespace

extern "C" mocap_status mocap_chunk_attn_noalloc(const void *q, const void *k_cache,
                                                 const void *v_cache, int64_t prefix, int64_t len,
                                                 int32_t n_q_heads, int32_t n_kv_heads,
                                                 int32_t head_dim, float scale, void *out,
                                                 float *lse, mocap_stream_t stream) {
  const mocap::Shape sh{n_q_heads, n_kv_heads, head_dim};
  const mocap_status st = mocap::check_shape(sh, scale);
  if (st != MOCAP_OK) return st;
  if (prefix < 0 || len < 0 || prefix > mocap::kMaxRows - len) return MOCAP_EINVAL;
  if (!mocap::pointers_ok(q, k_cache, v_cache, out, lse)) return MOCAP_EINVAL;
  if (len == 0) return MOCAP_OK;
  // Exactly mocap_chunk_attn with a workspace of MOCAP_NOALLOC_SCRATCH_BYTES:
  // a split whose partials do not fit runs as the single-pass kernel.
  mocap::SplitPlan sp = plan_for(prefix, len, n_q_heads, n_kv_heads, head_dim);
  if (sp.splits > 1 && sp.bytes > MOCAP_NOALLOC_SCRATCH_BYTES) sp = mocap::SplitPlan();
  void *ws = nullptr;
  if (sp.splits > 1) {
    ws = noalloc_scratch();
    if (ws == nullptr) return MOCAP_ECUDA;
  }
  std::vector<HostItem> items{{0, 0, prefix, len}};
  return mocap::dispatch<1>(q, k_cache, v_cache, items, len, sh, scale, out, lse,
                            reinterpret_cast<cudaStream_t>(stream), sp, ws);
}
