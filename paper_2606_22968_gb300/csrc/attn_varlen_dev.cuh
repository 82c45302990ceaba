// attn_varlen_dev.cuh -- the prepare kernel of mocap_chunk_attn_varlen_dev:
// variable-length attention whose (request, chunk) items live in device
// memory, so a device-side scheduler or a CUDA graph can supply them.
//
// Sec. 2.2 / Eq. 1: one launch serves several (request, chunk) items, each a
// chunk's queries against its request's KV prefix plus itself.  The host
// cannot read the items without a synchronisation, so a one-block kernel
// turns them into what the attention kernel's DEV instantiation reads:
//   varlen_dev_prepare (one block): validates every item, counts its CTAs
//     (128-row blocks x KV groups x head pairs), scans the counts into each
//     item's first CTA, and builds the item's Q, K and V tensor maps from
//     templates over the whole buffers with tensormap.replace (global
//     address at the item's first row, row extent = its rows), so the TMA
//     zero-fills past the item exactly as the per-item maps of the host form
//     do; then publishes the CTA count (0 after an invalid item, with
//     MOCAP_EINVAL in the status word).
//   then, in the same block, the item of every CTA (binary search over the
//     first CTAs), so an attention CTA finds its item with one load.
// The attention launch's grid is an upper bound on the CTA count, from the
// caller's bound on the items' total rows; CTAs past the count exit at once.
#pragma once

#include <cuda.h>

#include "attn_kernel.cuh"

namespace mocap {
namespace {

constexpr int kPrepThreads = 1024;

struct DevPrep {
  CUtensorMap tq, tk, tv;          // templates over the whole Q / K / V buffers
  const mocap_varlen_item *items;  // device, n_items
  ItemDesc *descs;                 // [n_items]
  CUtensorMap *maps;               // [n_items][3]
  int32_t *cta_item;               // [max_ctas]: the item of each CTA
  int32_t *total;                  // CTA count of the launch
  uint32_t *status;
  const uint8_t *q, *k, *v;
  int64_t q_rows_total, kv_rows_total;
  int64_t qrow_bytes, kvrow_bytes;
  int64_t max_ctas;                // the attention grid
  int32_t n_items;
  int32_t ctas_per_block;          // KV groups x head pairs
};

__device__ __forceinline__ void tmap_copy_replace(CUtensorMap *dst, const CUtensorMap &tmpl,
                                                  const void *addr, uint32_t rows) {
  const uint4 *s = reinterpret_cast<const uint4 *>(&tmpl);
  uint4 *d = reinterpret_cast<uint4 *>(dst);
#pragma unroll
  for (int i = 0; i < 8; ++i) d[i] = s[i];
  asm volatile("tensormap.replace.tile.global_address.global.b1024.b64 [%0], %1;" ::"l"(
                   reinterpret_cast<uint64_t>(dst)),
               "l"(reinterpret_cast<uint64_t>(addr))
               : "memory");
  asm volatile("tensormap.replace.tile.global_dim.global.b1024.b32 [%0], 2, %1;" ::"l"(
                   reinterpret_cast<uint64_t>(dst)),
               "r"(rows)
               : "memory");
}

__global__ void __launch_bounds__(kPrepThreads) varlen_dev_prepare(const __grid_constant__ DevPrep a) {
  __shared__ int64_t scan[kPrepThreads];
  __shared__ int64_t carry;
  __shared__ int bad;
  const int tid = static_cast<int>(threadIdx.x);
  if (tid == 0) {
    carry = 0;
    bad = 0;
  }
  __syncthreads();
  for (int64_t first = 0; first < a.n_items; first += kPrepThreads) {
    const int64_t i = first + tid;
    int64_t count = 0;
    if (i < a.n_items) {
      const mocap_varlen_item x = a.items[i];
      const bool ok = x.q_row >= 0 && x.kv_row >= 0 && x.prefix >= 0 && x.len >= 0 &&
                      x.prefix <= 0x7fffffffLL - x.len && x.q_row <= a.q_rows_total - x.len &&
                      x.kv_row <= a.kv_rows_total - (x.prefix + x.len);
      if (!ok) {
        atomicExch(&bad, 1);
      } else if (x.len > 0) {
        const int64_t q_blocks = (x.len + kBlockM - 1) / kBlockM;
        count = q_blocks * a.ctas_per_block;
        ItemDesc &d = a.descs[i];
        d.q_row = x.q_row;
        d.prefix = static_cast<int32_t>(x.prefix);
        d.len = static_cast<int32_t>(x.len);
        d.q_blocks = static_cast<int32_t>(q_blocks);
        CUtensorMap *m = a.maps + 3 * i;
        const uint32_t kv_rows = static_cast<uint32_t>(x.prefix + x.len);
        tmap_copy_replace(m + 0, a.tq, a.q + x.q_row * a.qrow_bytes, static_cast<uint32_t>(x.len));
        tmap_copy_replace(m + 1, a.tk, a.k + x.kv_row * a.kvrow_bytes, kv_rows);
        tmap_copy_replace(m + 2, a.tv, a.v + x.kv_row * a.kvrow_bytes, kv_rows);
      }
    }
    // inclusive scan of the counts (the items' first CTAs follow from it)
    scan[tid] = count;
    __syncthreads();
    for (int off = 1; off < kPrepThreads; off <<= 1) {
      const int64_t add = tid >= off ? scan[tid - off] : 0;
      __syncthreads();
      scan[tid] += add;
      __syncthreads();
    }
    if (i < a.n_items) {
      // every item gets its first CTA, empty ones too (the CTA table's
      // search needs them non-decreasing); clamped, the count check decides
      const int64_t begin = carry + scan[tid] - count;
      a.descs[i].cta_begin = static_cast<int32_t>(begin < 0x7fffffffLL ? begin : 0x7fffffffLL);
    }
    __syncthreads();
    if (tid == 0) carry += scan[kPrepThreads - 1];
    __syncthreads();
  }
  // the maps' generic-proxy writes before any later tensormap-proxy use
  asm volatile("fence.proxy.tensormap::generic.release.gpu;" ::: "memory");
  const bool ok = bad == 0 && carry <= a.max_ctas;
  const int64_t total = ok ? carry : 0;
  if (tid == 0) {
    *a.total = static_cast<int32_t>(total);
    if (!ok) atomicCAS(a.status, 0u, static_cast<uint32_t>(MOCAP_EINVAL));
  }
  // cta_item[c] = the last item whose first CTA is <= c (items without CTAs
  // share their successor's first CTA, so the last such item owns c); the
  // descriptors' first CTAs were written by this block before the barrier
  // above, and __syncthreads orders them for every thread of it
  __syncthreads();
  for (int64_t c = tid; c < total; c += kPrepThreads) {
    int lo = 0, hi = a.n_items - 1;  // descs[0].cta_begin == 0 <= c
    while (lo < hi) {
      const int mid = lo + (hi - lo + 1) / 2;
      if (a.descs[mid].cta_begin <= c) {
        lo = mid;
      } else {
        hi = mid - 1;
      }
    }
    a.cta_item[c] = lo;
  }
}

}  // namespace
}  // namespace mocap
