// last_row_attn.cu -- attention of each request's last query row only.
//
// Sec. 2.1: a prefill-only request produces one output token, so the final
// layer needs the attention output of the last prompt row alone: one query
// row per q-head against every key of the request.  Each K/V byte serves
// only the Hq/Hkv query heads of its group, so the work is memory-bound; the
// kernel streams K/V tiles through TMA and lets the tensor core do the small
// products in transposed form, so the 128 keys (or 128 dims) of a tile sit on
// the 128 TMEM lanes:
//   S^T[key, h]   = K[key, :] . q_h          (M=128 keys, N=16 padded heads)
//   O_t^T[dim, h] = sum_key V[key, dim] p_h[key]   (M=128 dims, A = V^T MN-major)
// Thread t owns key t for the softmax (per-head max / sum by block
// reductions, fp32, log2 domain) and dimension t for the output accumulator
// (registers, rescaled per tile).  grid = (key-range split, request, KV
// group); each CTA writes an fp32 partial (O / l, LSE) and bumps a counter of
// its (request, group); the CTA that completes the count merges the group's
// partials (the split-KV combine, O = sum_s e^(LSE_s - LSE) O_s) in the same
// launch, so no second kernel and no launch gap follow.
#include <cmath>
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <vector>

#include "internal.h"
#include "sm103_ptx.cuh"

namespace mocap {
namespace {

constexpr int kKeys = 128;     // keys per tile = TMEM lanes of S^T
// One K+V tile in flight per CTA; several CTAs per SM (76 KB of shared
// memory each) overlap each other's loads and small MMAs.  Measured on
// GB300 against 2 stages x 2 CTAs/SM: 4.1 vs 3.5 TB/s (131072 keys).
constexpr int kStages = 1;
constexpr int kCtasPerSm = 3;
constexpr int kThreads = 128;
constexpr int kMaxGroup = 16;  // q-heads per KV head (MMA N = 16)
constexpr int kN = 16;
constexpr int kMaxReq = 64;
constexpr int kMaxParts = 512;  // key-range splits of one request (merge scratch)
constexpr uint32_t kTmemCols = 32;  // S^T [0, 16), O^T tile [16, 32)

struct LastRowParams {
  CUtensorMap tk[kMaxReq];  // K of request r: [kv_len_r, Hkv, D], box {64, 1, 128}, 128B swizzle
  CUtensorMap tv[kMaxReq];  // V of request r: same
  const __nv_bfloat16 *q;   // [n_req, Hq, D]
  float *o_part;            // [splits, n_req, Hq, D]
  float *lse_part;          // [splits, Hq, n_req]
  uint32_t *arrived;        // [n_req, Hkv] CTAs done per (request, group); zero at launch
  __nv_bfloat16 *out;       // [n_req, Hq, D]
  float *lse;               // [Hq, n_req]
  uint32_t *status;
  int32_t kv_len[kMaxReq];
  int32_t n_req, n_q_heads, n_kv_heads, group, splits, tiles_per_cta;
  float scale_log2;
};

template <int D>
struct LrLayout {
  static constexpr int kTile = kKeys * D * 2;     // one K or V tile (bf16)
  static constexpr int kStage = 2 * kTile;        // K + V
  static constexpr int kRing = 0;
  static constexpr int kQ = kStages * kStage;     // Q_g: [16 heads x D] K-major, swizzled
  static constexpr int kP = kQ + kN * D * 2;      // P:   [16 heads x 128 keys] K-major
  static constexpr int kRed = kP + kN * kKeys * 2;  // fp32 [4 warps][16]
  static constexpr int kBars = kRed + 4 * kN * 4;   // full[kStages], mma
  static constexpr int kTmemSlot = kBars + 8 * (kStages + 1);
  static constexpr int kBytes = kTmemSlot + 8 + 1024;  // + alignment slack
};
static_assert(LrLayout<128>::kBytes <= 232448, "shared memory");

// Byte offset of element (row, col) in a K-major bf16 operand of `rows`
// rows stored as 64-column boxes with the 128-byte swizzle.
__device__ __forceinline__ uint32_t sw_off(int row, int col, int rows) {
  const int box = col >> 6, c = col & 63;
  return box * rows * 128 + row * 128 + ((((c >> 3) ^ (row & 7)) << 4) | ((c & 7) << 1));
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
}

// Split-KV merge of one (request, group) by one CTA, with the weights in
// shared memory below the `red` area (the drained K/V ring, Q_g and P):
//   1. one warp per head reads the parts' LSEs (lanes over the parts),
//      takes their maximum M_h, and keeps w[k][h] = exp(LSE_kh - M_h) and
//      their sum W_h;
//   2. each thread owns (head, 4 dims) pairs and sums w * O_k over the parts,
//      eight parts at a time, then scales by 1 / W_h.  With exactly two
//      pairs per thread (8 heads at d = 128, 16 at d = 64) both pairs' loads
//      go out together, sixteen in flight per thread.
// Every merged part holds at least one key, so each LSE_kh is finite.
template <int D>
__device__ __forceinline__ void merge_group(const LastRowParams &p, uint8_t *sm, int r, int g,
                                            int n_parts) {
  constexpr int kCols = D / 4;  // float4 columns of a head row
  static_assert(kMaxParts * kMaxGroup * 4 + 2 * kMaxGroup * 4 <= LrLayout<D>::kRed, "merge scratch");
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int G = p.group, Hq = p.n_q_heads;
  float *w = reinterpret_cast<float *>(sm);   // [n_parts][16]
  float *mh = w + kMaxParts * kMaxGroup;      // [16]
  float *wh = mh + kMaxGroup;                 // [16]
  for (int h = warp; h < G; h += kThreads / 32) {
    const float *lse_h = p.lse_part + static_cast<int64_t>(g * G + h) * p.n_req + r;
    const int64_t part_step = static_cast<int64_t>(Hq) * p.n_req;
    float m = -INFINITY;
    for (int k = lane; k < n_parts; k += 64) {  // two independent loads per lane and round
      const float a = __ldcg(lse_h + k * part_step);
      const float b = k + 32 < n_parts ? __ldcg(lse_h + (k + 32) * part_step) : -INFINITY;
      w[k * kMaxGroup + h] = a;
      if (k + 32 < n_parts) w[(k + 32) * kMaxGroup + h] = b;
      m = fmaxf(m, fmaxf(a, b));
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    float sum = 0.0f;
    for (int k = lane; k < n_parts; k += 32) {  // entries this lane wrote itself
      const float e = expf(w[k * kMaxGroup + h] - m);
      w[k * kMaxGroup + h] = e;
      sum += e;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
    if (lane == 0) {
      mh[h] = m;
      wh[h] = sum;
    }
  }
  __syncthreads();
  const float4 *o4 = reinterpret_cast<const float4 *>(p.o_part);
  const int64_t part_stride = static_cast<int64_t>(p.n_req) * Hq * kCols;  // float4s per part
  auto src_of = [&](int h, int c) {
    return o4 + (static_cast<int64_t>(r) * Hq + g * G + h) * kCols + c;
  };
  auto store = [&](int h, int c, float4 acc) {
    const float inv = 1.0f / wh[h];
    const int head = g * G + h;
    __nv_bfloat162 *dst = reinterpret_cast<__nv_bfloat162 *>(
        p.out + (static_cast<int64_t>(r) * Hq + head) * D + 4 * c);
    dst[0] = __floats2bfloat162_rn(acc.x * inv, acc.y * inv);
    dst[1] = __floats2bfloat162_rn(acc.z * inv, acc.w * inv);
    if (c == 0) p.lse[static_cast<int64_t>(head) * p.n_req + r] = mh[h] + logf(wh[h]);
  };
  auto fma4 = [](float4 &acc, float wk, const float4 &v) {
    acc.x += wk * v.x;
    acc.y += wk * v.y;
    acc.z += wk * v.z;
    acc.w += wk * v.w;
  };
  if (G * kCols == 2 * kThreads) {
    // pairs t and t + kThreads: same dims, heads h0 and h0 + kThreads / kCols
    const int c = t % kCols, h0 = t / kCols, h1 = h0 + kThreads / kCols;
    const float4 *s0 = src_of(h0, c), *s1 = src_of(h1, c);
    float4 a0 = make_float4(0.0f, 0.0f, 0.0f, 0.0f), a1 = a0;
    for (int k0 = 0; k0 < n_parts; k0 += 8) {
      float4 v0[8], v1[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const bool in = k0 + u < n_parts;
        v0[u] = in ? __ldcg(s0 + (k0 + u) * part_stride) : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        v1[u] = in ? __ldcg(s1 + (k0 + u) * part_stride) : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const bool in = k0 + u < n_parts;
        fma4(a0, in ? w[(k0 + u) * kMaxGroup + h0] : 0.0f, v0[u]);
        fma4(a1, in ? w[(k0 + u) * kMaxGroup + h1] : 0.0f, v1[u]);
      }
    }
    store(h0, c, a0);
    store(h1, c, a1);
    return;
  }
  for (int pair = t; pair < G * kCols; pair += kThreads) {
    const int h = pair / kCols, c = pair % kCols;
    const float4 *src = src_of(h, c);
    float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    for (int k0 = 0; k0 < n_parts; k0 += 8) {
      float4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        v[u] = k0 + u < n_parts ? __ldcg(src + (k0 + u) * part_stride)
                                : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
      for (int u = 0; u < 8; ++u) fma4(acc, k0 + u < n_parts ? w[(k0 + u) * kMaxGroup + h] : 0.0f, v[u]);
    }
    store(h, c, acc);
  }
}

template <int D>
__global__ void __launch_bounds__(kThreads, kCtasPerSm) last_row_kernel(const __grid_constant__ LastRowParams p) {
  using L = LrLayout<D>;
  extern __shared__ uint8_t sm_raw[];
  uint8_t *sm = sm_raw + ((1024u - (smem_u32(sm_raw) & 1023u)) & 1023u);
  const int split = blockIdx.x, r = blockIdx.y, g = blockIdx.z;
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int G = p.group;
  const int kv_len = p.kv_len[r];
  const int tiles = (kv_len + kKeys - 1) / kKeys;
  const int t0 = min(tiles, split * p.tiles_per_cta), t1 = min(tiles, t0 + p.tiles_per_cta);
  const int n = t1 - t0;
  const uint32_t base = smem_u32(sm);
  float *red = reinterpret_cast<float *>(sm + L::kRed);
  auto full = [&](int s) { return base + L::kBars + 8u * s; };
  const uint32_t mma_bar = base + L::kBars + 8u * kStages;
  const int64_t prow = static_cast<int64_t>(split) * p.n_req + r;

  // TMEM first.  Per-CTA timestamps on GB300 showed an SM starting its next
  // CTA of this kernel only once the CTA before it had given up its TMEM
  // allocation permit, so anything placed before the relinquish delays every
  // later CTA on the SM (Q staging there cost the third CTA ~10 us).
  if (warp == 0) {
    tmem_alloc(base + L::kTmemSlot, kTmemCols);
    tmem_relinquish();
  }
  __shared__ uint32_t abort_flag;
  if (t == 0) abort_flag = *reinterpret_cast<volatile uint32_t *>(p.status);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // an aborted launch, or a split past the request's keys, takes no part
  if (abort_flag != 0u || n <= 0) {
    if (warp == 0) tmem_dealloc(*reinterpret_cast<volatile uint32_t *>(sm + L::kTmemSlot), kTmemCols);
    return;
  }
  const int n_parts = (tiles + p.tiles_per_cta - 1) / p.tiles_per_cta;  // splits with keys

  // Q_g (unscaled bf16) and a zeroed P tile, in the MMA's swizzled layout;
  // 16-byte pieces (8 dims of one head), which the swizzle keeps whole.
  for (int i = t; i < kN * D / 8; i += kThreads) {
    const int h = i / (D / 8), c = (i % (D / 8)) * 8;
    const uint4 v = h < G ? *reinterpret_cast<const uint4 *>(
                                p.q + (static_cast<int64_t>(r) * p.n_q_heads + g * G + h) * D + c)
                          : make_uint4(0, 0, 0, 0);
    *reinterpret_cast<uint4 *>(sm + L::kQ + sw_off(h, c, kN)) = v;
  }
  for (int i = t; i < kN * kKeys / 8; i += kThreads)
    reinterpret_cast<uint4 *>(sm + L::kP)[i] = make_uint4(0, 0, 0, 0);
  if (t == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(full(s), 1);
    mbar_init(mma_bar, 1);
    fence_mbar_init();
  }
  fence_proxy_async_shared();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(sm + L::kTmemSlot);
  const uint32_t lane_addr = tmem + ((static_cast<uint32_t>(warp) * 32u) << 16);

  const CUtensorMap *mk = &p.tk[r];
  const CUtensorMap *mv = &p.tv[r];
  auto issue = [&](int tile, int s) {
    const uint32_t dst = base + L::kRing + s * L::kStage;
    mbar_arrive_expect_tx(full(s), L::kStage);
    for (int c = 0; c < D / 64; ++c) {
      tma_load_3d(dst + c * (kKeys * 128), mk, full(s), c * 64, g, tile * kKeys);
      tma_load_3d(dst + L::kTile + c * (kKeys * 128), mv, full(s), c * 64, g, tile * kKeys);
    }
  };
  int issued = 0;
  if (t == 0)
    for (; issued < min(n, kStages); ++issued) issue(t0 + issued, issued);

  // V^T as the M=128 A operand: dims 64..127 are the tile's second 64-dim
  // box (16 KB on).  With D = 64 there is no second box, so it aliases the
  // first (leading offset 0): those lanes of O^T are never read, and every
  // operand read stays inside this stage's V tile.
  constexpr uint32_t kVAtomStride = D == 128 ? kKeys * 128 : 0;
  constexpr uint32_t idesc_s = idesc_bf16_f32(128, kN, false, false);
  constexpr uint32_t idesc_o = idesc_bf16_f32(128, kN, true, false);
  const float sl2 = p.scale_log2;
  float m[kMaxGroup], lsum[kMaxGroup], o[kMaxGroup];
#pragma unroll
  for (int h = 0; h < kMaxGroup; ++h) {
    m[h] = -INFINITY;
    lsum[h] = 0.0f;
    o[h] = 0.0f;
  }
  bool ok = true;
  int mma_phase = 0;
  for (int j = 0; j < n; ++j) {
    const int s = j % kStages;
    const uint32_t kt = base + L::kRing + s * L::kStage, vt = kt + L::kTile;
    if (!__syncthreads_and(mbar_wait(full(s), (j / kStages) & 1, p.status))) {
      ok = false;
      break;
    }
    // ---- S^T = K . Q_g^T (keys on the lanes)
    if (t == 0) {
      tc_fence_after();
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t off = (kk / 4) * (kKeys * 128) + (kk % 4) * 32;
        const uint32_t qoff = (kk / 4) * (kN * 128) + (kk % 4) * 32;
        mma_ss(tmem, sdesc_sw128(kt + off, 16, 1024), sdesc_sw128(base + L::kQ + qoff, 16, 1024),
               idesc_s, kk > 0 ? 1u : 0u);
      }
      tc_commit(mma_bar);
    }
    if (!__syncthreads_and(mbar_wait(mma_bar, mma_phase & 1, p.status))) {
      ok = false;
      break;
    }
    ++mma_phase;
    tc_fence_after();
    uint32_t sr[16];
    tmem_ld16(lane_addr, sr);
    const bool valid_key = (t0 + j) * kKeys + t < kv_len;
    float sc[kMaxGroup];
#pragma unroll
    for (int h = 0; h < kMaxGroup; ++h) {
      sc[h] = valid_key ? __uint_as_float(sr[h]) * sl2 : -INFINITY;
      float v = sc[h];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
      if (lane == 0) red[warp * kN + h] = v;
    }
    __syncthreads();
    float alpha[kMaxGroup];
#pragma unroll
    for (int h = 0; h < kMaxGroup; ++h) {
      const float tm = fmaxf(fmaxf(red[h], red[kN + h]), fmaxf(red[2 * kN + h], red[3 * kN + h]));
      const float mn = fmaxf(m[h], tm);  // finite: each tile holds a valid key
      alpha[h] = ex2_approx(m[h] - mn);  // 0 on the first tile (m = -inf)
      m[h] = mn;
      const float pr = ex2_approx(sc[h] - mn);
      lsum[h] = lsum[h] * alpha[h] + pr;
      if (h < G)
        *reinterpret_cast<__nv_bfloat16 *>(sm + L::kP + sw_off(h, t, kN)) = __float2bfloat16_rn(pr);
    }
    fence_proxy_async_shared();
    tc_fence_before();
    __syncthreads();
    // ---- O_t^T = V^T . P^T (dims on the lanes)
    if (t == 0) {
      tc_fence_after();
#pragma unroll
      for (int kk = 0; kk < kKeys / 16; ++kk) {
        const uint32_t poff = (kk / 4) * (kN * 128) + (kk % 4) * 32;
        mma_ss(tmem + kN, sdesc_sw128(vt + kk * 2048, kVAtomStride, 1024),
               sdesc_sw128(base + L::kP + poff, 16, 1024), idesc_o, kk > 0 ? 1u : 0u);
      }
      tc_commit(mma_bar);
    }
    if (!__syncthreads_and(mbar_wait(mma_bar, mma_phase & 1, p.status))) {
      ok = false;
      break;
    }
    ++mma_phase;
    tc_fence_after();
    uint32_t orr[16];
    tmem_ld16(lane_addr + kN, orr);
#pragma unroll
    for (int h = 0; h < kMaxGroup; ++h) o[h] = o[h] * alpha[h] + __uint_as_float(orr[h]);
    tc_fence_before();
    __syncthreads();  // stage s, P and TMEM are free again
    if (t == 0 && issued < n) {
      issue(t0 + issued, issued % kStages);
      ++issued;
    }
  }
  if (!ok) {
    if (t == 0) {
      for (int j = max(0, issued - kStages); j < issued; ++j)
        mbar_wait(full(j % kStages), (j / kStages) & 1, p.status, 20000000ull, false);
      tc_commit(mma_bar);  // drain issued MMAs before TMEM is released
      mbar_wait(mma_bar, mma_phase & 1, p.status, 20000000ull, false);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
      tc_fence_after();
      tmem_dealloc(tmem, kTmemCols);
    }
    return;
  }
  // ---- row sums over the block; write this split's partial
#pragma unroll
  for (int h = 0; h < kMaxGroup; ++h) {
    float v = lsum[h];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    if (lane == 0) red[warp * kN + h] = v;
  }
  __syncthreads();
#pragma unroll
  for (int h = 0; h < kMaxGroup; ++h) {
    if (h < G) {
      const float l = red[h] + red[kN + h] + red[2 * kN + h] + red[3 * kN + h];
      const int head = g * G + h;
      if (t < D) p.o_part[(prow * p.n_q_heads + head) * D + t] = o[h] / l;
      if (t == 0)
        p.lse_part[(static_cast<int64_t>(split) * p.n_q_heads + head) * p.n_req + r] =
            (m[h] + log2f(l)) * 0.69314718055994530942f;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }

  // ---- the last of the group's n_parts CTAs merges their partials
  __shared__ uint32_t is_last;
  __threadfence();  // this CTA's partial is visible device-wide before the count
  __syncthreads();
  if (t == 0) {
    const uint32_t before = atomicAdd(p.arrived + r * p.n_kv_heads + g, 1u);
    is_last = before + 1u == static_cast<uint32_t>(n_parts) ? 1u : 0u;
  }
  __syncthreads();
  if (is_last == 0u) return;
  __threadfence();  // order the partial reads after the count that completed
  merge_group<D>(p, sm, r, g, n_parts);
}

// [rows, heads, d] bf16, box {64, 1, 128}: row t of a 64-dim box sits at
// t * 128 bytes, its 16-byte chunks permuted by t & 7 when swizzled.
bool make_kv_map(CUtensorMap *map, const void *ptr, int64_t rows, int heads, int d,
                 bool swizzle) {
  auto fn = tensor_map_encoder();
  if (fn == nullptr) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(heads),
                        static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(d) * 2,
                           static_cast<cuuint64_t>(heads) * static_cast<cuuint64_t>(d) * 2};
  cuuint32_t box[3] = {64u, 1u, static_cast<cuuint32_t>(kKeys)};
  cuuint32_t elem[3] = {1u, 1u, 1u};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), dims, strides, box,
            elem, CU_TENSOR_MAP_INTERLEAVE_NONE,
            swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tiles per CTA so that all (request, group) key ranges give about
// kCtasPerSm CTAs per SM in total; the split count is what the longest
// request needs.
struct LrPlan {
  int tiles_per_cta = 1, splits = 1;
};
LrPlan plan_splits(const int64_t *kv_len, int n_req, int n_kv_heads) {
  int64_t total = 0, max_tiles = 1;
  for (int r = 0; r < n_req; ++r) {
    const int64_t tr = std::max<int64_t>(1, (kv_len[r] + kKeys - 1) / kKeys);
    total += tr;
    max_tiles = std::max(max_tiles, tr);
  }
  const int64_t target_ctas = static_cast<int64_t>(kCtasPerSm) * device_sm_count();
  int64_t per = (total * n_kv_heads + target_ctas - 1) / target_ctas;
  per = std::max<int64_t>(1, per);
  per = std::max<int64_t>(per, (max_tiles + kMaxParts - 1) / kMaxParts);
  LrPlan pl;
  pl.tiles_per_cta = static_cast<int>(per);
  pl.splits = static_cast<int>((max_tiles + per - 1) / per);  // <= kMaxParts
  return pl;
}

}  // namespace
}  // namespace mocap

extern "C" size_t mocap_last_row_attn_workspace_size(const int64_t *kv_len, int32_t n_req,
                                                     int32_t n_q_heads, int32_t n_kv_heads,
                                                     int32_t head_dim) {
  if (kv_len == nullptr || n_req < 1 || n_req > mocap::kMaxReq || n_q_heads < 1 ||
      n_kv_heads < 1)
    return 0;
  const size_t splits = static_cast<size_t>(mocap::plan_splits(kv_len, n_req, n_kv_heads).splits);
  const size_t o = splits * n_req * n_q_heads * head_dim * sizeof(float);
  const size_t l = splits * n_q_heads * n_req * sizeof(float);
  return (o + 255) / 256 * 256 + (l + 255) / 256 * 256 +
         static_cast<size_t>(n_req) * n_kv_heads * sizeof(uint32_t);
}

extern "C" mocap_status mocap_last_row_attn(const void *q_last, const void *k_cache,
                                            const void *v_cache, const int64_t *kv_row,
                                            const int64_t *kv_len, int32_t n_req,
                                            int64_t kv_rows_total, int32_t n_q_heads,
                                            int32_t n_kv_heads, int32_t head_dim, float scale,
                                            void *out, float *lse, void *workspace,
                                            size_t workspace_bytes, mocap_stream_t stream) {
  using namespace mocap;
  if (!q_last || !k_cache || !v_cache || !kv_row || !kv_len || !out || !lse || !workspace)
    return MOCAP_EINVAL;
  if (!aligned16(q_last) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(out) ||
      !aligned16(workspace) || (reinterpret_cast<uintptr_t>(lse) & 3u))
    return MOCAP_EINVAL;
  if (n_req < 1 || n_req > kMaxReq) return MOCAP_EINVAL;
  if (n_q_heads < 1 || n_kv_heads < 1 || n_q_heads % n_kv_heads) return MOCAP_EINVAL;
  if (n_q_heads / n_kv_heads > kMaxGroup) return MOCAP_EUNSUPPORTED;
  if (head_dim != 64 && head_dim != 128) return MOCAP_EUNSUPPORTED;
  if (!(scale > 0.0f) || !std::isfinite(scale)) return MOCAP_EINVAL;
  for (int r = 0; r < n_req; ++r)
    if (kv_len[r] < 1 || kv_row[r] < 0 || kv_len[r] > 0x7fffffffLL ||
        kv_row[r] > kv_rows_total - kv_len[r])
      return MOCAP_EINVAL;
  const size_t need =
      mocap_last_row_attn_workspace_size(kv_len, n_req, n_q_heads, n_kv_heads, head_dim);
  if (workspace_bytes < need) return MOCAP_EINVAL;
  uint32_t *status = device_status_ptr();
  if (status == nullptr) return MOCAP_ECUDA;

  static LastRowParams prm;
  static std::mutex mu;
  std::lock_guard<std::mutex> lock(mu);
  std::memset(&prm, 0, sizeof(prm));
  const size_t row_bytes = static_cast<size_t>(n_kv_heads) * head_dim * 2;
  for (int r = 0; r < n_req; ++r) {
    const auto *kb = static_cast<const uint8_t *>(k_cache) + kv_row[r] * row_bytes;
    const auto *vb = static_cast<const uint8_t *>(v_cache) + kv_row[r] * row_bytes;
    if (!make_kv_map(&prm.tk[r], kb, kv_len[r], n_kv_heads, head_dim, true) ||
        !make_kv_map(&prm.tv[r], vb, kv_len[r], n_kv_heads, head_dim, true))
      return MOCAP_ECUDA;
    prm.kv_len[r] = static_cast<int32_t>(kv_len[r]);
  }
  const LrPlan plan = plan_splits(kv_len, n_req, n_kv_heads);
  const int splits = plan.splits;
  const size_t o_bytes = static_cast<size_t>(splits) * n_req * n_q_heads * head_dim * sizeof(float);
  const size_t l_bytes = static_cast<size_t>(splits) * n_q_heads * n_req * sizeof(float);
  auto *ws = static_cast<uint8_t *>(workspace);
  prm.q = static_cast<const __nv_bfloat16 *>(q_last);
  prm.o_part = reinterpret_cast<float *>(ws);
  prm.lse_part = reinterpret_cast<float *>(ws + (o_bytes + 255) / 256 * 256);
  prm.arrived = reinterpret_cast<uint32_t *>(ws + (o_bytes + 255) / 256 * 256 +
                                             (l_bytes + 255) / 256 * 256);
  prm.out = static_cast<__nv_bfloat16 *>(out);
  prm.lse = lse;
  prm.status = status;
  prm.n_req = n_req;
  prm.n_q_heads = n_q_heads;
  prm.n_kv_heads = n_kv_heads;
  prm.group = n_q_heads / n_kv_heads;
  prm.splits = splits;
  prm.tiles_per_cta = plan.tiles_per_cta;
  prm.scale_log2 = static_cast<float>(static_cast<double>(scale) * 1.4426950408889634074);
  const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(prm.arrived, 0, static_cast<size_t>(n_req) * n_kv_heads * sizeof(uint32_t),
                      st) != cudaSuccess)
    return MOCAP_ECUDA;
  const dim3 grid(splits, n_req, n_kv_heads);
  const uint64_t ctx = current_context();
  if (ctx == 0) return MOCAP_ECUDA;
  // the shared-memory size is a per-context attribute of each kernel
  auto prepare = [&](auto kern, int smem, ContextOnce &once) -> bool {
    if (once.done(ctx)) return true;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
        cudaSuccess)
      return false;
    once.mark(ctx);
    return true;
  };
  if (head_dim == 128) {
    static ContextOnce once;
    if (!prepare(last_row_kernel<128>, LrLayout<128>::kBytes, once)) return MOCAP_ECUDA;
    last_row_kernel<128><<<grid, kThreads, LrLayout<128>::kBytes, st>>>(prm);
  } else {
    static ContextOnce once;
    if (!prepare(last_row_kernel<64>, LrLayout<64>::kBytes, once)) return MOCAP_ECUDA;
    last_row_kernel<64><<<grid, kThreads, LrLayout<64>::kBytes, st>>>(prm);
  }
  return cudaGetLastError() == cudaSuccess ? MOCAP_OK : MOCAP_ECUDA;
}
