// last_row_attn.cu -- attention of each request's last query row only.
//
// Sec. 2.1: a prefill-only request produces one output token, so the final
// layer needs the attention output of the last prompt row alone: one query
// row per q-head against every key of the request.  That is memory-bound
// (each K/V byte is used by the Hq/Hkv query heads of its group only), so
// this kernel streams K/V at HBM speed instead of running the 128-row tensor
// core tiles of the chunk kernel:
//   grid  = (key-range split, request, KV group); 128 threads per CTA
//   TMA   K and V tiles of 128 keys through a 3-stage ring (bounded waits)
//   S     thread t owns key t: s_h = scale * q_h . k_t for the group's heads
//   soft  per-head online softmax in fp32 (block reductions, log2 domain)
//   P.V   thread t owns dimension t: o_h[t] += sum_keys p_h[key] v[key][t]
// Each CTA writes an fp32 partial (O / l, LSE) for its key range; the
// split-KV combine kernel merges them.
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

// Shared with the chunk kernel's translation unit: merges split partials.
mocap_status launch_attn_combine(const float *o_part, const float *lse_part, int splits,
                                 int64_t len, int n_q_heads, int head_dim, void *out, float *lse,
                                 int64_t lse_stride, cudaStream_t stream);

namespace {

constexpr int kKeys = 128;        // keys per tile
constexpr int kStages = 3;
constexpr int kThreads = 128;
constexpr int kMaxGroup = 16;     // q-heads per KV head
constexpr int kMaxReq = 64;
constexpr int kTilesPerSplit = 16;  // 2048 keys per CTA at most

struct LastRowParams {
  CUtensorMap tk[kMaxReq];  // K of request r: [kv_len_r, Hkv, D], box {64, 1, 128}, 128B swizzle
  CUtensorMap tv[kMaxReq];  // V of request r: same box, no swizzle
  const __nv_bfloat16 *q;   // [n_req, Hq, D]
  float *o_part;            // [splits, n_req, Hq, D]
  float *lse_part;          // [splits, Hq, n_req]
  uint32_t *status;
  int32_t kv_len[kMaxReq];
  int32_t n_req, n_q_heads, n_kv_heads, group, splits;
  float scale_log2;
};

template <int D>
struct LrLayout {
  static constexpr int kTile = kKeys * D * 2;          // one K or V tile (bf16)
  static constexpr int kStage = 2 * kTile;             // K + V
  static constexpr int kRing = 0;
  static constexpr int kQ = kStages * kStage;          // fp32 [G][D]
  static constexpr int kP = kQ + kMaxGroup * D * 4;    // fp32 [G][128]
  static constexpr int kRed = kP + kMaxGroup * kKeys * 4;  // fp32 [4 warps][G]
  static constexpr int kBars = kRed + 4 * kMaxGroup * 4;
  static constexpr int kBytes = kBars + 8 * 2 * kStages + 1024;  // + alignment slack
};
static_assert(LrLayout<128>::kBytes <= 232448, "shared memory");

template <int D>
__global__ void __launch_bounds__(kThreads) last_row_kernel(const __grid_constant__ LastRowParams p) {
  using L = LrLayout<D>;
  extern __shared__ uint8_t sm_raw[];
  // 1024-byte aligned base: swizzled TMA tiles start on a swizzle period
  uint8_t *sm = sm_raw + ((1024u - (smem_u32(sm_raw) & 1023u)) & 1023u);
  const int split = blockIdx.x, r = blockIdx.y, g = blockIdx.z;
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int G = p.group;
  const int kv_len = p.kv_len[r];
  const int tiles = (kv_len + kKeys - 1) / kKeys;
  const int per = (tiles + p.splits - 1) / p.splits;
  const int t0 = min(tiles, split * per), t1 = min(tiles, t0 + per);
  float *q_s = reinterpret_cast<float *>(sm + L::kQ);
  float *p_s = reinterpret_cast<float *>(sm + L::kP);
  float *red = reinterpret_cast<float *>(sm + L::kRed);
  const uint32_t base = smem_u32(sm);
  auto full = [&](int s) { return base + L::kBars + 8u * s; };

  __shared__ uint32_t abort_flag;
  if (t == 0) abort_flag = *reinterpret_cast<volatile uint32_t *>(p.status);
  __syncthreads();
  if (abort_flag != 0u) return;

  // the group's query rows, fp32, pre-scaled by scale * log2(e)
  for (int i = t; i < G * D; i += kThreads) {
    const int h = i / D, c = i % D;
    q_s[i] = __bfloat162float(p.q[(static_cast<int64_t>(r) * p.n_q_heads + g * G + h) * D + c]) *
             p.scale_log2;
  }
  if (t == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(full(s), 1);
    fence_mbar_init();
  }
  __syncthreads();

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
  const int n = t1 - t0;
  int issued = 0;  // tiles whose loads were started (thread 0)
  if (t == 0)
    for (; issued < min(n, kStages); ++issued) issue(t0 + issued, issued);

  float m[kMaxGroup], lsum[kMaxGroup], o[kMaxGroup];
#pragma unroll
  for (int h = 0; h < kMaxGroup; ++h) {
    m[h] = -INFINITY;
    lsum[h] = 0.0f;
    o[h] = 0.0f;
  }
  bool ok = true;
  for (int j = 0; j < n; ++j) {
    const int s = j % kStages;
    const bool landed = mbar_wait(full(s), (j / kStages) & 1, p.status);
    if (!__syncthreads_and(landed)) {  // the whole CTA agrees before unwinding
      ok = false;
      break;
    }
    const uint8_t *kt = sm + L::kRing + s * L::kStage;  // box c: [128 keys][64 dims]
    const uint8_t *vt = kt + L::kTile;
    const int key = (t0 + j) * kKeys + t;
    // ---- scores: thread t = key t
    float sc[kMaxGroup];
#pragma unroll
    for (int h = 0; h < kMaxGroup; ++h) sc[h] = 0.0f;
    for (int c = 0; c < D / 64; ++c) {
      // key t's 64 dims of box c: 16-byte chunk v8 sits at (v8 ^ (t & 7)) * 16
      const uint8_t *krow = kt + c * (kKeys * 128) + t * 128;
#pragma unroll
      for (int v8 = 0; v8 < 8; ++v8) {
        const uint4 kv = *reinterpret_cast<const uint4 *>(krow + ((v8 ^ (t & 7)) << 4));
        const __nv_bfloat162 *k2 = reinterpret_cast<const __nv_bfloat162 *>(&kv);
        float kf[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __bfloat1622float2(k2[e]);
          kf[2 * e] = f.x;
          kf[2 * e + 1] = f.y;
        }
        const int d0 = c * 64 + v8 * 8;
#pragma unroll
        for (int h = 0; h < kMaxGroup; ++h) {
          if (h < G) {
            const float *qh = q_s + h * D + d0;
#pragma unroll
            for (int e = 0; e < 8; ++e) sc[h] = fmaf(qh[e], kf[e], sc[h]);
          }
        }
      }
    }
    if (key >= kv_len)
#pragma unroll
      for (int h = 0; h < kMaxGroup; ++h) sc[h] = -INFINITY;
    // ---- per-head tile max (warp shuffle, then across the 4 warps)
#pragma unroll
    for (int h = 0; h < kMaxGroup; ++h) {
      if (h < G) {
        float v = sc[h];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
        if (lane == 0) red[warp * kMaxGroup + h] = v;
      }
    }
    __syncthreads();
    float alpha[kMaxGroup];
#pragma unroll
    for (int h = 0; h < kMaxGroup; ++h) {
      alpha[h] = 1.0f;
      if (h < G) {
        const float tm = fmaxf(fmaxf(red[h], red[kMaxGroup + h]),
                               fmaxf(red[2 * kMaxGroup + h], red[3 * kMaxGroup + h]));
        const float mn = fmaxf(m[h], tm);  // finite: key tile j contains a valid key
        alpha[h] = ex2_approx(m[h] - mn);  // m = -inf at the first tile: alpha = 0
        m[h] = mn;
        const float pr = ex2_approx(sc[h] - mn);
        p_s[h * kKeys + t] = pr;
        lsum[h] = lsum[h] * alpha[h] + pr;
      }
    }
    __syncthreads();
    // ---- P.V: thread t = dimension t (D == 128; for D == 64 threads >= 64 idle)
    if (t < D) {
      const int c = t / 64, dd = t % 64;
      const uint8_t *vcol = vt + c * (kKeys * 128) + dd * 2;
#pragma unroll
      for (int h = 0; h < kMaxGroup; ++h)
        if (h < G) o[h] *= alpha[h];
      for (int kk = 0; kk < kKeys; ++kk) {
        const float vv = __bfloat162float(*reinterpret_cast<const __nv_bfloat16 *>(vcol + kk * 128));
#pragma unroll
        for (int h = 0; h < kMaxGroup; ++h)
          if (h < G) o[h] = fmaf(p_s[h * kKeys + kk], vv, o[h]);
      }
    }
    __syncthreads();  // stage s and p_s free again
    if (t == 0 && j + kStages < n) {
      issue(t0 + j + kStages, s);
      ++issued;
    }
  }
  if (!ok) {
    // copies still in flight land before the CTA exits
    if (t == 0)
      for (int j = max(0, issued - kStages); j < issued; ++j)
        mbar_wait(full(j % kStages), (j / kStages) & 1, p.status, 20000000ull, false);
    return;
  }
  // ---- row sums: per-thread partials (same rescales) -> block totals
#pragma unroll
  for (int h = 0; h < kMaxGroup; ++h) {
    if (h < G) {
      float v = lsum[h];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      if (lane == 0) red[warp * kMaxGroup + h] = v;
    }
  }
  __syncthreads();
  const int64_t prow = static_cast<int64_t>(split) * p.n_req + r;
#pragma unroll
  for (int h = 0; h < kMaxGroup; ++h) {
    if (h < G) {
      const float l = red[h] + red[kMaxGroup + h] + red[2 * kMaxGroup + h] + red[3 * kMaxGroup + h];
      const bool any = n > 0 && l > 0.0f;
      const int head = g * G + h;
      if (t < D) p.o_part[(prow * p.n_q_heads + head) * D + t] = any ? o[h] / l : 0.0f;
      if (t == 0)
        p.lse_part[(static_cast<int64_t>(split) * p.n_q_heads + head) * p.n_req + r] =
            any ? (m[h] + log2f(l)) * 0.69314718055994530942f : -INFINITY;
    }
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn3() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// [rows, heads, d] bf16, box {64, 1, 128}: row t of a 64-dim box sits at
// t * 128 bytes, its 16-byte chunks permuted by t & 7 when swizzled.
bool make_kv_map(CUtensorMap *map, const void *ptr, int64_t rows, int heads, int d,
                 bool swizzle) {
  auto fn = encode_fn3();
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

int plan_splits(const int64_t *kv_len, int n_req) {
  int64_t max_tiles = 1;
  for (int r = 0; r < n_req; ++r) max_tiles = std::max<int64_t>(max_tiles, (kv_len[r] + kKeys - 1) / kKeys);
  return static_cast<int>((max_tiles + kTilesPerSplit - 1) / kTilesPerSplit);
}

}  // namespace
}  // namespace mocap

extern "C" size_t mocap_last_row_attn_workspace_size(const int64_t *kv_len, int32_t n_req,
                                                     int32_t n_q_heads, int32_t head_dim) {
  if (kv_len == nullptr || n_req < 1 || n_req > mocap::kMaxReq || n_q_heads < 1) return 0;
  const size_t splits = static_cast<size_t>(mocap::plan_splits(kv_len, n_req));
  const size_t o = splits * n_req * n_q_heads * head_dim * sizeof(float);
  return (o + 255) / 256 * 256 + splits * n_q_heads * n_req * sizeof(float);
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
  const size_t need = mocap_last_row_attn_workspace_size(kv_len, n_req, n_q_heads, head_dim);
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
        !make_kv_map(&prm.tv[r], vb, kv_len[r], n_kv_heads, head_dim, false))
      return MOCAP_ECUDA;
    prm.kv_len[r] = static_cast<int32_t>(kv_len[r]);
  }
  const int splits = plan_splits(kv_len, n_req);
  const size_t o_bytes = static_cast<size_t>(splits) * n_req * n_q_heads * head_dim * sizeof(float);
  prm.q = static_cast<const __nv_bfloat16 *>(q_last);
  prm.o_part = static_cast<float *>(workspace);
  prm.lse_part = reinterpret_cast<float *>(static_cast<uint8_t *>(workspace) + (o_bytes + 255) / 256 * 256);
  prm.status = status;
  prm.n_req = n_req;
  prm.n_q_heads = n_q_heads;
  prm.n_kv_heads = n_kv_heads;
  prm.group = n_q_heads / n_kv_heads;
  prm.splits = splits;
  prm.scale_log2 = static_cast<float>(static_cast<double>(scale) * 1.4426950408889634074);
  const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const dim3 grid(splits, n_req, n_kv_heads);
  if (head_dim == 128) {
    static bool attr = false;
    if (!attr) {
      if (cudaFuncSetAttribute(last_row_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               LrLayout<128>::kBytes) != cudaSuccess)
        return MOCAP_ECUDA;
      attr = true;
    }
    last_row_kernel<128><<<grid, kThreads, LrLayout<128>::kBytes, st>>>(prm);
  } else {
    static bool attr = false;
    if (!attr) {
      if (cudaFuncSetAttribute(last_row_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               LrLayout<64>::kBytes) != cudaSuccess)
        return MOCAP_ECUDA;
      attr = true;
    }
    last_row_kernel<64><<<grid, kThreads, LrLayout<64>::kBytes, st>>>(prm);
  }
  if (cudaGetLastError() != cudaSuccess) return MOCAP_ECUDA;
  return launch_attn_combine(prm.o_part, prm.lse_part, splits, n_req, n_q_heads, head_dim, out,
                             lse, n_req, st);
}
