/*
 * mocap.h -- C ABI of the GB300 (sm_103a) chunked causal prefill attention
 * library: the data-parallel hot path of MOCAP's prefill-only method
 * (arXiv 2606.22968).
 *
 * The method (Sec. 2.2, Sec. 3.2 / Eq. 1, Sec. 4.2): a long prompt of S
 * tokens is split into M chunks with boundaries 0 = b_0 < b_1 < ... < b_M = S.
 * Chunk i (rows [b_i, b_{i+1})) attends to the keys/values of all earlier
 * chunks plus a causal block over itself, so its attention cost grows with
 * its prefix; Latency-Balanced Chunk Partitioning picks boundaries that
 * balance that cost.  The library exposes:
 *
 *   mocap_lbcp_partition      chunk boundaries (host, exact integers)
 *   mocap_lbcp_partition_dp   boundaries from Algorithm 1's stage-1 DP (host)
 *   mocap_lbcp_partition_dp_latency  the same DP with the kernel's latency model
 *   mocap_lbcp_gemm_weight    the DP's GEMM-term weight from measured rates (host)
 *   mocap_kv_append           chunk K/V -> contiguous bf16 KV cache (device)
 *   mocap_kv_append_overlap   the same, sized to run beside an attention launch
 *   mocap_copy_from_host, mocap_copy_to_host
 *                             host <-> device copies by the SMs (a prompt's
 *                             inputs up, its results back)
 *   mocap_qkv_rope_append     QKV projection + RoPE + KV append (device GEMM)
 *   mocap_chunk_attn          one chunk's GQA attention over cache[0, prefix+len)
 *   mocap_chunk_attn_varlen   the same for many (request, chunk) items in one launch
 *   mocap_chunk_attn_varlen_dev  the same with the items in device memory
 *   mocap_chunk_attn_append, mocap_chunk_attn_varlen_append
 *                             the same with the next chunk's KV append in the launch
 *   mocap_last_row_attn       each request's last row only (prefill-only output)
 *   mocap_last_device_status  bounded-wait timeouts reported by the kernels
 *   mocap_selftest_bounded_wait  drives that timeout path on purpose (tests)
 *   mocap_status_string       text for a status code
 *
 * Conventions for every entry point:
 *   - Tensor pointers are DEVICE pointers owned by the caller.  The library
 *     never allocates, frees or retains caller memory.
 *   - Layouts are dense row-major with no padding:
 *       Q, O      bf16 [rows, n_q_heads, head_dim]
 *       K, V      bf16 [rows, n_kv_heads, head_dim]   (chunk input or cache)
 *       LSE       fp32 [n_q_heads, rows]
 *     Device pointers must be 16-byte aligned.
 *   - Work is enqueued on `stream` (NULL = legacy default stream) and the
 *     call returns without synchronising.  No hidden host<->device traffic.
 *   - Arguments are validated before any launch; on MOCAP_EINVAL or
 *     MOCAP_EUNSUPPORTED nothing was enqueued.  MOCAP_ECUDA reports a failed
 *     CUDA call or launch (the launch error is consumed).
 *   - Calls run in the CUDA context current on the calling thread: the
 *     device's primary context (the CUDA runtime API's), or one the caller
 *     made current with the driver API.  State that belongs to a context
 *     (the status word's address, kernel attributes set on first use, the
 *     no-allocation scratch address) is set up once per context, on its
 *     first call, which should come before any stream capture.
 *   - Entry points may be called from several host threads; launches that
 *     share a caller workspace must not overlap on the GPU.
 */
#ifndef MOCAP_H_
#define MOCAP_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *mocap_stream_t; /* same object as cudaStream_t */

typedef enum {
  MOCAP_OK = 0,
  MOCAP_EINVAL = 1,        /* bad argument (null, range, alignment, shape)   */
  MOCAP_ECUDA = 2,         /* a CUDA runtime/driver call failed              */
  MOCAP_EUNSUPPORTED = 3,  /* valid request this build does not implement    */
  MOCAP_ETIMEOUT = 4       /* a device-side bounded wait expired             */
} mocap_status;

typedef enum {
  MOCAP_PART_UNIFORM = 0,  /* n_i = round_half_up(i * U / M)                 */
  MOCAP_PART_LBCP = 1      /* n_i = round_half_up(U * sqrt(i / M))           */
} mocap_part_mode;

/*
 * mocap_lbcp_partition -- chunk boundaries with equal attention cost.
 *
 * Sec. 3.2, Eq. 1: chunk i of length c_i with prefix p_i costs attention work
 * that grows with c_i * (keys seen).  We balance cost_i = c_i * (p_i + c_i/2),
 * the causal pair count up to its O(c_i) term; since 2 * cost_i =
 * b_{i+1}^2 - b_i^2 the equal-cost split is b_i = S * sqrt(i / M) (the
 * compute-balanced initialisation of Sec. 4.2 / Algorithm 1 stage 1, for the
 * attention term).  Boundaries are snapped to multiples of `granularity` g:
 * with U = seq_len / g (floor), n_i = round_half_up(U * sqrt(i / M)) computed
 * exactly in integers, b_i = g * n_i, then in one forward pass
 * b_i = min(max(b_i, b_{i-1} + g), g * (U - (M - i))), b_0 = 0, b_M = seq_len.
 * MOCAP_PART_UNIFORM uses n_i = round_half_up(i * U / M) with the same clamps.
 * Every chunk has at least g tokens; the last absorbs seq_len % g.
 *
 *   seq_len      S, tokens, 1 <= S
 *   num_chunks   M >= 1, with M * granularity <= S and S / g < 2^31
 *   granularity  g >= 1 (128 matches the attention kernel's row tile)
 *   boundaries   HOST array of num_chunks + 1 int64, written on success
 *
 * Pure host integer code: deterministic and bit-exact, no CUDA calls.
 * Returns MOCAP_EINVAL for a null pointer or out-of-range argument.
 */
mocap_status mocap_lbcp_partition(int64_t seq_len, int32_t num_chunks,
                                  int32_t granularity, mocap_part_mode mode,
                                  int64_t *boundaries);

typedef enum {
  MOCAP_COST_CAUSAL = 0,   /* chunk cost c (p + c/2): causal (query, key) pairs */
  MOCAP_COST_EQ1 = 1       /* chunk cost c (p + c): Eq. 1 as printed            */
} mocap_cost_model;

/*
 * mocap_lbcp_partition_dp -- chunk boundaries from the dynamic program of
 * Algorithm 1, stage 1 (Sec. 4.2): the compute-balanced initialisation that
 * minimises t_sum + (N - 1) t_max for an N-stage chunked pipeline.
 *
 * Positions and sizes are counted in units of `granularity` (U = seq_len /
 * g; the last chunk absorbs seq_len % g).  EvaluateChunk(k, s), the cost of a
 * chunk of k units starting at unit s, is k (2 s + k) (MOCAP_COST_CAUSAL,
 * twice c (p + c/2)) or 2 k (s + k) (MOCAP_COST_EQ1, twice Eq. 1's c (p + c)),
 * plus gemm_weight * k for the GEMM term of Eq. 1.  The loops run as in the
 * algorithm: chunk index m from M down to 1, start s from U-1 down to 0,
 * size k upward; state (m, s) keeps the first k that gives the smallest
 * t_sum + (N - 1) max(t, t_max) over its suffix.  Exact integer arithmetic:
 * bit-exact on every platform.  The stage-2 simulated annealing of
 * Algorithm 1 needs the paper's multi-stage execution model and is not
 * provided.
 *
 *   num_stages   N >= 1 pipeline stages
 *   gemm_weight  0 .. 2^40, weight of the linear term (same doubled units)
 *   boundaries   HOST array of num_chunks + 1 int64, written on success
 * MOCAP_EINVAL for bad arguments, including N (2 U^2 + gemm_weight U) >=
 * 2^62 (the compared objective t_sum + (N - 1) t_max could leave int64);
 * MOCAP_EUNSUPPORTED when M * U^2 > 4e9 (the O(M U^2) host work would be too
 * long; use a coarser granularity).
 */
mocap_status mocap_lbcp_partition_dp(int64_t seq_len, int32_t num_chunks,
                                     int32_t granularity, int32_t num_stages,
                                     mocap_cost_model model, int64_t gemm_weight,
                                     int64_t *boundaries);

/*
 * mocap_lbcp_partition_dp_latency -- Algorithm 1's stage-1 DP (Sec. 4.2) with
 * EvaluateChunk as the compute latency of this library's chunk attention
 * kernel on a GPU with `num_sms` SMs, in 128-row units.
 *
 * The latency model (integer picoseconds, so the result is bit-exact on
 * every platform): the chunk's CTAs -- n_kv_heads * ceil((n_q_heads /
 * n_kv_heads) / 2) per 128-row query block, block qb seeing
 * ceil(min(prefix + 128 (qb + 1), prefix + len) / 128) key tiles -- are
 * list-scheduled, heaviest block first, each onto a least-loaded SM; a CTA
 * costs 4 us plus 1.4 us * (head_dim / 128) per key tile it covers; with
 * the key range split in s = 2..4 parts (considered only below 8 CTAs per SM)
 * each CTA covers floor((j+1) T / s) - floor(j T / s) tiles and the merge
 * adds 3 us + (bytes moved) / (5 bytes per ps); the chunk takes its fastest
 * split.  These are the costs the split planner of mocap_chunk_attn uses.
 * Unlike the causal pair count, the model sees how a chunk's CTAs fill the
 * SMs' waves (measured on GB300: it tracks per-chunk attention latency with
 * correlation 0.92, the pair count 0.59).
 *
 * Loops and tie rule as mocap_lbcp_partition_dp (m down, s down, k up,
 * strict improvement of t_sum + (N - 1) t_max), with each interior boundary
 * limited to `window` units either side of mocap_lbcp_partition's
 * closed-form LBCP boundary (window 0 returns that split).  The last chunk
 * absorbs seq_len % 128.
 *
 *   num_stages   N >= 1;  n_q_heads a multiple of n_kv_heads (<= 4096)
 *   head_dim     64 or 128 (else MOCAP_EUNSUPPORTED);  num_sms 1 .. 4096
 *   window       >= 0 units of 128 rows
 *   boundaries   HOST array of num_chunks + 1 int64, written on success
 * MOCAP_EINVAL for bad arguments (seq_len < 2^31, num_chunks * 128 <=
 * seq_len); MOCAP_EUNSUPPORTED when the windows' chunk evaluations would be
 * too much host work (use a smaller window).  Pure host code.
 */
mocap_status mocap_lbcp_partition_dp_latency(int64_t seq_len, int32_t num_chunks,
                                             int32_t num_stages, int32_t n_q_heads,
                                             int32_t n_kv_heads, int32_t head_dim,
                                             int32_t num_sms, int32_t window,
                                             int64_t *boundaries);

/*
 * mocap_lbcp_gemm_weight -- the gemm_weight argument of
 * mocap_lbcp_partition_dp for chunk stages whose measured cost is
 * a * (causal query-key pairs) + b * (rows): Eq. 1's attention term plus its
 * GEMM term (Sec. 3.2).  A chunk of k units of `granularity` g rows starting
 * at unit s has about g^2 k (s + k/2) pairs and g k rows, so in the DP's
 * doubled units its cost is proportional to k (2 s + k) + w k with
 * w = 2 b / (g a), rounded half up.
 *
 *   attn_s_per_pair  a > 0 (seconds, or any unit shared with b)
 *   gemm_s_per_row   b >= 0
 *   weight           HOST int64, written on success
 * MOCAP_EINVAL for a null pointer, granularity < 1, a <= 0, b < 0, NaN, or a
 * weight above 2^40.  Pure host arithmetic.
 */
mocap_status mocap_lbcp_gemm_weight(double attn_s_per_pair, double gemm_s_per_row,
                                    int32_t granularity, int64_t *weight);

/*
 * mocap_kv_append -- write a chunk's K and V into the KV cache.
 *
 * Sec. 2.2 / Sec. 3.1: the KV of every earlier chunk stays live for later
 * chunks.  Copies rows [0, len) of k_chunk/v_chunk (bf16 [len, n_kv_heads,
 * head_dim]) to rows [offset, offset + len) of k_cache/v_cache (bf16
 * [cache_capacity, n_kv_heads, head_dim]), bit-exact; no other cache byte is
 * touched.  Source and destination must not overlap.
 *
 * MOCAP_EINVAL: null pointer, misaligned pointer, offset < 0, len < 0,
 * offset + len > cache_capacity, n_kv_heads < 1, head_dim < 1 or
 * n_kv_heads * head_dim not a multiple of 8.  len == 0 is a no-op.
 */
mocap_status mocap_kv_append(const void *k_chunk, const void *v_chunk,
                             void *k_cache, void *v_cache,
                             int64_t cache_capacity, int64_t offset, int64_t len,
                             int32_t n_kv_heads, int32_t head_dim,
                             mocap_stream_t stream);

/*
 * mocap_kv_append_overlap -- mocap_kv_append with a kernel sized to run
 * beside a concurrently running attention launch (Sec. 2.2: chunk i + 1's
 * K/V can be written while chunk i attends, since chunk i never reads those
 * rows).  Its CTAs are one warp of at most 32 registers per thread and use
 * no shared memory: that fits in what an attention CTA (384 threads x 168
 * registers) leaves free on an SM, so the copy proceeds on every SM while
 * the attention runs instead of waiting for SMs to drain.  Meant for a
 * second stream whose work is joined (event) before the attention that
 * reads the rows.  Same arguments, checks and results as mocap_kv_append;
 * its own bandwidth is lower (a few TB/s at most), by design.
 */
mocap_status mocap_kv_append_overlap(const void *k_chunk, const void *v_chunk,
                                     void *k_cache, void *v_cache,
                                     int64_t cache_capacity, int64_t offset, int64_t len,
                                     int32_t n_kv_heads, int32_t head_dim,
                                     mocap_stream_t stream);

/*
 * One host -> device copy of mocap_copy_from_host: `bytes` bytes (a multiple
 * of 16) from page-locked host memory at `src` to device memory at `dst`,
 * both 16-byte aligned.
 */
typedef struct {
  void *dst;
  const void *src;
  int64_t bytes;
} mocap_copy_item;

#define MOCAP_COPY_MAX_ITEMS 8

/*
 * mocap_copy_from_host -- up to MOCAP_COPY_MAX_ITEMS host -> device copies
 * in one kernel launch on `stream`, done by the SMs reading the host pages
 * through their device mapping (a prompt's Q/K/V on their way to the chunk
 * pipeline, Sec. 2.2).  On GB300 the copy engines' uploads from page-locked
 * memory ran at about 20 GB/s right after heavy device work in most trials,
 * where SM loads of the same pages kept the link's ~200 GB/s.
 *
 *   beside_kernels  0: all SMs (the GPU otherwise idle, e.g. a prompt's
 *                   first chunk); nonzero: one warp per SM with at most 32
 *                   registers and no shared memory, which fits beside a
 *                   running attention launch (as mocap_kv_append_overlap).
 *
 * Each source range must lie in one page-locked allocation (cudaHostAlloc,
 * cudaMallocHost or cudaHostRegister) that the device sees at the same
 * address (unified addressing), each destination in device memory; both
 * ends of every range are checked with cudaPointerGetAttributes.  The host
 * memory must stay valid and unchanged until the copy has run.
 * MOCAP_EINVAL: n_items outside [0, MOCAP_COPY_MAX_ITEMS], a null item
 * array, a null or misaligned pointer, bytes < 0 or not a multiple of 16, a
 * source that is not such host memory or a destination that is not device
 * memory.  Items of 0 bytes are skipped.
 */
mocap_status mocap_copy_from_host(const mocap_copy_item *items, int32_t n_items,
                                  int32_t beside_kernels, mocap_stream_t stream);

/*
 * mocap_copy_to_host -- the same in the other direction: each item copies
 * `bytes` from device memory at `src` to page-locked host memory at `dst`
 * (a chunk's O and LSE on their way back), with the SMs storing through the
 * host pages' device mapping; the copy engines' returns slowed the same way
 * after heavy device work.  Same launch forms, checks (device source,
 * mapped page-locked destination) and errors as mocap_copy_from_host.
 */
mocap_status mocap_copy_to_host(const mocap_copy_item *items, int32_t n_items,
                                int32_t beside_kernels, mocap_stream_t stream);

/*
 * mocap_qkv_rope_append -- a chunk's QKV projection, rotary embedding and KV
 * append in one kernel.
 *
 * Sec. 3.2 / Eq. 1: each chunk also pays GEMM work that grows with its
 * length alone; the QKV projection is the one attention depends on.  For the
 * chunk's hidden states X (bf16 [len, hidden]) and the packed weights W (bf16
 * [(Hq + 2 Hkv) d, hidden]; rows 0 .. Hq d - 1 produce Q, the next Hkv d
 * produce K, the last Hkv d produce V):
 *   [Q | K | V] = X W^T                                   (fp32 accumulate)
 *   Q and K rotated at positions offset + r (rotate-half RoPE: dims j and
 *   j + d/2 of each head turn by (offset + r) * rope_theta^(-2j/d))
 *   q_out[r]                 <- Q (bf16 [len, Hq, d])
 *   k_cache[offset + r], v_cache[offset + r] <- K, V (bf16 [capacity, Hkv, d])
 * so the attention of the same chunk can run right after it.  Cache rows
 * outside [offset, offset + len) are not touched.
 *
 * Requirements: head_dim in {64, 128} and (Hq + 2 Hkv) * head_dim a multiple
 * of 256 (else MOCAP_EUNSUPPORTED); hidden a multiple of 8; rope_theta > 1;
 * 16-byte aligned pointers; offset + len <= cache_capacity.  len == 0 is a
 * no-op.  Persistent tcgen05 GEMM: 128 x 256 output tiles, K steps of 64.
 */
mocap_status mocap_qkv_rope_append(const void *x, const void *w_qkv, void *q_out,
                                   void *k_cache, void *v_cache, int64_t cache_capacity,
                                   int64_t offset, int64_t len, int32_t hidden,
                                   int32_t n_q_heads, int32_t n_kv_heads, int32_t head_dim,
                                   float rope_theta, mocap_stream_t stream);

/*
 * mocap_chunk_attn -- attention of one chunk against its KV prefix.
 *
 * Sec. 2.2 / Eq. 1: the chunk's queries (global rows prefix .. prefix+len-1)
 * attend to cache rows 0 .. prefix+len-1 with a causal mask: query row t sees
 * key rows j <= t.  For query head h the KV head is h / (n_q_heads /
 * n_kv_heads) (contiguous GQA groups).  With s_j = scale * q_t . k_j:
 *   out[i, h, :] = sum_j softmax(s)_j * v[j, kv(h), :]       (bf16, RNE)
 *   lse[h, i]    = ln sum_j exp(s_j)                          (fp32)
 * Softmax statistics and accumulation are fp32; the probabilities are
 * rounded to bf16 for the P.V product.
 *
 *   q         bf16 [len, n_q_heads, head_dim]
 *   k_cache   bf16 [>= prefix+len, n_kv_heads, head_dim]; rows >= prefix+len
 *   v_cache   are never read (their contents may be anything, NaN included)
 *   out       bf16 [len, n_q_heads, head_dim]
 *   lse       fp32 [n_q_heads, len]
 *   workspace, workspace_bytes: optional caller-owned device scratch
 *             (16-byte aligned).  With at least
 *             mocap_chunk_attn_workspace_size(...) bytes the key range may
 *             be split (same results up to fp32 rounding order); with less,
 *             or NULL, the single-pass kernel runs.  Contents on entry are
 *             ignored; it must not be used by overlapping work.
 *
 * Requirements: head_dim in {64, 128} (else MOCAP_EUNSUPPORTED); n_q_heads a
 * multiple of n_kv_heads; scale > 0 and finite; prefix >= 0; len >= 0
 * (0 = no-op); prefix + len < 2^31; 16-byte aligned pointers.
 * Device-side bounded waits that expire are reported by
 * mocap_last_device_status(); the kernel never traps.
 * With head_dim 128 and a multiple of four query heads per KV head the
 * kernel runs on pairs of CTAs (thread-block clusters of two, tcgen05
 * cta_group::2; results equal to the single-CTA kernel up to fp32 rounding
 * order).  Environment: MOCAP_ATTN_PAIR=0 selects the single-CTA kernel for
 * every shape; it is read on every call.
 */
mocap_status mocap_chunk_attn(const void *q, const void *k_cache, const void *v_cache,
                              int64_t prefix, int64_t len,
                              int32_t n_q_heads, int32_t n_kv_heads, int32_t head_dim,
                              float scale, void *out, float *lse,
                              void *workspace, size_t workspace_bytes,
                              mocap_stream_t stream);

/*
 * mocap_chunk_attn_workspace_size -- bytes of caller-owned device scratch that
 * let mocap_chunk_attn split the chunk's key range (split-KV) for this shape.
 *
 * Late chunks of a long prompt have few 128-row query blocks but long
 * prefixes, so their CTAs are few and long and the last wave leaves SMs idle
 * (wave quantisation).  With enough workspace the kernel splits each query
 * block's key tiles into 2..4 contiguous ranges, writes per-range fp32
 * partials (O / l and the range's LSE) to the workspace, and a second kernel
 * merges them: O = sum_k exp(LSE_k - LSE) O_k, LSE = ln sum_k exp(LSE_k).
 * The split count is chosen on the host by a list-scheduling estimate over
 * the device's SM count; 0 means no split helps (or invalid arguments).
 * Environment: MOCAP_SPLIT_KV=0 disables splitting, MOCAP_SPLIT_KV=1..4
 * forces that split count (capped so the first 128-row block keeps at least
 * one key tile per split); it is read on every call.
 * Layout: o_part [splits, len, Hq, d] fp32, then (256-byte aligned)
 * lse_part [splits, Hq, len] fp32.
 */
size_t mocap_chunk_attn_workspace_size(int64_t prefix, int64_t len, int32_t n_q_heads,
                                       int32_t n_kv_heads, int32_t head_dim);

/*
 * mocap_chunk_attn_noalloc -- mocap_chunk_attn for callers that cannot
 * allocate device memory.  The paper has no counterpart: this entry point
 * exists only for how some applications manage memory.
 *
 * Who needs it: a host program that owns all device memory through its own
 * pool and does not let libraries call cudaMalloc behind its back (the pool
 * may already hold nearly all of the GPU, or it must account for every
 * byte), and serving loops where the latency and stalls of cudaMalloc /
 * cudaFree are not acceptable.  Such callers cannot provide the split-KV
 * workspace of mocap_chunk_attn.  This entry point takes the same arguments
 * without the workspace and keeps the split-KV partials in a fixed
 * MOCAP_NOALLOC_SCRATCH_BYTES (32 MiB) array compiled into the library: it
 * calls no cudaMalloc, cudaFree or other allocating routine.
 *
 *   - Results: bitwise those of mocap_chunk_attn given a workspace of
 *     MOCAP_NOALLOC_SCRATCH_BYTES bytes (same split plan, same kernels).
 *   - Limit: when the split the library would use for this shape needs more
 *     than MOCAP_NOALLOC_SCRATCH_BYTES (see mocap_chunk_attn_workspace_size;
 *     e.g. 2 splits of a 2048-row chunk with 64 query heads need 135 MB), the
 *     call runs the single-pass kernel instead, as mocap_chunk_attn does with
 *     too small a workspace: the same results up to fp32 rounding order, but
 *     a late chunk's last wave may leave SMs idle.  Shapes that need no split
 *     run the single-pass kernel too and use no scratch.
 *   - Every CUDA context that loads the library holds its own copy of the
 *     array until the context ends.  The first call in a context looks up
 *     the array's device address (cudaGetSymbolAddress, once per context);
 *     make that first call before any stream capture.
 *   - All calls in a context share the array.  A call writes every scratch
 *     byte it reads, so nothing has to start at zero, but calls whose work
 *     overlaps on the GPU (e.g. on different streams) race on the array.
 */
#define MOCAP_NOALLOC_SCRATCH_BYTES (32u * 1024u * 1024u)
mocap_status mocap_chunk_attn_noalloc(const void *q, const void *k_cache, const void *v_cache,
                                      int64_t prefix, int64_t len,
                                      int32_t n_q_heads, int32_t n_kv_heads, int32_t head_dim,
                                      float scale, void *out, float *lse,
                                      mocap_stream_t stream);

/*
 * One (request, chunk) item of a varlen launch.  All offsets are in rows.
 *   q_row     first row of this chunk's queries in the packed q / out buffers
 *   kv_row    first cache row of the item's request (its key 0)
 *   prefix    keys of earlier chunks of the request (cache rows kv_row ..
 *             kv_row + prefix - 1)
 *   len       the chunk's length; its own keys are cache rows
 *             kv_row + prefix .. kv_row + prefix + len - 1
 */
typedef struct {
  int64_t q_row;
  int64_t kv_row;
  int64_t prefix;
  int64_t len;
} mocap_varlen_item;

#define MOCAP_VARLEN_MAX_ITEMS 64

/*
 * mocap_chunk_attn_varlen -- mocap_chunk_attn over up to
 * MOCAP_VARLEN_MAX_ITEMS independent items in a single launch (e.g. chunk k
 * of every request of a prefill batch).  Semantics per item are exactly
 * mocap_chunk_attn with q = q + q_row rows, k/v_cache = cache + kv_row rows,
 * out = out + q_row rows, and lse row block [h, q_row .. q_row+len) of the
 * packed fp32 [n_q_heads, q_rows_total] array.
 *
 *   items        HOST array of n_items descriptors (read during the call only)
 *   q_rows_total rows of the packed q / out buffers and row stride of lse
 *   kv_rows_total rows of the packed caches (bounds check only)
 *   workspace, workspace_bytes: optional caller-owned device scratch
 *                (16-byte aligned).  Used only when exactly one item has
 *                rows: with at least mocap_chunk_attn_workspace_size(prefix,
 *                len, ...) bytes for that item, its key range may be split
 *                as in mocap_chunk_attn (a late chunk of one long request
 *                fills the GPU's SMs instead of leaving a second, almost
 *                empty wave).  Several items never split.
 * Items must not write overlapping output rows.  Same requirements and
 * errors as mocap_chunk_attn; n_items == 0 is a no-op.
 */
mocap_status mocap_chunk_attn_varlen(const void *q, const void *k_cache, const void *v_cache,
                                     const mocap_varlen_item *items, int32_t n_items,
                                     int64_t q_rows_total, int64_t kv_rows_total,
                                     int32_t n_q_heads, int32_t n_kv_heads, int32_t head_dim,
                                     float scale, void *out, float *lse,
                                     void *workspace, size_t workspace_bytes,
                                     mocap_stream_t stream);

#define MOCAP_VARLEN_DEV_MAX_ITEMS 65536

/*
 * mocap_chunk_attn_varlen_dev_workspace_size -- bytes of device scratch that
 * mocap_chunk_attn_varlen_dev needs for n_items items whose lengths add up
 * to at most max_rows: per item its three TMA tensor maps (384 B) and
 * descriptor, one 4-byte entry per CTA of the launch's grid, which has
 * (ceil(max_rows / 128) + n_items) x n_kv_heads x
 * ceil(n_q_heads / n_kv_heads / 2) CTAs, and the CTA count.  0 when
 * n_items == 0 or an argument is out of range (max_rows outside
 * [0, 2^31 - 1], n_items above MOCAP_VARLEN_DEV_MAX_ITEMS, a bad shape).
 */
size_t mocap_chunk_attn_varlen_dev_workspace_size(int32_t n_items, int64_t max_rows,
                                                  int32_t n_q_heads, int32_t n_kv_heads,
                                                  int32_t head_dim);

/*
 * mocap_chunk_attn_varlen_dev -- mocap_chunk_attn_varlen with the item array
 * in DEVICE memory (Sec. 2.2: chunk k of every request of a batch in one
 * launch), so a device-side scheduler, or a CUDA graph replayed with new
 * item values, supplies the (request, chunk) items without a host round
 * trip.  Up to MOCAP_VARLEN_DEV_MAX_ITEMS items.
 *
 *   items        DEVICE array of n_items mocap_varlen_item (8-byte aligned),
 *                read by the launch; the caller keeps it unchanged until the
 *                work queued on `stream` has started past it
 *   max_rows     an upper bound on the sum of the items' len (a step's token
 *                budget; q_rows_total always serves).  It sizes the launch
 *                grid and the workspace: a tight bound spares the launch
 *                CTAs that find no work and exit.
 *   workspace, workspace_bytes: caller-owned device scratch, 128-byte
 *                aligned, at least mocap_chunk_attn_varlen_dev_workspace_size
 *                (n_items, max_rows, ...) bytes; overwritten by the call
 *   other arguments as mocap_chunk_attn_varlen.
 *
 * Two launches on `stream`: a one-block kernel validates the items, counts
 * and scans their CTAs, builds each item's tensor maps (tensormap.replace
 * of the global address and row extent of templates the host encodes over
 * the whole buffers) and fills the CTA -> item table; then the attention
 * kernel, on the grid above, whose CTAs past the items' count exit at once.
 * Per item the results are bitwise those of
 * mocap_chunk_attn_varlen with two or more items (this form never splits a
 * key range).  CTAs follow the items in the order given: put the items with
 * the most keys first (the host-array form sorts them so itself).
 *
 * Errors: the host-side checks of mocap_chunk_attn_varlen on the shape,
 * pointers and totals, n_items outside [0, MOCAP_VARLEN_DEV_MAX_ITEMS], a
 * null or misaligned items array, a missing, misaligned or short workspace
 * -> MOCAP_EINVAL.  An item that fails mocap_chunk_attn_varlen's item checks
 * (negative field, rows outside q_rows_total / kv_rows_total,
 * prefix + len >= 2^31), or items that need more CTAs than the grid has
 * (their lengths exceed max_rows), are found on the device: the call then
 * writes nothing and records
 * MOCAP_EINVAL in the status word that mocap_last_device_status returns (and
 * clears); until then later launches do nothing, as after an expired wait.
 * Items must not write overlapping output rows.  n_items == 0 is a no-op.
 */
mocap_status mocap_chunk_attn_varlen_dev(const void *q, const void *k_cache, const void *v_cache,
                                         const mocap_varlen_item *items, int32_t n_items,
                                         int64_t q_rows_total, int64_t kv_rows_total,
                                         int64_t max_rows,
                                         int32_t n_q_heads, int32_t n_kv_heads, int32_t head_dim,
                                         float scale, void *out, float *lse, void *workspace,
                                         size_t workspace_bytes, mocap_stream_t stream);

/*
 * One KV append that an attention launch carries out (see
 * mocap_chunk_attn_append): rows [0, rows) of k_src / v_src (bf16
 * [rows, n_kv_heads, head_dim], 16-byte aligned, device) are written to cache
 * rows [dst_row, dst_row + rows), as mocap_kv_append would.
 */
typedef struct {
  const void *k_src;
  const void *v_src;
  int64_t dst_row;
  int64_t rows;
} mocap_kv_append_item;

#define MOCAP_FUSED_APPEND_MAX 64

/*
 * mocap_chunk_attn_append -- mocap_chunk_attn plus KV appends done in the same
 * launch: the chunked prefill walks its chunks in order (Sec. 2.2), and
 * chunk i + 1's K/V rows, which chunk i's attention never reads, are written
 * to the cache by warps of chunk i's attention kernel that would otherwise
 * idle.  The copy's HBM traffic overlaps tensor-bound work, and a prompt of
 * M chunks needs M attention launches plus one append (chunk 0's) instead of
 * M of each.
 *
 * Attention arguments and results as mocap_chunk_attn (split-KV workspace
 * included).  Then:
 *   appends        HOST array of n_appends descriptors (read during the call)
 *   n_appends      0 .. MOCAP_FUSED_APPEND_MAX
 *   cache_capacity rows of k_cache / v_cache (>= prefix + len)
 * Each append must lie inside the cache and write only rows outside
 * [0, prefix + len) (the rows this call reads) and outside the other
 * appends' rows; sources must not overlap the cache rows written.  Else
 * MOCAP_EINVAL, with nothing enqueued.  The appended rows are complete, like
 * the outputs, when work queued after the call on `stream` starts.  With
 * len == 0 the appends run as plain append launches.  After an expired
 * bounded wait (see mocap_last_device_status) the call does nothing, appends
 * included.
 */
mocap_status mocap_chunk_attn_append(const void *q, const void *k_cache, const void *v_cache,
                                     int64_t prefix, int64_t len,
                                     int32_t n_q_heads, int32_t n_kv_heads, int32_t head_dim,
                                     float scale, void *out, float *lse,
                                     void *workspace, size_t workspace_bytes,
                                     const mocap_kv_append_item *appends, int32_t n_appends,
                                     int64_t cache_capacity, mocap_stream_t stream);

/*
 * mocap_chunk_attn_varlen_append -- mocap_chunk_attn_varlen plus KV appends
 * done in the same launch (e.g. chunk k + 1 of every request while chunk k
 * of every request attends).  Appends as in mocap_chunk_attn_append, with
 * destination rows in the packed caches (kv_rows_total rows): each must
 * avoid every item's rows [kv_row, kv_row + prefix + len).
 */
mocap_status mocap_chunk_attn_varlen_append(const void *q, const void *k_cache,
                                            const void *v_cache,
                                            const mocap_varlen_item *items, int32_t n_items,
                                            int64_t q_rows_total, int64_t kv_rows_total,
                                            int32_t n_q_heads, int32_t n_kv_heads,
                                            int32_t head_dim, float scale, void *out, float *lse,
                                            void *workspace, size_t workspace_bytes,
                                            const mocap_kv_append_item *appends,
                                            int32_t n_appends, mocap_stream_t stream);

/*
 * mocap_last_row_attn -- attention of each request's last prompt row only.
 *
 * Sec. 2.1: a prefill-only request emits a single token, so its final layer
 * needs the attention output of the last row alone: for request r and query
 * head h, the row at position kv_len[r] - 1 attends to every key of the
 * request (keys 0 .. kv_len[r] - 1), with the same definition as
 * mocap_chunk_attn.  This is memory-bound (each K/V byte serves only the
 * n_q_heads / n_kv_heads heads of its group), so a dedicated kernel streams
 * K/V tiles through TMA, lets the tensor core form the small products in
 * transposed form (keys, then dimensions, on the 128 TMEM lanes), and splits
 * the requests' keys into ranges (about three CTAs per SM in total) whose
 * fp32 partials are merged like split-KV, in the same launch: the last CTA
 * of each (request, KV group) to finish merges the group's partials.
 *
 *   q_last    bf16 [n_req, Hq, d]: the last row's queries of each request
 *   k_cache,  bf16 [kv_rows_total, Hkv, d]: request r's keys are rows
 *   v_cache   kv_row[r] .. kv_row[r] + kv_len[r] - 1 (rows past them unread)
 *   kv_row, kv_len  HOST arrays of n_req int64 (kv_len[r] >= 1)
 *   out       bf16 [n_req, Hq, d];  lse fp32 [Hq, n_req]
 *   workspace at least mocap_last_row_attn_workspace_size(...) bytes, 16-byte
 *             aligned: fp32 partials plus n_req * Hkv arrival counters, which
 *             the call zeroes with a memset on `stream` before its launch.
 *             Calls that may run concurrently need separate workspaces.
 * Enqueues one memset and one kernel.
 * 1 <= n_req <= 64; Hq / Hkv <= 16; head_dim in {64, 128}.
 */
size_t mocap_last_row_attn_workspace_size(const int64_t *kv_len, int32_t n_req,
                                          int32_t n_q_heads, int32_t n_kv_heads,
                                          int32_t head_dim);
mocap_status mocap_last_row_attn(const void *q_last, const void *k_cache, const void *v_cache,
                                 const int64_t *kv_row, const int64_t *kv_len, int32_t n_req,
                                 int64_t kv_rows_total, int32_t n_q_heads, int32_t n_kv_heads,
                                 int32_t head_dim, float scale, void *out, float *lse,
                                 void *workspace, size_t workspace_bytes, mocap_stream_t stream);

/*
 * mocap_last_device_status -- synchronises `stream`, then reads and clears
 * the device status word that the kernels set when a bounded wait expires
 * (MOCAP_ETIMEOUT) instead of hanging, or when mocap_chunk_attn_varlen_dev
 * finds an invalid device item (MOCAP_EINVAL); the first recorded value
 * stays.  MOCAP_OK when nothing was recorded; MOCAP_ECUDA if the
 * synchronisation itself failed.
 */
mocap_status mocap_last_device_status(mocap_stream_t stream);

/*
 * mocap_selftest_bounded_wait -- exercises the kernels' failure path without
 * a fault.  Every wait in this library's kernels is bounded: past its limit
 * it records MOCAP_ETIMEOUT in the device status word and the kernel unwinds
 * (no trap, no hang).  This launches a one-thread kernel that waits, with
 * the same bounded wait, on a barrier nothing ever completes, for limit_us
 * microseconds (1 .. 1000000, else MOCAP_EINVAL).  Afterwards
 * mocap_last_device_status() reports MOCAP_ETIMEOUT, and until it is read
 * every attention launch (split-KV combine included) returns without doing
 * work, leaving its outputs as they were.  No counterpart in the
 * paper: failure detection for shared GPUs.
 */
mocap_status mocap_selftest_bounded_wait(uint32_t limit_us, mocap_stream_t stream);

/* Static, NUL-terminated name of a status code. */
const char *mocap_status_string(mocap_status status);

#ifdef __cplusplus
}
#endif

#endif /* MOCAP_H_ */
