/*
 * refadapt.h — C ABI of the RefAdapt-DiT hot path on one GB300 (sm_103a).
 *
 * RefAdapt-DiT (training-free reference reuse for reference-conditioned
 * diffusion transformers): every DiT block runs joint attention over
 * [text; reference; target] tokens. A block that reuses skips the reference
 * query rows and lets text and target queries attend to reference K/V cached
 * at the block's last materialisation; the first block whose head-mean score
 * D x M reaches theta reactivates and every deeper block recomputes
 * (paper Sec. 4, Algorithm 1).
 *
 * Conventions for every entry point:
 *  - All device pointers are caller-owned; the library allocates no device
 *    memory. Every call is asynchronous on `stream` (a cudaStream_t passed as
 *    void*; NULL = the legacy default stream) and performs no host sync.
 *  - Invalid arguments return RA_EINVAL before anything is launched;
 *    refadapt_last_error() then holds a one-line reason (thread-local).
 *  - A failed launch returns RA_ECUDA. A device-side wait that exceeded its
 *    time budget sets bit 0 of the caller's error word (see
 *    refadapt_check_error), never traps, and leaves the context usable.
 *  - No exceptions cross the ABI; nothing calls exit().
 *  - Calls may come from several host threads and target several GPUs: each
 *    works on the device current in the calling thread, and the library's
 *    one-time set-up (kernel shared-memory limits, SM counts, cluster
 *    occupancy) is kept per device under a mutex, the no-allocation scratch
 *    address per device and CUDA context. Work on one device follows the
 *    stream order the caller gives.
 *  - bf16 tensors are described by ra_seg: element (b, h, n, c) lives at
 *    ptr + b*stride_b + h*stride_h + n*stride_n + c (strides in elements,
 *    c contiguous). ptr and every stride must be 16-byte aligned
 *    (strides multiples of 8 elements).
 */
#ifndef REFADAPT_H
#define REFADAPT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  RA_OK = 0,
  RA_EINVAL = 1,        /* bad argument; nothing launched */
  RA_EUNSUPPORTED = 2,  /* valid but not supported here (e.g. no sm_103 device) */
  RA_ECUDA = 3,         /* a CUDA call failed */
  RA_ETIMEOUT = 4       /* a device-side wait ran out of its budget */
} ra_status;

/* Block execution modes (paper Sec. 4 "Execution and cache state";
 * Algorithm 1). REUSE: reference query rows skipped, text and target rows
 * attend to cached reference K/V. BOUNDARY: the first crossing block; every
 * row runs, reference K/V still from the cache, the cache is not updated.
 * COMPUTE: a block deeper than the boundary; fresh reference K/V are written
 * to the cache (a_b = t) and every row runs. FULL: bounded-age or step-0 full
 * refresh; same work as COMPUTE. */
typedef enum {
  RA_MODE_REUSE = 0,
  RA_MODE_BOUNDARY = 1,
  RA_MODE_COMPUTE = 2,
  RA_MODE_FULL = 3
} ra_mode;

/* Token roles (paper Sec. 3 "Setting"): R = reference rows, Y = the
 * remaining active-generation rows, split here into text and target. */
enum { RA_TEXT = 0, RA_REF = 1, RA_TGT = 2 };

/* Rows of one Q tile of the attention kernel; mass partials come per tile. */
#define RA_MASS_TILE_ROWS 128

typedef struct {
  void* ptr;          /* device, bf16 */
  int64_t stride_b;   /* elements */
  int64_t stride_h;   /* elements */
  int64_t stride_n;   /* elements */
  int32_t n;          /* rows (tokens) in this segment, >= 0 */
  int32_t reserved;   /* set to 0 */
} ra_seg;

/* ------------------------------------------------------------------ attention
 * refadapt_joint_attn — joint attention of one DiT block with the reference
 * mass as a by-product.
 *
 * Computes, per sample b and head h, O = Softmax(scale * Q K^T + bias) V
 * (paper Sec. 3.3, Attn(Q,K,V) = Softmax(QK^T / sqrt(d_h)) V) over the keys
 * [text; ref; target], bidirectional, no mask. Query rows: text and target
 * when mode[b] == RA_MODE_REUSE (reference rows skipped, their O rows left
 * untouched; App. A.4 removes the two reference-query score regions), every
 * row otherwise. The reference K/V segments are whatever the caller points
 * k[RA_REF] / v[RA_REF] at — normally the block's cache slot, so reuse costs
 * no copy.
 *
 * Mass (paper Eq. 4): for every executed query row q in the mass row set,
 * the softmax probability summed over reference keys, l_ref(q) / l(q), is
 * accumulated per 128-row Q tile into mass_partial[b][h][i] (fp32), i over
 * the text tiles (ceil(n_text/128)) then the target tiles
 * (ceil(n_tgt/128)), n counting query rows; refadapt_mass_partial_len()
 * gives the length. Mass row
 * set: target rows (mass_rows = 0), or text + target rows (mass_rows = 1);
 * partials of tiles outside the set are written as 0. M_{t,b,h} is the sum of
 * a (b, h) row of partials divided by the number of mass rows (the gate does
 * this). Every partial is written on every call, in a fixed reduction order
 * (deterministic).
 *
 * Arguments:
 *  q, k, v, o [3]   segments per role (RA_TEXT, RA_REF, RA_TGT). Per role q
 *                   and o share n (query rows) and k and v share n (key
 *                   rows); query and key rows of a role may differ (e.g. a
 *                   row sample of the queries). The target segment needs at
 *                   least one key row. q[RA_REF] / o[RA_REF] with ptr NULL:
 *                   the reference query rows are not computed, whatever the
 *                   mode.
 *  B, H, d          batch, heads, head dim; d in {64, 128}.
 *  softmax_scale    > 0; pass 0 for 1/sqrt(d).
 *  ref_logit_bias   device [H] fp32 or NULL: added to the logits of target
 *                   query rows against reference keys (natural-log units).
 *  mode             device [B] int32 (ra_mode) or NULL (= every row runs).
 *  mass_partial     device [B][H][refadapt_mass_partial_len(n_text, n_tgt)].
 *  mass_row_stride  the "sampled target-query rows" of Eq. 4 / Algorithm 1:
 *                   0 or 1 counts every mass row; k > 1 counts rows 0, k,
 *                   2k, ... of the target segment (and of the text segment
 *                   when mass_rows = 1); the partials then sum the sampled
 *                   rows only (divide by their count). O is unaffected.
 *  err_word         device int32 or NULL; bit 0 set on a device timeout.
 *
 * Fused reference-cache update (paper Eq. 11; Algorithm 1's compute and full
 * branches), optional: off when ref_fresh_q/k/v.ptr and a_b are all NULL
 * (the zero-initialised struct). Otherwise, for
 * every sample whose mode is RA_MODE_COMPUTE or RA_MODE_FULL, the reference
 * K/V (and the reference query) are read from ref_fresh_k / ref_fresh_v /
 * ref_fresh_q (this step's reference projections) instead of k/v/q[RA_REF],
 * and copied into k/v/q[RA_REF] (the block's cache slot) as a by-product:
 * the first CTA of each (sample, head) bulk-stores every reference K/V tile
 * it streams through shared memory for its MMAs, each reference-row CTA its
 * own query tiles, and a_b[b] = step. Samples in REUSE or BOUNDARY read the
 * cache slot as before and leave it untouched. This replaces a separate
 * refadapt_ref_cache_update (and its reads of the fresh tensors) on the
 * attention's own pass over them.
 *  ref_fresh_k/v    segments with n = k[RA_REF].n (16-byte aligned as above;
 *                   ptr NULL only when n = 0).
 *  ref_fresh_q      n = q[RA_REF].n when q[RA_REF] is given; ptr NULL and
 *                   n = 0 otherwise.
 *  a_b              device [B] int32 or NULL: materialisation step per sample.
 *  step             the step index written into a_b.
 * A fresh segment whose ptr equals its cache segment's (same strides) is read
 * in place and not copied; K and V are both in place or both copied. The
 * cache segments must not overlap the fresh ones otherwise. Errors
 * (RA_EINVAL, nothing queued): n or stride mismatches as above.
 */
typedef struct {
  int32_t B, H, d;
  int32_t mass_rows;
  ra_seg q[3], k[3], v[3], o[3];
  float softmax_scale;
  int32_t mass_row_stride;  /* 0 or 1: every mass row; k > 1: rows 0, k, 2k, ... of each mass segment */
  const float* ref_logit_bias;
  const int32_t* mode;
  float* mass_partial;
  int32_t* err_word;
  ra_seg ref_fresh_q, ref_fresh_k, ref_fresh_v;  /* fused cache update; off when these ptrs and a_b are NULL */
  int32_t* a_b;
  int32_t step;
  int32_t reserved;  /* set to 0 */
} ra_attn_args;

ra_status refadapt_joint_attn(const ra_attn_args* args, void* stream);

int32_t refadapt_mass_partial_len(int32_t n_text, int32_t n_tgt);

/* ------------------------------------------------------------------ Q change
 * refadapt_q_delta — consecutive relative drift of the post-RoPE target
 * query, per sample and head (paper Eq. 1 applied to Q^{Y,h}, Sec. 4
 * "Runtime cues"):
 *   D[b][h] = ||q_cur - q_prev||_F / (||q_prev||_F + eps)
 * over the segment's n rows x d columns. Bandwidth-bound: reads both tensors
 * once through bulk copies into shared memory; fp32 per-thread sums and
 * butterflies, then compensated two-float sums across units, warps and
 * blocks, all in a fixed order (deterministic; relative error of D ~1e-7).
 *
 * Each slab (one sample and head) is reduced by one thread-block cluster of
 * up to 8 CTAs through distributed shared memory, leaving the workspace
 * untouched, when a slab has at most 8 x 384 units of 8 KB per tensor
 * (n <= 98304 rows at d = 128, 196608 at d = 64), all B * H clusters fit on
 * the GPU at once, and they fill at least 60 % of the SMs (or of the units,
 * for tiny inputs). Otherwise a
 * multi-block path spreads the units over all SMs; its ticket counters and
 * partial sums live in the workspace.
 *
 *  q_cur, q_prev    segments with equal n (>= 1); d in {64, 128}.
 *  d_out            device [B][H] fp32.
 *  workspace        device scratch of refadapt_q_delta_workspace_size(B, H)
 *                   bytes, 16-byte aligned, zero-filled once before its first
 *                   use; every call leaves it ready for the next. Calls that
 *                   share a workspace must be stream-ordered. Required (not
 *                   NULL) whatever the slab length.
 */
size_t refadapt_q_delta_workspace_size(int32_t B, int32_t H);
ra_status refadapt_q_delta(const ra_seg* q_cur, const ra_seg* q_prev, int32_t B, int32_t H, int32_t d,
                           float eps, float* d_out, void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------ Q change, no allocation
 * refadapt_q_delta_noalloc — the same D as refadapt_q_delta, for callers that
 * cannot allocate device memory and have no workspace to hand over: for
 * example a plugin inside a host framework that owns the whole device memory
 * pool and forbids direct cudaMalloc, or a latency-critical loop that must not
 * pay cudaMalloc's implicit device synchronisation. The paper has no
 * counterpart; this is an interface convenience only.
 *
 * The scratch that the long-slab path needs (ticket counters and per-block
 * partial sums; slabs that fit one cluster use none) lives in a
 * file-scope static device array inside the library, sized for at most
 * RA_Q_DELTA_NOALLOC_MAX_BH (= B * H) slabs, about 193 KB; every GPU that loads
 * the library holds it until the process exits. Larger B * H returns RA_EINVAL
 * (use refadapt_q_delta with a workspace). The call allocates nothing: no
 * cudaMalloc, no cudaFree, no allocating library routine. Its first call on a
 * device looks the array's device address up (cudaGetSymbolAddress with that
 * device current) and caches it for the CUDA context current at that moment;
 * a later call in another context (for instance after cudaDeviceReset tore
 * the primary context down) looks it up again. Make the first call, and the
 * first call after a reset, before any stream capture. A call that takes the
 * multi-block path clears that path's ticket counters on `stream` right
 * before its kernel, after every argument check; a call that returns
 * RA_EINVAL queues nothing. All calls share the one array, so calls that
 * overlap on the GPU (different streams, or different host threads without
 * ordering) race and must not be issued. Arguments and results are those of
 * refadapt_q_delta.
 */
#define RA_Q_DELTA_NOALLOC_MAX_BH 96
ra_status refadapt_q_delta_noalloc(const ra_seg* q_cur, const ra_seg* q_prev, int32_t B, int32_t H, int32_t d,
                                   float eps, float* d_out, void* stream);

/* ------------------------------------------------------------------ gate
 * Controller state of Algorithm 1 for one trajectory (opaque, device
 * resident): a_full (step of the last full refresh), whether the current
 * step is a full refresh, and per sample the reactivated latch and boundary.
 */
typedef struct ra_state ra_state;
size_t refadapt_state_size(int32_t B);
ra_status refadapt_state_init(ra_state* state, int32_t B, void* stream);

/* refadapt_gate — one block's decision (paper Eqs. 12-13, App. A.2 head
 * mean, bounded-age refresh of Sec. 4 / Algorithm 1), on the device.
 *
 * Must be called for blocks 0, 1, ... in order within a step. At b == 0 it
 * opens step t: t == 0 forces FULL (and a_full = 0); else t - a_full >=
 * delta_max forces FULL for every block of the step (and a_full = t); else
 * the reactivated latch is cleared. Per sample: g_h = D[b][h] * M_{t-1,b,h}
 * (M from the previous step's mass partials of this block), gbar = mean_h
 * g_h; FULL if the step is a full refresh, COMPUTE if already reactivated,
 * else BOUNDARY (and latch) if gbar >= theta — or b >= forced_boundary when
 * forced_boundary >= 0 — else REUSE.
 *
 * cue selects the per-head trigger of the controller ablation (paper Sec. 5.3,
 * Tab. 4; App. A.2), everything else unchanged: RA_CUE_PRODUCT g_h = D_h M_h
 * (the method), RA_CUE_CHANGE g_h = D_h (target-Q change only),
 * RA_CUE_EXPOSURE g_h = M_h (exposure only). The anchor-relative variant is
 * RA_CUE_PRODUCT fed with the change to the block's last materialisation
 * (c^anchor of App. A.2) in q_delta; the fixed-interval baseline is
 * theta = +inf with delta_max = the interval.
 *
 *  q_delta            device [B][H] (refadapt_q_delta for this step/block);
 *                     may be NULL at t == 0.
 *  mass_partial_prev  device [B][H][mass_partial_len] from step t-1, block b;
 *                     may be NULL at t == 0.
 *  mass_row_count     number of rows the partials cover (n_tgt, or
 *                     n_text + n_tgt when mass_rows = 1).
 *  mode_out           device [B] int32, read by refadapt_joint_attn and
 *                     refadapt_ref_cache_update.
 *  gbar_out, m_out    device [B] and [B][H] fp32 or NULL (logging; gbar is
 *                     NaN at t == 0).
 */
typedef struct {
  double theta;
  int32_t t, b, B, H;
  int32_t delta_max;
  int32_t forced_boundary;
  int32_t mass_partial_len;
  int32_t mass_row_count;
  int32_t cue;         /* ra_cue */
  int32_t reserved;    /* set to 0 */
  const float* q_delta;
  const float* mass_partial_prev;
  ra_state* state;
  int32_t* mode_out;
  float* gbar_out;
  float* m_out;
} ra_gate_args;

typedef enum { RA_CUE_PRODUCT = 0, RA_CUE_CHANGE = 1, RA_CUE_EXPOSURE = 2 } ra_cue;

ra_status refadapt_gate(const ra_gate_args* args, void* stream);

/* refadapt_q_delta_gate — refadapt_q_delta, then refadapt_gate on the D it
 * produced (paper Eq. 1, then Eqs. 12-13 / App. A.2 / Algorithm 1), with the
 * results of the two calls, bit for bit. When the Q change takes its cluster
 * path this is one launch: each cluster's leader writes its slab's D and takes
 * a ticket from the workspace; the leader that takes the last one runs the
 * decision on all B x H values in its CTA. No CTA waits for another. On the
 * multi-block path the gate is a second launch behind the Q change.
 *
 *  q_cur ... workspace_bytes   as for refadapt_q_delta (the workspace also
 *                              holds the ticket; same size function).
 *  gate                        as for refadapt_gate with gate->B == B,
 *                              gate->H == H, gate->t >= 1 (step 0 has no Q
 *                              change: call refadapt_gate), and gate->q_delta
 *                              NULL or equal to d_out.
 * Errors: RA_EINVAL for either call's argument errors, nothing queued.
 */
ra_status refadapt_q_delta_gate(const ra_seg* q_cur, const ra_seg* q_prev, int32_t B, int32_t H, int32_t d,
                                float eps, float* d_out, void* workspace, size_t workspace_bytes,
                                const ra_gate_args* gate, void* stream);

/* ------------------------------------------------------------------ cache
 * refadapt_ref_cache_update — materialise a block's reference K/V into its
 * cache slot (paper Eq. 11, Z_b = (H_b, K_b, V_b, a_b); Algorithm 1: a
 * COMPUTE or FULL block updates K_b, V_b and sets a_b = t).
 *
 * For each sample b with mode[b] in {COMPUTE, FULL}: copies k_src -> k_cache,
 * v_src -> v_cache and, when x_src is not NULL, x_src -> x_cache (the
 * block's cached reference hidden state, any bf16 [B, x_heads, n, x_width]
 * tensor), then sets a_b[b] = t. Samples in other modes are untouched. A copy
 * whose source and destination pointers are equal is skipped (in-place
 * producer). 16-byte vector copies.
 *
 *  k_*, v_*      segments [B, H, n_ref, d]; all n equal; d in {64, 128}.
 *  x_src/x_cache optional segments [B, x_heads, n_ref, x_width];
 *                x_width a multiple of 8.
 *  mode          device [B] int32.
 *  a_b           device [B] int32 or NULL.
 */
ra_status refadapt_ref_cache_update(const ra_seg* k_src, const ra_seg* v_src, const ra_seg* k_cache,
                                    const ra_seg* v_cache, int32_t B, int32_t H, int32_t d,
                                    const ra_seg* x_src, const ra_seg* x_cache, int32_t x_heads,
                                    int32_t x_width, const int32_t* mode, int32_t t, int32_t* a_b,
                                    void* stream);

/* ------------------------------------------------------------------ DiT block around the attention
 * The paper's models are DiTs whose blocks run joint attention over
 * [text; reference; target] rows (Sec. 3, "Setting"). Under reuse the
 * reference-side QKV projections and the other reference-stream operations
 * are skipped because the layer-wise reference K/V are cached (App. A.4);
 * at the boundary the cached reference hidden state is restored, its query
 * runs against the current target and the reference output becomes the next
 * block's cached hidden state (Algorithm 1, App. A.3). The paper does not
 * give the block's layers; these entry points build a dual-stream MMDiT
 * block (text rows with one weight set, reference and target rows with
 * another) from: a modulated LayerNorm (refadapt_ln_modulate), linear layers
 * with fused epilogues (refadapt_gemm) and the RoPE table the QKV epilogue
 * reads (refadapt_rope_table).
 *
 * Rows come in up to three segments (text, reference, target), each with its
 * own pointers and strides; row r of sample s of a segment lives at
 * ptr + s * stride_s + r * stride_r (elements, features contiguous). A
 * segment with gated = 1 is skipped for samples whose mode (device [B],
 * written by refadapt_gate) is RA_MODE_REUSE. All calls are asynchronous on
 * `stream` and allocate nothing; invalid arguments return RA_EINVAL before
 * anything is launched.
 */

/* refadapt_rope_table — table[pos][i] = (cos, sin)(pos * base^(-2i/d)),
 * fp32, pos in [0, n_pos), i in [0, d/2): [n_pos][d/2][2] floats, 16-byte
 * aligned (device, caller-owned). Angles in fp64. d a multiple of 4. */
ra_status refadapt_rope_table(float* table, int32_t n_pos, int32_t d, double base, void* stream);

/* refadapt_ln_modulate — x = LN(h) * (1 + scale[s]) + shift[s] per row:
 * LN without affine over C features, fp32 mean and variance, eps added to
 * the variance; shift and scale are the block's AdaLN vectors for the row's
 * stream and sample, fp32 [B][C] (row stride mod_stride_s). bf16 in and out;
 * h and x must not overlap. C a multiple of 256, at most 4096; pointers
 * 16-byte aligned, row strides >= C and multiples of 8 elements. */
typedef struct {
  const void* h;
  int64_t h_stride_s, h_stride_r;
  void* x;
  int64_t x_stride_s, x_stride_r;
  const float* shift;
  const float* scale;
  int64_t mod_stride_s;
  int32_t rows;       /* rows per sample, >= 0 */
  int32_t gated;
} ra_lnmod_seg;

typedef struct {
  int32_t B, C, n_seg, reserved;
  float eps, reserved2;
  ra_lnmod_seg seg[3];
  const int32_t* mode;  /* device [B]; required when a segment is gated */
} ra_lnmod_args;

ra_status refadapt_ln_modulate(const ra_lnmod_args* args, void* stream);

/* refadapt_gemm — out = epilogue(A W^T + bias) on tcgen05 tensor cores:
 * A bf16 rows of each segment (K features), W bf16 [N][K] (nn.Linear
 * layout, one weight matrix per segment, so text and image streams differ),
 * bias fp32 [N] or NULL, fp32 accumulation. N a multiple of 256, K of 64.
 * Epilogues (fp32 until one final rounding to bf16):
 *   RA_EPI_STORE  out = acc + bias
 *   RA_EPI_GELU   out = gelu_tanh(acc + bias)
 *   RA_EPI_RESID  out = resid + gate[s] * (acc + bias); gate fp32 [B][N]
 *                 (row stride gate_stride_s); resid may equal out
 *                 (in-place update of a residual stream) but must not
 *                 partially overlap it.
 *   RA_EPI_QKV    N = 3 H d, columns [q | k | v], head h at h*d within each
 *                 part: q and k of each head are RMS-normalised over d
 *                 (fp32, norm_eps added to the mean square) and scaled by
 *                 q_norm / k_norm [d], then rotated by RoPE on interleaved
 *                 pairs (2i, 2i+1) at position pos_offset + r, reading
 *                 rope[pos][i] (refadapt_rope_table, rope_len rows); v gets
 *                 the bias only. Written head-major to q_out, k_out, v_out
 *                 (ra_seg, n = rows): for a gated segment (the reference
 *                 rows) the K and V tiles are also skipped when the mode is
 *                 RA_MODE_BOUNDARY (the block keeps its cached K/V), so k_out
 *                 and v_out can point straight at the block's cache slot.
 * Pointers 16-byte aligned; row strides multiples of 8 elements; out rows
 * hold N columns (out_stride_r >= N); A rows K (a_stride_r >= K).
 * err_word: device int32 or NULL; bit 0 set if a device wait timed out.
 * tile_mode: 0 picks CTA pairs (a cluster of two SMs running one
 * cta_group::2 MMA on a 256 x 256 tile, each SM staging half of the operands)
 * when the call has at least a wave of such tiles, else one CTA per 128 x 256
 * tile; 1 and 2 force either (results are the same; tests use both).
 */
typedef enum { RA_EPI_STORE = 0, RA_EPI_GELU = 1, RA_EPI_RESID = 2, RA_EPI_QKV = 3 } ra_epilogue;

typedef struct {
  const void* a;
  int64_t a_stride_s, a_stride_r;
  int32_t rows;        /* rows per sample, >= 0 */
  int32_t gated;
  const void* w;       /* bf16 [N][K] */
  const float* bias;   /* [N] or NULL */
  void* out;           /* STORE / GELU / RESID */
  int64_t out_stride_s, out_stride_r;
  const void* resid;   /* RESID */
  int64_t resid_stride_s, resid_stride_r;
  const float* gate;   /* RESID: [B][N] */
  int64_t gate_stride_s;
  ra_seg q_out, k_out, v_out;          /* QKV: [B, H, rows, d] */
  const float* q_norm;                 /* QKV: [d] */
  const float* k_norm;                 /* QKV: [d] */
  int32_t pos_offset;                  /* QKV: RoPE position of row 0 */
  int32_t reserved;
} ra_gemm_seg;

typedef struct {
  int32_t B, N, K, epilogue;
  int32_t H, d, n_seg, rope_len;       /* H, d, rope_len: QKV only */
  ra_gemm_seg seg[3];
  const int32_t* mode;                 /* device [B]; required when a segment is gated */
  const float* rope;                   /* QKV: [rope_len][d/2][2] */
  float norm_eps;
  int32_t tile_mode;                   /* 0 auto, 1 one CTA per 128 x 256 tile, 2 CTA pairs on 256 x 256 */
  int32_t* err_word;
} ra_gemm_args;

ra_status refadapt_gemm(const ra_gemm_args* args, void* stream);

/* ------------------------------------------------------------------ misc */
const char* refadapt_status_string(ra_status s);
const char* refadapt_last_error(void);

/* Budget, in nanoseconds, of every device-side mbarrier wait of kernels
 * launched afterwards by this process (default 2e9). */
void refadapt_set_wait_budget_ns(uint64_t ns);

/* Synchronises `stream`, reads the device error word, clears it and returns
 * RA_ETIMEOUT if a device wait ran out, RA_ECUDA on a CUDA error, else RA_OK. */
ra_status refadapt_check_error(int32_t* err_word, void* stream);

int32_t refadapt_version(void);

/* Diagnostic for the timeout path: launches one thread that waits, with the
 * given budget, on an mbarrier that nothing ever arrives at — the same bounded
 * wait every kernel uses. The wait gives up, sets bit 0 of *err_word and the
 * kernel returns normally, so refadapt_check_error then reports RA_ETIMEOUT
 * with the context still usable. budget_ns is capped at 1e9. */
ra_status refadapt_selftest_wait_timeout(int32_t* err_word, uint64_t budget_ns, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* REFADAPT_H */
