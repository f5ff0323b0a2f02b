/*
 * evisel.h - C ABI of the GB300 (sm_103a) sparse-prefill evidence probe.
 *
 * The probe is the paper's evidence-grounding pass (Sec. 3.2, "Sparse Evidence
 * Probing", Eq. 1): block-sparse, causal, grouped-query prefill attention over
 * a packed batch of videos, each laid out as X = [X_vis; X_Q] (pooled visual
 * tokens, then the query's text tokens; Appendix "Detailed Sparse
 * Prefilling"), followed by the attention evidence read off the text rows
 * (Sec. 3.2, "Evidence Decomposition"): the softmax mass from the text rows
 * onto every visual token, reduced per token, per frame and per head, and the
 * query-frame cue A_qf.
 *
 * Conventions for every entry point:
 *   - Pointers marked "device" are CUDA device pointers owned by the caller;
 *     pointers marked "host" are ordinary host memory read during the call only.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     All device work is enqueued asynchronously on it; nothing blocks the host
 *     except evisel_status() and evisel_free().
 *   - Return value 0 = success, negative = an EVISEL_E* code below; on failure
 *     nothing has been enqueued and evisel_last_error() describes the cause
 *     (thread-local string).
 *   - Thread safety: calls are reentrant provided each thread uses its own
 *     workspace.
 */
#ifndef EVISEL_H
#define EVISEL_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define EVISEL_OK             0
#define EVISEL_EINVAL        -1  /* null pointer, bad count, misaligned pointer   */
#define EVISEL_EUNSUPPORTED  -2  /* head_dim, tile, hq % hkv or N_v outside the set */
#define EVISEL_EMASK         -3  /* unsorted / out-of-range / non-causal CSR, missing diagonal */
#define EVISEL_ECUDA         -4  /* a CUDA runtime/driver call failed             */
#define EVISEL_ENOMEM        -5  /* device or pinned allocation failed            */
#define EVISEL_ETIMEOUT      -6  /* device-side: a bounded wait gave up           */
#define EVISEL_EBOUNDS       -7  /* reserved for device-side index checks; every index is
                                     validated on the host before launch, and no kernel of
                                     this library records it */
#define EVISEL_ESTATE        -8  /* evidence requested before any probe on the workspace */

/* Opaque workspace owned by the library: work list, device copy of the mask,
 * split-KV partials and the text-row logit spill. Created by the first
 * evisel_probe_attention() call that receives *ws == NULL; reused (grown if
 * needed) by later calls; released only by evisel_free(). */
typedef struct evisel_ws evisel_ws;

/* Description of one probe call (one transformer layer).
 *
 * Token layout (Appendix, "Detailed Sparse Prefilling"): videos are packed back
 * to back; video b spans global tokens [cu_seqlens[b], cu_seqlens[b+1]), its
 * first n_vis[b] tokens are visual (n_vis[b] = T_b * tokens_per_frame), the rest
 * are its text tokens. Visual tokens are cut into tiles of `tile` tokens from the
 * visual start and text tokens independently from the text start; the last tile
 * of each may be short. tile must be a multiple of tokens_per_frame so that no
 * frame crosses a tile (Eq. 1: block boundaries align with frame boundaries).
 *
 * Mask (Sec. 3.2: block-sparse attention keeps only retained blocks): a CSR over
 * the visual row tiles of all videos in video order; row r lists, sorted
 * ascending, the video-local visual kv-tile ids its queries may attend to. Each
 * row must contain its own (diagonal) tile and only tiles <= it. Text rows are
 * implicitly dense and causal over their own video. Within a kept tile, keys are
 * causal (key position <= query position).
 *
 * Softmax (Eq. 8, Eq. 11): logits s_ij = softmax_scale * q_i . k_j with query
 * head h reading KV head h / (hq / hkv); LSE_i = ln sum_j exp(s_ij).
 */
typedef struct {
  int32_t num_videos;            /* B >= 1                                         */
  const int32_t* cu_seqlens_h;   /* host [B+1], cu_seqlens[0] = 0, non-decreasing   */
  const int32_t* n_vis_h;        /* host [B], 0 <= n_vis[b] <= seqlen_b, a multiple of
                                    tokens_per_frame; a video may have no text tokens
                                    (its evidence is then zero) or no visual tokens  */
  int32_t tokens_per_frame;      /* N_v: a power of two, 4 <= N_v <= tile          */
  int32_t hq;                    /* query heads                                     */
  int32_t hkv;                   /* KV heads, hq % hkv == 0                         */
  int32_t head_dim;              /* d in {64, 128}                                  */
  int32_t tile;                  /* t_s in {64, 128}                                */
  float softmax_scale;           /* 0 => 1/sqrt(head_dim)                           */
  const void* q;                 /* device bf16 [N_tot, hq, d], contiguous, 16-B aligned */
  const void* k;                 /* device bf16 [N_tot, hkv, d]                     */
  const void* v;                 /* device bf16 [N_tot, hkv, d]                     */
  const int32_t* mask_row_ptr_h; /* host [R+1], R = sum_b ceil(n_vis[b] / tile)      */
  const int32_t* mask_col_idx_h; /* host [row_ptr[R]]                               */
  void* o;                       /* device bf16 [N_tot, hq, d] (written)            */
  float* lse;                    /* device fp32 [hq, N_tot], natural log (written); must
                                    stay alive until evisel_evidence_reduce() ran  */
  int32_t cross_frame;           /* 1: the probe also keeps, per visual row, kept kv
                                    tile and key frame, the log-sum of the row's
                                    attention on that frame, for
                                    evisel_cross_frame_evidence() (needs
                                    tokens_per_frame >= 16; workspace grows by
                                    hq * nnz(mask) * tile * (tile / min(N_v, 64))
                                    * 4 bytes).
                                    0: not kept. Ignored by evisel_intra_frame_evidence. */
  int32_t text_evidence;         /* how evisel_evidence_reduce() forms the text-row
                                    probabilities: 0 = from the text rows' logits the
                                    probe spills into the workspace (hq * n_text *
                                    n_vis * 4 bytes per video); 1 = recomputed from
                                    q and k (no spill; q and k, like lse, must stay
                                    alive until evisel_evidence_reduce() ran). Same
                                    outputs within fp32 rounding. */
  const uint32_t* keep;          /* NULL, or device per-row block masks from
                                    evisel_topp_mask(): row i of head h attends only
                                    the keys of blocks whose bit is set (its top-p
                                    set S_i and its own block, causally), within the
                                    kv tiles the mask above keeps (pass the row
                                    tiles' union). Not with cross_frame or
                                    text_evidence; evisel_intra_frame_evidence and
                                    evisel_cross_frame_evidence refuse such a probe. */
  int32_t keep_words;            /* W of keep [hq, W, N_tot]                        */
  int32_t keep_block;            /* the block size B the masks were built with      */
} evisel_probe_args;

/* Block-sparse causal GQA varlen attention (Eq. 1; Appendix Eq. 8 and Eq. 11
 * with exact token logits on every kept tile). Writes O and LSE for every
 * token, and spills the text rows' logits onto their video's visual tokens into
 * the workspace for evisel_evidence_reduce().
 *   args      : the call description above (host struct, read during the call).
 *   stream    : cudaStream_t as void*.
 *   ws_inout  : in/out. *ws_inout == NULL -> a workspace is created and stored;
 *               otherwise it is reused (grown when too small). The caller must not
 *               use one workspace from two streams concurrently.
 * Errors: EVISEL_EINVAL, EVISEL_EUNSUPPORTED, EVISEL_EMASK (validated on the host
 * before any launch), EVISEL_ENOMEM, EVISEL_ECUDA. Device-side timeouts surface
 * through evisel_status(). */
int evisel_probe_attention(const evisel_probe_args* args, void* stream, evisel_ws** ws_inout);

/* Evidence reduction over the text rows of the last probe on `ws` (Sec. 3.2,
 * "Evidence Decomposition"; head averaging and the query-frame cue A_qf):
 *   tok[h, m]   = sum_{text rows i} exp(s_im - LSE_i)      device fp32 [hq, sum_b n_vis[b]]
 *   frame[h, t] = sum_{m in frame t} tok[h, m]             device fp32 [hq, sum_b T_b]
 *   head[b, h]  = sum_{t in video b} frame[h, t]           device fp32 [B, hq]
 *   aqf[t]      = sum_h frame[h, t] / (hq * n_text_b)      device fp32 [sum_b T_b]
 *                 (0 for a video without text tokens)
 * Columns of tok and frame are the videos' visual tokens / frames in video order.
 * accumulate != 0 adds tok and frame into the existing contents (sum over
 * layers); head and aqf are always recomputed from the resulting frame map, so
 * they accumulate too. Must be enqueued on the probe's stream (or after it).
 * Errors: EVISEL_EINVAL, EVISEL_ESTATE, EVISEL_ECUDA. */
int evisel_evidence_reduce(const evisel_ws* ws, float* tok, float* frame, float* head, float* aqf,
                           int accumulate, void* stream);

/* Synchronises the stream of the workspace's last call, releases every device
 * and host buffer of the workspace. NULL-safe. */
void evisel_free(evisel_ws* ws);

/* Synchronises the stream of the workspace's last call and returns the device
 * status word (EVISEL_OK or EVISEL_ETIMEOUT; EVISEL_EBOUNDS is reserved), then
 * clears it.
 * Returns EVISEL_ECUDA if the synchronisation itself failed. */
int evisel_status(evisel_ws* ws);

/* Static description of a status code. */
const char* evisel_strerror(int code);

/* Detail of the last failure on the calling thread ("" if none). */
const char* evisel_last_error(void);

/* Bytes of device memory currently held by the workspace (0 for NULL). */
int64_t evisel_workspace_bytes(const evisel_ws* ws);

/* Identity of this binary: a hash of the sources, headers, compiler flags,
 * compiler version and machine type it was built from (a static string owned
 * by the library). The paper has no counterpart; it lets a log show which
 * build ran. */
const char* evisel_build_id(void);

/* ---- Entry point that allocates nothing ---------------------------------------
 * The paper has no counterpart to this call. It serves callers of this library
 * that cannot call cudaMalloc on their serving path: servers that hand all device
 * memory to their own pool up front, real-time paths where an allocation (and the
 * device synchronisation that cudaFree implies) is not acceptable, or hosts that
 * forbid the library any allocator use of its own.
 *
 * It computes exactly what evisel_probe_attention() followed by
 * evisel_evidence_reduce() compute, with the same arguments and outputs (O and
 * LSE through `args`, the four evidence maps through tok/frame/head/aqf), but it
 * allocates nothing: no cudaMalloc, cudaFree, pinned memory or workspace. All of
 * its scratch -- the work plan, the split-KV partials of the text rows and the
 * text-row logit spill -- lives in one static device array of
 * EVISEL_NOALLOC_SCRATCH_BYTES (64 MiB), which every GPU that loads this library
 * holds until the process exits.
 *   - Limit: a problem whose scratch does not fit is rejected with EVISEL_ENOMEM
 *     (evisel_last_error() states the bytes needed) before anything is enqueued.
 *     The spill dominates: about hq * n_text * n_vis * 4 bytes per video, e.g.
 *     28 heads x 64 text x 4096 visual tokens = 29 MiB fits; the 65,664-token
 *     probe (940 MiB) does not -- use evisel_probe_attention() for it.
 *   - Set-up: the first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress, with that device current) and caches it; make that
 *     first call before any stream capture begins.
 *   - Sharing: all calls use the same array, which keeps the previous call's
 *     contents; each call clears what must start at zero (the device status
 *     word). Calls whose GPU work overlaps (different streams, or host threads
 *     without ordering) race on the array: order them on one stream.
 *   - device_status: NULL -> the call is asynchronous on `stream`; otherwise it
 *     waits for `stream` and stores the device status word there (EVISEL_OK or
 *     EVISEL_ETIMEOUT). With NULL a device-side timeout is not reported: the
 *     status word lives in the shared array, no other call reads it, and the
 *     next call clears it. Callers that need to know pass a pointer.
 * Errors: as evisel_probe_attention() and evisel_evidence_reduce(). */
#define EVISEL_NOALLOC_SCRATCH_BYTES (64LL << 20)
int evisel_probe_evidence_noalloc(const evisel_probe_args* args, float* tok, float* frame, float* head,
                                  float* aqf, int accumulate, void* stream, int* device_status);

/* ---------------------------------------------------------------------------
 * evisel_intra_frame_evidence: the intra-frame cue A_if of Sec. 3.2
 * ("Evidence Decomposition"): for every frame t (over the videos in order),
 * the head-averaged token-level causal attention among its N_v visual tokens,
 *     A_if[t, i, j] = (1 / hq) sum_h exp(s^h_ij - LSE^h_i),  j <= i,  0 above,
 * with s = scale q_i k_j (Eq. 8) recomputed from Q/K and LSE the row's
 * normaliser saved by the probe (Eq. 11), so each frame row sums to the share
 * of its attention that stays inside the frame. E_if, the selector's
 * intra-frame input, is A_if flattened per timestamp (and stacked over layers
 * by the caller).
 *   args   the arguments of the evisel_probe_attention() call that ran on `ws`
 *          (q, k, cu_seqlens_h, n_vis_h, tokens_per_frame, hq, hkv, head_dim,
 *          softmax_scale; args->lse is that call's LSE output, read here);
 *          o/v/mask are not read but must be valid as for the probe.
 *   ws     the workspace of that probe (its plan is read; the call records
 *          its stream there, so that evisel_status(ws) waits for it).
 *   aif    device fp32 [sum_b T_b, N_v, N_v], T_b = n_vis_h[b] / N_v.
 *   accumulate  0: overwrite aif; 1: add to it (sum over layers).
 * Asynchronous on `stream` (cudaStream_t, NULL = legacy default). Device-side
 * timeouts are reported through evisel_status(ws).
 * Errors: EVISEL_EINVAL (NULL aif or args as for the probe), EVISEL_ESTATE (no
 * probe has run on ws), EVISEL_ECUDA. */
int evisel_intra_frame_evidence(const evisel_probe_args* args, const evisel_ws* ws, float* aif, int accumulate,
                                void* stream);

/* ---------------------------------------------------------------------------
 * evisel_cross_frame_evidence: the cross-frame cue A_ff of Sec. 3.2 ("Evidence
 * Decomposition") and its timestamp-aligned evidence E_ff. For frames b < a of
 * one video,
 *     A_ff[a-1, b] = (1 / (N_v hq)) sum_h sum_{i in frame a} sum_{j in frame b} P^h_ij,
 * the attention frame a's visual rows give to frame b, averaged over a's rows
 * and over heads (P the probe's probability, Eq. 11: pairs whose kv tile the
 * mask does not keep are 0), and
 *     E_ff[t] = ( sum_{b<t} A_ff[t-1, b] + sum_{a>t} A_ff[a-1, t] ) / 2,
 * the attention frame t gives to earlier frames and the attention it receives
 * from later ones, averaged.
 *   args   the arguments of the evisel_probe_attention() call that ran on `ws`,
 *          which must have had cross_frame = 1 (args->lse is read).
 *   ws     that workspace (its plan and cross-frame partials are read; the call
 *          records its stream there for evisel_status()).
 *   aff    device fp32, the videos' [(T_b - 1), (T_b - 1)] row-major blocks back
 *          to back in video order (sum_b (T_b - 1)^2 floats; entries b >= a are 0).
 *   eff    device fp32 [sum_b T_b], or NULL to skip it. Always recomputed from
 *          the resulting aff (so it follows aff's accumulation).
 *   accumulate  0: overwrite aff (every entry is written); 1: add to it (sum
 *          over layers).
 * Asynchronous on `stream`. Errors: EVISEL_EINVAL (NULL aff when sum_b
 * (T_b - 1)^2 > 0, args not matching the probe), EVISEL_ESTATE (no probe on
 * ws, or it ran without cross_frame), EVISEL_ECUDA. */
int evisel_cross_frame_evidence(const evisel_probe_args* args, evisel_ws* ws, float* aff, float* eff,
                                int accumulate, void* stream);

/* ---------------------------------------------------------------------------
 * evisel_topp_mask: the top-p block retention of the sparse prefill (Appendix,
 * "Detailed Sparse Prefilling", Eq. 6-9 and the retention rule after Eq. 9).
 * Blocks: per video, visual blocks of `block` tokens from the visual start,
 * then the text tokens in blocks of `block` from the text start (the last may
 * be short); block ids count the visual blocks first. For row i: H_i = the
 * blocks of its video that end before i; k_bar_j = mean key of block j (Eq. 7,
 * per KV head, rounded to bf16); g_ij = softmax_scale q_i k_bar_j (Eq. 8);
 * p_ij = softmax over H_i (Eq. 9); S_i = the shortest prefix of H_i ordered by
 * p descending (ties: lower block id) whose mass reaches tau_p. Logits closer
 * than (max - min) / 16384 over H_i may be taken as ties.
 *   args   q, k, cu_seqlens_h, n_vis_h, tokens_per_frame, hq, hkv, head_dim,
 *          tile, softmax_scale as for the probe (the mask, v, o, lse are not read).
 *   block  B: a power of two, 16 <= B <= tokens_per_frame (so B divides N_v).
 *   tau_p  in (0, 1] (the paper uses 0.97).
 *   keep   device uint32 [hq, W, N_tot], W = ceil(max_b blocks_b / 32): bit j of
 *          word w of (h, row) is block 32 w + j of the row's video, set for S_i
 *          and for the row's own block (whose causal prefix it attends).
 *   tile_union  device uint32 [R, ceil(max_b ceil(n_vis_b / tile) / 32)] or NULL:
 *          for each visual row tile of the probe's tiling (R as the mask's rows),
 *          bit c of the video-local visual kv tile c, set when some row of the
 *          tile keeps a block of that tile for some head. Read as a CSR (each row
 *          lists its set bits ascending), it is a valid mask for
 *          evisel_probe_attention() whose kept tiles cover every row's S_i.
 *   ws_inout  a workspace (created when *ws_inout == NULL) that holds the
 *          call's metadata and the k_bar scratch.
 * Asynchronous on `stream`. Errors: EVISEL_EINVAL, EVISEL_EUNSUPPORTED,
 * EVISEL_ENOMEM, EVISEL_ECUDA; device timeouts through evisel_status(). */
int evisel_topp_mask(const evisel_probe_args* args, int32_t block, float tau_p, uint32_t* keep,
                     uint32_t* tile_union, void* stream, evisel_ws** ws_inout);

/* ---------------------------------------------------------------------------
 * evisel_coarse_evidence: the evidence maps of the coarse token-level map of the
 * sparse prefill (Appendix, "Detailed Sparse Prefilling", Eq. 10-11). For a text
 * row i of head h: a_im = softmax_scale q_i k_m for the keys of its own block up
 * to i, a_im = g_ij = softmax_scale q_i k_bar_j for the tokens of each block j of
 * S_i, -inf elsewhere; A~_i = softmax(a_i). Then, over the text rows,
 *   tok[h, m] = sum_i A~_im (visual m), frame[h, t], head[b, h], aqf[t]
 * as evisel_evidence_reduce() defines them (same layouts).
 *   args   as for the evisel_topp_mask() call that ran on `ws` (q, k, videos, N_v,
 *          heads, head_dim, softmax_scale); `block` its block size.
 *   keep   that call's per-row bits (S_i and the own block).
 *   ws     the workspace of that call (its k_bar is read; coarse scratch grows
 *          by about hq * n_text_total * 32 * W * 4 bytes).
 *   accumulate  0: overwrite tok and frame; 1: add (sum over layers); head and
 *          aqf are recomputed from the resulting frame map.
 * Asynchronous on `stream` after a short synchronous upload of the per-video
 * offsets. Errors: EVISEL_EINVAL, EVISEL_ESTATE (no evisel_topp_mask on ws),
 * EVISEL_ENOMEM, EVISEL_ECUDA. */
int evisel_coarse_evidence(const evisel_probe_args* args, evisel_ws* ws, int32_t block, const uint32_t* keep,
                           float* tok, float* frame, float* head, float* aqf, int accumulate, void* stream);

/* ---------------------------------------------------------------------------
 * evisel_selftest_wait: failure detection check (no counterpart in the paper).
 * Every wait in the library's kernels is bounded: it gives up after a time
 * limit, records EVISEL_ETIMEOUT in a device status word and lets the kernel
 * drain and exit, so that a stuck pipeline ends as an error the host can read
 * instead of a hung GPU. This call runs that same bounded wait in a one-warp
 * kernel on a barrier of its own, with a short limit:
 *   - arrive = 0: nothing ever completes the barrier's phase, so the wait must
 *     give up after about timeout_us microseconds: *device_status = EVISEL_ETIMEOUT;
 *   - arrive = 1: the kernel completes the phase before waiting:
 *     *device_status = EVISEL_OK.
 * timeout_us: 1 .. 1000000. stream: cudaStream_t (NULL = legacy default).
 * The call waits for `stream` and stores the kernel's status in *device_status
 * (required). The device keeps working afterwards (nothing faults or traps).
 * Returns EVISEL_OK, EVISEL_EINVAL (bad timeout or NULL device_status) or
 * EVISEL_ECUDA. */
int evisel_selftest_wait(int timeout_us, int arrive, void* stream, int* device_status);

#ifdef __cplusplus
}
#endif

#endif /* EVISEL_H */
