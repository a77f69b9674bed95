/*
 * mk_attn.h -- C ABI of the GB300 (sm_103a) attention library: forward and
 * backward passes and a paged decode step.
 *
 * The operation is the fused attention forward pass whose reference the
 * paper's Flash Attention and GQA Attention kernels reproduce (Table 2; the
 * contract of Section 2.1 and Section 3.1: take the same input arrays as the
 * reference operation and return the same outputs).  For each sequence b,
 * query head h (key/value head g = h / (Hq / Hkv), contiguous groups) and
 * query position i of the sequence:
 *
 *   K_i    = { j : 0 <= j < L_b  and  (not causal  or  j <= i) }
 *   o[i]   = sum_{j in K_i} softmax_j(scale * q[i] . k[j]) * v[j]
 *   lse[i] = ln( sum_{j in K_i} exp(scale * q[i] . k[j]) )        (natural log)
 *
 * Causal masking is aligned top-left: query and key sequences have the same
 * length, so row i sees keys 0..i.
 *
 * Everything here is plain C: device pointers, sizes and a CUDA stream handle
 * passed as void*.  No symbol takes a PyTorch type.
 */
#ifndef MK_ATTN_H
#define MK_ATTN_H

#include <stdint.h>

#if defined(__GNUC__)
#define MK_API __attribute__((visibility("default")))
#else
#define MK_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes returned by every entry point. */
typedef enum {
    MK_OK = 0,
    MK_ERR_INVALID_ARG = -1,  /* null pointer, non-positive size, Hq % Hkv != 0 */
    MK_ERR_UNSUPPORTED = -2,  /* head dimension other than 64 or 128 */
    MK_ERR_ALIGNMENT = -3,    /* a base pointer not 16-byte aligned */
    MK_ERR_CUDA = -4,         /* a CUDA runtime/driver call failed */
    MK_ERR_TIMEOUT = -5,      /* a kernel wait ran out; reported by mk_attn_check_status */
    MK_ERR_SCRATCH_LIMIT = -6, /* sizes need more than MK_ATTN_DECODE_STATIC_SCRATCH_BYTES of
                                  scratch (mk_attn_decode_paged_noalloc only) */
    MK_ERR_BOUNDS = -7         /* a kernel's store index fell outside its output; checked
                                  only by the check build (MK_DEBUG), reported by
                                  mk_attn_check_status */
} mk_status;

/*
 * Check mode and check build.
 *
 *   MK_ATTN_DEBUG  environment variable, read once at the first call.  Set
 *                  to a nonzero value, every entry point that enqueued work
 *                  synchronises its stream before returning and returns what
 *                  mk_attn_check_status reports (MK_OK, MK_ERR_TIMEOUT,
 *                  MK_ERR_INVALID_ARG, MK_ERR_BOUNDS, MK_ERR_CUDA) instead of
 *                  MK_OK: a device-side error is then tied to the call that
 *                  caused it.  Such calls are no longer asynchronous, so the
 *                  check mode cannot be used while a stream is being captured
 *                  into a CUDA graph (the synchronisation would fail the call
 *                  with MK_ERR_CUDA).
 *   MK_DEBUG       compile definition of the check build of this library
 *                  (libmk_attn_debug.so).  Every kernel then checks the index
 *                  of each global-memory store of its outputs, partials and
 *                  workspace against the sizes of the call; an index out of
 *                  range skips the store and records MK_ERR_BOUNDS for
 *                  mk_attn_check_status.  Nothing traps.  The release build
 *                  carries none of these checks.
 */

/*
 * Streams and CUDA graphs.  Every entry point only enqueues work on the
 * caller's stream (host-side checks and tensor-map encoding aside), so a call
 * can be captured into a CUDA graph and replayed, with these conditions:
 *   - make one call of each entry point and head dimension outside the
 *     capture first (it sets the kernels' shared-memory limits once per
 *     device);
 *   - no check mode (MK_ATTN_DEBUG) during the capture;
 *   - mk_attn_decode_paged_noalloc: see its scratch lookup below;
 *   - MK_SCHED_DYNAMIC (mk_attn_tuning): see the schedule's counter slot.
 * Where one call launches two kernels (the decode and latent decode merges),
 * the second is a programmatic dependent launch: it may be scheduled while the
 * first drains and waits on the device for its results.
 */

/*
 * mk_attn_fwd -- attention forward pass (causal or not, GQA, optional varlen).
 *
 * Arguments (all pointers are DEVICE pointers owned by the caller):
 *   q          bf16, fixed length [B, S, Hq, D]; varlen [T, Hq, D]. Read only.
 *   k, v       bf16, fixed length [B, S, Hkv, D]; varlen [T, Hkv, D]. Read only.
 *   o          bf16 output, same layout as q.  Fully overwritten.
 *   lse        fp32 output, fixed length [B, Hq, S]; varlen [Hq, T].  Fully
 *              overwritten with the natural-log row log-sum-exp (scale included).
 *   B          number of sequences (>= 1).
 *   Hq, Hkv    query and key/value heads (>= 1, Hq % Hkv == 0).
 *   S          fixed length: tokens per sequence (>= 1);
 *              varlen: total tokens T = cu_seqlens[B] (>= 1).
 *   D          head dimension, 64 or 128.
 *   causal     nonzero: row i attends to keys 0..i of its sequence.
 *   scale      multiplier of q . k before the softmax (e.g. 1/sqrt(D)).
 *   cu_seqlens NULL for fixed length; otherwise a DEVICE int32 array [B+1]
 *              of sequence start offsets into the packed token dimension:
 *              cu_seqlens[0] = 0, non-decreasing, cu_seqlens[B] = T.  It is
 *              read only on the device, so the call never synchronises.
 *              Values outside [0, T] are clamped on the device: a malformed
 *              array gives unspecified results but no access outside q, k, v,
 *              o and lse.
 *   stream     cudaStream_t (NULL = legacy default stream).
 *
 * Layout: every tensor is contiguous, innermost dimension last; each base
 * pointer must be 16-byte aligned.
 *
 * Behaviour: the call validates its arguments on the host, encodes TMA
 * descriptors and enqueues one kernel on `stream`; it returns without
 * synchronising.  On any error it returns a negative mk_status and enqueues
 * nothing, so o and lse are left untouched.  The library allocates no device
 * memory.  Results are deterministic: each output element is computed by one
 * CTA in a fixed order, under every schedule, so repeated calls on the same
 * inputs are bitwise identical.  Sequences of length 0 (varlen) produce no
 * rows.  Every internal wait of the kernel is bounded; if one runs out the
 * kernel records MK_ERR_TIMEOUT for mk_attn_check_status and exits.
 */
MK_API int mk_attn_fwd(const void *q, const void *k, const void *v, void *o, float *lse,
                       int B, int Hq, int Hkv, int S, int D, int causal, float scale,
                       const int32_t *cu_seqlens, void *stream);

/*
 * mk_attn_fwd_stall_test -- test support for the failure path only.  Same
 * arguments, checks and return value as mk_attn_fwd, but no CTA loads its
 * first query tile: the kernel's bounded wait for it runs out (about 2 s), all
 * roles of the CTA unwind (in-flight copies and MMAs are drained, tensor
 * memory is freed), o and lse are left incomplete,
 * and the next mk_attn_check_status on the stream returns MK_ERR_TIMEOUT.
 * No fault is raised; the CUDA context stays usable.  Never needed for
 * computing attention.
 */
MK_API int mk_attn_fwd_stall_test(const void *q, const void *k, const void *v, void *o,
                                  float *lse, int B, int Hq, int Hkv, int S, int D, int causal,
                                  float scale, const int32_t *cu_seqlens, void *stream);

/*
 * mk_attn_bwd_workspace_bytes -- bytes of device workspace mk_attn_bwd needs
 * (one fp32 per query row and head: Delta_i = dO_i . o_i), or -1 for invalid
 * sizes.  varlen: nonzero when cu_seqlens will be passed (S = total tokens).
 */
MK_API int64_t mk_attn_bwd_workspace_bytes(int B, int Hq, int S, int varlen);

/*
 * mk_attn_bwd -- attention backward pass: the gradients of the mk_attn_fwd
 * operation with respect to q, k and v for an output gradient dO (the
 * training step of the paper's attention kernels, Table 2).  With
 * P_ij = exp(scale * q_i . k_j - lse_i) over the keys row i sees:
 *   dv_j = sum_{h in group(j)} sum_i P_ij dO_i
 *   dS_ij = P_ij (dO_i . v_j - Delta_i),   Delta_i = dO_i . o_i
 *   dq_i = scale * sum_j dS_ij k_j
 *   dk_j = scale * sum_{h in group(j)} sum_i dS_ij q_i
 *
 * Arguments (all pointers are DEVICE pointers owned by the caller):
 *   q, k, v, B, Hq, Hkv, S, D, causal, scale, cu_seqlens
 *              exactly as passed to mk_attn_fwd.
 *   o, lse     the outputs of that mk_attn_fwd call (bf16 o, fp32 lse).
 *   dO         bf16 gradient of o, layout of q.  Read only.
 *   dq         bf16 output, layout of q.  Fully overwritten.
 *   dk, dv     bf16 outputs, layout of k and v.  Fully overwritten; rows of
 *              keys that no query sees are zero.
 *   workspace  device buffer of at least mk_attn_bwd_workspace_bytes()
 *              bytes, 16-byte aligned; scratch, contents on entry do not
 *              matter.  Calls that share a workspace must not overlap.
 *   stream     cudaStream_t; two kernels are enqueued (dQ, which also
 *              writes Delta_i = dO_i . o_i to the workspace, then dK/dV,
 *              which reads it); the call never synchronises.
 * Layout and alignment: as mk_attn_fwd; dO, dq, dk, dv and workspace 16-byte
 * aligned, lse 4-byte aligned.
 * Returns MK_OK, or MK_ERR_INVALID_ARG (null pointer, sizes, too small a
 * workspace), MK_ERR_UNSUPPORTED (D, or Hq above 65535), MK_ERR_ALIGNMENT,
 * MK_ERR_CUDA; on any
 * error nothing is enqueued.  Deterministic: no atomics, repeated calls give
 * bitwise identical gradients.  Internal waits are bounded as in mk_attn_fwd
 * (MK_ERR_TIMEOUT through mk_attn_check_status).
 */
MK_API int mk_attn_bwd(const void *q, const void *k, const void *v, const void *o,
                       const float *lse, const void *dO, void *dq, void *dk, void *dv, int B,
                       int Hq, int Hkv, int S, int D, int causal, float scale,
                       const int32_t *cu_seqlens, void *workspace, int64_t workspace_bytes,
                       void *stream);

/* Stages of the backward pass, for mk_attn_bwd_stages. */
#define MK_BWD_DELTA 1 /* Delta_i = dO_i . o_i into the workspace (a kernel of its own) */
#define MK_BWD_DKDV 2  /* dk and dv (reads Delta from the workspace) */
#define MK_BWD_DQ 4    /* dq; also computes Delta and writes it to the workspace */
#define MK_BWD_ALL 7

/*
 * mk_attn_bwd_stages -- mk_attn_bwd, enqueuing only the stages in `stages`
 * (a nonzero OR of the MK_BWD_* flags), in the order Delta, dQ, dK/dV; the
 * Delta kernel is skipped when dQ is enqueued (dQ writes Delta itself).
 * Arguments, checks and errors are those of mk_attn_bwd.  MK_BWD_DKDV reads
 * the Delta that an earlier MK_BWD_DELTA or MK_BWD_DQ stage wrote into the
 * same workspace for the same o and dO.  Outputs of stages not enqueued are
 * left untouched.
 */
MK_API int mk_attn_bwd_stages(const void *q, const void *k, const void *v, const void *o,
                              const float *lse, const void *dO, void *dq, void *dk, void *dv,
                              int B, int Hq, int Hkv, int S, int D, int causal, float scale,
                              const int32_t *cu_seqlens, void *workspace,
                              int64_t workspace_bytes, int stages, void *stream);

/*
 * mk_attn_decode_workspace_bytes -- bytes of device workspace that
 * mk_attn_decode_paged needs for these sizes on the current device (0: none),
 * or -1 for invalid sizes.  Depends on the device's SM count only through the
 * number of KV splits it chooses.
 */
MK_API int64_t mk_attn_decode_workspace_bytes(int B, int Hq, int Hkv, int D, int page_size,
                                              int max_pages);

/*
 * mk_attn_decode_paged -- one decode step against a paged key/value cache
 * (the Paged Attention row of the paper's Table 2).  For each sequence b and
 * query head h (key/value head h / (Hq/Hkv)), the newest query attends to all
 * L_b = seq_lens[b] cached positions of its sequence (no mask: the query is
 * the last position):
 *   o[b,h,:] = sum_j softmax_j(scale * q[b,h,:] . k_j) v_j
 *   lse[b,h] = ln sum_j exp(scale * q[b,h,:] . k_j)
 * where position j is slot j % page_size of physical page
 * page_table[b, j / page_size].
 *
 * Arguments (all pointers are DEVICE pointers owned by the caller):
 *   q            bf16 [B, Hq, D].  Read only.
 *   k_cache,     bf16 [num_pages, page_size, Hkv, D].  Read only.
 *   v_cache
 *   page_table   int32 [B, max_pages]; entries j < ceil(L_b / page_size)
 *                must lie in [0, num_pages).  Read only, on the device.
 *   seq_lens     int32 [B], each in [0, max_pages * page_size].  Read only.
 *   o            bf16 [B, Hq, D] output, fully overwritten.
 *   lse          fp32 [B, Hq] output, fully overwritten (natural log, scale
 *                included); L_b = 0 gives o = 0 and lse = -inf.
 *   D            64 or 128.   page_size  16, 32, 64 or 128.
 *   Hq / Hkv     any; Hkv * ceil(Hq / Hkv / 8) at most 65535, B at most
 *                65535.
 *   workspace    device buffer of at least mk_attn_decode_workspace_bytes()
 *                bytes, 16-byte aligned, or NULL when that is 0.  Scratch
 *                for the per-split partial results; its contents on entry
 *                do not matter.  Launches that share a workspace must not
 *                overlap in time.
 *   stream       cudaStream_t; the call is asynchronous and never syncs.
 * Returns MK_OK; MK_ERR_INVALID_ARG (null pointer, sizes out of range, a
 * missing or too small workspace), MK_ERR_UNSUPPORTED (D, page_size, or a
 * grid beyond those limits), MK_ERR_ALIGNMENT (q, caches, o or workspace not
 * 16-byte aligned; page_table, seq_lens or lse not 4-byte aligned), or
 * MK_ERR_CUDA.  On any error nothing is launched.  Page-table entries or
 * lengths out of range, which only the device sees, leave o and lse undefined
 * and make the next mk_attn_check_status return MK_ERR_INVALID_ARG.
 */
MK_API int mk_attn_decode_paged(const void *q, const void *k_cache, const void *v_cache,
                                const int32_t *page_table, const int32_t *seq_lens, void *o,
                                float *lse, int B, int Hq, int Hkv, int D, int page_size,
                                int max_pages, int num_pages, float scale, void *workspace,
                                int64_t workspace_bytes, void *stream);

/* Size of the library's own decode scratch array (16 MiB).  It belongs to
 * the code of the paged decode step, and a GPU reserves it when that code is
 * loaded on it: at the first decode call on the device (either decode entry
 * point), or at context creation when the CUDA runtime loads modules eagerly
 * (CUDA_MODULE_LOADING=EAGER).  It stays reserved until the process exits.
 * Callers that never run a decode step do not load that code and do not
 * hold the array (mk_attn_check_status reads only the status words of the
 * kernel families that have run on the device). */
#define MK_ATTN_DECODE_STATIC_SCRATCH_BYTES (16 * 1024 * 1024)

/*
 * mk_attn_decode_paged_noalloc -- mk_attn_decode_paged for callers that
 * cannot allocate device memory: code that runs where cudaMalloc is not
 * allowed or not wanted (inside a host callback, under an allocator that
 * another runtime owns, or in a plugin that must not touch the device heap).
 * The paper has no counterpart; it is an addition of this library.
 *
 * Arguments, layouts, results and errors are those of mk_attn_decode_paged
 * without `workspace` and `workspace_bytes`: the per-split partial results
 * go to a scratch array of MK_ATTN_DECODE_STATIC_SCRATCH_BYTES bytes that
 * the library declares in device memory (one per GPU).  The call allocates
 * nothing and calls no allocating routine; the array itself is reserved when
 * the decode code loads on the device (see MK_ATTN_DECODE_STATIC_SCRATCH_BYTES),
 * which the first call does if nothing loaded it before.  A caller whose
 * device memory another allocator will take should therefore make one call
 * at start-up, before that allocator claims the device: if the device has no
 * room left for the array when the code loads, that call returns MK_ERR_CUDA.
 *
 *   - Checks run in this order, and the first that fails decides the
 *     status: the host argument checks of mk_attn_decode_paged (no CUDA
 *     call); then the scratch size: sizes for which
 *     mk_attn_decode_workspace_bytes() exceeds
 *     MK_ATTN_DECODE_STATIC_SCRATCH_BYTES return MK_ERR_SCRATCH_LIMIT and
 *     launch nothing (use mk_attn_decode_paged with a workspace for those);
 *     then the array's address.
 *   - The first valid call on each device looks up that device's address of
 *     the array (with the device current) and keeps it; make that first call
 *     before any stream capture on the device.  A failed lookup returns
 *     MK_ERR_CUDA.
 *   - Every call on a device shares the one array, which keeps whatever the
 *     last call left there (nothing in it needs to start at zero: each call
 *     writes every partial it reads).  Calls whose kernels can overlap on the
 *     GPU -- on different streams with no ordering between them, or from
 *     several host threads -- race on it; order them (one stream, or events).
 */
MK_API int mk_attn_decode_paged_noalloc(const void *q, const void *k_cache, const void *v_cache,
                                        const int32_t *page_table, const int32_t *seq_lens,
                                        void *o, float *lse, int B, int Hq, int Hkv, int D,
                                        int page_size, int max_pages, int num_pages, float scale,
                                        void *stream);

/* Latent (MLA) decode: row width of the latent cache (512 latent + 64 rotary
 * components) and of the values (the first 512 components). */
#define MK_MLA_DQK 576
#define MK_MLA_DV 512

/*
 * mk_attn_mla_decode_workspace_bytes -- bytes of device workspace that
 * mk_attn_mla_decode_paged needs for these sizes on the current device (0:
 * none), or -1 for invalid sizes.
 */
MK_API int64_t mk_attn_mla_decode_workspace_bytes(int B, int Hq, int page_size, int max_pages);

/*
 * mk_attn_mla_decode_paged -- one decode step of multi-head latent attention
 * in its absorbed form (the paper's MLA Attention row, Table 2 and Table 3):
 * every query head attends to one shared latent cache, whose rows are the
 * keys in full (MK_MLA_DQK components) and the values through their first
 * MK_MLA_DV components.  For sequence b and query head h:
 *   o[b,h,:] = sum_j softmax_j(scale * q[b,h,:] . c_j) c_j[:MK_MLA_DV]
 *   lse[b,h] = ln sum_j exp(scale * q[b,h,:] . c_j)
 * over the L_b = seq_lens[b] cached positions, position j being slot
 * j % page_size of page page_table[b, j / page_size].
 *
 * Arguments (all pointers are DEVICE pointers owned by the caller):
 *   q           bf16 [B, Hq, MK_MLA_DQK].  Read only.
 *   cache       bf16 [num_pages, page_size, MK_MLA_DQK].  Read only.  Slots
 *               of a sequence's last page past L_b are read (with weight
 *               zero) and must hold finite values.
 *   page_table  int32 [B, max_pages]; entries j < ceil(L_b / page_size) in
 *               [0, num_pages).  seq_lens int32 [B], each in
 *               [0, max_pages * page_size].
 *   o           bf16 [B, Hq, MK_MLA_DV] output; lse fp32 [B, Hq] output
 *               (natural log, scale included); L_b = 0 gives o = 0 and
 *               lse = -inf.
 *   Hq          any (groups of 128 heads), B * ceil(Hq / 128) <= 2^29.
 *   page_size   16, 32, 64 or 128.
 *   workspace   device buffer of at least mk_attn_mla_decode_workspace_bytes()
 *               bytes, 16-byte aligned, or NULL when that is 0 (scratch for
 *               the per-split partials; calls sharing it must not overlap).
 *   stream      cudaStream_t; asynchronous, never synchronises.
 * Returns MK_OK, MK_ERR_INVALID_ARG, MK_ERR_UNSUPPORTED (page_size, grid
 * limits), MK_ERR_ALIGNMENT (q, cache, o, workspace not 16-byte aligned;
 * page_table, seq_lens, lse not 4-byte aligned) or MK_ERR_CUDA; on any
 * error nothing is launched.  Device-side inputs out of range make the next
 * mk_attn_check_status return MK_ERR_INVALID_ARG.
 */
MK_API int mk_attn_mla_decode_paged(const void *q, const void *cache, const int32_t *page_table,
                                    const int32_t *seq_lens, void *o, float *lse, int B, int Hq,
                                    int page_size, int max_pages, int num_pages, float scale,
                                    void *workspace, int64_t workspace_bytes, void *stream);

/* Schedules of work units over the persistent CTAs (mk_attn_tuning.schedule).
 * Units are numbered heaviest first (causal: the query tiles that see the most
 * keys, or the key tiles seen by the most queries). */
#define MK_SCHED_SNAKE 0       /* round k: CTA c takes unit kG + c, or kG + G-1-c in odd rounds */
#define MK_SCHED_ROUND_ROBIN 1 /* round k: CTA c takes unit kG + c */
#define MK_SCHED_BLOCKED 2     /* CTA c takes units c*ceil(n/G) .. (c+1)*ceil(n/G) - 1 */
#define MK_SCHED_DYNAMIC 3     /* forward: CTA c takes unit c, then claims the next
                                  unclaimed unit from a device counter shortly before
                                  each of its units ends (greedy, heaviest first).  The
                                  counters are a ring of 1024 per device, one per launch,
                                  reset by each launch's last CTA: at most 1024 forward
                                  launches may execute at once on a device.  A launch
                                  captured in a CUDA graph keeps its slot, so two
                                  instances of that graph must not run at once.  The
                                  backward kernels take it as MK_SCHED_SNAKE. */

/*
 * Launch parameters that change speed but never results beyond rounding:
 * the knobs of the config autotuner (the paper's Autotuning Agent, Section
 * 2.1, searches kernel configurations the same way: time each candidate,
 * keep the fastest correct one).  Tile shapes and pipeline depths are fixed
 * at compile time by TMEM and shared-memory capacity and are not tunable.
 */
typedef struct {
  int ctas;              /* forward / backward: persistent CTAs, 0 = one per SM;
                            otherwise 1..65535 (capped at the number of units) */
  int schedule;          /* forward / backward: MK_SCHED_* */
  float rescale_log2;    /* forward: the running row max moves (and O is rescaled)
                            only when it rises by more than this, in log2 units;
                            0..16, exact for every value (default 8) */
  int split_ctas_per_sm; /* decode: KV splits are planned for about this many
                            CTAs per SM, 1..64 (default 24) */
  int split_min_pages;   /* decode: fewest pages per KV split, 1..4096 (default 2) */
  int mla_split_ctas_per_sm; /* latent decode: KV splits planned for about this many
                                CTAs per SM (one CTA fits an SM), 1..64 (default 3) */
} mk_attn_tuning;

/*
 * mk_attn_set_tuning -- sets the process-wide tuning used by every later
 * call of mk_attn_fwd, mk_attn_bwd(_stages), mk_attn_decode_paged(_noalloc)
 * and mk_attn_decode_workspace_bytes (the decode split plan, and so its
 * workspace size, depends on it).  NULL restores the defaults.  Returns
 * MK_OK, or MK_ERR_INVALID_ARG for a value out of range (the settings are
 * then unchanged).  Host only; thread-safe, but a call racing a launch on
 * another thread may apply to it or not.
 */
MK_API int mk_attn_set_tuning(const mk_attn_tuning *tuning);

/* mk_attn_get_tuning -- copies the current tuning into *tuning (MK_OK), or
 * returns MK_ERR_INVALID_ARG for NULL. */
MK_API int mk_attn_get_tuning(mk_attn_tuning *tuning);

/* Short static description of a status code.  Never NULL. */
MK_API const char *mk_attn_error_string(int status);

/*
 * mk_attn_check_status -- synchronises `stream`, then reads and clears the
 * device status words written by kernels (forward, backward, decode, latent
 * decode) whose internal waits ran out, that met device-side inputs out of
 * range (decode page tables, lengths), or (check build only) whose store
 * index checks failed.  Only the families that have enqueued a kernel on the
 * current device are read, so the call loads no kernel code of its own.
 * Returns MK_OK, MK_ERR_TIMEOUT, MK_ERR_INVALID_ARG, MK_ERR_BOUNDS, or
 * MK_ERR_CUDA if synchronisation failed.
 */
MK_API int mk_attn_check_status(void *stream);

/* Library version, major * 10000 + minor * 100 + patch. */
MK_API int mk_attn_version(void);

#ifdef __cplusplus
}
#endif

#endif /* MK_ATTN_H */
