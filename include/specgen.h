/*
 * specgen.h -- C ABI of the GB300 fork-decode attention library.
 *
 * The operation.  SpecGen forks K non-reasoning generations off a running
 * reasoning generation; every fork's prompt is the iteration prompt followed by
 * the reasoning prefix pi (Algorithm 1, "Fork K spec. generations"; Section
 * 6.1.1), so the forks share that prefix's KV cache (Section 4.2; Section 8.6,
 * prefix-cache reuse).  Decoding one token for every fork means: for fork f of
 * trace t and query head h (kv head g = h / (hq / hkv)),
 *
 *     keys/values = prefix tokens 0..P_t-1 of trace t, then suffix tokens
 *                   0..S_f-1 of fork f (logical order)
 *     s_i  = scale * <q[f,h,:], k_i[g,:]>
 *     O    = sum_i softmax(s)_i v_i[g,:]        LSE = ln sum_i exp(s_i)
 *
 * The library splits this into a prefix stage (all forks of a trace read the
 * shared prefix pages once), a per-fork suffix stage, and a log-sum-exp merge of
 * the partial results; the answer is the plain definition above up to fp32
 * rounding.
 *
 * Paged KV layout (caller-owned device memory, never freed by the library):
 *     k_pages  bf16 [num_pages][hkv][page_size x head_dim_qk block]
 *     v_pages  bf16 [num_pages][hkv][page_size x head_dim_v block]
 *              (block element order: args->kv_layout, see SPECGEN_KV_*)
 *              or NULL: latent KV, value row = first head_dim_v columns of the
 *              key row (MLA-style absorbed attention, hkv = 1 typically).
 *     Token j of a sequence lives in page table[j / page_size] at slot
 *     j % page_size.  A suffix starts at slot 0 of its own first page.  Slots
 *     past a sequence's length are never read (they may hold anything,
 *     including NaN).
 * Block tables are CSR int32 arrays on the device:
 *     prefix pages of trace t: prefix_block_table[prefix_bt_offsets[t] + i]
 *     suffix pages of fork f:  suffix_block_table[suffix_bt_offsets[f] + i]
 * Forks of trace t are forks fork_offsets[t] .. fork_offsets[t+1]-1 (host).
 *
 * Conventions.  Every call is asynchronous on the caller's CUDA stream
 * (cudaStream_t passed as void*, NULL = legacy default stream), performs no
 * device synchronisation and allocates no device memory: scratch lives in the
 * caller's workspace.  Errors are status codes, never exceptions or aborts.
 * Kernels never trap: a page id outside [0, num_pages) is skipped and recorded
 * in the workspace status word (read it with specgen_workspace_status).
 */
#ifndef SPECGEN_H
#define SPECGEN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SPECGEN_OK = 0,
  SPECGEN_ERR_NULL = -1,        /* a required pointer is NULL */
  SPECGEN_ERR_SHAPE = -2,       /* inconsistent sizes (e.g. hq % hkv != 0, negative length) */
  SPECGEN_ERR_UNSUPPORTED = -3, /* head dims / page size / group size not built */
  SPECGEN_ERR_WORKSPACE = -4,   /* workspace too small or misaligned (256 B) */
  SPECGEN_ERR_INDEX = -5,       /* device saw a page id outside [0, num_pages) */
  SPECGEN_ERR_CUDA = -6,        /* a CUDA runtime call or launch failed */
  SPECGEN_ERR_TIMEOUT = -7      /* a device-side wait hit its iteration limit */
} specgen_status;

/* Device-side arguments of one fork-decode call (all pointers device memory). */
typedef struct {
  int num_traces;               /* T >= 1 */
  int total_forks;              /* F >= 1, sum over traces */
  int hq, hkv;                  /* query / kv heads, hq % hkv == 0 */
  int head_dim_qk, head_dim_v;  /* (64,64), (128,128) or (576,512) with v_pages == NULL */
  int page_size;                /* 16 or 64 tokens */
  int num_pages;                /* pool size; page ids are checked against it */
  float scale;                  /* softmax scale sigma applied to q.k, finite and > 0 */
  const void* q;                /* bf16 [total_forks][hq][head_dim_qk]; q and the pools
                                   16-byte aligned (else SPECGEN_ERR_SHAPE) */
  const void* k_pages;          /* bf16, layout above */
  const void* v_pages;          /* bf16, layout above, or NULL (latent KV) */
  const int32_t* prefix_block_table;
  const int32_t* prefix_bt_offsets;  /* [num_traces + 1] */
  const int32_t* suffix_block_table;
  const int32_t* suffix_bt_offsets;  /* [total_forks + 1] */
  void* out;                    /* bf16 [total_forks][hq][head_dim_v] (written) */
  float* lse;                   /* fp32 [total_forks][hq] natural-log LSE (written) */
  void* workspace;              /* >= specgen_fork_attn_workspace_size bytes, 256-B aligned */
  size_t workspace_bytes;
  int kv_layout;                /* SPECGEN_KV_ROWS or SPECGEN_KV_TILED (see below) */
  const int32_t* suffix_lens;   /* optional device [total_forks]: the suffix lengths to use,
                                   each <= the host length the plan was made for; NULL =
                                   the planned lengths.  Lets one plan serve several decode
                                   steps (plan for the lengths a few steps ahead, advance
                                   this array on the device after each append). */
} specgen_fork_attn_args;

/* Layout of one (page, kv head) block of page_size x head_dim values in the
 * separate K and V pools:
 *   SPECGEN_KV_ROWS   token-major rows: element (t, d) at t * head_dim + d.
 *   SPECGEN_KV_TILED  8 x 8 tiles: element (t, d) at
 *                     ((t/8) * (head_dim/8) + d/8) * 64 + (t%8) * 8 + d%8,
 *                     so the block is exactly the tensor cores' operand layout
 *                     and moves with one bulk copy.  Requires the tensor-core
 *                     path (separate V pool, head_dim 64 or 128, page_size 16).
 * The latent pool (v_pages == NULL) is always token-major (kv_layout must be
 * SPECGEN_KV_ROWS there).  Any other value: SPECGEN_ERR_SHAPE; TILED on a
 * shape outside the tensor-core path: SPECGEN_ERR_UNSUPPORTED. */
#define SPECGEN_KV_ROWS 0
#define SPECGEN_KV_TILED 1

/* Host copies of the lengths: planning reads them, so no device->host copy is
 * needed.  The device block tables must hold at least ceil(len/page_size)
 * pages for every sequence.  The two block-table offset arrays are optional
 * host copies of args->prefix_bt_offsets / suffix_bt_offsets; when given (both
 * non-NULL) the kernels skip one dependent device load per work item. */
typedef struct {
  const int32_t* prefix_lens;   /* host [num_traces], >= 0 */
  const int32_t* fork_offsets;  /* host [num_traces + 1], non-decreasing, [0]=0, [T]=F */
  const int32_t* suffix_lens;   /* host [total_forks], >= 0 */
  const int32_t* prefix_bt_offsets;  /* host [num_traces + 1] or NULL */
  const int32_t* suffix_bt_offsets;  /* host [total_forks + 1] or NULL */
} specgen_host_lens;

/* Result of planning: work counts and workspace offsets.  Treat as opaque;
 * valid for the args/lens it was made from while the workspace is unchanged. */
typedef struct {
  int32_t valid;
  int32_t n_tc_items;           /* tensor-core work items (prefix and suffix chunks) */
  int32_t n_tc_ctas;            /* persistent CTAs of the tensor-core kernel */
  int32_t n_split_items;        /* split-K paged-decode work items */
  int32_t n_rows;               /* total_forks * hq */
  int32_t total_slots;          /* partial (O, LSE) slots */
  int32_t flags;
  int32_t n_part_groups;        /* head groups with their own partial count per fork */
  int64_t plan_bytes;           /* plan bytes copied into the workspace */
  int64_t ws_plan_off, ws_part_o_off, ws_part_lse_off, ws_end;
  int64_t offsets[8];           /* internal offsets inside the plan region */
  int32_t n_sfx_items;          /* suffix-stage work items (per-fork suffix page ranges) */
  int32_t n_sfx_ctas;           /* CTAs of the suffix-stage kernel */
  int64_t sfx_offsets[2];       /* internal offsets inside the plan region */
} specgen_plan;

/* Bytes of workspace one call needs (0 on invalid input).  Depends only on the
 * sizes in args (pointers may be NULL) and on the host lengths. */
size_t specgen_fork_attn_workspace_size(const specgen_fork_attn_args* args,
                                        const specgen_host_lens* lens);

/* Plan the call on the host and copy the plan into the workspace (one
 * cudaMemcpyAsync on `stream` from library-owned host memory that stays valid
 * until the next plan call from this thread).  Also resets the workspace status
 * word.  `plan` receives the launch shapes used by specgen_fork_attn_run. */
specgen_status specgen_fork_attn_plan(const specgen_fork_attn_args* args,
                                      const specgen_host_lens* lens,
                                      specgen_plan* plan, void* cuda_stream);

/* specgen_fork_attn_plan into host memory (no counterpart in the paper: a
 * convenience for callers that stage their own uploads, and a way to check a
 * plan on the host).  Writes the plan region -- exactly the
 * plan->ws_plan_off + plan->plan_bytes bytes that specgen_fork_attn_plan copies
 * to the start of args->workspace: a zeroed header holding the status word,
 * then the work list -- to host_dst, and fills `plan`.  Nothing is copied to
 * the device: the caller uploads those bytes to the start of the workspace
 * before specgen_fork_attn_run.  Same checks and status codes as
 * specgen_fork_attn_plan; SPECGEN_ERR_WORKSPACE if host_bytes is too small. */
specgen_status specgen_fork_attn_plan_host(const specgen_fork_attn_args* args,
                                           const specgen_host_lens* lens, void* host_dst,
                                           size_t host_bytes, specgen_plan* plan);

/* Launch the kernels of a planned call (no host-device copies; capturable in a
 * CUDA graph).  The data pointers in args may differ from the planning call;
 * the sizes and workspace may not. */
specgen_status specgen_fork_attn_run(const specgen_fork_attn_args* args,
                                     const specgen_plan* plan, void* cuda_stream);

/* The two stages of specgen_fork_attn_run, for callers that schedule them
 * apart (or time each kernel alone).  _partials launches the attention kernels
 * (tensor-core and/or split-K), which write every work item's partial (O
 * normalised by its own softmax sum, LSE) into the workspace; _merge launches
 * the log-sum-exp merge that combines each (fork, head) row's partials into
 * out / lse (exact merge of attention over disjoint key sets, the prefix and
 * suffix stages above).  _partials then _merge on one stream equals one
 * specgen_fork_attn_run.  (No separate counterpart in the paper: a scheduling
 * and timing convenience.)  Same arguments, checks and status codes as
 * specgen_fork_attn_run. */
specgen_status specgen_fork_attn_run_partials(const specgen_fork_attn_args* args,
                                              const specgen_plan* plan, void* cuda_stream);
specgen_status specgen_fork_attn_run_merge(const specgen_fork_attn_args* args,
                                           const specgen_plan* plan, void* cuda_stream);

/* specgen_fork_attn_run with timing marks for per-kernel measurement: records
 * events[0] on `cuda_stream` before the first kernel and events[i] after the
 * i-th kernel (i = 1 .. n_events-1; extra launches get no mark).  `events`
 * holds cudaEvent_t handles created by the caller.  Runs exactly the same
 * kernels as specgen_fork_attn_run; *n_launches (if not NULL) receives how
 * many kernels were launched. */
specgen_status specgen_fork_attn_run_profiled(const specgen_fork_attn_args* args,
                                              const specgen_plan* plan, void* cuda_stream,
                                              void* const* events, int n_events,
                                              int* n_launches);

/* Fork-decode attention for every fork and query head: plan + run. */
specgen_status specgen_fork_attn_decode(const specgen_fork_attn_args* args,
                                        const specgen_host_lens* lens,
                                        void* cuda_stream);

/* One decode step from host memory, in one call (no counterpart in the paper:
 * a serving convenience).  On `cuda_stream`: copies in_bytes from host_in to
 * dev_in, then does specgen_fork_attn_decode(args, lens), then copies
 * out_bytes from dev_out to host_out.  The caller lays the step's device
 * inputs (Q and the block-table arrays) out inside dev_in and points args at
 * them, and likewise out / lse inside dev_out, so that each direction is a
 * single copy.  Host buffers should be pinned for the copies to be
 * asynchronous; host_out is valid once the stream reaches the end of the
 * call.  in_bytes or out_bytes may be 0 (that copy is skipped).  The plan is
 * uploaded from a page-locked staging ring that the library keeps per host
 * thread (4 slots, grown on demand, kept until the process exits), so the call
 * does not wait for its copies; a slot is reused only once the copy that read
 * it has run, so the host blocks when it is 4 calls ahead of the GPU.  Status
 * codes as specgen_fork_attn_decode (a shape error queues nothing);
 * SPECGEN_ERR_NULL for a missing buffer of a non-empty copy; SPECGEN_ERR_CUDA
 * if a copy cannot be queued. */
specgen_status specgen_fork_attn_decode_staged(const specgen_fork_attn_args* args,
                                               const specgen_host_lens* lens,
                                               const void* host_in, void* dev_in,
                                               size_t in_bytes, const void* dev_out,
                                               void* host_out, size_t out_bytes,
                                               void* cuda_stream);

/* specgen_fork_attn_decode_staged with the plan in the caller's input
 * buffers (no counterpart in the paper: a serving convenience).  host_in and
 * dev_in are in_capacity bytes long (dev_in 256-byte aligned); the caller's
 * packed inputs occupy their first in_bytes, as for
 * specgen_fork_attn_decode_staged.  The call plans on the host, writes the
 * plan region (a zeroed status header, then the plan:
 * specgen_plan.ws_plan_off + plan_bytes bytes, as the workspace would hold
 * it) into host_in at offset r (in_bytes rounded up to 256) and sends the
 * first r + region bytes of host_in to dev_in: in one copy after the planning
 * when the stream still has work queued, or, when the stream is idle (the
 * GPU is waiting for this host), the inputs at once, overlapping the
 * planning, and the plan region after it.  The kernels read the plan there,
 * and keep their partials in args->workspace (still
 * specgen_fork_attn_workspace_size bytes).  The call's status word is the
 * first word at dev_in + r: read it with specgen_workspace_status(dev_in + r,
 * stream).  host_in is written by the call, so, as for the inputs the caller
 * stores there, no copy still queued may read it (reuse it only after the
 * stream has passed the previous call's copy).  Returns SPECGEN_ERR_WORKSPACE
 * when r + region > in_capacity or args->workspace_bytes is too small (the
 * inputs may have been copied to dev_in already; nothing else is queued), the
 * shape and pointer checks of specgen_fork_attn_decode and SPECGEN_ERR_SHAPE
 * for a dev_in not 256-byte aligned (nothing queued), SPECGEN_ERR_NULL for a
 * missing buffer, SPECGEN_ERR_CUDA if a copy or launch cannot be queued. */
specgen_status specgen_fork_attn_decode_staged_inline(const specgen_fork_attn_args* args,
                                                      const specgen_host_lens* lens,
                                                      void* host_in, void* dev_in,
                                                      size_t in_bytes, size_t in_capacity,
                                                      const void* dev_out, void* host_out,
                                                      size_t out_bytes, void* cuda_stream);

/* specgen_fork_attn_decode for callers that cannot allocate device memory.
 * (No counterpart in the paper: this is a deployment convenience.)  Some
 * callers cannot call cudaMalloc at all -- for example a plugin inside a host
 * engine that owns the whole device memory pool, or code on a latency-critical
 * path where an allocation (which may synchronise the device) is not allowed --
 * so they cannot supply args->workspace.  This entry point ignores
 * args->workspace / workspace_bytes and uses a library-owned scratch array of
 * 16 MiB (SPECGEN_STATIC_WORKSPACE_BYTES) that every GPU loading the library
 * keeps until the process exits; it allocates nothing.  Each call is planned
 * once on the host; a call that needs more scratch than the array holds
 * (specgen_fork_attn_workspace_size above 16 MiB) returns SPECGEN_ERR_WORKSPACE
 * before any CUDA call.  Every call then asks the runtime for the array's
 * device address on the calling thread's current device (a host-side query;
 * nothing is cached, so a context created again is handled).  All calls share
 * the one array and each leaves its contents behind (the plan upload resets
 * the status word): calls that may overlap on the GPU (different streams, or
 * host threads) race and must be serialised by the caller.  The status word of
 * the array (a page id outside the pool was skipped, or a device-side wait hit
 * its limit and the outputs are not valid) is read with
 * specgen_static_workspace_status; without that read both go unnoticed. */
#define SPECGEN_STATIC_WORKSPACE_BYTES (16u << 20)
specgen_status specgen_fork_attn_decode_static(const specgen_fork_attn_args* args,
                                               const specgen_host_lens* lens,
                                               void* cuda_stream);

/* specgen_workspace_status for the scratch array of
 * specgen_fork_attn_decode_static on the current device: synchronises
 * `cuda_stream` and returns SPECGEN_OK, SPECGEN_ERR_INDEX or
 * SPECGEN_ERR_TIMEOUT for the last static call that ran (SPECGEN_ERR_CUDA if
 * the array's address cannot be had).  (No counterpart in the paper.) */
specgen_status specgen_static_workspace_status(void* cuda_stream);

/* Standalone log-sum-exp merge of two partial attentions over disjoint key
 * sets (the combination step of the split computation):
 *     m = max(lse_a, lse_b); w_x = exp(lse_x - m)
 *     out = (w_a out_a + w_b out_b) / (w_a + w_b);  lse = m + ln(w_a + w_b)
 * An input row with lse = -inf is empty; both empty gives out = 0, lse = -inf.
 * out_a, out_b, out: [rows][dv] of dtype (0 = bf16, 1 = fp32); lse_*: fp32 [rows].
 * out/lse may alias out_a/lse_a (in-place).  Device pointers. */
specgen_status specgen_lse_merge(const void* out_a, const float* lse_a,
                                 const void* out_b, const float* lse_b,
                                 void* out, float* lse, int rows, int dv,
                                 int dtype, void* cuda_stream);

/* ---- Fork prefill ---------------------------------------------------------
 * Before a fork decodes, its new prompt tokens (the iteration prompt after the
 * shared reasoning prefix, Algorithm 1 and Section 6.1.1) are prefilled: fork f
 * appends chunk_lens[f] tokens after its suffix_lens[f] existing suffix tokens
 * (their K/V rows already written into its suffix pages, e.g. by the caller's
 * projection), and query j of the chunk attends to the trace's prefix, the
 * fork's existing suffix and, causally, chunk tokens 0..j: exactly a decode
 * query whose suffix length is suffix_lens[f] + j + 1.  The call plans one row
 * block per chunk token (fork by fork, trace by trace), so the prefix stage
 * still reads each prefix page once for up to 128 / (hq / hkv) query rows.
 * args: as for decode except total_forks = sum of chunk_lens (query rows):
 * q, out, lse are [rows][hq][...] in that order, while the block tables and
 * suffix_bt_offsets stay per fork (fork_offsets[num_traces] forks);
 * args->suffix_lens must be NULL.  Run the plan with specgen_fork_attn_run
 * (or _partials / _merge); same status codes as the decode entry points. */
typedef struct {
  const int32_t* prefix_lens;       /* host [num_traces] */
  const int32_t* fork_offsets;      /* host [num_traces + 1] over forks */
  const int32_t* suffix_lens;       /* host [forks]: suffix tokens before the chunk */
  const int32_t* chunk_lens;        /* host [forks]: new tokens of each fork (>= 0) */
  const int32_t* prefix_bt_offsets; /* host [num_traces + 1] or NULL */
  const int32_t* suffix_bt_offsets; /* host [forks + 1] or NULL */
} specgen_prefill_lens;

size_t specgen_fork_prefill_workspace_size(const specgen_fork_attn_args* args,
                                           const specgen_prefill_lens* lens);
specgen_status specgen_fork_prefill_plan(const specgen_fork_attn_args* args,
                                         const specgen_prefill_lens* lens, specgen_plan* plan,
                                         void* cuda_stream);
/* specgen_fork_prefill_plan into host memory, as specgen_fork_attn_plan_host
 * does for decode (no counterpart in the paper). */
specgen_status specgen_fork_prefill_plan_host(const specgen_fork_attn_args* args,
                                              const specgen_prefill_lens* lens, void* host_dst,
                                              size_t host_bytes, specgen_plan* plan);

/* ---- Nested-prefix cascade -------------------------------------------------
 * Fork events taken repeatedly along one reasoning trace, at growing prefixes
 * pi_1, pi_2, ... (Algorithm 1 triggers speculation again and again), give a
 * tree of shared prefix segments.  Segment s holds segment_lens[s] tokens in
 * prefix table s (args->prefix_block_table / prefix_bt_offsets are indexed by
 * segment; token 0 sits at slot 0 of the segment's first page, so a fork point
 * inside a page leaves that page's tail to each fork's own suffix) and serves
 * the forks [segment_rows[2s], segment_rows[2s+1]).  Fork f attends to every
 * segment that serves it, then to its own suffix.  The ranges must be laminar
 * (any two nested or disjoint: number the forks depth-first); each segment's
 * pages are then read once for up to 128 / (hq / hkv) forks, not once per fork
 * event.  args: num_traces = num_segments, everything else as for decode
 * (args->suffix_lens may cut suffixes).  Run the plan with
 * specgen_fork_attn_run; same status codes as the decode entry points. */
typedef struct {
  int num_segments;
  const int32_t* segment_lens;       /* host [num_segments], >= 0 */
  const int32_t* segment_rows;       /* host [2 * num_segments]: [begin, end) of forks */
  const int32_t* suffix_lens;        /* host [total_forks], >= 0 */
  const int32_t* segment_bt_offsets; /* host [num_segments + 1] or NULL */
  const int32_t* suffix_bt_offsets;  /* host [total_forks + 1] or NULL */
} specgen_cascade_lens;

size_t specgen_fork_cascade_workspace_size(const specgen_fork_attn_args* args,
                                           const specgen_cascade_lens* lens);
specgen_status specgen_fork_cascade_plan(const specgen_fork_attn_args* args,
                                         const specgen_cascade_lens* lens, specgen_plan* plan,
                                         void* cuda_stream);
/* specgen_fork_cascade_plan into host memory, as specgen_fork_attn_plan_host
 * does for decode (no counterpart in the paper). */
specgen_status specgen_fork_cascade_plan_host(const specgen_fork_attn_args* args,
                                              const specgen_cascade_lens* lens, void* host_dst,
                                              size_t host_bytes, specgen_plan* plan);

/* ---- Decode-step append --------------------------------------------------
 * After a fork event every fork decodes its own continuation while the prefix
 * stays shared (Algorithm 1, "Fork K spec. generations"; Section 4.2), so each
 * decode step adds one key/value row per fork to the fork's private suffix,
 * before that step's attention reads it.  Fork f with n = suffix_lens[f]
 * tokens already in its suffix writes its rows to slot n % page_size of page
 * suffix_block_table[suffix_bt_offsets[f] + n / page_size]; when
 * n % page_size == 0 that page is new: the fork takes free_pages[j], where j
 * counts the forks before f that also start a page in this call (fork order),
 * and the id is written into the fork's block table.  All inputs are device
 * memory and nothing is planned on the host, so the call can be captured in a
 * CUDA graph; the caller then adds 1 to every suffix length (host and device
 * copies) and drops the j ids taken from the front of its free list.  With
 * suffix_lens_next the kernel writes the advanced device lengths itself, into
 * a second array (another fork's count still reads the first one), which the
 * step's attention and the next append then take as their suffix_lens; the
 * two arrays swap roles every step.  The kernel is launched as a programmatic
 * dependent of the stream's previous kernel (it reads nothing before that
 * kernel has completed) and lets the next kernel start its prologue early.
 * A fork whose block table has no room (n / page_size >= its CSR capacity),
 * whose free-list entry does not exist, or whose page id is outside
 * [0, num_pages) writes nothing and ORs SPECGEN_ERR_INDEX's bit (1) into
 * *status (when status is not NULL; a fork-attention workspace's first word
 * serves, read back with specgen_workspace_status).  Rows are copied bit for
 * bit.  (An extension of the decode path; the paper shows no kernel for it.) */
typedef struct {
  int total_forks, hkv, head_dim_qk, head_dim_v, page_size, num_pages;
  int kv_layout;                    /* layout of the pools: SPECGEN_KV_ROWS / _TILED */
  const void* k_new;                /* bf16 [total_forks][hkv][head_dim_qk], 16-B aligned */
  const void* v_new;                /* bf16 [total_forks][hkv][head_dim_v]; NULL iff v_pages is */
  void* k_pages;                    /* pools as in specgen_fork_attn_args (written), 16-B aligned */
  void* v_pages;                    /* NULL: latent pool, only the key row is stored */
  int32_t* suffix_block_table;      /* CSR with spare capacity per fork; new ids written */
  const int32_t* suffix_bt_offsets; /* [total_forks + 1] */
  const int32_t* suffix_lens;       /* [total_forks] tokens already in each suffix */
  const int32_t* free_pages;        /* [num_free] page ids handed out in fork order */
  int num_free;
  uint32_t* status;                 /* device status word, or NULL */
  int32_t* suffix_lens_next;        /* optional [total_forks]: receives the lengths after
                                       this call (suffix_lens[f] + 1 where fork f appended,
                                       suffix_lens[f] where it could not); NULL: not
                                       written.  Must not be suffix_lens itself. */
} specgen_append_args;

/* Head dims must be multiples of 8 (rows move in 16-byte pieces); page_size a power of
 * two <= 1024; the tiled layout needs page_size % 8 == 0 and a value pool.
 * Returns SPECGEN_OK after launching (asynchronous on cuda_stream),
 * SPECGEN_ERR_NULL / _SHAPE / _UNSUPPORTED on bad arguments (nothing
 * launched; SPECGEN_ERR_UNSUPPORTED for suffix_lens_next == suffix_lens),
 * SPECGEN_ERR_CUDA if the launch fails. */
specgen_status specgen_append_kv(const specgen_append_args* args, void* cuda_stream);

/* ---- Prefix page pack / unpack ----------------------------------------------
 * The remote prefix cache (Section 6.2.3) moves a suspended trace's prefix KV
 * off the GPU and back.  On the device that is a gather of the sequence's pages
 * into one contiguous buffer and a scatter back under a new block table:
 *   specgen_pack_pages    packed = K[table[0]] .. K[table[n-1]] V[table[0]] .. V[table[n-1]]
 *   specgen_unpack_pages  page table[i] of each pool <- page i of packed
 * where a page block is hkv x page_size x head_dim bf16 in the pool's own block
 * layout (bytes are copied as they are: rows and tiled pools both work; the
 * latent pool has no V section).  Pools hold num_pages blocks.  A page id
 * outside [0, num_pages) is skipped and ORs SPECGEN_ERR_INDEX's bit (1) into
 * *status (when status is not NULL).  table, packed and the pools are device
 * memory (16-byte aligned); asynchronous on cuda_stream, capturable.
 * (An extension for the remote prefix cache; the paper shows no kernel for it.) */
typedef struct {
  int hkv, head_dim_qk, head_dim_v, page_size, num_pages;
  void* k_pages;                    /* bf16 [num_pages][hkv][page_size][head_dim_qk] */
  void* v_pages;                    /* bf16 [num_pages][hkv][page_size][head_dim_v] or NULL */
  uint32_t* status;                 /* device status word, or NULL */
} specgen_pool_desc;

/* Bytes of the packed buffer for n_pages pages (0 on invalid input; a page
 * block must be a multiple of 16 bytes). */
size_t specgen_packed_bytes(const specgen_pool_desc* pool, int n_pages);
specgen_status specgen_pack_pages(const specgen_pool_desc* pool, const int32_t* table,
                                  int n_pages, void* packed, void* cuda_stream);
specgen_status specgen_unpack_pages(const specgen_pool_desc* pool, const int32_t* table,
                                    int n_pages, const void* packed, void* cuda_stream);

/* Read the workspace status word written by the kernels (synchronises
 * `cuda_stream`).  Returns SPECGEN_OK, SPECGEN_ERR_INDEX or SPECGEN_ERR_TIMEOUT. */
specgen_status specgen_workspace_status(const void* workspace, void* cuda_stream);

/* Static text for a status code. */
const char* specgen_status_string(specgen_status status);

/* Library version (major * 10000 + minor * 100 + patch). */
int specgen_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SPECGEN_H */
