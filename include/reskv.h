/*
 * reskv.h -- C ABI of the GB300 (sm_103a) ResKV decode library.
 *
 * ResKV ("Reconstructing Omitted Attention Contributions for Fixed-Budget KV
 * Cache Compression") keeps, per (layer, KV head), a fixed budget of b cache
 * slots split as b = m + r (Sec. 5.1): m exact main-cache tokens (Sec. 5.2,
 * Eq. main_selection) and r residual entries (k_bar_j, v_bar_j, c_j) that
 * summarise the evicted tokens (Sec. 5.3, Eq. summary).  Decoding attends with
 * one shared softmax over both (Sec. 5.4, Eqs. residual_logit, reskv_den,
 * reskv_num, reskv) with the residual logits shifted by log g(q), the dynamic
 * gate of Sec. 5.5.2 (Eq. gate).  r is chosen per (layer, KV head) by the
 * validation proxy of Sec. 5.5.1 (Eqs. valloss, valproxy).  Alg. 1 is the
 * construction, Alg. 2 the decode step.
 *
 * Conventions for every entry point:
 *  - Pointers named "device" are CUDA device pointers of the current device;
 *    "host" pointers are ordinary host memory.  The library never takes
 *    ownership of caller buffers.
 *  - `stream` is a cudaStream_t (NULL = legacy default stream).  Work is
 *    enqueued asynchronously on it; callers must not free inputs before the
 *    stream has passed the call.
 *  - Every function returns a status; nothing aborts or throws across the ABI.
 *    On error the output handle is left untouched and reskv_last_error()
 *    returns a message (thread-local, valid until the next call on the thread).
 *  - Arguments are validated on the host before any launch.
 *  - Calls that share one cache handle must be ordered (same stream, or
 *    synchronised): the handle's decode workspace is reused by every call.
 */
#ifndef RESKV_H
#define RESKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  RESKV_OK = 0,
  RESKV_ERR_INVALID_ARG = 1,   /* bad pointer, size or configuration        */
  RESKV_ERR_UNSUPPORTED = 2,   /* valid but outside what the kernels cover   */
  RESKV_ERR_OOM = 3,           /* cudaMalloc failed                          */
  RESKV_ERR_CUDA = 4,          /* a CUDA runtime call or launch failed       */
  RESKV_ERR_DEVICE_STATUS = 5  /* a kernel reported a fault (bounded wait
                                  timed out or an index left its range)      */
} reskv_status;

enum { RESKV_SCORE_OBS_POOL = 0, RESKV_SCORE_KEYNORM = 1 };
enum { RESKV_GATE_DYNAMIC = 0, RESKV_GATE_FIXED = 1 };
/* RESKV_SOFTMAX_SHARED: Eq. reskv, one softmax over main and residual entries
 * (the method).  RESKV_SOFTMAX_SEPARATE: the "w/o shared softmax" ablation
 * (Table ablation_main); the paper prints no combination rule, and the one
 * built is o^ = (1 - g) o_M + g o_R with each branch normalised on its own
 * (o^ = o_M without residual mass).  It applies to decode and to the
 * validation proxy of reskv_build_cache. */
enum { RESKV_SOFTMAX_SHARED = 0, RESKV_SOFTMAX_SEPARATE = 1 };
enum { RESKV_DECODE_AUTO = 0, RESKV_DECODE_FMA = 1, RESKV_DECODE_MMA = 2, RESKV_DECODE_CLUSTER = 3,
       RESKV_DECODE_LSE_MERGE = 4 };
/* RESKV_BUDGET_UNIFORM: every (layer, batch, KV head) unit gets `budget` (or
 * its entry of unit_budgets).  RESKV_BUDGET_ADAKV: reskv_build_cache splits the
 * H_kv * budget slots of each (layer, batch element) between its KV heads as
 * AdaKV does (App. B, "AdaKV": token scores as importance, safeguard
 * coefficient 0.2), then builds every head with its own budget b_h (the
 * "+ResKV" rows of Table ruler_paper and Table longbench_paper).  The paper
 * prints no formula; the rule built: every head keeps its recent window P and
 * its own f = floor(adakv_safeguard * (budget - |P|)) best-ranked tokens; the
 * other H_kv * (budget - |P| - f) slots go to the highest scores among all
 * heads' remaining evictable tokens (ties: lower head, then lower position);
 * b_h = |P| + f + head h's share.  With budget >= seq_len nothing is evicted
 * and every head keeps `budget`. */
enum { RESKV_BUDGET_UNIFORM = 0, RESKV_BUDGET_ADAKV = 1 };

/* What reskv_append does when a unit's append_capacity slots are taken.
 * RESKV_APPEND_FAIL: the call fails (RESKV_ERR_UNSUPPORTED, nothing written).
 * RESKV_APPEND_RING_DROP, RESKV_APPEND_RING_FOLD: the A appended slots are a
 * ring of the unit's A most recent tokens; the oldest leaves the exact window
 * to make room.  DROP: it leaves the cache.  FOLD: it becomes a member of its
 * nearest residual entry (least squared distance between keys, decided
 * exactly, ties to the lower entry; the nearest-centre rule of Eq.
 * residual_partition) whose stored means and count are updated as a running
 * mean (Eq. summary): k_bar <- (c k_bar + k) / (c + 1) and v_bar likewise,
 * evaluated in fp64 and stored in bf16 (round to nearest even), c <- c + 1,
 * log-count beta ln(c + 1); a unit without residual entries drops it.  The
 * paper leaves refreshing residual entries during generation to future work
 * (App. E); this is the reading built. */
enum { RESKV_APPEND_FAIL = 0, RESKV_APPEND_RING_DROP = 1, RESKV_APPEND_RING_FOLD = 2 };

#define RESKV_MAX_GRID 8

/*
 * Construction and decode settings.  reskv_config_default() fills the paper's
 * values (App. B, "ResKV Construction Settings"; App. B.2 SnapKV): recent
 * window 64, pooling kernel 5, 96 fit + 32 validation queries, ratio grid
 * {0, .05, .10, .15, .20}, 4 Lloyd iterations, delta 0.01, beta 1.0,
 * tau 0.25, alpha (= 1/T_g) 12, g_min 0.
 */
typedef struct reskv_config {
  int32_t batch;           /* B                                              */
  int32_t n_layers;        /* L                                              */
  int32_t n_kv_heads;      /* H_kv                                           */
  int32_t group;           /* G query heads per KV head (GQA); 1, 2 or 4     */
  int32_t head_dim;        /* d; must be 128                                 */
  int64_t seq_len;         /* s, cached tokens per (batch, layer, KV head)   */
  int32_t budget;          /* b slots per (layer, KV head) (Sec. 3.2)        */
  int32_t recent_window;   /* |P|, always kept (Eq. main_selection)          */
  int32_t n_obs;           /* observation queries per query head             */
  int32_t n_fit;           /* first n_fit rows score tokens (Sec. 5.5.1)     */
  int32_t n_val;           /* last n_val rows validate (Sec. 5.5.1)          */
  int32_t pool_kernel;     /* SnapKV average-pooling width, odd (App. B.2)   */
  int32_t score_mode;      /* RESKV_SCORE_*                                  */
  int32_t n_grid;          /* entries used in grid_ratios                    */
  float grid_ratios[RESKV_MAX_GRID]; /* candidates r = floor(ratio * b)      */
  int32_t lloyd_iters;     /* T rounds of (assign, update) (App. B)          */
  float delta;             /* margin of Eq. valproxy                         */
  float beta;              /* count exponent: logit term beta * log c_j      */
  const int32_t* residual_override; /* host [L*B*H_kv] fixed r per unit, or
                              NULL to run the validation proxy               */
  int32_t gate_mode;       /* RESKV_GATE_DYNAMIC (Eq. gate) or _FIXED        */
  float tau;               /* gate threshold                                 */
  float alpha;             /* gate slope 1/T_g                               */
  float g_min;             /* gate floor                                     */
  float g_fixed;           /* gate value for RESKV_GATE_FIXED (0 = main-only,
                              1 = the paper's "w/o dynamic gate" ablation)   */
  int32_t keep_debug;      /* nonzero: keep construction intermediates for
                              reskv_export_debug (scores, ranking, losses)   */
  int32_t decode_warps;    /* 0: automatic.  Otherwise the number of equal
                              pieces (one warp each) a decode call cuts its
                              slot range into, capped at 8 warps per SM; the
                              result does not depend on it beyond rounding   */
  int32_t decode_kernel;   /* RESKV_DECODE_*: 0 automatic (tensor cores:
                              cluster kernel when a launch's units fit on the
                              device in one wave and decode_warps is 0, else
                              stream-K), 1 CUDA-core fp32x2 FMA, 2 tensor-core
                              stream-K over the launch's slot range, 3
                              tensor-core with one thread-block cluster of 1..8
                              CTAs per unit (decode_warps ignored), 4 the
                              paper's decode structure for comparison (Sec.
                              6.1, App. B): main-cache pass and residual pass
                              merged through log-sum-exp statistics, three
                              launches (decode_warps ignored)                */
  int32_t softmax_mode;    /* RESKV_SOFTMAX_*                                */
  int32_t append_capacity; /* A >= 0: slots per unit reserved for tokens
                              appended at decode time (reskv_append); the
                              unit stride of the layout is budget + A        */
  const int32_t* unit_budgets; /* host [L*B*H_kv] per-unit budgets b_u (AdaKV-
                              style allocation across heads, App. B), or NULL
                              for `budget` everywhere.  Unit u then owns
                              b_u + A slots starting at sum_{v<u} (b_v + A).
                              reskv_build_cache needs b_u >= min(|P|, s)     */
  int32_t budget_mode;     /* RESKV_BUDGET_*; ADAKV needs unit_budgets NULL
                              and is a construction setting (import ignores
                              it).  The built layout is ragged: read the
                              budgets with reskv_get_unit_budgets            */
  float adakv_safeguard;   /* AdaKV safeguard coefficient in [0, 1] (0.2)    */
  int32_t append_policy;   /* RESKV_APPEND_* (reskv_config_default:
                              RESKV_APPEND_RING_FOLD)                        */
} reskv_config;

/* Fill *cfg with the paper's defaults; shape fields are zeroed. */
void reskv_config_default(reskv_config* cfg);

/* Opaque handle; owns every device buffer of the compressed cache. */
typedef struct reskv_cache reskv_cache;

/*
 * Alg. 1 for every (layer, batch, KV head) unit: token scores (App. B.2 rule
 * from the fit observation queries, or the query-free key-norm score), main
 * selection (Eq. main_selection), Lloyd residual entries (Eqs.
 * residual_partition, summary), validation proxy (Eqs. valloss, valproxy) and
 * packing into the ragged main+residual layout.
 *
 *   K_layers[l], V_layers[l] : device bf16 [B, H_kv, s, d] (row-major)
 *   Qobs_layers[l]           : device bf16 [B, H_kv*G, n_obs, d], or the
 *                              array itself NULL with RESKV_SCORE_KEYNORM and
 *                              residual_override set
 *   out                      : receives a new handle on success
 *
 * Inputs may be freed once the stream has passed the call.  The call
 * allocates the handle's device memory (cudaMalloc) and temporary workspace.
 */
reskv_status reskv_build_cache(const reskv_config* cfg, const void* const* K_layers,
                               const void* const* V_layers, const void* const* Qobs_layers,
                               void* stream, reskv_cache** out);

/*
 * Alg. 2 (shared-softmax decode with the dynamic gate) for one decode query
 * per query head.
 *
 *   layer in [0, L) : Q device bf16 [B, H_kv*G, d], O device fp32 [B, H_kv*G, d]
 *   layer == -1     : all layers in one launch, Q [L, B, H_kv*G, d], O likewise
 *
 * Query head hq attends with KV head hq / G.  O must not alias Q.
 */
reskv_status reskv_decode_attn(const reskv_cache* c, int32_t layer, const void* Q, void* O,
                               void* stream);

/*
 * Alg. 2 for the contiguous layers layer0 .. layer0 + n_layers - 1 in one
 * launch (reskv_decode_attn is this call with one layer or all layers): the
 * layers a pipeline stage owns, or a group of layers whose queries and
 * outputs a caller moves between host and device while the next group
 * decodes.  Q device bf16 [n_layers, B, H_kv*G, d], O device fp32, same
 * shape, 16-byte aligned.  RESKV_ERR_INVALID_ARG unless 0 <= layer0 and
 * 1 <= n_layers <= L - layer0.
 */
reskv_status reskv_decode_attn_layers(const reskv_cache* c, int32_t layer0, int32_t n_layers,
                                      const void* Q, void* O, void* stream);

/*
 * Alg. 2 for all layers with the queries and outputs in host memory.
 *
 *   Q_host : host bf16 [L, B, H_kv*G, d]
 *   O_host : host fp32, same shape; must not overlap Q_host
 *
 * With page-locked buffers the device can address (cudaHostAlloc,
 * cudaMallocHost, cudaHostRegister with mapping), the one decode launch reads
 * Q from and writes O to host memory itself, so the transfers overlap the
 * streaming of the cache.  Pageable buffers are staged: a copy in, the
 * decode, a copy out on `stream` (the first such call allocates the handle's
 * staging buffers, device Q and O of all layers, kept until reskv_free).
 * Asynchronous on `stream`: O_host holds the result once the stream has
 * passed the call (cudaStreamSynchronize).  Results equal reskv_decode_attn's
 * bit for bit.  The caller keeps both buffers.  RESKV_ERR_INVALID_ARG for a
 * NULL pointer or overlapping buffers, RESKV_ERR_OOM when the staging buffers
 * cannot be allocated, RESKV_ERR_CUDA when a copy or the launch fails.
 */
reskv_status reskv_decode_attn_host(const reskv_cache* c, const void* Q_host, void* O_host,
                                    void* stream);

/* Release every device buffer of the handle (synchronises the device). NULL-safe. */
void reskv_free(reskv_cache* c);

/* Message of the last failing call on this thread ("" if none). */
const char* reskv_last_error(void);

/* Read the kernels' device status word; RESKV_ERR_DEVICE_STATUS if a kernel
 * reported a fault since the handle was made (synchronises the device). */
reskv_status reskv_check_status(const reskv_cache* c);

/* Shape of a handle's cache. */
typedef struct reskv_cache_info {
  int64_t n_units;         /* U = L*B*H_kv, unit u = (l*B + b)*H_kv + h      */
  int32_t budget;          /* b, main + residual slots per unit              */
  int32_t head_dim;
  int64_t slot_bytes;      /* bytes of one K row + one V row                 */
  int64_t cache_bytes;     /* device bytes of K/V slots + log-counts         */
  int32_t layer_cluster;   /* CTAs per unit of an automatic one-layer decode
                              launch (cluster kernel); 0: stream-K kernel     */
  int32_t layer_cluster_warps; /* warps per CTA of that cluster launch       */
  int32_t all_cluster;     /* the same for an all-layer launch (layer = -1)  */
  int32_t all_cluster_warps;
  float build_ms[6];       /* device time of reskv_build_cache per stage of
                              Alg. 1, summed over layers (ms): token scores,
                              ranking, validation targets o_S, Lloyd residual
                              entries, validation losses + choice of r,
                              packing; zero for an imported cache          */
  int32_t append_capacity; /* A, slots per unit for appended tokens          */
  int32_t stride;          /* b + A, slots per unit in the layout; 0 with
                              per-unit budgets                               */
  int32_t max_appended;    /* most tokens appended to any unit so far        */
  int32_t ragged;          /* 1 with per-unit budgets                        */
  int64_t total_slots;     /* slots of the layout (sum over units)           */
  int32_t n_candidates;    /* candidate columns of the validation proxy (the
                              losses array has 1 + n_candidates per unit)    */
  int32_t ranked_width;    /* entries per unit of RESKV_DEBUG_RANKED         */
  int32_t all_units_per_warp;   /* tensor-core stream-K plan of an all-layer
                              call: k > 0 when every warp takes k whole units
                              (short units), 0 for equal slot pieces or when
                              that call runs another kernel                 */
  int32_t layer_units_per_warp; /* the same for a one-layer call (layer 0)   */
  int32_t kv_copy_rank;    /* rank of the TMA copies of the tensor-core
                              kernels: 3 (one copy per 16-row K or V chunk)
                              or 2 (two 64-dim copies, when the driver
                              refuses the 3-D map)                           */
  int32_t reserved0;
} reskv_cache_info;

reskv_status reskv_get_info(const reskv_cache* c, reskv_cache_info* info);

/* Budget b_u of every unit of the layout (unit u owns b_u + append_capacity
 * slots): `budget` everywhere, the caller's unit_budgets, or the allocation
 * reskv_build_cache made with RESKV_BUDGET_ADAKV.  host_budgets: int32
 * [n_units]; n_units must equal the handle's. */
reskv_status reskv_get_unit_budgets(const reskv_cache* c, int32_t* host_budgets, int64_t n_units);

/*
 * Host-side view of a cache layout, used by reskv_import_cache (read) and
 * reskv_export_cache (written).  Unit u owns S_u = b_u + append_capacity
 * consecutive slots (b_u = budget, or unit_budgets[u]), starting at slot
 * sum_{v<u} S_v (= u*S with one budget): its first n_main[u] slots are
 * main-cache tokens, the next n_res[u] residual entries, the next n_app[u]
 * tokens appended at decode time (exact main rows, reskv_append); the rest is
 * unused.  With N = sum_u S_u slots:
 *   n_main, n_res : int32 [U]
 *   kslots, vslots: bf16 bit patterns, uint16 [N, d]
 *   logc          : fp32 [N]; beta*log c_j at residual slots (-inf for an
 *                   empty entry), ignored at main slots
 *   slot_pos      : int32 [N]; original token position of main slots
 *                   (appended tokens: s, s+1, ...), -1 at residual slots (may
 *                   be NULL on import)
 *   counts        : int32 [N]; c_j at residual slots, 0 at main slots
 *                   (may be NULL on import)
 *   n_app         : int32 [U] (may be NULL on import: none appended)
 */
typedef struct reskv_host_cache {
  int32_t* n_main;
  int32_t* n_res;
  uint16_t* kslots;
  uint16_t* vslots;
  float* logc;
  int32_t* slot_pos;
  int32_t* counts;
  int32_t* n_app;
} reskv_host_cache;

/* Build a handle from host arrays (an externally constructed cache; only the
 * shape, gate, budget, unit_budgets and append_capacity fields of cfg are
 * used).  Requires 1 <= n_main[u], n_main[u] + n_res[u] <= b_u and
 * 0 <= n_app[u] <= append_capacity. */
reskv_status reskv_import_cache(const reskv_config* cfg, const reskv_host_cache* h,
                                void* stream, reskv_cache** out);

/* Copy the handle's layout to host arrays (every pointer non-NULL, sized as
 * above).  Synchronises `stream`. */
reskv_status reskv_export_cache(const reskv_cache* c, reskv_host_cache* h, void* stream);

/*
 * Append the newest decoded token to the cache: one exact K row and V row per
 * (batch, KV head) unit of `layer`, into the unit's append_capacity slots after
 * its main and residual slots (Sec. 3.1: each decode step appends the new
 * token's key and value; Alg. 2 attends over the cache as it stands).
 * Appended tokens are main-cache tokens for every later decode: exact rows in
 * the shared softmax, counted in p_max of the gate.  When the slots are taken,
 * cfg.append_policy decides (RESKV_APPEND_*): refuse, or drop the oldest
 * appended token, or fold it into its nearest residual entry.  The slots then
 * hold the A most recent tokens in ring order (reskv_export_cache gives each
 * its position; an imported cache's appended rows count as appended in slot
 * order).
 *
 *   layer in [0, L) : K_new, V_new device bf16 [B, H_kv, d]
 *   layer == -1     : every layer, K_new, V_new [L, B, H_kv, d]
 *
 * RESKV_ERR_UNSUPPORTED (nothing written) when append_capacity is 0, or when a
 * unit of the call has append_capacity tokens already under
 * RESKV_APPEND_FAIL.  The rows are complete when the stream reaches the next
 * call on it.
 */
reskv_status reskv_append(reskv_cache* c, int32_t layer, const void* K_new, const void* V_new,
                          void* stream);

enum {
  RESKV_DEBUG_SCORES = 0,  /* fp64 [U, s]: token scores                      */
  RESKV_DEBUG_RANKED = 1,  /* int32 [U, W]: top of the ranking of S\P, W =
                              info.ranked_width (b - |P| with one budget);
                              with per-unit budgets unit u fills its first
                              min(b_u, s) - |P| entries, the rest is -1      */
  RESKV_DEBUG_LOSSES = 2,  /* fp64 [U, 1 + n_cand]: L_0 then L_r per candidate
                              column; +inf where a unit has no such candidate */
  RESKV_DEBUG_CANDIDATES = 3, /* int32 [n_cand]: candidate r values, ascending
                              (one budget for every unit only)               */
  RESKV_DEBUG_UNIT_CANDIDATES = 4 /* int32 [U, n_cand]: r of every candidate
                              column per unit, 0 where the unit has none.
                              With per-unit budgets the columns are the
                              positive grid ratios in ascending order and
                              r = floor(ratio * b_u), dropped (0) when zero,
                              equal to the previous column's r, or leaving
                              less than |P| main slots                        */
};

/* Copy a construction intermediate (cfg.keep_debug was set) to host memory.
 * `bytes` must equal the size of the array.  Synchronises the device. */
reskv_status reskv_export_debug(const reskv_cache* c, int32_t what, void* host_dst,
                                size_t bytes);

/*
 * Fault injection, for testing the failure paths without faulting a GPU (no
 * counterpart in the paper).  Process-wide; takes effect on the next calls:
 *   RESKV_TEST_FAIL_FIRST_WAIT, n >= 0: the next n decode launches (any decode
 *     entry point) run with every warp giving up its first ring wait as if
 *     the wait's bound had run out: the kernel sets its status word (code 1),
 *     waits for its own copies in flight and returns with the output
 *     incomplete.  The handle's partial-result tickets are then not reset:
 *     free the handle after reskv_check_status reports the fault.  A
 *     reskv_build_cache call takes one of the n instead: in its first
 *     persistent Lloyd assignment, CTA 0's certifier gives up its first
 *     wait; that CTA stops at a tile boundary, the build completes with the
 *     entries of that run incomplete, and the new handle's status word
 *     reports code 1.
 *   RESKV_TEST_FAIL_ALLOC, n >= 1: the n-th device allocation of the library
 *     from now on fails as cudaMalloc out of memory would (nothing is
 *     allocated for it; the call returns RESKV_ERR_OOM and frees what it had
 *     allocated).  n = 0 cancels.
 * RESKV_ERR_INVALID_ARG for another `what` or n < 0.
 */
enum { RESKV_TEST_FAIL_FIRST_WAIT = 1, RESKV_TEST_FAIL_ALLOC = 2 };
reskv_status reskv_test_inject(int32_t what, int64_t n);

/*
 * Decode that allocates nothing.  The paper has no counterpart: this entry
 * point exists for callers that cannot allocate device memory at decode time
 * -- code running inside a host application whose memory manager owns every
 * GPU allocation, or latency-critical paths that must not call cudaMalloc
 * (it may block and synchronise the device).  Such callers hold the
 * compressed cache in memory of their own and describe it here with plain
 * device pointers (the layout of reskv_import_cache, on the device).
 *
 * The per-call scratch (partial results of units split between warps, their
 * tickets, a status word) lives in one static device array of 16 MiB inside
 * the library; every GPU that loads the library holds it until the process
 * exits.  A call whose scratch would exceed it fails with
 * RESKV_ERR_UNSUPPORTED before launching anything; decode fewer units per call
 * (one layer at a time) in that case.  Roughly, a call needs
 * (n_units + 8 * SMs) * 2 * group * 528 bytes plus 4 bytes per unit.
 *
 * Every call looks up the array's device address (cudaGetSymbolAddress, with
 * the caller's device current; it allocates nothing).  The first call on a
 * device may also load the library's device code, so make it before any
 * stream capture.  Every call shares the array and clears the parts that must
 * start at zero, so calls that overlap on the GPU race: order them on one
 * stream (or synchronise between them).  A kernel fault (a bounded wait that
 * gave up, leaving O partly unwritten, or an index out of range) is ORed into
 * a device status word that only reskv_noalloc_check_status reads and clears.
 *
 * The cache has no appended tokens (budget here is the unit stride).
 *   kslots, vslots : device bf16 [n_units, budget, 128], 16-byte aligned
 *   logc           : device fp32 [n_units, budget] (beta*log c at residual slots)
 *   n_main, n_res  : device int32 [n_units]; the caller guarantees
 *                    1 <= n_main[u] and n_main[u] + n_res[u] <= budget
 *   Q              : device bf16 [n_units / n_kv_heads, n_kv_heads*group, 128]
 *   O              : device fp32, same shape as Q
 * When budget is a multiple of 16, logc is 16-byte aligned and the cache holds
 * fewer than 2^31 slots, the call runs the tensor-core kernel of
 * reskv_decode_attn (its 16-slot copies then stay inside these arrays; the
 * copy descriptors are encoded on the host per call, which allocates
 * nothing); otherwise the CUDA-core kernel, which reads slot by slot.  Either
 * reads only inside these arrays.
 */
typedef struct reskv_device_cache {
  const void* kslots;
  const void* vslots;
  const float* logc;
  const int32_t* n_main;
  const int32_t* n_res;
  int64_t n_units;
  int32_t budget;
  int32_t n_kv_heads;
  int32_t group;
  int32_t gate_mode;
  float tau, alpha, g_min, g_fixed;
} reskv_device_cache;

reskv_status reskv_decode_attn_noalloc(const reskv_device_cache* c, const void* Q, void* O,
                                       void* stream);

/*
 * Status of the no-allocation decode (no counterpart in the paper; it
 * allocates nothing either).  Synchronises `stream`, reads the current
 * device's status word of reskv_decode_attn_noalloc -- the codes of every
 * kernel fault since the last check, ORed together -- and clears it.
 * RESKV_ERR_DEVICE_STATUS when a fault was recorded (the message names the
 * codes: 1 = bounded wait timed out, 2 = index out of range), else RESKV_OK.
 * last_kernel (may be NULL) receives the kernel that the calling thread's
 * last successful reskv_decode_attn_noalloc launched: RESKV_DECODE_MMA (the
 * tensor-core stream-K kernel) or RESKV_DECODE_FMA (the CUDA-core kernel,
 * taken when budget is not a multiple of 16 or logc is not 16-byte aligned);
 * 0 before the first call.
 */
reskv_status reskv_noalloc_check_status(void* stream, int32_t* last_kernel);

#ifdef __cplusplus
}
#endif

#endif /* RESKV_H */
