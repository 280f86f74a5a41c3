/*
 * scone.h — C ABI of the SCONE inference-time input-embedding path on one
 * NVIDIA GB300 (sm_103a).
 *
 * The path (Algorithm 1, inference branch, Sec. 3 of "Scaling Embedding
 * Layers in Language Models"): for every position i of a token sequence
 * (sigma_1 .. sigma_m), take the smallest j < i such that the n-gram
 * (sigma_j .. sigma_i) is an f-gram, i.e. the longest f-gram ending at i,
 * and emit that f-gram's precomputed embedding F(sigma_j .. sigma_i); if no
 * f-gram ends at i, emit the token embedding T(sigma_i). f-grams have
 * lengths 2..K (V_fgram is a subset of V_token^[2,K], Sec. 3).
 *
 * F is stored as "a dense embedding matrix paired with a hash dictionary
 * that maps f-grams to matrix indices" (Sec. 2, "Efficient Indexing for
 * Large Embedding Layers"). Here the dictionary is a GPU bucketized cuckoo
 * hash table (two candidate buckets of two slots per key; a lookup reads the
 * second bucket only when the first is full without the key) built once by
 * scone_table_build; the dense matrix stays
 * caller-owned in HBM or in host-pinned, device-mapped memory (the paper's
 * off-accelerator tier, Sec. 4.3).
 *
 * Conventions shared by every call
 *  - Pointers are plain addresses; "device" means a CUDA device address
 *    (cudaMalloc / torch CUDA tensor), "host" an ordinary host address.
 *    No call takes ownership of a caller buffer.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default).
 *    Calls marked "async" only enqueue work on it and return.
 *  - Embedding rows are bf16, passed as raw 16-bit words (scone_bf16), rows
 *    of d elements, row-major, no padding between rows.
 *  - Token batches are dense [B x L] int32, sequence-major. n-grams never
 *    cross a sequence boundary; the first position of every sequence always
 *    takes T.
 *  - Errors the host can see (null or misaligned pointers, bad sizes, K or
 *    vocab that the key format cannot hold) are returned at once and nothing
 *    is enqueued. Errors only the device can see (a token outside
 *    [0, vocab), a lookup that exceeded the probe limit) never trap: the
 *    position gets a zero row, row = -1 and len = 0, and a sticky status
 *    word in the table records the first such error; scone_status reads it.
 *  - Return values are SCONE_OK (0) or a negative scone_err code.
 */
#ifndef SCONE_H_
#define SCONE_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct scone_table scone_table;   /* opaque; owns its slot array and status word */
typedef struct scone_decode scone_decode; /* opaque; owns the device history ring */
typedef struct scone_discover scone_discover; /* opaque; reusable workspace of f-gram discovery */
typedef uint16_t scone_bf16;              /* raw bf16 bits */

enum scone_err {
  SCONE_OK = 0,
  SCONE_ERR_INVALID_ARG = -1,     /* bad pointer, size, alignment or location */
  SCONE_ERR_TOKEN_RANGE = -2,     /* a token outside [0, vocab) (device-detected, sticky) */
  SCONE_ERR_DUPLICATE_FGRAM = -3, /* the f-gram list holds the same n-gram twice */
  SCONE_ERR_TABLE_FULL = -4,      /* an insert found no free slot (cannot happen below LF 1) */
  SCONE_ERR_PROBE_LIMIT = -5,     /* a lookup read more buckets than the limit (sticky) */
  SCONE_ERR_UNSUPPORTED = -6,     /* outside what the call supports: K * ceil(log2 vocab)
                                     wider than the key format, a size past the call's
                                     documented limit, or a copy mode it cannot use */
  SCONE_ERR_CUDA = -7,            /* a CUDA runtime call failed */
  SCONE_ERR_NOMEM = -8            /* device or host allocation failed */
};

enum scone_rows_location {
  SCONE_ROWS_DEVICE = 0,      /* F is device memory (HBM) */
  SCONE_ROWS_HOST_MAPPED = 1  /* F is host memory from cudaHostAlloc(..., cudaHostAllocMapped)
                                 or cudaHostRegister(..., Mapped); the GPU reads it over the
                                 host link */
};

/*
 * scone_table_build — the f-gram dictionary of Sec. 2 ("hash dictionary that
 * maps f-grams to matrix indices"), built on the GPU. Synchronous.
 *
 *  fgram_tok  host int32 [n_fgrams * K]: f-gram r is fgram_tok[r*K .. r*K+len-1],
 *             oldest token first; entries past the length are ignored.
 *  fgram_len  host uint8 [n_fgrams], each in [2, K] (1-grams are not f-grams, Sec. 3).
 *  n_fgrams   >= 0. Row r of F belongs to f-gram r (its index in this list).
 *  K          maximum f-gram length, 2..8.
 *  vocab      token ids are [0, vocab); every f-gram token must be in range.
 *  d          embedding width (elements per row), >= 1.
 *  F          [n_fgrams * d] bf16 rows; a device address, or a host address of
 *             mapped pinned memory when F_location = SCONE_ROWS_HOST_MAPPED.
 *             May be NULL only when n_fgrams = 0.
 *  T          device [vocab * d] bf16 token embeddings (Sec. 2: T stays on the
 *             accelerator).
 *  load_factor  target fill of the slot array, in (0, 0.85]; 0 selects 0.5.
 *  stream     used for the build kernels; the call synchronizes it.
 *  out        receives the table.
 *
 * The table borrows F and T (they must outlive it) and owns only its slot
 * array (16- or 32-byte slots, two per bucket), a status word and a zero row.
 * Insertion may retry with new hash seeds; TABLE_FULL means eight seeds
 * failed (not expected below load factor 0.85). Errors: INVALID_ARG (bad
 * list, length, token or pointer), DUPLICATE_FGRAM, TABLE_FULL,
 * UNSUPPORTED (key does not fit: K*ceil(log2 vocab) > 220), NOMEM, CUDA.
 *
 * Tables with 16-byte slots and 3 <= K <= 5 also get a suffix index (see
 * scone_fgram_suffix_index): every suffix of length >= 2 of a listed f-gram
 * is findable, as an f-gram or as a marker slot without a row, and carries
 * a bit saying that a longer f-gram ends with it. The fused embed can then
 * look the lengths up one at a time and stop at the first absent window.
 * The markers count towards the load factor (scone_table_info.n_markers);
 * results are the same with or without the index.
 */
int scone_table_build(const int32_t* fgram_tok, const uint8_t* fgram_len, int64_t n_fgrams,
                      int32_t K, int32_t vocab, int32_t d, const scone_bf16* F,
                      int32_t F_location, const scone_bf16* T, float load_factor, void* stream,
                      scone_table** out);

/*
 * scone_fgram_suffix_index — the suffix index that scone_table_build adds to
 * a table (host only, no GPU needed). Algorithm 1 (Sec. 3) takes the longest
 * window ending at a position that is an f-gram. If every suffix of length
 * >= 2 of every listed f-gram can be found, with a bit saying that a longer
 * f-gram ends with it, a lookup may try n = 2, 3, ... and stop at the first
 * window that is absent or lacks the bit: no longer window is an f-gram.
 *
 *  fgram_tok, fgram_len, n_fgrams, K  the list, as for scone_table_build.
 *  ext         host uint8 [n_fgrams] or NULL: ext[r] = 1 when f-gram r is a
 *              suffix of a longer listed f-gram, else 0.
 *  marker_tok  host int32 [marker_cap * K] or NULL: the suffixes that are not
 *              listed, each once, padded with -1 (oldest token first).
 *  marker_len  host uint8 [marker_cap] or NULL: their lengths.
 *  marker_cap  markers the caller has room for (0: count only); the first
 *              min(cap, count) markers are written.
 *  n_markers   receives the number of markers.
 *
 * Markers are listed in the order the f-grams reach them (f-gram order,
 * longest suffix first). Errors: INVALID_ARG (bad pointer, K or length),
 * DUPLICATE_FGRAM, UNSUPPORTED (more than 2^32 - 2 entries), NOMEM.
 */
int scone_fgram_suffix_index(const int32_t* fgram_tok, const uint8_t* fgram_len,
                             int64_t n_fgrams, int32_t K, uint8_t* ext, int32_t* marker_tok,
                             uint8_t* marker_len, int64_t marker_cap, int64_t* n_markers);

/* Frees the slot array and status word (after a device synchronize). NULL is a no-op. */
int scone_table_destroy(scone_table* table);

/*
 * scone_table_rebuild_noalloc — puts a new f-gram list (and its rows F) into
 * a table made by scone_table_build, without allocating any memory. The
 * paper has no counterpart: it is for callers that cannot allocate at the
 * moment they swap lists, e.g. a serving process whose device memory is
 * owned by another allocator (cudaMalloc would fail or fragment it), or a
 * latency-bound thread that must not pay for cudaMalloc / cudaFree, which can
 * synchronize the whole device.
 *
 * It reuses the table's own slot array, so the new list must fit it: at most
 * 0.85 * n_slots f-grams (see scone_table_get_info). K, vocab, d, T and the F
 * location stay those of the original build. The rebuilt table has no
 * suffix index (n_markers 0: computing one needs host memory), so the fused
 * embed looks every length up; results are the same. The build kernels' scratch (a
 * device copy of the list plus three flags) lives in one file-scope device
 * array of SCONE_REBUILD_SCRATCH_BYTES, which every GPU that loads the library
 * holds until the process exits. A list of n f-grams needs
 *     256 + round256(n) + round256(4 * K * n)
 * bytes of it (round256 rounds up to a multiple of 256; a list of
 * SCONE_REBUILD_MAX_FGRAMS(K) f-grams always fits: 1,290,496 at K = 3), and a
 * larger list is rejected with SCONE_ERR_INVALID_ARG before any device work.
 * The first call on a device looks the array's address up (once per device);
 * make that first call before any stream capture begins.
 *
 * All calls share that array and it keeps the last call's contents; the
 * flags are cleared by each call. Calls whose device work overlaps (other
 * streams, other threads) race on it, and so do lookups on this table from
 * other streams during the call. Synchronous: it synchronizes `stream`.
 *
 * Launches take the table's state (F, row count, hash seed) by value when
 * they are enqueued. Work enqueued or captured before this call (a CUDA graph
 * of embed or decode launches, in particular) keeps the old state and would
 * read the new slots against the old F: capture such graphs again after the
 * call returns.
 *
 * Errors: INVALID_ARG (table NULL, list too large for the table or the
 * scratch, bad list or F; the table is unchanged), DUPLICATE_FGRAM or
 * TABLE_FULL (the table is then left empty: every position falls back to T),
 * CUDA (one attempt is made to leave the table empty; if scone_table_get_info
 * then still reports the old n_fgrams the table is inconsistent and must be
 * destroyed).
 */
#define SCONE_REBUILD_SCRATCH_BYTES (16u << 20)
/* A list size that always fits the scratch: since each rounding adds at most
 * 255 bytes, n = floor((SCONE_REBUILD_SCRATCH_BYTES - 768) / (4*K + 1)) satisfies
 * 256 + round256(n) + round256(4*K*n) <= SCONE_REBUILD_SCRATCH_BYTES, and the
 * exact limit exceeds it by fewer than 510 / (4*K + 1) + 1 f-grams. */
#define SCONE_REBUILD_MAX_FGRAMS(K) \
  ((int64_t)(((int64_t)SCONE_REBUILD_SCRATCH_BYTES - 768) / (4 * (int64_t)(K) + 1)))
int scone_table_rebuild_noalloc(scone_table* table, const int32_t* fgram_tok,
                                const uint8_t* fgram_len, int64_t n_fgrams, const scone_bf16* F,
                                void* stream);

/* Host-side description of a built table (sizes are in bytes). */
typedef struct scone_table_info {
  int64_t n_fgrams;
  int64_t n_slots;
  int64_t n_buckets;
  int32_t slot_bytes;        /* 16 or 32 */
  int32_t key_bits;          /* K * bits_per_token + 4 length bits */
  int32_t bits_per_token;
  int32_t K;
  int32_t vocab;
  int32_t d;
  int32_t F_location;
  int32_t max_insert_probe;  /* most cuckoo evictions any f-gram insert needed */
  int64_t table_bytes;       /* slot array */
  int64_t F_bytes;           /* n_fgrams * d * 2 (borrowed) */
  int64_t T_bytes;           /* vocab * d * 2 (borrowed) */
  int64_t n_markers;         /* marker slots of the suffix index (0 without one) */
  int32_t suffix_index;      /* 1: the table has a suffix index (see scone_table_build) */
} scone_table_info;

int scone_table_get_info(const scone_table* table, scone_table_info* info);

/*
 * Diagnostic: caps the buckets one lookup may read. A lookup normally reads
 * both candidate buckets (2, the default); with 1 it reads only the first,
 * and a key not found there makes the position an error position with
 * SCONE_ERR_PROBE_LIMIT recorded. max_buckets >= 1 (values above 2 act as 2).
 */
int scone_table_set_probe_limit(scone_table* table, int64_t max_buckets);

/* How scone_embed moves rows (a tuning knob; results are identical). scone_embed_varlen
   reads it too: REGISTERS keeps its register kernel, AUTO and PIPELINED take the walk
   over the suffix index where that applies, BULK and SPLIT act as REGISTERS there. So
   does scone_match: REGISTERS looks every length up, any other mode walks the lengths
   on a table with a suffix index. */
enum scone_copy_mode {
  SCONE_COPY_AUTO = 0,       /* the library picks per call: PIPELINED where it applies and the
                                table has a suffix index or 3 < K <= 5, REGISTERS otherwise */
  SCONE_COPY_REGISTERS = 1,  /* 16-byte loads and streaming stores through registers */
  SCONE_COPY_BULK = 2,       /* cp.async.bulk (TMA) through a shared-memory ring; needs rows of a
                                multiple of 16 bytes, 16-byte aligned F, T and out, and F in
                                device memory, else scone_embed returns SCONE_ERR_UNSUPPORTED */
  SCONE_COPY_SPLIT = 3,      /* register copies by warps that only copy, fed through a
                                shared-memory ring by warps that only match */
  SCONE_COPY_PIPELINED = 4   /* register copies with the next tile's match interleaved into
                                the current tile's copy (on a table with a suffix index the
                                match walks the lengths one bucket at a time); for 16-byte
                                slots, K <= 5 and 16-byte-aligned rows, else as
                                SCONE_COPY_REGISTERS */
};

int scone_table_set_copy_mode(scone_table* table, int32_t mode);

/*
 * scone_match — the selection step of Algorithm 1 (Sec. 3): for each
 * position, the length of the longest f-gram ending there and its row of F.
 * Probes lengths 2..min(K, i+1), i.e. at most K-1 lookups per token, the
 * bound Sec. 4.3 states ("up to four queries per token" for K = 5). On a
 * table with a suffix index and tokens in device memory the lengths are
 * walked in turn, stopping at the first absent or unextended window (fewer
 * lookups; see the copy modes).
 * Otherwise all lengths read their first buckets in one round trip, and the
 * lengths whose first bucket is full without the key, and that are longer
 * than the best first-round hit, read their second buckets in a second one.
 * Async.
 *
 *  tok  int32 [B * L]; row int32 [B * L] (F row, or -1 when T is used or on
 *  error); len uint8 [B * L] or NULL (n in 2..K for an f-gram, 1 for the
 *  token fallback, 0 for an error position). All three are device-accessible
 *  addresses: device memory, or host memory from scone_host_alloc, which the
 *  kernel then reads and writes over the host link. The latter is the
 *  training-time pre-scan of Appendix F (tag every corpus token with its
 *  longest matching length): a corpus too large for HBM is tagged in place.
 *  B * L may exceed 2^31.
 */
int scone_match(const scone_table* table, const int32_t* tok, int32_t B, int32_t L,
                int32_t* row, uint8_t* len, void* stream);

/*
 * scone_prescan — the training-time pre-scan of Appendix F (tag every token
 * of a corpus with its longest f-gram's length and row) for a corpus in host
 * memory, staged through HBM: chunks of whole sequences are copied in, tagged
 * by the match kernel (scone_match on device memory) and their tags copied
 * out, each on its own stream, so the host link carries bulk copies in both
 * directions while the kernel works on the chunk before. Same results as
 * scone_match on the host addresses.
 *
 *  tok        host int32 [B * L]; row host int32 [B * L]; len host uint8
 *             [B * L] or NULL. Pinned memory (scone_host_alloc or registered)
 *             lets the copies overlap; pageable memory works, more slowly.
 *  B, L       B sequences of L >= 1 tokens (B * L may exceed 2^31).
 *  chunk_tokens  tokens per chunk, rounded down to whole sequences (at least
 *             one); 0 selects 32 Mi. The first call on a table allocates two
 *             chunks of device buffers (9 bytes per token each, 5 without
 *             len) and three streams, which the table keeps (a later call
 *             with larger chunks, or with len after calls without it,
 *             reallocates them) and scone_table_destroy frees.
 *  stream     work queued on it before the call comes first; the call
 *             returns when the tags are in host memory (synchronous).
 *
 * Calls on one table must not overlap (they share its buffers). Device-
 * detected errors are recorded in the table's status word as for
 * scone_match. Errors: INVALID_ARG, NOMEM (the device buffers), CUDA.
 */
int scone_prescan(scone_table* table, const int32_t* tok, int64_t B, int32_t L, int32_t* row,
                  uint8_t* len, int64_t chunk_tokens, void* stream);

/*
 * scone_fgram_discover — constructs V_fgram from a corpus: Algorithm 3
 * ("Constructing a set of f-grams", Appendix A) by the K-1 counting scans of
 * Sec. 3.2. C_w is the number of windows equal to the n-gram w, n = 2..K,
 * over every sequence of the dense [B x L] corpus (windows never span two
 * sequences; overlapping windows count separately). Only n-grams with
 * C_w >= min_count are eligible (Sec. 3.2 uses 5; 1 gives Algorithm 3
 * exactly). The S eligible n-grams with the largest C_w are returned; ties
 * go to the shorter n-gram, then to the earlier first occurrence (start
 * position in the flattened corpus). The list is ordered by length, then by
 * first occurrence, so it can be passed to scone_table_build as is (f-gram
 * r gets row r). If fewer than S n-grams are eligible, all are returned.
 *
 *  ws           a workspace from scone_discover_create, or NULL. The call's
 *               device buffers (and a small pinned host area for its reads of
 *               counters) are taken from it and stay allocated there (grown as
 *               needed, never shrunk) until scone_discover_destroy, so
 *               repeated calls allocate nothing; with NULL they are
 *               allocated and freed inside the call.
 *  tok          int32 [B * L], device-accessible (device memory, or host
 *               memory from scone_host_alloc read over the host link);
 *               every token in [0, vocab). B * L <= 2^30.
 *  fgram_tok    int32 [S * K], padded with -1 after each n-gram's tokens;
 *  fgram_len    uint8 [S]; fgram_count uint32 [S] or NULL. Device-accessible
 *               (device or host-mapped); entries past *n_out are untouched.
 *  n_out        host; receives the number of f-grams written (<= S).
 *  stats        host or NULL; per length n (index n): windows counted after
 *               pruning, distinct n-grams among them, eligible n-grams,
 *               global table updates and the device time of each pass
 *               (binning, counting, flagging, whole scan); the count of the
 *               S-th f-gram and how many f-grams at that count were taken;
 *               the largest counting table allocated; the device time of
 *               the call.
 *
 * Synchronous: returns when the lists are written. Working memory: about
 * 15 bytes per token for K = 2, 19 for K = 3 and 23 for K >= 4 (binned
 * window records and the names of the previous scan), a counting table of
 * 64 bytes per distinct n-gram of the largest scan (see
 * scone_discover_set_table_slack), and the lists of eligible n-grams
 * (4 (n + 1) bytes each). Errors: SCONE_ERR_INVALID_ARG (K outside [2, 8],
 * min_count < 1, S < 0, null pointers), SCONE_ERR_UNSUPPORTED (B * L > 2^30),
 * SCONE_ERR_TOKEN_RANGE (a token outside [0, vocab); nothing is written),
 * SCONE_ERR_TABLE_FULL (a worst-case counting table filled up, which only a
 * corpus built to collide in the hash can cause), SCONE_ERR_NOMEM,
 * SCONE_ERR_CUDA.
 */
typedef struct scone_discover_stats {
  int64_t candidates[9];      /* windows counted in scan n (after pruning for n >= 3) */
  int64_t distinct[9];        /* distinct n-grams among them */
  int64_t frequent[9];        /* n-grams with count >= min_count */
  int64_t flushes[9];         /* global table updates of scan n: binned windows plus
                                 entries of the per-block hot-key caches */
  int64_t threshold;          /* count of the last-ranked selected f-gram; 0 when all taken */
  int64_t selected_at_threshold; /* f-grams taken at that count (0 when all taken) */
  int64_t table_bytes_max;    /* largest counting table of a scan */
  double ms_bin[9];           /* device time of scan n's binning pass (CUDA events) */
  double ms_count[9];         /* ... of its counting pass */
  double ms_flag[9];          /* ... of its flagging pass (lookups and names) */
  double ms_scan[9];          /* device time of the whole scan n */
  int64_t estimate[9];        /* sketch estimate of the distinct n-grams of scan n, which
                                 sizes its counting table */
  int64_t table_rebuilds;     /* scans whose table turned out too small for the estimate
                                 and were counted again in a worst-case table */
  double ms_select;           /* device time of the selection and the emission */
  double ms_total;            /* device time of the whole call, first launch to last */
  double ms_alloc_host;       /* host time spent in the call's allocations */
  int64_t workspace_bytes;    /* device bytes held by the workspace after the call */
} scone_discover_stats;

int scone_fgram_discover(scone_discover* ws, const int32_t* tok, int32_t B, int32_t L,
                         int32_t vocab, int32_t K, int64_t S, int32_t min_count,
                         int32_t* fgram_tok, uint8_t* fgram_len, uint32_t* fgram_count,
                         int64_t* n_out, scone_discover_stats* stats, void* stream);

/* An empty discovery workspace on the current device (no device memory yet). */
int scone_discover_create(scone_discover** out);
/* Frees the workspace and its device buffers (NULL is a no-op). */
int scone_discover_destroy(scone_discover* ws);
/*
 * Sizing of the counting tables of the calls that use ws: slots per
 * estimated distinct n-gram (default 4, i.e. load factor 0.25). Each scan
 * estimates its distinct n-grams with a HyperLogLog sketch (standard error
 * 1.6%) before it counts. A table that still fills up (probe sequences past
 * 4096 slots) is rebuilt at the worst-case size, two slots per counted
 * window, and the scan counted again: results never depend on the setting,
 * only memory and time do. Errors: SCONE_ERR_INVALID_ARG (ws NULL,
 * slots_per_key not in (0, 1e6]).
 */
int scone_discover_set_table_slack(scone_discover* ws, double slots_per_key);

/*
 * scone_embed_gather — the emission step of Algorithm 1 (Sec. 3): for each
 * of n_tok positions, out[t] = F[row[t]] if row[t] >= 0, else T[tok[t]]
 * (a zero row when tok[t] is out of range or row[t] >= n_fgrams, which also
 * sets the sticky status). tok, row device [n_tok]; out device [n_tok * d].
 * Async.
 */
int scone_embed_gather(const scone_table* table, const int32_t* tok, const int32_t* row,
                       int64_t n_tok, scone_bf16* out, void* stream);

/*
 * scone_embed — Algorithm 1 end to end (Sec. 3, inference branch) in one
 * launch: match and gather fused, no intermediate row array in memory.
 * tok int32 [B * L], device-accessible: device memory, or page-locked host
 * memory mapped for the device (cudaHostAlloc, cudaHostRegister,
 * scone_host_alloc), which the kernel then reads over the host link with no
 * staging copy; out device [B * L * d]; row / len as in scone_match, each
 * may be NULL. Async; host tokens must stay unchanged until the call's work
 * on the stream is done.
 */
int scone_embed(const scone_table* table, const int32_t* tok, int32_t B, int32_t L,
                scone_bf16* out, int32_t* row, uint8_t* len, void* stream);

/*
 * scone_embed_varlen — Algorithm 1 over a packed ragged batch, optionally
 * continuing sequences held in a decode state: chunked prefill, decode, and
 * batches that mix them in one launch. Async.
 *
 *  tok         device int32 [n_tok]: n_seq sequences packed back to back.
 *  cu_seqlens  device int32 [n_seq + 1]: sequence b is tok[cu[b] .. cu[b+1]);
 *              cu[0] = 0, nondecreasing, cu[n_seq] = n_tok (empty sequences
 *              allowed). Not checked on the host.
 *  state       NULL: every sequence starts at its first token (with equal
 *              lengths L this is scone_embed). Otherwise a decode state of the
 *              same table: sequence b continues slot seq_slot[b] (device int32
 *              [n_seq], distinct slots; NULL = slot b, then n_seq <= S). The
 *              slot's history (its last K-1 tokens so far) precedes the chunk,
 *              so windows reach back into it; after the launch the history is
 *              the last K-1 tokens of history ++ chunk. A slot outside [0, S)
 *              is a device-detected INVALID_ARG: zero rows, row -1, len 0.
 *  out, row, len  as in scone_embed, one entry per packed position.
 * n_tok <= 2^31 - 1.
 */
int scone_embed_varlen(const scone_table* table, const int32_t* tok, int64_t n_tok,
                       const int32_t* cu_seqlens, int32_t n_seq, scone_decode* state,
                       const int32_t* seq_slot, scone_bf16* out, int32_t* row, uint8_t* len,
                       void* stream);

/*
 * scone_gemm_bf16 — the tensor-core (tcgen05) GEMM behind the f-gram model's
 * dense layers (exported for testing): C = epilogue(A B^T) with A [M x K] and
 * B [N x K] bf16, row-major, K contiguous; fp32 accumulation. Epilogues:
 * SCONE_GEMM_STORE (C [M x N] = A B^T), SCONE_GEMM_RESIDUAL (C = R + A B^T,
 * R [M x N], C may equal R), SCONE_GEMM_SWIGLU (C [M x N/2]: in every group of
 * 32 columns of A B^T, the first 16 are gates g and the next 16 ups u of 16
 * consecutive outputs, C = silu(g) u). N must be a multiple of 256, K of 64,
 * all pointers device memory aligned to 16 bytes. status: device int that
 * receives SCONE_ERR_CUDA if a pipeline wait timed out (left untouched
 * otherwise). Async.
 */
enum scone_gemm_epilogue { SCONE_GEMM_STORE = 0, SCONE_GEMM_RESIDUAL = 1, SCONE_GEMM_SWIGLU = 2 };
int scone_gemm_bf16(const scone_bf16* A, const scone_bf16* B, const scone_bf16* R, scone_bf16* C,
                    int32_t M, int32_t N, int32_t K, int32_t epilogue, int* status, void* stream);
/* The same with the kernel chosen (for tests and measurements): variant 0 =
 * default, 1 = one SM per 128 x 256 tile, 2 = pairs of SMs per 256 x 256 tile
 * (a 2-CTA cluster, tcgen05 cta_group::2). */
int scone_gemm_bf16_variant(const scone_bf16* A, const scone_bf16* B, const scone_bf16* R,
                            scone_bf16* C, int32_t M, int32_t N, int32_t K, int32_t epilogue,
                            int32_t variant, int* status, void* stream);

/*
 * Precomputing F with the f-gram model (Sec. 3.2: after training F is
 * precomputed and stored; Algorithm 1 embeds an f-gram by A_fgram(T(s_j), ..,
 * T(s_i)) in training). The model is a pre-LN transformer over the f-gram's
 * token rows plus absolute position embeddings: x_0[j] = T(s_j) + P[j],
 * j = 0..n-1 from the f-gram's first token (Appendix F, Implementation
 * Details: an absolute position embedding layer whose size is the longest
 * f-gram). Per layer h = x + Attn(LN(x)), x = h + MLP(LN(h)); LN is the
 * non-parametric layer norm (eps 1e-5); Attn is causal multi-head attention
 * scaled by 1/sqrt(hd); MLP is SwiGLU. F(w) = LN of the last position's final
 * state. A model created with SCONE_FGRAM_POS_ROTARY has no P and applies
 * rotary embeddings to q and k instead (rotate-half pairs (i, i + hd/2),
 * angle pos * 10000^(-2i/hd)); that option is not the paper's scheme.
 *
 * scone_fgram_model_create: d (multiple of 256, d/256 a power of two up to
 * 16), n_heads (head size d/n_heads in {64, 128, 256}), ffw (multiple of 128),
 * n_layers, max_pos (rows of P, 1..8; ignored for rotary), position;
 * weights: device bf16, packed per layer as qkv [3d x d] (query, key, value
 * rows), o [d x d], gu [2 ffw x d] (rows 32g..32g+15 are the gates of
 * features 16g..16g+15, the next 16 rows their ups), down [d x ffw],
 * row-major, followed (absolute positions) by P [max_pos x d]; borrowed, must
 * outlive the model. batch: f-grams per internal batch (0 = 16384); the
 * workspace grows with the tokens of a batch. Synchronous.
 */
enum scone_fgram_position { SCONE_FGRAM_POS_ABSOLUTE = 0, SCONE_FGRAM_POS_ROTARY = 1 };
typedef struct scone_fgram_model scone_fgram_model;
int scone_fgram_model_create(int32_t d, int32_t n_heads, int32_t ffw, int32_t n_layers,
                             int32_t max_pos, int32_t position, const scone_bf16* weights,
                             int64_t batch, scone_fgram_model** out);
int scone_fgram_model_destroy(scone_fgram_model* model);

/*
 * scone_fgram_precompute: F rows of n f-grams. fgram_tok device int32 [n * K]
 * (f-gram r's tokens first, padding ignored), fgram_len device uint8 [n] in
 * [2, K] (lengths outside [1, K] are read as 1 and reported), T device
 * [vocab * d], F device or host-mapped [n * d] (16-byte aligned). The f-grams
 * of a batch are packed without padding and every dense layer is a
 * tensor-core GEMM over all their tokens (f-grams are not padded: with the
 * padding of Appendix F after the last token and causal attention, the last
 * token's output is the same). K above max_pos (absolute positions) is
 * INVALID_ARG before any device work. Synchronous; returns SCONE_OK or the
 * first device-detected error (TOKEN_RANGE: that token's input row is zero;
 * INVALID_ARG: a length outside [1, K]; CUDA: a GEMM pipeline timed out).
 */
int scone_fgram_precompute(scone_fgram_model* model, const int32_t* fgram_tok,
                           const uint8_t* fgram_len, int64_t n, int32_t K, const scone_bf16* T,
                           int32_t vocab, scone_bf16* F, void* stream);

/*
 * Row store: F in a file, beyond host memory (the paper's storage tier:
 * f-gram embeddings on solid-state drives, Sec. 4.3). The file holds F row
 * after row (n_rows x d bf16, no header). The store caches rows in HBM
 * (cache_rows slots, direct-mapped by row id); a gather copies hits from the
 * cache, reads misses from the file (pread on `threads` reader threads, 0 =
 * one per core; O_DIRECT when a row is a multiple of 4 KiB) and fills the
 * cache with them.
 *
 * scone_rowstore_open: d a multiple of 8; the file must hold n_rows rows.
 * Synchronous. scone_rowstore_gather: out[t] = F[row[t]] (row[t] >= 0) or
 * T[tok[t]] (row[t] < 0, T from the table, whose d must equal the store's);
 * row as written by scone_match, scone_embed_varlen or scone_decode_step;
 * tok, row device [n]; out device [n * d], 16-byte aligned. A table used only
 * to select rows for a store (scone_match, or scone_decode_step with out =
 * NULL) never reads its F, and may be built with a placeholder F of one row;
 * the calls that copy f-gram rows (scone_embed, scone_embed_gather,
 * scone_embed_varlen, scone_decode_step with out) need the full F. Synchronous (the
 * host reads the misses). A row id >= n_rows or a token outside the vocab is
 * a device-detected error (zero row, sticky table status); a failed read
 * returns SCONE_ERR_CUDA.
 */
typedef struct scone_rowstore scone_rowstore;
typedef struct scone_rowstore_stats {
  int64_t positions;   /* positions gathered since open */
  int64_t misses;      /* positions whose row was not in the cache */
  int64_t rows_read;   /* distinct rows read from the file */
  int64_t bytes_read;
  int32_t direct_io;   /* 1 if the file is read with O_DIRECT */
} scone_rowstore_stats;
int scone_rowstore_open(const char* path, int64_t n_rows, int32_t d, int64_t cache_rows,
                        int32_t threads, scone_rowstore** out);
int scone_rowstore_gather(scone_rowstore* store, const scone_table* table, const int32_t* tok,
                          const int32_t* row, int64_t n, scone_bf16* out, void* stream);
int scone_rowstore_get_stats(const scone_rowstore* store, scone_rowstore_stats* out);
int scone_rowstore_close(scone_rowstore* store);
/*
 * scone_rowstore_probe_reads — the storage device's own rate for this store:
 * n_reads rows drawn uniformly (a counter hash of `seed`) from the store's
 * file, read with the store's reader threads and I/O mode (O_DIRECT where the
 * gather uses it) into host buffers that are then discarded; no GPU work and
 * no cache involvement. *rows_per_s and *bytes_per_s receive the rates over
 * the host's steady clock. The roofline of the storage tier (Sec. 4.3: F on
 * solid-state drives, one read per missed row). Synchronous; a failed read
 * returns SCONE_ERR_CUDA, a failed buffer allocation SCONE_ERR_NOMEM.
 */
int scone_rowstore_probe_reads(scone_rowstore* store, int64_t n_reads, uint64_t seed,
                               double* rows_per_s, double* bytes_per_s);

/*
 * Decode (Sec. 3.2: T stays on the accelerator "for decoding", F is looked
 * up per generated token). A decode state holds, per live sequence, its last
 * K-1 tokens on the device, which is all Algorithm 1 needs for the next
 * position.
 *
 * scone_decode_create: S live sequences. hist host int32 [S * (K-1)]: the
 * sequence's known tokens right-aligned in its row (entries left of the last
 * hist_len[s] are ignored); hist_len host int32 [S] in [0, K-1]. Synchronous.
 */
int scone_decode_create(const scone_table* table, int32_t S, const int32_t* hist,
                        const int32_t* hist_len, scone_decode** out);

/*
 * scone_decode_step: appends new_tok[s] (int32 [S], device memory or
 * page-locked host memory mapped for the device, which the kernel then reads
 * over the host link) to sequence s, embeds it by Algorithm 1 over the
 * sequence so far, and writes out device [S * d]; row device int32 [S] and
 * len device uint8 [S] may be NULL. out may be NULL when row is given: the
 * step then only selects (for rows gathered from a row store,
 * scone_rowstore_gather). Async; steps on one state must be ordered on one
 * stream, and host tokens must stay unchanged until the step is done.
 */
int scone_decode_step(scone_decode* state, const int32_t* new_tok, scone_bf16* out, int32_t* row,
                      uint8_t* len, void* stream);

/* Copies the device history back: hist host [S * (K-1)], hist_len host [S]. Synchronous. */
int scone_decode_get_history(const scone_decode* state, int32_t* hist, int32_t* hist_len);

int scone_decode_destroy(scone_decode* state);

/*
 * scone_status: synchronizes `stream`, returns the first device-detected
 * error recorded since the last call (SCONE_OK if none) and clears it. The
 * kernel that records an error also writes it to a host-mapped word of the
 * table, so when no error was recorded the call is the sync and one read of
 * host memory; after an error it clears that word and launches one 1-thread
 * kernel that moves the status word to the host and clears it. An error that
 * a kernel on another stream records during the call is returned by the next
 * call. Calls on one table must not overlap.
 */
int scone_status(const scone_table* table, void* stream);

/*
 * Host memory for the offloaded tier: pinned and mapped into the device
 * address space, so kernels read it over the host link. Use it for F with
 * SCONE_ROWS_HOST_MAPPED. Where the OS offers transparent huge pages the
 * buffer is a huge-page-aligned anonymous mapping advised MADV_HUGEPAGE,
 * touched, then registered (cudaHostRegister, Mapped | Portable): scattered
 * row reads over tens of GB then need far fewer GPU address translations
 * (measured on GB300: 2x the random-row read rate of cudaHostAlloc memory at
 * 82 GB). Otherwise it is cudaHostAlloc(Mapped | Portable). The contents
 * start as zeros only in the first case. Synchronous. Errors: INVALID_ARG
 * (bytes < 1 or out NULL), NOMEM (no pinned allocation succeeded; *out is NULL).
 */
int scone_host_alloc(int64_t bytes, void** out);

/* Frees memory from scone_host_alloc (after a device synchronize). NULL is a no-op. */
int scone_host_free(void* p);

/* Static description of an error code. */
const char* scone_strerror(int code);

/* ABI version, (major << 16) | minor. */
int scone_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SCONE_H_ */
