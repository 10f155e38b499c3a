/*
 * kvg.h — C ABI of libkvg: byte-exact KV-state graft and GQA decode attention
 * on one GB300 (sm_103a).
 *
 * The operations follow the problem statement of "Byte-Exact KV-State
 * Grafting" (arxiv 2607.14431):
 *   - deposit: a computed KV state is captured once, with its positions, as a
 *     persistent block (Sec. 3.3, deposit step of the flywheel; Sec. 4.4);
 *   - graft: the block is installed into a fresh context at the positions it
 *     was captured at, [0, N), and new queries are computed on top at
 *     [N, N+q) (Sec. 3.2, "position consistency");
 *   - relocate: optionally the block is re-based to another absolute offset,
 *     which re-rotates its keys and is not byte-exact (Sec. 4.2);
 *   - decode: attention of a new query over the grafted context (Sec. 3.2,
 *     Sec. 4.3);
 *   - digest: SHA-256 of raw bytes, the paper's byte-exactness test (Sec. 3.2)
 *     and its per-block integrity check (Sec. 4.11).
 *
 * Conventions for every call:
 *   - No exceptions cross the ABI and nothing aborts the process: each call
 *     returns a kvg_status.  Arguments are checked on the host before any GPU
 *     work is enqueued; a call that fails a host check changes no state.
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *     stream).  GPU work is enqueued on it and the call returns without
 *     waiting unless a flag asks for it.  Errors that only the GPU can see
 *     (a digest mismatch, a failed device-side bounds check) are recorded in
 *     the cache's device status word and reported by kvg_sync().
 *   - Element types: inputs and outputs (k, v, q, out) are bf16 (raw 16-bit
 *     patterns); a cache and its blocks hold bf16 or, when kvg_dims.kv_dtype
 *     asks for it, fp8 E4M3 codes.  Sizes are in elements unless a name ends
 *     in _bytes.
 *   - Ownership: stores, caches and their device memory belong to the
 *     library; buffers passed in (k, v, q, out, positions) belong to the
 *     caller and must stay valid until the enqueued work completes.
 *   - Threads: a store or cache must not be used from two host threads at
 *     once.  Different caches are independent.
 */
#ifndef KVG_H
#define KVG_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum kvg_status {
    KVG_OK = 0,
    KVG_ERR_ARG = -1,          /* bad argument or unsupported geometry */
    KVG_ERR_OOM = -2,          /* device or pinned-host allocation failed */
    KVG_ERR_CUDA = -3,         /* a CUDA runtime call failed */
    KVG_ERR_NOT_FOUND = -4,    /* no such block id */
    KVG_ERR_CAPACITY = -5,     /* not enough free pages, slots or store bytes */
    KVG_ERR_POSITION = -6,     /* position tag + delta outside [0, 2^31) */
    KVG_ERR_DIGEST = -7,       /* a page digest did not match the stored one */
    KVG_ERR_FORMAT = -8,       /* serialized block header or layout invalid */
    KVG_ERR_TIMEOUT = -9,      /* kvg_sync gave up waiting */
    KVG_ERR_DEVICE_CHECK = -10 /* a kernel's own bounds/wait check failed */
} kvg_status;

enum { KVG_RESIDENCY_HBM = 0, KVG_RESIDENCY_PINNED_HOST = 1, KVG_RESIDENCY_CACHE_POOL = 2 };
enum { KVG_ROPE_HALF = 0, KVG_ROPE_INTERLEAVED = 1 };
enum { KVG_GRAFT_VERIFY = 1u, KVG_GRAFT_SYNC = 2u };
enum { KVG_SHA256_PLAIN = 0, KVG_SHA256_PAGED = 1 };
enum { KVG_DECODE_MERGE = 1u };
/* KV element types (kvg_dims.kv_dtype). */
enum { KVG_KV_BF16 = 0, KVG_KV_E4M3 = 1 };

/* Leaf size of the two-level page digest (bytes). */
#define KVG_DIGEST_LEAF_BYTES 4096
/* Most page indices a graft report lists. */
#define KVG_REPORT_MAX_PAGES 64

/* KV geometry shared by a store and the caches it grafts into.
 * A page holds page_size consecutive token slots of every KV head:
 * [n_kv_heads][page_size][head_dim] elements per layer and per K or V, so
 * page_bytes = elem_bytes * n_kv_heads * page_size * head_dim.
 * Supported: head_dim in {64, 128, 256}; page_size >= 1; page_bytes a
 * multiple of 16.  rope_theta / rope_style only matter for relocation:
 * the rotation pairs dimension i with i + head_dim/2 (KVG_ROPE_HALF) or
 * 2i with 2i+1 (KVG_ROPE_INTERLEAVED) at frequency rope_theta^(-2i/head_dim).
 * Element type (quantized KV blocks: a block's size depends on the cache's
 * quantization, Sec. 4.4):
 *   KVG_KV_BF16 (0): bf16, elem_bytes 2; k_scale, v_scale ignored.
 *   KVG_KV_E4M3 (1): fp8 E4M3 codes, elem_bytes 1, with per-tensor fp32
 *     scales (finite, > 0): a K element is its code's value * k_scale, a V
 *     element * v_scale.  Appends quantize bf16 input: the fp32 value times
 *     r = fp32(1 / scale) (IEEE fp32 division, then one fp32 product),
 *     rounded to nearest-even on the E4M3 grid, saturating at +-448.
 *     Relocation (delta != 0) is not supported; decode needs head_dim 128 or
 *     256.  Blocks carry the scales; a block grafts only into a cache with
 *     the same element type and scales. */
typedef struct kvg_dims {
    int32_t n_layers;
    int32_t n_kv_heads;
    int32_t head_dim;
    int32_t page_size;
    double rope_theta;
    int32_t rope_style;
    int32_t kv_dtype;
    float k_scale;
    float v_scale;
} kvg_dims;

typedef struct kvg_store kvg_store;
typedef struct kvg_cache kvg_cache;

/* ---------------------------------------------------------------- store -- */

/* A store holds serialized blocks (the paper's persistent artifacts, Sec. 3.3,
 * Sec. 4.4) in HBM or in pinned host memory, up to capacity_bytes.  Block ids
 * are 0, 1, 2, ... in deposit/import order.  Pinned-host stores are carved
 * from 1 GiB (or larger, for larger blocks) page-locked slabs allocated on
 * demand; a block never straddles two slabs.
 * device: CUDA ordinal used for HBM stores and for the store's kernels. */
kvg_status kvg_store_create(const kvg_dims *dims, int32_t residency, uint64_t capacity_bytes,
                            int32_t device, kvg_store **out);
void kvg_store_destroy(kvg_store *store);

/* A store whose blocks live inside `cache`'s own page pool (residency
 * KVG_RESIDENCY_CACHE_POOL), for a zero-copy graft.  A deposit copies the rows
 * into pool pages that the block owns from then on (taken from the cache's
 * free list for good); an own-position graft then writes only the sequence's
 * page-table entries, fills and position tags, pointing at the block's full
 * pages (shared and read-only: appends never write a full page), and copies a
 * partially filled last page into a page of the sequence, which its appends
 * fill.  A release never frees a block's pages.  Deposits and grafts must use
 * this cache; relocation (delta != 0) needs a copying store (KVG_ERR_ARG);
 * blocks have at most 1024 pages.  capacity_bytes bounds the blocks'
 * metadata (header, position tags, digests, page ids) kept in HBM.
 * kvg_store_block_info's `bytes` points at that metadata; export, save and
 * import produce and accept the same serialized bytes as other stores.
 * Destroy such a store before its cache; its pages return to the free list
 * unless a sequence still points at them. */
kvg_status kvg_store_create_in_cache(kvg_cache *cache, uint64_t capacity_bytes, kvg_store **out);

/* Serialized block layout (little-endian), one contiguous region:
 *   [0, 256)      header: magic "KVGBLK01", u32 version = 1, u32 header bytes
 *                 = 256, i32 n_layers, n_kv_heads, head_dim, page_size,
 *                 i64 n_tokens, i64 n_pages, f64 rope_theta, i32 rope_style,
 *                 i32 dtype (1 = bf16, 2 = E4M3), u64 positions_offset,
 *                 digests_offset, pages_offset, total_bytes; at byte 96 the
 *                 32-byte block digest; for E4M3 the fp32 k_scale and v_scale
 *                 at bytes 128 and 132; the rest zero.
 *   positions     int32 [n_tokens] position tags (offset 256)
 *   digests       [n_layers][2][n_pages][32] page digests (256-aligned)
 *   pages         bf16 (or E4M3 codes)
 *                 [n_layers][2][n_pages][n_kv_heads][page_size][head_dim]
 *                 (4096-aligned), kv 0 = K, 1 = V; token t of the block is row
 *                 t % page_size of page t / page_size; rows past n_tokens in
 *                 the last page are zero.
 * Page digest = SHA-256 over the concatenated SHA-256 digests of the page's
 * consecutive 4096-byte leaves (the last leaf may be shorter).  Block digest =
 * SHA-256 over the position tags (int32 LE) followed by all page digests. */
typedef struct kvg_block_info {
    int64_t n_tokens;
    int64_t n_pages;           /* pages per layer per K/V */
    int32_t residency;
    int32_t reserved;
    const void *bytes;         /* device pointer (HBM store) or host pointer */
    uint64_t total_bytes;
    uint64_t positions_offset;
    uint64_t digests_offset;
    uint64_t pages_offset;
    uint8_t block_digest[32];  /* read back from the block header (synchronous) */
} kvg_block_info;

/* Describes block `block_id`.  Synchronizes the device (it reads the header
 * the deposit kernels wrote).  KVG_ERR_NOT_FOUND for an unknown id. */
kvg_status kvg_store_block_info(kvg_store *store, uint64_t block_id, kvg_block_info *out);

/* Copies a serialized block (host memory, e.g. read from a block file) into
 * the store.  The header is validated against the store's geometry
 * (KVG_ERR_FORMAT); with KVG_GRAFT_VERIFY every page digest and the block
 * digest are recomputed on the GPU and compared (KVG_ERR_DIGEST; the block is
 * then not added).  Synchronous.  This is how a block file moves between
 * machines (Sec. 4.11). */
kvg_status kvg_store_import(kvg_store *store, const void *bytes, uint64_t n_bytes, uint32_t flags,
                            uint64_t *block_id_out);

/* Copies block `block_id`'s serialized bytes to host memory `dst` (capacity
 * dst_bytes >= total_bytes).  Synchronous. */
kvg_status kvg_store_export(kvg_store *store, uint64_t block_id, void *dst, uint64_t dst_bytes);

/* Writes block `block_id` to the file `path` in the serialized layout above:
 * one plain file per block, the paper's persistent medium (Sec. 4.4) that is
 * copied between machines as is (Sec. 4.11).  Synchronous; KVG_ERR_ARG if the
 * file cannot be written.  An HBM store's block passes through two of the
 * store's pinned 16 MiB bounce buffers (allocated by its first file transfer
 * and kept until kvg_store_destroy), the next chunk's copy to the host
 * overlapping the current chunk's write. */
kvg_status kvg_store_save(kvg_store *store, uint64_t block_id, const char *path);

/* Reads a block file into the store, validating it like kvg_store_import;
 * with KVG_GRAFT_VERIFY every page digest and the block digest are recomputed
 * on the GPU and compared (KVG_ERR_DIGEST: the block is not added and its
 * space is given back).  KVG_ERR_FORMAT for a short or malformed file.
 * Synchronous.  The file is read in 16 MiB chunks by up to 8 threads: into a
 * pinned-host store directly, into an HBM store through the store's pinned
 * bounce buffers, each chunk's copy to HBM overlapping the next reads. */
kvg_status kvg_store_load(kvg_store *store, const char *path, uint32_t flags, uint64_t *block_id_out);

/* Readies a pinned-host store's block for a later graft (Sec. 4.4's restore
 * from a deep store, where the next block to restore is known ahead): enqueues
 * on `stream` one 4-byte read per host page of the block, which makes the GPU
 * resolve the address translations of all its pages.  A graft reads a block
 * at the host link's rate only when they are resolved; the GPU keeps those of
 * the last several GB of host memory it touched, so a graft of a block not
 * read recently otherwise takes up to about three times as long.  Issue it
 * on a stream other than the graft's while the previous graft runs (one
 * small read per host page).  No effect on HBM and cache-pool stores.
 * Errors: KVG_ERR_ARG (null store), KVG_ERR_NOT_FOUND. */
kvg_status kvg_store_prefetch(kvg_store *store, uint64_t block_id, void *stream);

/* ---------------------------------------------------------------- cache -- */

/* A paged KV cache on `device`: the "fresh inference context" a block is
 * installed into (Sec. 3.2: a fresh process or serving slot whose live
 * context holds the restored prefix at [0, N); Sec. 3.3: the serving side of
 * the deposit/graft cycle).  Pool of elements (bf16, or E4M3 codes for an
 * fp8 cache) [n_layers][2][n_pages][n_kv_heads][page_size][head_dim] (one
 * page id names the same token rows in every layer), and per sequence a page table, per-page fill counts, position tags
 * per slot and a slot high-water mark.  The pool is not initialised.
 * Free pages are handed out from the front of an ordered free list,
 * initially 0, 1, ..., n_pages-1; a released sequence's pages go to its back
 * in page-table order.  max_slots bounds one sequence's slots.  The first
 * cache created on a device also makes the 16 MiB static scratch of
 * kvg_decode_attention_noalloc resident there (KVG_ERR_CUDA if that fails). */
kvg_status kvg_cache_create(const kvg_dims *dims, int32_t n_pages, int32_t max_seqs,
                            int32_t max_slots, int32_t device, kvg_cache **out);
void kvg_cache_destroy(kvg_cache *cache);

/* Replaces the free-list order by the permutation order[0..n_pages).  Only
 * while every page is free (KVG_ERR_ARG otherwise).  Physical placement never
 * changes any result: attention reduces in logical token order. */
kvg_status kvg_cache_set_free_order(kvg_cache *cache, const int32_t *order, int32_t n_pages);

/* Sliding-window layers over a full-size cache (Sec. 4.3: a sliding-window
 * model resumes exactly from a restored block once its windowed layers keep
 * full-size KV).  Every layer keeps every row, so deposits and grafts stay
 * byte-exact; decode attention on layer l reads only the last windows[l]
 * valid rows of each sequence (counted back over its pages' fills, so the
 * window spans an unfilled tail of a page left by a page-aligned graft), or
 * every row when windows[l] == 0.  With consecutive position tags over the
 * valid rows, as after an own-position graft followed by appends, this is the
 * usual window over positions (query position q sees keys q-W+1 .. q, its
 * own row appended before the decode).
 * windows: host array of n_layers values >= 0; n == 0 (windows ignored)
 * resets every layer to 0.  Takes effect for later decode calls; changes no
 * cache contents.  Errors: KVG_ERR_ARG (n not 0 or n_layers, a negative
 * window). */
kvg_status kvg_cache_set_layer_windows(kvg_cache *cache, const int32_t *windows, int32_t n);

/* Device-side layout, for inspection and for interop with other kernels. */
typedef struct kvg_cache_view {
    void *pool;            /* elements [L][2][n_pages][Hkv][P][D] (bf16 or E4M3 codes) */
    int32_t *page_table;   /* int32 [max_seqs][max_pages], -1 = no page */
    int32_t *page_fill;    /* int32 [max_seqs][max_pages], valid rows (a prefix) */
    int32_t *positions;    /* int32 [max_seqs][max_slots], -1 = unwritten */
    uint64_t pool_bytes;
    uint64_t page_bytes;
    int32_t n_pages;
    int32_t max_seqs;
    int32_t max_slots;
    int32_t max_pages;     /* ceil(max_slots / page_size) */
} kvg_cache_view;
kvg_status kvg_cache_view_get(const kvg_cache *cache, kvg_cache_view *out);

/* Host-side bookkeeping of sequence `seq`: slot high-water mark and pages held. */
kvg_status kvg_cache_seq_info(const kvg_cache *cache, int32_t seq, int32_t *n_slots,
                              int32_t *n_pages);

/* Fresh write (the "fresh" arm the graft must reproduce, Sec. 3.2): rows
 * t = 0..n-1 of k and v (device, bf16 [n_layers][n][n_kv_heads][head_dim],
 * post-RoPE as a prefill produced them) and positions (device int32 [n]) go
 * to slots s = n_slots + t of `seq`, allocating pages as needed.
 * KVG_ERR_CAPACITY if slots or pages run out (nothing is written). */
kvg_status kvg_cache_append(kvg_cache *cache, int32_t seq, const void *k, const void *v,
                            const int32_t *positions, int32_t n, void *stream);

/* Decode-step append: one new row per sequence for B sequences in one
 * launch.  Row b of k and v (device, bf16 [n_layers][B][n_kv_heads]
 * [head_dim]) and positions[b] (device int32 [B]) go to slot n_slots of
 * sequence seq_ids[b] (host array, distinct ids, B <= 256), allocating a page
 * where a sequence's last page is full.  KVG_ERR_CAPACITY if slots or pages
 * run out (nothing is written); KVG_ERR_ARG on repeated ids. */
kvg_status kvg_cache_append_batch(kvg_cache *cache, const int32_t *seq_ids, int32_t B, const void *k,
                                  const void *v, const int32_t *positions, void *stream);

/* Returns the sequence's pages to the free list and clears its page table,
 * fills and position tags: the serving slot is empty again, ready for the
 * next graft into a fresh context (Sec. 3.2; Sec. 4.4, where the movable
 * window swaps which block is resident in the live prefix).  Enqueued on
 * `stream`; the host bookkeeping changes at once, so the next graft or
 * append may be given these pages: work on other streams that still reads
 * them must be ordered before that call's stream (an event), as on one
 * stream it is by itself. */
kvg_status kvg_cache_release(kvg_cache *cache, int32_t seq, void *stream);

/* ----------------------------------------------------------- deposit -- */

/* Captures slots [slot0, slot0+n) of `seq` (slot0 a multiple of page_size,
 * slot0 + n <= n_slots) with their position tags into a new block of `store`
 * (layout above), computing every page digest and the block digest on the
 * GPU.  Sec. 3.3 deposit; the block is byte-identical to one built from the
 * same rows anywhere else.  KVG_ERR_CAPACITY if the store is full.
 * Ordering: the call returns once the rows are gathered (it reads the
 * position tags back to bound later relocations).  The page digests follow
 * on `stream`, so work enqueued later on `stream` (a graft, a verification)
 * sees the whole block but its block digest, which one serial SHA-256 chain
 * computes on a library stream; kvg_store_block_info, kvg_store_export and
 * kvg_store_save wait for it.  A pinned-host store's block is assembled and
 * hashed in an HBM staging buffer (grown to the largest block deposited into
 * that store) and copied out: everything but the 256-byte header in `stream`
 * order, the header after the block digest. */
kvg_status kvg_deposit(kvg_store *store, const kvg_cache *cache, int32_t seq, int32_t slot0,
                       int32_t n, void *stream, uint64_t *block_id_out);

/* -------------------------------------------------------------- graft -- */

typedef struct kvg_graft_report {
    int32_t seq;
    int32_t n_pages_checked;   /* pages hashed (L * 2 * n_pages) */
    int32_t n_mismatch;        /* pages whose digest differed */
    int32_t n_listed;
    int32_t mismatch_pages[KVG_REPORT_MAX_PAGES]; /* index (l * 2 + kv) * n_pages + j */
} kvg_graft_report;

/* Own-position graft (Sec. 3.2): installs block `block_id` into sequence
 * `seq` at slot dst_slot, which must be the sequence's next page boundary
 * (ceil(n_slots / page_size) * page_size; pass -1 for that).  The block's
 * pages are copied whole into freshly allocated cache pages, its position
 * tags are written to the slots, and n_slots becomes dst_slot + n_tokens.
 * The graft is a byte copy: restored rows equal the deposited rows bit for
 * bit, so attention over them equals attention over the same rows written
 * fresh.
 * delta != 0 re-bases the block (Sec. 4.2): position tags become tag + delta,
 * and each valid key row is rotated by delta positions (fp32 arithmetic on a
 * host-fp64 cos/sin table, rounded to bf16 RNE); value rows and padding rows
 * are copied unchanged.  delta == 0 is the pure copy.
 * Blocks of a pinned-host store are read by the GPU directly from host memory.
 * flags: KVG_GRAFT_VERIFY hashes every page the graft read and compares with
 * the stored digests.  With delta == 0 this is one pass: each 4 KiB leaf is
 * read from the store once, written to its cache page and hashed from the same
 * registers, so the digest covers exactly the restored bytes; with delta != 0
 * the store's pages are hashed after the copy.  Verifying calls on one cache
 * (this flag, kvg_verify) share its leaf-digest scratch, so they must not run
 * concurrently on different streams.  KVG_GRAFT_SYNC waits for completion, fills `report`
 * (nullable) and returns KVG_ERR_DIGEST on a mismatch.  Without SYNC a
 * mismatch surfaces at the next kvg_sync().
 * Errors (no state change): KVG_ERR_NOT_FOUND, KVG_ERR_ARG (geometry or
 * dst_slot), KVG_ERR_CAPACITY (pages or slots), KVG_ERR_POSITION. */
kvg_status kvg_graft(kvg_store *store, uint64_t block_id, kvg_cache *cache, int32_t seq,
                     int32_t dst_slot, int64_t delta, uint32_t flags, void *stream,
                     kvg_graft_report *report);

/* kvg_graft with a completion event per chunk of the copy, for a caller that
 * works on the restored rows while the rest of the block is still being
 * copied (Sec. 4.4's restore: a split decode over each chunk's slots with
 * kvg_decode_attention_range while the next chunk crosses the host link).
 * Same arguments, checks, effects and errors as kvg_graft, plus:
 * events: host array of max_events (>= 1) caller-created CUDA events
 * (cudaEvent_t, on the cache's device; timing may be disabled).  The graft
 * copies the block in page-range chunks (one chunk for most HBM-store
 * blocks; up to 16 for a verified graft from a pinned-host store, the last
 * two short); chunk k of C maps to event k * E / C with E = min(max_events,
 * C).  On KVG_OK, *n_chunks = E, and for j < E events[j] is recorded on
 * `stream` once every chunk that maps to j has its rows (all layers, K and V)
 * and position tags in the cache; chunk_end_slot[j] (host array of at least
 * E) is the slot just past those rows, so event j covers slots
 * [dst_slot, chunk_end_slot[j]) and chunk_end_slot[E - 1] = dst_slot +
 * n_tokens.  An event does not wait for the digest check (KVG_GRAFT_VERIFY):
 * that verdict covers the whole block and is known only when all of the
 * call's work on `stream` is done (KVG_GRAFT_SYNC, or kvg_sync), so work
 * started from an event must not publish its result before then.
 * KVG_ERR_ARG if events, chunk_end_slot or n_chunks is null, an event is
 * null, or max_events < 1. */
kvg_status kvg_graft_chunked(kvg_store *store, uint64_t block_id, kvg_cache *cache, int32_t seq,
                             int32_t dst_slot, int64_t delta, uint32_t flags, void *stream,
                             kvg_graft_report *report, void *const *events, int32_t max_events,
                             int32_t *chunk_end_slot, int32_t *n_chunks);

/* A batch of grafts in one call: graft i installs block block_ids[i] into
 * sequence seq_ids[i] at that sequence's next page boundary, in order,
 * exactly as n kvg_graft calls with delta = deltas[i] would (a sequence may
 * appear several times: its blocks land one after another, each
 * page-aligned).  deltas: host array of n, or NULL for own-position grafts
 * throughout (Sec. 3.2).  A nonzero delta re-bases that graft (Sec. 4.2):
 * position tags + delta, keys rotated with the same fp32 cos/sin and the
 * same operation order as kvg_graft, so the restored bytes equal those of a
 * kvg_graft with that delta.  With deltas equal to the tokens already in the
 * sequence, a sequence's blocks get consecutive position tags (the
 * sequential composition of Sec. 4.8 at the KV level).  The page copies of
 * all grafts run as one launch, so the GPU stays full across graft
 * boundaries.  block_ids, seq_ids: host arrays of n (1 <= n <= 4096); each
 * block at most 1,024 pages per (layer, K/V).  Every argument, capacity,
 * page count and position range is checked first: on an error nothing is
 * grafted (KVG_ERR_POSITION when tags + delta leave [0, 2^31), KVG_ERR_ARG
 * for a nonzero delta on an fp8 cache).  Not for pool-resident stores
 * (KVG_ERR_ARG; use kvg_graft).  flags as for kvg_graft: KVG_GRAFT_VERIFY
 * hashes each own-position graft's restored pages, and each re-based
 * graft's stored pages, after the copies; the report's seq is the (last)
 * failing graft's sequence and mismatch_pages its block page indices.  The
 * call stages its job table in library-owned pinned memory and waits for
 * the previous batch's table copy on this cache before reusing it. */
kvg_status kvg_graft_batch(kvg_store *store, const uint64_t *block_ids, kvg_cache *cache, const int32_t *seq_ids,
                           const int64_t *deltas, int32_t n, uint32_t flags, void *stream,
                           kvg_graft_report *report);

/* Re-checks a grafted range: hashes the cache pages that hold slots
 * [slot0, slot0 + n_tokens(block)) of `seq` (slot0 page-aligned) on the GPU
 * and compares each page digest with block `block_id`'s stored digest
 * (Sec. 4.11 integrity check, applied to the live copy).  Only meaningful for
 * own-position grafts (relocated key pages differ by design), and only until
 * rows are appended into a ragged block's last page: its digest covers the
 * block's zero padding rows, which appends overwrite.  Flags and reporting as
 * for kvg_graft (KVG_GRAFT_SYNC waits and fills `report`). */
kvg_status kvg_verify(kvg_store *store, uint64_t block_id, kvg_cache *cache, int32_t seq,
                      int32_t slot0, uint32_t flags, void *stream, kvg_graft_report *report);

/* ------------------------------------------------------------- decode -- */

/* Decode attention of one query token per sequence (Sec. 3.2, Sec. 4.3):
 * for batch row b (sequence seq_ids[b], host array), query head h and KV head
 * g = h / (n_q_heads / n_kv_heads):
 *     o[h] = sum_t softmax_t(scale * q[h] . k_t[g]) v_t[g]
 * over every valid row of the sequence (pages in logical order, rows below
 * their fill) — on a windowed layer (kvg_cache_set_layer_windows) over its
 * last W valid rows — accumulated in fp32 and rounded to bf16 (RNE).  An
 * empty sequence gives o = 0.  Layers with different windows run as separate
 * launches on the stream.
 * q, out: device bf16 [n_layers_run][B][n_q_heads][head_dim] where
 * layer >= 0 runs that layer only (n_layers_run = 1) and layer == -1 runs all
 * layers in one launch.  The reduction order depends only on the logical
 * token index, never on physical page placement, so results are bitwise
 * reproducible and identical for grafted and freshly written rows.
 * n_q_heads must be a multiple of n_kv_heads with group size in {1, 2, 4, 8}
 * and group * head_dim <= 512.  B <= 4096.
 * The split-K partials live in per-cache scratch shared by every decode of
 * the cache (this call and kvg_decode_attention_range): a decode enqueued on
 * another stream than the previous one first waits on the GPU for that one,
 * so decodes of one cache on several streams run one after another. */
kvg_status kvg_decode_attention(kvg_cache *cache, int32_t layer, const int32_t *seq_ids,
                                int32_t B, const void *q, int32_t n_q_heads, void *out,
                                float scale, void *stream);

/* Split decode: the attention of kvg_decode_attention over only the rows in
 * slots [slot_begin, slot_end) of each sequence, kept as a softmax state that
 * calls over other slot ranges merge into, so that the part of a context that
 * is already resident is attended to while the rest is still being restored
 * (the decode step of Sec. 3.2 on top of a block that a graft from the host
 * store, Sec. 4.4, is still copying).  The paper has no split decode of its
 * own; the state is the usual one of an online softmax.
 * Rows: the valid rows (below their page's fill) of the sequence's pages
 * slot_begin / page_size ... slot_end / page_size - 1, and on a windowed
 * layer only those that are also among its last W valid rows (the window is
 * taken over the whole sequence as it stands at the call).
 * slot_begin, slot_end: multiples of page_size, 0 <= slot_begin <= slot_end;
 * slot_end >= max_slots means "to the end of the sequence".
 * state: device fp32 [n_layers_run][B][n_q_heads][head_dim + 4], 16-byte
 * aligned, caller-owned; per query head: o[head_dim] (the weighted sum of
 * value rows, times v_scale for an fp8 cache), m (the running maximum of
 * scale * log2(e) * q.k), l (the sum of 2^(scale * log2(e) * q.k - m)), two
 * unused floats.  A head with no rows has l = 0, o = 0, m = -inf.
 * flags: 0 overwrites the state with this call's part; KVG_DECODE_MERGE
 * merges this call's part into the state already there (written by earlier
 * calls with the same layer, batch rows and heads): m' = max(m0, m),
 * o' = o0 2^(m0 - m') + o 2^(m - m'), l' = l0 2^(m0 - m') + l 2^(m - m').
 * Parts that cover disjoint slot ranges whose union is every row give, after
 * kvg_decode_state_finish, the attention over all rows within the rounding
 * of the merge; the result is bitwise reproducible for the same sequence of
 * calls.  Other arguments and errors as for kvg_decode_attention, plus
 * KVG_ERR_ARG for a range that is not page-aligned or unknown flags. */
kvg_status kvg_decode_attention_range(kvg_cache *cache, int32_t layer, const int32_t *seq_ids, int32_t B,
                                      const void *q, int32_t n_q_heads, float scale, int32_t slot_begin,
                                      int32_t slot_end, uint32_t flags, float *state, void *stream);

/* Output of a split decode: out[r][d] = bf16_rne(o[d] / l) for each of the
 * n_rows = n_layers_run * B * n_q_heads state rows (out = 0 where l = 0),
 * written as bf16 [n_rows][head_dim] (the layout of kvg_decode_attention's
 * out).  state and out are device pointers, 16-byte aligned; head_dim 64,
 * 128 or 256.  Runs on `stream` on the current device. */
kvg_status kvg_decode_state_finish(const float *state, int64_t n_rows, int32_t head_dim, void *out,
                                   void *stream);

/* The same decode attention, for callers that cannot allocate GPU memory.
 * (The paper has no counterpart: this is a deployment variant.)
 * kvg_decode_attention() grows per-cache scratch for its split-K partial
 * results with cudaMalloc when a call first needs it; cudaMalloc/cudaFree
 * synchronise the whole device and can fail once another allocator has
 * reserved the memory, which latency-bound serving loops and processes with a
 * fixed memory footprint cannot accept.  This entry point instead keeps the
 * partials in one file-scope device array of 16 MiB that every GPU loading
 * the library holds until the process exits, and calls no allocating routine
 * (no cudaMalloc, cudaFree or library allocator).  Arguments, results and
 * errors are those of kvg_decode_attention, with these differences:
 *   - the partials take (units + workers) * G * (4 * head_dim + 8) bytes,
 *     units = (layers of one launch: those sharing a window, at most 256)
 *     * min(B, 256) * n_kv_heads, G = n_q_heads /
 *     n_kv_heads; the number of decode workers (warps) is capped so they fit
 *     in 16 MiB - 256 bytes, and a call that does not fit even with one
 *     worker returns KVG_ERR_CAPACITY with an explanatory kvg_last_error()
 *     and enqueues nothing;
 *   - the array's device address is looked up (cudaGetSymbolAddress, with
 *     the device current) by kvg_cache_create, once per device: that is when
 *     the module holding the array is made resident on the device and its
 *     16 MiB are taken, also under lazy module loading.  This entry point
 *     itself only reads the stored address, so its first call allocates
 *     nothing either;
 *   - every call on a device shares the one array, and the array keeps the
 *     previous call's contents (each partial the call reads is first written
 *     by the same call, so nothing needs clearing): calls whose GPU work
 *     overlaps in time, on different streams or from different threads, race
 *     and give wrong results.  Serialise them (one stream, or events). */
kvg_status kvg_decode_attention_noalloc(kvg_cache *cache, int32_t layer, const int32_t *seq_ids,
                                        int32_t B, const void *q, int32_t n_q_heads, void *out,
                                        float scale, void *stream);

/* ------------------------------------------------------------- digest -- */

/* SHA-256 (FIPS 180-4) on the GPU.
 * KVG_SHA256_PLAIN: out[32] = SHA-256 of bytes[0, n): one serial chain (one
 *   warp expands each block's message schedule while another runs the
 *   rounds when bytes is 4-byte aligned), about 0.85 us per 64-byte block
 *   (~75 MB/s; 1.5 us unaligned) — meant for short messages such as
 *   headers and test vectors; page contents use KVG_SHA256_PAGED.
 * KVG_SHA256_PAGED: n must be a multiple of page_bytes; out[32 * i] = the
 *   two-level digest of page i = bytes[i * page_bytes, (i+1) * page_bytes).
 * bytes and out are device pointers (or pinned host memory the GPU can
 * reach).  Paged calls use the library's per-device scratch (leaf digests):
 * each one's stream first waits for the previous paged call on the device,
 * so calls on different streams run one after another on the GPU, in the
 * order they were made (calls from several host threads take a lock). */
kvg_status kvg_digest(const void *bytes, uint64_t n, int32_t mode, uint64_t page_bytes,
                      uint8_t *out, void *stream);

/* --------------------------------------------------------------- misc -- */

/* Waits (up to timeout_s seconds, polling) for `stream`, then reads and clears
 * the cache's device status word.  This is where the outcome of the
 * asynchronous digest gate arrives on the host: a graft is accepted only
 * when every restored page's SHA-256 matches the deposited one (Sec. 3.2's
 * byte-equality test; Sec. 4.11's per-block integrity check).  Returns KVG_ERR_TIMEOUT if the stream is
 * still busy, KVG_ERR_DIGEST after a failed verification (report, nullable,
 * gets the details), KVG_ERR_DEVICE_CHECK if a kernel's own check failed. */
kvg_status kvg_sync(kvg_cache *cache, void *stream, double timeout_s, kvg_graft_report *report);

/* Failure-detection self-test: enqueues a kernel whose wait (an mbarrier
 * that nothing completes — the same bounded wait every kernel uses for its
 * asynchronous copies) gives up after limit_ns (at most 10 s) and records
 * KVG_ERR_DEVICE_CHECK in the cache's status word; the next kvg_sync returns
 * it and the context stays usable.  Nothing faults or hangs. */
kvg_status kvg_selftest_bounded_wait(kvg_cache *cache, uint64_t limit_ns, void *stream);

/* Name of a status code (a static string; "unknown status" for values not
 * in kvg_status).  The codes are the failure modes of the problem statement:
 * digest mismatch (Sec. 3.2, Sec. 4.11), position tags out of range after a
 * re-base (Sec. 4.2), a block that does not fit the cache (Sec. 3.3). */
const char *kvg_status_string(kvg_status status);

/* Human-readable detail of the last failed call on this host thread (empty if
 * none); valid until the next call on the thread. */
const char *kvg_last_error(void);

/* Library version, e.g. 0x000200 for 0.2.0 (0.2: kv_dtype and fp8 scales in kvg_dims). */
uint32_t kvg_version(void);

/* Number of CUDA kernel launches this library has issued since it was
 * loaded (all devices, all threads).  A diagnostic for benchmarks. */
uint64_t kvg_launch_count(void);

#ifdef __cplusplus
}
#endif
#endif /* KVG_H */
