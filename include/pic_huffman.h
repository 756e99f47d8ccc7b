/*
 * pic_huffman.h -- C ABI of the GPU Huffman decoder (arxiv 2609.09020, Sec.
 * 3.3: image-specific Huffman tables, O(1) decoding of a symbol from a table
 * of 2^p entries (p = the longest code), that table stored run-length
 * compressed with one entry per coded symbol; Sec. 4.1: the decoder follows
 * the self-synchronising parallel decoding of GPUHD, Weissenberger & Schmidt
 * 2018).
 *
 * Code and stream conventions (the readings the oracle shares):
 *   - canonical prefix code, lengths 1..p, p <= 12; the stored table lists
 *     the coded symbols' values and lengths in canonical order (by length,
 *     then value); codes are assigned in that order, each the previous plus
 *     one, shifted left when the length grows;
 *   - bits most significant first in 32-bit words;
 *   - a batch holds B streams back to back, each starting on a multiple of
 *     PIC_HUFF_WORDS_PER_SUBSEQ words (the encoder pads), each with its own
 *     table and its own symbol count (from the container header).
 * Device pointers owned by the caller, asynchronous on `stream`, pic_status
 * codes, no traps.
 */
#ifndef PIC_HUFFMAN_H
#define PIC_HUFFMAN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Bits decoded per thread before synchronisation: 8 words = 256 bits. */
#define PIC_HUFF_WORDS_PER_SUBSEQ 8
#define PIC_HUFF_MAX_PRECISION 12

/* Device workspace bytes for a batch of B streams in n_words words with
 * code precision p (the decode tables and the per-256-bit bookkeeping);
 * -1 for arguments out of range. */
int64_t pic_huffman_workspace_bytes(int64_t n_words, int B, int p);

/*
 * Decodes B streams on `stream`:
 *   words       : uint32, device, [n_words] (16-byte aligned)
 *   n_words     : total words, a multiple of PIC_HUFF_WORDS_PER_SUBSEQ
 *   word_off    : int64, device, [B + 1]: stream b is words
 *                 [word_off[b], word_off[b + 1]), each a multiple of
 *                 PIC_HUFF_WORDS_PER_SUBSEQ, word_off[B] = n_words
 *   n_bits      : int64, device, [B]: coded bits of stream b
 *                 (<= 32 (word_off[b + 1] - word_off[b]))
 *   tab_value   : int32, device, [B][max_table]: the stored tables' symbol
 *                 values (any int32), canonical order
 *   tab_len     : int32, device, [B][max_table]: code lengths, 1..p; the
 *                 first 0 (or max_table) ends an image's table
 *   p           : the precision, 1..12: every length <= p
 *   sym_off     : int64, device, [B + 1]: stream b decodes to
 *                 out[sym_off[b] .. sym_off[b + 1])
 *   out         : int32, device, [sym_off[B]]
 *   workspace   : device, >= pic_huffman_workspace_bytes, 16-byte aligned
 * A stream that is not a sequence of codewords of its table, a symbol count
 * different from sym_off's, or a table whose lengths violate Kraft's
 * inequality is reported by pic_huffman_status (nothing is written out of
 * bounds; the output is then unspecified), as is a stream whose parallel
 * decodings do not synchronise within 64 passes (never seen on Huffman codes;
 * the result is then unspecified too).
 * Errors: PIC_ERR_INVALID_ARG, PIC_ERR_UNSUPPORTED (no cooperative launch on
 * this device), PIC_ERR_CUDA.
 */
int pic_huffman_decode(const uint32_t *words, int64_t n_words, const int64_t *word_off,
                       const int64_t *n_bits, int B, const int32_t *tab_value,
                       const int32_t *tab_len, int max_table, int p, const int64_t *sym_off,
                       int32_t *out, void *workspace, size_t workspace_bytes, void *stream);

/* Synchronises `stream`; PIC_OK if the last decode with this workspace found
 * every stream well formed, PIC_ERR_INVALID_ARG if not, PIC_ERR_CUDA. */
int pic_huffman_status(const void *workspace, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* PIC_HUFFMAN_H */
