// stream_order.h -- what this library last put on each CUDA stream, as far as
// the next attention call needs to know it.  Not part of the ABI.
//
// A decode grid may start without waiting for the grid before it (chain 3 in
// the attention kernel) only when that grid is one of this library's split-K
// combines: a combine releases the next grid only after its own wait, so
// every grid before it has completed by then, and the decode grid defers its
// writes of the output and the workspace (which the combine uses) until its
// own wait.  Every kernel launch and copy the library issues records itself
// here, so a sync kernel, an append or a table copy between two attention
// calls turns the start-without-waiting off for the next call.
#pragma once

// record the library's latest launch on `stream` (a combine or anything else)
void kvp_note_stream(void *stream, bool combine);
// true when the library's latest launch on `stream` was a split-K combine
bool kvp_stream_after_combine(void *stream);
